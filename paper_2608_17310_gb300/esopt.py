"""Python binding of the ES-step C ABI (``include/esopt.h``).

Argument marshalling only: every function forwards to the function of the same
name in ``libesopt.so``; all arithmetic of the step runs in the library's CUDA
kernels (device entry points) or its C++ host code (reward normalisation,
sigma schedule, coefficients). There is no fallback: if the library is not
built, importing the functions raises.

Device pointers are plain integers; torch tensors are accepted wherever a
device buffer is expected and are passed by ``data_ptr()``. ``stream`` is a
``cudaStream_t`` as an integer, a ``torch.cuda.Stream``, or None for torch's
current stream (the legacy default stream if torch is not in use).
"""
from __future__ import annotations

import ctypes
import os
import sys
from dataclasses import dataclass
from typing import Iterable, Sequence

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "_build", "libesopt.so")

ES_MAX_SEEDS = 1024
ES_STATIC_MAX_SEGMENTS = 1024

ES_OK = 0
ES_ERR_INVALID_ARG = 1
ES_ERR_ALIGNMENT = 2
ES_ERR_OVERLAP = 3
ES_ERR_NONFINITE = 4
ES_ERR_TOO_MANY_SEEDS = 5
ES_ERR_CUDA = 6
ES_ERR_NO_MEMORY = 7
ES_ERR_WRONG_DEVICE = 8

ES_BF16 = 0
ES_FP32 = 1
ES_FP8_E4M3 = 2

ES_SCALE_PAPER = 0
ES_SCALE_CANONICAL = 1


class es_segment_t(ctypes.Structure):
    _fields_ = [("data", ctypes.c_void_p), ("numel", ctypes.c_uint64),
                ("index_base", ctypes.c_uint64)]


class EsError(RuntimeError):
    def __init__(self, status: int, func: str, detail: str):
        self.status = status
        super().__init__(f"{func}: {detail or _status_string(status)} (status {status})")


_lib = None


def _load() -> ctypes.CDLL:
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(
            f"{LIB_PATH} is missing: build the CUDA library first "
            "(python -m paper_2608_17310_gb300.build)")
    L = ctypes.CDLL(LIB_PATH)
    vp, u64, f32, f64, i32 = (ctypes.c_void_p, ctypes.c_uint64, ctypes.c_float,
                              ctypes.c_double, ctypes.c_int)
    P = ctypes.POINTER
    sigs = {
        "es_plan_create": (i32, [P(es_segment_t), i32, i32, P(vp)]),
        "es_plan_create_scaled": (i32, [P(es_segment_t), P(f32), i32, i32, P(vp)]),
        "es_plan_destroy": (i32, [vp]),
        "es_plan_numel": (u64, [vp]),
        "es_assign_index_bases": (u64, [P(es_segment_t), i32]),
        "es_noise_fill": (i32, [u64, u64, u64, vp, vp]),
        "es_noise_bits": (i32, [u64, u64, u64, vp, vp]),
        "es_box_muller": (i32, [vp, u64, vp, vp]),
        "es_perturb": (i32, [vp, u64, f32, vp]),
        "es_restore": (i32, [vp, u64, f32, vp]),
        "es_restore_perturb": (i32, [vp, u64, f32, u64, f32, vp]),
        "es_update": (i32, [vp, P(u64), P(f32), i32, vp]),
        "es_update_perturb": (i32, [vp, P(u64), P(f32), i32, u64, f32, vp]),
        "es_replay": (i32, [vp, P(u64), P(f32), P(i32), i32, vp]),
        "es_normalize_rewards": (i32, [P(f64), i32, f64, P(f64)]),
        "es_sigma_cosine": (f64, [f64, f64, i32, i32]),
        "es_update_coeffs": (i32, [P(f64), i32, f64, f64, i32, P(f32)]),
        "es_fold_antithetic": (i32, [P(f64), P(f64), i32, f64, f64, i32, P(f32)]),
        "es_perturb_noalloc": (i32, [P(es_segment_t), i32, i32, u64, f32, vp]),
        "es_status_string": (ctypes.c_char_p, [i32]),
        "es_last_error": (ctypes.c_char_p, []),
    }
    for name, (res, args) in sigs.items():
        fn = getattr(L, name)
        fn.restype = res
        fn.argtypes = args
    _lib = L
    return L


def lib() -> ctypes.CDLL:
    return _load()


def _status_string(status: int) -> str:
    return _load().es_status_string(status).decode()


def es_status_string(status: int) -> str:
    return _status_string(status)


def es_last_error() -> str:
    return _load().es_last_error().decode()


def _check(status: int, func: str) -> None:
    if status != ES_OK:
        raise EsError(status, func, es_last_error())


def _stream(stream) -> int:
    if stream is None:
        torch = sys.modules.get("torch")
        if torch is not None and torch.cuda.is_available() and torch.cuda.is_initialized():
            return torch.cuda.current_stream().cuda_stream
        return 0
    if isinstance(stream, int):
        return stream
    return int(stream.cuda_stream)


def _ptr(buf) -> int:
    if isinstance(buf, int):
        return buf
    return int(buf.data_ptr())


def _f64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.float64)


# --- plan -------------------------------------------------------------------

@dataclass
class Segment:
    """One parameter tensor: device pointer, element count, global index base."""
    data: int
    numel: int
    index_base: int = 0


class Plan:
    """Owns an ``es_plan_t``. Keeps the objects that own the memory alive."""

    def __init__(self, handle: int, numel: int, dtype: int, keepalive=(), scales=None):
        self.handle = handle
        self.numel = numel
        self.dtype = dtype
        self.scales = None if scales is None else [float(x) for x in scales]
        self._keepalive = tuple(keepalive)

    def close(self) -> None:
        if self.handle:
            h, self.handle = self.handle, None
            _check(_load().es_plan_destroy(h), "es_plan_destroy")

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()


def _seg_array(segments: Sequence[Segment]):
    arr = (es_segment_t * len(segments))()
    for k, s in enumerate(segments):
        arr[k].data = s.data
        arr[k].numel = s.numel
        arr[k].index_base = s.index_base
    return arr


def es_assign_index_bases(segments: Sequence[Segment]) -> int:
    """Fills ``index_base`` in place (8-aligned, in order); returns the index end."""
    arr = _seg_array(segments)
    end = _load().es_assign_index_bases(arr, len(segments))
    for k, s in enumerate(segments):
        s.index_base = int(arr[k].index_base)
    return int(end)


def es_plan_create(segments: Sequence[Segment], dtype: int, keepalive: Iterable = ()) -> Plan:
    arr = _seg_array(segments)
    handle = ctypes.c_void_p()
    _check(_load().es_plan_create(arr, len(segments), dtype, ctypes.byref(handle)),
           "es_plan_create")
    return Plan(handle.value, int(_load().es_plan_numel(handle)), dtype, keepalive)


def es_plan_create_scaled(segments: Sequence[Segment], scales, dtype: int,
                          keepalive: Iterable = ()) -> Plan:
    """A plan whose segment j holds values scales[j] * stored (ES_FP8_E4M3)."""
    arr = _seg_array(segments)
    sc = np.ascontiguousarray(scales, dtype=np.float32)
    if sc.size != len(segments):
        raise ValueError("one scale per segment")
    handle = ctypes.c_void_p()
    _check(_load().es_plan_create_scaled(arr, sc.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                                         len(segments), dtype, ctypes.byref(handle)),
           "es_plan_create_scaled")
    return Plan(handle.value, int(_load().es_plan_numel(handle)), dtype, keepalive, sc)


def segments_from_tensors(tensors, index_bases=None):
    """Segments for a list of contiguous CUDA tensors (bases assigned if None)."""
    segs = []
    for t in tensors:
        if not t.is_cuda:
            raise ValueError("parameter tensors must be CUDA tensors")
        if not t.is_contiguous():
            raise ValueError("parameter tensors must be contiguous")
        segs.append(Segment(int(t.data_ptr()), int(t.numel()), 0))
    if index_bases is None:
        es_assign_index_bases(segs)
    else:
        for s, b in zip(segs, index_bases):
            s.index_base = int(b)
    return segs


def plan_from_tensors(tensors, index_bases=None, scales=None) -> Plan:
    """es_plan_create over torch tensors of one dtype: bf16, fp32, or FP8 E4M3
    (torch.float8_e4m3fn, or uint8 holding E4M3 codes), the latter with one
    scale per tensor (es_plan_create_scaled; all 1 if scales is None)."""
    import torch  # only for the dtype check
    tensors = list(tensors)
    dts = {t.dtype for t in tensors}
    if dts == {torch.bfloat16}:
        dtype = ES_BF16
    elif dts == {torch.float32}:
        dtype = ES_FP32
    elif dts <= {torch.float8_e4m3fn, torch.uint8}:
        dtype = ES_FP8_E4M3
    else:
        raise ValueError(f"all tensors must be bfloat16, float32 or FP8 E4M3, got {dts}")
    segs = segments_from_tensors(tensors, index_bases)
    if scales is not None:
        return es_plan_create_scaled(segs, scales, dtype, keepalive=tensors)
    return es_plan_create(segs, dtype, keepalive=tensors)


# --- device entry points ----------------------------------------------------------

def es_noise_fill(seed: int, index_base: int, n: int, out, stream=None) -> None:
    _check(_load().es_noise_fill(seed, index_base, n, _ptr(out), _stream(stream)),
           "es_noise_fill")


def es_noise_bits(seed: int, block_base: int, nblocks: int, out, stream=None) -> None:
    _check(_load().es_noise_bits(seed, block_base, nblocks, _ptr(out), _stream(stream)),
           "es_noise_bits")


def es_box_muller(words, npairs: int, out, stream=None) -> None:
    _check(_load().es_box_muller(_ptr(words), npairs, _ptr(out), _stream(stream)),
           "es_box_muller")


def es_perturb(plan: Plan, seed: int, sigma: float, stream=None) -> None:
    _check(_load().es_perturb(plan.handle, seed, sigma, _stream(stream)), "es_perturb")


def es_restore(plan: Plan, seed: int, sigma: float, stream=None) -> None:
    _check(_load().es_restore(plan.handle, seed, sigma, _stream(stream)), "es_restore")


def es_restore_perturb(plan: Plan, restore_seed: int, sigma_restore: float, perturb_seed: int,
                       sigma_perturb: float, stream=None) -> None:
    _check(_load().es_restore_perturb(plan.handle, restore_seed, sigma_restore, perturb_seed,
                                      sigma_perturb, _stream(stream)), "es_restore_perturb")


def es_update(plan: Plan, seeds, coeffs, stream=None) -> None:
    s = np.ascontiguousarray(seeds, dtype=np.uint64)
    c = np.ascontiguousarray(coeffs, dtype=np.float32)
    if s.size != c.size:
        raise ValueError("seeds and coeffs differ in length")
    _check(_load().es_update(plan.handle, s.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64)),
                             c.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), s.size,
                             _stream(stream)), "es_update")


def es_perturb_noalloc(segments: Sequence[Segment], dtype: int, seed: int, sigma: float,
                       stream=None) -> None:
    """Perturb (or, with -sigma, restore) without a plan and without any device
    allocation; the segment table goes to the library's static device array."""
    arr = _seg_array(segments)
    _check(_load().es_perturb_noalloc(arr, len(segments), dtype, seed, sigma, _stream(stream)),
           "es_perturb_noalloc")


def es_update_perturb(plan: Plan, seeds, coeffs, next_seed: int, sigma_next: float,
                      stream=None) -> None:
    s = np.ascontiguousarray(seeds, dtype=np.uint64)
    c = np.ascontiguousarray(coeffs, dtype=np.float32)
    if s.size != c.size:
        raise ValueError("seeds and coeffs differ in length")
    _check(_load().es_update_perturb(plan.handle, s.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64)),
                                     c.ctypes.data_as(ctypes.POINTER(ctypes.c_float)), s.size,
                                     next_seed, sigma_next, _stream(stream)), "es_update_perturb")


def es_replay(plan: Plan, seeds, coeffs, counts, stream=None) -> None:
    """Replays generations back to back: counts[g] seeds/coefficients each."""
    s = np.ascontiguousarray(seeds, dtype=np.uint64)
    c = np.ascontiguousarray(coeffs, dtype=np.float32)
    n = np.ascontiguousarray(counts, dtype=np.int32)
    if s.size != c.size or int(n.sum()) != s.size:
        raise ValueError("seeds, coeffs and counts do not agree")
    _check(_load().es_replay(plan.handle, s.ctypes.data_as(ctypes.POINTER(ctypes.c_uint64)),
                             c.ctypes.data_as(ctypes.POINTER(ctypes.c_float)),
                             n.ctypes.data_as(ctypes.POINTER(ctypes.c_int)), n.size,
                             _stream(stream)), "es_replay")


# --- host-side generation control ---------------------------------------------------

def es_normalize_rewards(rewards, eps_z: float = 1e-8) -> np.ndarray:
    r = _f64(rewards)
    out = np.empty_like(r)
    P = ctypes.POINTER(ctypes.c_double)
    _check(_load().es_normalize_rewards(r.ctypes.data_as(P), r.size, eps_z,
                                        out.ctypes.data_as(P)), "es_normalize_rewards")
    return out


def es_sigma_cosine(sigma0: float, sigmaT: float, t: int, T: int) -> float:
    return float(_load().es_sigma_cosine(sigma0, sigmaT, t, T))


def es_update_coeffs(rhat, alpha: float, sigma: float, mode: int = ES_SCALE_PAPER) -> np.ndarray:
    r = _f64(rhat)
    out = np.empty(r.size, dtype=np.float32)
    _check(_load().es_update_coeffs(r.ctypes.data_as(ctypes.POINTER(ctypes.c_double)), r.size,
                                    alpha, sigma, mode,
                                    out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
           "es_update_coeffs")
    return out


def es_fold_antithetic(rhat_pos, rhat_neg, alpha: float, sigma: float,
                       mode: int = ES_SCALE_PAPER) -> np.ndarray:
    p, m = _f64(rhat_pos), _f64(rhat_neg)
    if p.size != m.size:
        raise ValueError("rhat_pos and rhat_neg differ in length")
    out = np.empty(p.size, dtype=np.float32)
    P = ctypes.POINTER(ctypes.c_double)
    _check(_load().es_fold_antithetic(p.ctypes.data_as(P), m.ctypes.data_as(P), p.size, alpha,
                                      sigma, mode,
                                      out.ctypes.data_as(ctypes.POINTER(ctypes.c_float))),
           "es_fold_antithetic")
    return out
