"""ctypes wrapper around the plain-C ES-step oracle (``esopt_oracle.c``).

TEST INFRASTRUCTURE ONLY: the test suite, the package smoke check and the
benchmark's CPU-baseline leg are the only callers. The product path never
imports this module.

Every function takes and returns numpy arrays; the arithmetic is all in the C
file, in double precision, following the paper's statement of the step.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "esopt_oracle.c")
_BUILD_DIR = os.path.join(_HERE, "_build")
_LIB_PATH = os.path.join(_BUILD_DIR, "liboracle.so")
_lock = threading.Lock()
_lib = None

_u64p = ctypes.POINTER(ctypes.c_uint64)
_u32p = ctypes.POINTER(ctypes.c_uint32)
_u16p = ctypes.POINTER(ctypes.c_uint16)
_u8p = ctypes.POINTER(ctypes.c_uint8)
_f32p = ctypes.POINTER(ctypes.c_float)
_f64p = ctypes.POINTER(ctypes.c_double)


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/_build/liboracle.so`` with gcc."""
    os.makedirs(_BUILD_DIR, exist_ok=True)
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".{os.getpid()}.tmp"
    cmd = ["gcc", "-O2", "-std=gnu11", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            L = ctypes.CDLL(build())
            L.oracle_philox4x32_10.argtypes = [_u32p, _u32p, _u32p]
            L.oracle_noise_block.argtypes = [ctypes.c_uint64, ctypes.c_uint64, _u32p]
            L.oracle_noise_blocks.argtypes = [ctypes.c_uint64, ctypes.c_uint64, ctypes.c_uint64,
                                              _u32p]
            L.oracle_uniform.argtypes = [ctypes.c_uint32]
            L.oracle_uniform.restype = ctypes.c_double
            L.oracle_box_muller_fill.argtypes = [_u32p, ctypes.c_uint64, _f64p]
            L.oracle_gaussian.argtypes = [ctypes.c_uint64, ctypes.c_uint64]
            L.oracle_gaussian.restype = ctypes.c_double
            L.oracle_noise_fill.argtypes = [ctypes.c_uint64, ctypes.c_uint64,
                                            ctypes.c_uint64, _f64p]
            L.oracle_noise_at.argtypes = [ctypes.c_uint64, _u64p, ctypes.c_uint64, _f64p]
            L.oracle_bf16_to_double.argtypes = [ctypes.c_uint16]
            L.oracle_bf16_to_double.restype = ctypes.c_double
            L.oracle_bf16_from_double.argtypes = [ctypes.c_double]
            L.oracle_bf16_from_double.restype = ctypes.c_uint16
            L.oracle_f32_from_double.argtypes = [ctypes.c_double]
            L.oracle_f32_from_double.restype = ctypes.c_float
            L.oracle_e4m3_to_double.argtypes = [ctypes.c_uint8]
            L.oracle_e4m3_to_double.restype = ctypes.c_double
            L.oracle_e4m3_from_double.argtypes = [ctypes.c_double]
            L.oracle_e4m3_from_double.restype = ctypes.c_uint8
            L.oracle_axpy_noise_e4m3.argtypes = [_u8p, _u64p, ctypes.c_uint64,
                                                 ctypes.c_uint64, ctypes.c_float, ctypes.c_float]
            L.oracle_update_e4m3.argtypes = [_u8p, _u64p, ctypes.c_uint64, _u64p,
                                             _f32p, ctypes.c_int, ctypes.c_float]
            L.oracle_axpy_noise_f32.argtypes = [_f32p, _u64p, ctypes.c_uint64,
                                                ctypes.c_uint64, ctypes.c_float]
            L.oracle_axpy_noise_bf16.argtypes = [_u16p, _u64p, ctypes.c_uint64,
                                                 ctypes.c_uint64, ctypes.c_float]
            L.oracle_update_f32.argtypes = [_f32p, _u64p, ctypes.c_uint64, _u64p,
                                            _f32p, ctypes.c_int]
            L.oracle_update_bf16.argtypes = [_u16p, _u64p, ctypes.c_uint64, _u64p,
                                             _f32p, ctypes.c_int]
            L.oracle_zscore.argtypes = [_f64p, ctypes.c_int, ctypes.c_double, _f64p]
            L.oracle_zscore.restype = ctypes.c_int
            L.oracle_sigma_cosine.argtypes = [ctypes.c_double, ctypes.c_double,
                                              ctypes.c_int, ctypes.c_int]
            L.oracle_sigma_cosine.restype = ctypes.c_double
            L.oracle_update_coeffs.argtypes = [_f64p, ctypes.c_int, ctypes.c_double,
                                               ctypes.c_double, ctypes.c_int, _f32p]
            L.oracle_update_coeffs.restype = ctypes.c_int
            L.oracle_fold_antithetic.argtypes = [_f64p, _f64p, ctypes.c_int,
                                                 ctypes.c_double, ctypes.c_double,
                                                 ctypes.c_int, _f32p]
            L.oracle_fold_antithetic.restype = ctypes.c_int
            L.oracle_quadratic_reward.argtypes = [_f32p, _f32p, ctypes.c_uint64]
            L.oracle_quadratic_reward.restype = ctypes.c_double
            _lib = L
    return _lib


def _ptr(a: np.ndarray, ctype):
    assert a.flags["C_CONTIGUOUS"], "oracle arrays must be C-contiguous"
    return a.ctypes.data_as(ctype)


# --- generator ------------------------------------------------------------

def philox4x32_10(counter, key) -> np.ndarray:
    """Raw Philox4x32-10 block for a 4-word counter and 2-word key."""
    c = np.ascontiguousarray(counter, dtype=np.uint32)
    k = np.ascontiguousarray(key, dtype=np.uint32)
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_philox4x32_10(_ptr(c, _u32p), _ptr(k, _u32p), _ptr(out, _u32p))
    return out


def noise_block(seed: int, j: int) -> np.ndarray:
    out = np.zeros(4, dtype=np.uint32)
    lib().oracle_noise_block(seed, j, _ptr(out, _u32p))
    return out


def noise_blocks(seed: int, j0: int, n: int) -> np.ndarray:
    """Philox words of blocks j0 .. j0 + n - 1, shape (n, 4)."""
    out = np.zeros((n, 4), dtype=np.uint32)
    if n:
        lib().oracle_noise_blocks(seed, j0, n, _ptr(out, _u32p))
    return out


def uniform(x: int) -> float:
    return lib().oracle_uniform(x)


def box_muller(words: np.ndarray) -> np.ndarray:
    """Box-Muller of word pairs (words[2k] -> radius, words[2k+1] -> angle)."""
    w = np.ascontiguousarray(words, dtype=np.uint32)
    out = np.empty(w.size, dtype=np.float64)
    if w.size:
        lib().oracle_box_muller_fill(_ptr(w, _u32p), w.size // 2, _ptr(out, _f64p))
    return out


def gaussian(seed: int, g: int) -> float:
    return lib().oracle_gaussian(seed, g)


def noise_fill(seed: int, index_base: int, n: int) -> np.ndarray:
    out = np.empty(n, dtype=np.float64)
    if n:
        lib().oracle_noise_fill(seed, index_base, n, _ptr(out, _f64p))
    return out


def noise_at(seed: int, g: np.ndarray) -> np.ndarray:
    g = np.ascontiguousarray(g, dtype=np.uint64)
    out = np.empty(g.size, dtype=np.float64)
    if g.size:
        lib().oracle_noise_at(seed, _ptr(g, _u64p), g.size, _ptr(out, _f64p))
    return out


# --- storage rounding -----------------------------------------------------

def bf16_from_double(x: float) -> int:
    return lib().oracle_bf16_from_double(x)


def bf16_to_double(h: int) -> float:
    return lib().oracle_bf16_to_double(h)


def bf16_bits_to_f64(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> float64 values (exact widening)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << 16
    return b.view(np.float32).astype(np.float64)


def e4m3_to_double(c: int) -> float:
    return lib().oracle_e4m3_to_double(c)


def e4m3_from_double(x: float) -> int:
    return lib().oracle_e4m3_from_double(x)


def e4m3_codes_to_f64(codes: np.ndarray) -> np.ndarray:
    """E4M3 codes (uint8) -> float64 values, one oracle call per code."""
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    return np.array([lib().oracle_e4m3_to_double(int(v)) for v in c.ravel()],
                    dtype=np.float64).reshape(c.shape)


# --- step -----------------------------------------------------------------

def _indices(g, n):
    if g is None:
        raise ValueError("global indices are required")
    g = np.ascontiguousarray(g, dtype=np.uint64)
    if g.size != n:
        raise ValueError("index list and theta differ in length")
    return g


def axpy_noise_f32(theta: np.ndarray, g: np.ndarray, seed: int, scale: float) -> np.ndarray:
    """theta + scale * eps_seed[g], rounded once to fp32 (returns a new array)."""
    t = np.array(theta, dtype=np.float32, copy=True, order="C")
    g = _indices(g, t.size)
    if t.size:
        lib().oracle_axpy_noise_f32(_ptr(t, _f32p), _ptr(g, _u64p), t.size, seed,
                                    float(np.float32(scale)))
    return t


def axpy_noise_bf16(theta_bits: np.ndarray, g: np.ndarray, seed: int, scale: float) -> np.ndarray:
    """Same on bf16 bit patterns (uint16), rounded once to bf16."""
    t = np.array(theta_bits, dtype=np.uint16, copy=True, order="C")
    g = _indices(g, t.size)
    if t.size:
        lib().oracle_axpy_noise_bf16(_ptr(t, _u16p), _ptr(g, _u64p), t.size, seed,
                                     float(np.float32(scale)))
    return t


def axpy_noise_e4m3(codes: np.ndarray, g: np.ndarray, seed: int, scale: float,
                    seg_scale: float) -> np.ndarray:
    """E4M3 codes (uint8) of a segment with scale seg_scale: the nearest code of
    (seg_scale * value + scale * eps_seed[g]) / seg_scale (returns a new array)."""
    t = np.array(codes, dtype=np.uint8, copy=True, order="C")
    g = _indices(g, t.size)
    if t.size:
        lib().oracle_axpy_noise_e4m3(_ptr(t, _u8p), _ptr(g, _u64p), t.size, seed,
                                     float(np.float32(scale)), float(np.float32(seg_scale)))
    return t


def _axpy(theta, g, seed, scale, dtype, seg_scale):
    if dtype == "f32":
        return axpy_noise_f32(theta, g, seed, scale)
    if dtype == "bf16":
        return axpy_noise_bf16(theta, g, seed, scale)
    if dtype == "e4m3":
        return axpy_noise_e4m3(theta, g, seed, scale, seg_scale)
    raise ValueError(f"unknown storage type {dtype}")


def perturb(theta, g, seed, sigma, dtype="f32", seg_scale=1.0):
    return _axpy(theta, g, seed, float(np.float32(sigma)), dtype, seg_scale)


def restore(theta, g, seed, sigma, dtype="f32", seg_scale=1.0):
    return _axpy(theta, g, seed, -float(np.float32(sigma)), dtype, seg_scale)


def update(theta, g, seeds, coeffs, dtype="f32", seg_scale=1.0):
    """theta + sum_i coeffs[i] * eps_{seeds[i]}[g], summed in double, one rounding
    (for E4M3: of the scaled value, stored back divided by seg_scale)."""
    s = np.ascontiguousarray(seeds, dtype=np.uint64)
    c = np.ascontiguousarray(coeffs, dtype=np.float32)
    if s.size != c.size:
        raise ValueError("seeds and coeffs differ in length")
    if dtype == "e4m3":
        t = np.array(theta, dtype=np.uint8, copy=True, order="C")
        g = _indices(g, t.size)
        if t.size:
            lib().oracle_update_e4m3(_ptr(t, _u8p), _ptr(g, _u64p), t.size, _ptr(s, _u64p),
                                     _ptr(c, _f32p), s.size, float(np.float32(seg_scale)))
        return t
    if dtype == "f32":
        t = np.array(theta, dtype=np.float32, copy=True, order="C")
        g = _indices(g, t.size)
        if t.size:
            lib().oracle_update_f32(_ptr(t, _f32p), _ptr(g, _u64p), t.size,
                                    _ptr(s, _u64p), _ptr(c, _f32p), s.size)
    else:
        t = np.array(theta, dtype=np.uint16, copy=True, order="C")
        g = _indices(g, t.size)
        if t.size:
            lib().oracle_update_bf16(_ptr(t, _u16p), _ptr(g, _u64p), t.size,
                                     _ptr(s, _u64p), _ptr(c, _f32p), s.size)
    return t


# --- host-side generation control -------------------------------------------

def zscore(R, eps_z: float = 1e-8):
    r = np.ascontiguousarray(R, dtype=np.float64)
    out = np.empty_like(r)
    replaced = lib().oracle_zscore(_ptr(r, _f64p), r.size, eps_z, _ptr(out, _f64p))
    if replaced < 0:
        raise ValueError("invalid reward vector")
    return out


def sigma_cosine(sigma0: float, sigmaT: float, t: int, T: int) -> float:
    return lib().oracle_sigma_cosine(sigma0, sigmaT, t, T)


def update_coeffs(Rhat, alpha: float, sigma: float, mode: int) -> np.ndarray:
    r = np.ascontiguousarray(Rhat, dtype=np.float64)
    out = np.empty(r.size, dtype=np.float32)
    if lib().oracle_update_coeffs(_ptr(r, _f64p), r.size, alpha, sigma, mode,
                                  _ptr(out, _f32p)) != 0:
        raise ValueError("invalid coefficient arguments")
    return out


def fold_antithetic(Rhat_pos, Rhat_neg, alpha: float, sigma: float, mode: int) -> np.ndarray:
    p = np.ascontiguousarray(Rhat_pos, dtype=np.float64)
    m = np.ascontiguousarray(Rhat_neg, dtype=np.float64)
    out = np.empty(p.size, dtype=np.float32)
    if p.size != m.size or lib().oracle_fold_antithetic(
            _ptr(p, _f64p), _ptr(m, _f64p), p.size, alpha, sigma, mode,
            _ptr(out, _f32p)) != 0:
        raise ValueError("invalid antithetic arguments")
    return out


def quadratic_reward(theta: np.ndarray, theta_star: np.ndarray) -> float:
    t = np.ascontiguousarray(theta, dtype=np.float32)
    s = np.ascontiguousarray(theta_star, dtype=np.float32)
    return lib().oracle_quadratic_reward(_ptr(t, _f32p), _ptr(s, _f32p), t.size)
