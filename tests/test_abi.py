"""The C-ABI library loads on a machine without a GPU, exports every function
that include/esopt.h declares, and its host-only logic (reward z-score, cosine
schedule, coefficients, plan validation) agrees with the oracle. No device call
is made here."""
import math
import os
import re
import subprocess

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def E():
    from paper_2608_17310_gb300 import build, esopt
    build.build_library()
    esopt._load()
    return esopt


def _declared():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            text = open(os.path.join(ROOT, "include", fn)).read()
            text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
            names |= set(re.findall(r"\b(es_[a-z0-9_]+)\s*\(", text))
    return names


def test_library_exports_every_declared_function(E):
    declared = _declared()
    assert {"es_plan_create", "es_perturb", "es_restore", "es_update", "es_noise_fill"} <= declared
    out = subprocess.run(["nm", "-D", "--defined-only", E.LIB_PATH], capture_output=True,
                         text=True, check=True).stdout
    exported = set(re.findall(r"\bT (es_[a-z0-9_]+)$", out, flags=re.M))
    assert declared <= exported, declared - exported
    for name in declared:
        assert hasattr(E.lib(), name)


def test_header_compiles_as_c():
    src = '#include "esopt.h"\nint main(void){ es_segment_t s; (void)s; return ES_OK; }\n'
    r = subprocess.run(["gcc", "-std=c99", "-Wall", "-Werror", "-fsyntax-only",
                        f"-I{os.path.join(ROOT, 'include')}", "-x", "c", "-"],
                       input=src, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr


def test_plain_c_consumer_compiles_and_links(E, tmp_path):
    # tests/abi_c_consumer.c uses the library through the header alone; the GPU
    # tests run it. Here: it compiles as strict C99 and links.
    from parity import build_c_consumer
    assert os.path.exists(build_c_consumer(tmp_path))


def test_normalize_rewards_matches_oracle(E, oracle):
    rng = np.random.default_rng(0)
    cases = [rng.uniform(size=8), (rng.uniform(size=16) < 0.3).astype(float),
             rng.standard_normal(30), rng.standard_normal(128) * 100 + 5,
             np.full(16, 0.3), np.array([1.0]), np.array([0.2, np.nan, 0.9, -np.inf, 0.5]),
             np.array([np.nan, np.nan])]
    for R in cases:
        for eps in (1e-8, 0.0):
            got = E.es_normalize_rewards(R, eps)
            want = oracle.zscore(R, eps)
            assert np.allclose(got, want, rtol=1e-14, atol=1e-14), (R, got, want)


def test_sigma_cosine_matches_oracle(E, oracle):
    for s0, sT, T in [(1e-3, 2.5e-4, 100), (7e-4, 5e-4, 100), (0.05, 0.005, 200),
                      (1e-3, 0.0, 50), (1.5e-3, 1.5e-3, 70), (5e-4, 5e-4, 0)]:
        for t in list(range(-2, T + 3)) if T else [-1, 0, 1]:
            assert math.isclose(E.es_sigma_cosine(s0, sT, t, T), oracle.sigma_cosine(s0, sT, t, T),
                                rel_tol=1e-15, abs_tol=1e-300)


def test_update_coeffs_and_fold_match_oracle(E, oracle):
    rng = np.random.default_rng(1)
    for n in (1, 8, 30, 128):
        rhat = rng.standard_normal(n)
        for mode in (E.ES_SCALE_PAPER, E.ES_SCALE_CANONICAL):
            assert np.array_equal(E.es_update_coeffs(rhat, 5e-4, 1e-3, mode),
                                  oracle.update_coeffs(rhat, 5e-4, 1e-3, mode))
            rm = rng.standard_normal(n)
            assert np.array_equal(E.es_fold_antithetic(rhat, rm, 0.01, 0.05, mode),
                                  oracle.fold_antithetic(rhat, rm, 0.01, 0.05, mode))


def test_host_argument_errors(E):
    with pytest.raises(E.EsError) as ei:
        E.es_update_coeffs([1.0], 1e-3, 0.0, E.ES_SCALE_CANONICAL)
    assert ei.value.status == E.ES_ERR_INVALID_ARG
    with pytest.raises(E.EsError) as ei:
        E.es_update_coeffs([1.0], float("nan"), 1e-3, E.ES_SCALE_PAPER)
    assert ei.value.status == E.ES_ERR_NONFINITE
    with pytest.raises(E.EsError) as ei:
        E.es_update_coeffs([1.0], 1e-3, 1e-3, 7)
    assert ei.value.status == E.ES_ERR_INVALID_ARG
    with pytest.raises(E.EsError) as ei:
        E.es_normalize_rewards([1.0, 2.0], -1.0)
    assert ei.value.status == E.ES_ERR_INVALID_ARG
    with pytest.raises(E.EsError) as ei:
        E.es_normalize_rewards([], 1e-8)
    assert ei.value.status == E.ES_ERR_INVALID_ARG


def test_assign_index_bases(E):
    segs = [E.Segment(0, n) for n in (10, 3, 16, 8, 1)]
    end = E.es_assign_index_bases(segs)
    assert [s.index_base for s in segs] == [0, 16, 24, 40, 48]
    assert end == 49


def test_plan_validation_rejects_before_touching_the_device(E):
    # Only integers stand in for device pointers: validation runs before any
    # CUDA call, so these return their error without a GPU or driver.
    S = E.Segment
    cases = [
        ([S(0x1008, 16, 0)], E.ES_ERR_ALIGNMENT),                 # data not 16-B aligned
        ([S(0x1000, 16, 4)], E.ES_ERR_ALIGNMENT),                 # base not a multiple of 8
        ([S(0x1000, 0, 0)], E.ES_ERR_INVALID_ARG),                # empty segment
        ([S(0, 16, 0)], E.ES_ERR_INVALID_ARG),                    # NULL data
        ([S(0x1000, 16, 0), S(0x2000, 16, 8)], E.ES_ERR_OVERLAP),      # index ranges overlap
        ([S(0x1000, 16, 0), S(0x1010, 16, 16)], E.ES_ERR_OVERLAP),     # memory overlaps (bf16)
        ([S(0x1000, 16, 2**64 - 8)], E.ES_ERR_INVALID_ARG),       # index range past 2^64
    ]
    for segs, want in cases:
        with pytest.raises(E.EsError) as ei:
            E.es_plan_create(segs, E.ES_BF16)
        assert ei.value.status == want, (segs, ei.value)
    with pytest.raises(E.EsError) as ei:
        E.es_plan_create([S(0x1000, 16, 0)], 5)
    assert ei.value.status == E.ES_ERR_INVALID_ARG
    # Adjacent (touching) segments pass every host check; the device step then
    # fails: without a GPU at cudaGetDevice, with one at the device-memory check
    # (these addresses are not device memory).
    with pytest.raises(E.EsError) as ei:
        E.es_plan_create([S(0x1000, 16, 0), S(0x1020, 16, 16)], E.ES_BF16)
    assert ei.value.status in (E.ES_ERR_CUDA, E.ES_ERR_INVALID_ARG)
    if ei.value.status == E.ES_ERR_INVALID_ARG:
        assert "not device memory" in str(ei.value)


def test_product_path_has_no_cpu_fallback(E, monkeypatch, tmp_path):
    # With the library missing, the binding raises instead of computing anything.
    import importlib
    from paper_2608_17310_gb300 import esopt as mod
    fresh = importlib.reload(mod)
    monkeypatch.setattr(fresh, "LIB_PATH", str(tmp_path / "missing.so"))
    fresh._lib = None
    with pytest.raises(RuntimeError):
        fresh.es_sigma_cosine(1.0, 0.0, 0, 1)
    importlib.reload(mod)


def test_noalloc_validation_rejects_before_touching_the_device(E):
    S = E.Segment
    cases = [
        ([S(0x1000, 16, 0)] * (E.ES_STATIC_MAX_SEGMENTS + 1), E.ES_ERR_INVALID_ARG),
        ([S(0x1008, 16, 0)], E.ES_ERR_ALIGNMENT),
        ([S(0x1000, 16, 4)], E.ES_ERR_ALIGNMENT),
        ([S(0x1000, 16, 0), S(0x1010, 16, 16)], E.ES_ERR_OVERLAP),
        ([S(0x1000, 16, 0), S(0x2000, 16, 8)], E.ES_ERR_OVERLAP),
    ]
    for segs, want in cases:
        with pytest.raises(E.EsError) as ei:
            E.es_perturb_noalloc(segs, E.ES_BF16, 1, 1e-3)
        assert ei.value.status == want
    with pytest.raises(E.EsError) as ei:
        E.es_perturb_noalloc([S(0x1000, 16, 0)], E.ES_BF16, 1, float("nan"))
    assert ei.value.status == E.ES_ERR_NONFINITE


def test_normalize_rewards_in_place(E, oracle):
    import ctypes
    R = np.array([0.3, np.nan, 0.9, 0.1, 0.5, 0.5])
    want = oracle.zscore(R.copy(), 1e-8)
    buf = R.copy()
    P = ctypes.POINTER(ctypes.c_double)
    st = E.lib().es_normalize_rewards(buf.ctypes.data_as(P), buf.size, 1e-8, buf.ctypes.data_as(P))
    assert st == E.ES_OK
    assert np.allclose(buf, want, rtol=1e-14, atol=1e-14)


def test_assign_index_bases_overflow_returns_zero(E):
    segs = [E.Segment(0, 2**63), E.Segment(0, 2**63 + 16)]
    assert E.es_assign_index_bases(segs) == 0


def test_last_error_is_per_thread(E):
    # Each thread provokes a different validation error (no device call is
    # reached) and must read back its own detail, whatever the other threads
    # do meanwhile: es_last_error() is thread-local.
    import threading
    S = E.Segment
    cases = {
        "align": ([S(0x1001, 16, 0)], "16-byte aligned"),
        "base": ([S(0x1000, 16, 3)], "multiple of 8"),
        "overlap": ([S(0x1000, 16, 0), S(0x2000, 16, 8)], "overlap in index space"),
        "empty": ([S(0x1000, 0, 0)], "zero numel"),
    }
    errors = []
    barrier = threading.Barrier(len(cases))

    def worker(name, segs, expect):
        try:
            barrier.wait()
            for _ in range(200):
                try:
                    E.es_plan_create(segs, E.ES_BF16)
                except E.EsError:
                    pass
                msg = E.es_last_error()
                if expect not in msg:
                    errors.append((name, msg))
                    return
        except Exception as exc:  # pragma: no cover
            errors.append((name, repr(exc)))

    threads = [threading.Thread(target=worker, args=(k, s, e)) for k, (s, e) in cases.items()]
    for t in threads:
        t.start()
    for t in threads:
        t.join()
    assert not errors, errors


def test_scaled_plan_rejects_bad_scales_before_any_device_call(E):
    # The scales are checked before the segments are looked at, so this pointer
    # is never dereferenced.
    seg = [E.Segment(0x100000, 16, 0)]
    for bad in (0.0, -1.0, float("nan"), float("inf"), 1e-45):
        with pytest.raises(E.EsError) as ei:
            E.es_plan_create_scaled(seg, [bad], E.ES_FP8_E4M3)
        assert ei.value.status == E.ES_ERR_INVALID_ARG
    with pytest.raises(E.EsError) as ei:
        E.es_plan_create_scaled(seg, [1.0], E.ES_BF16)
    assert ei.value.status == E.ES_ERR_INVALID_ARG
