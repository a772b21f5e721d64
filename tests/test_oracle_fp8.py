"""Pins of the oracle's FP8 E4M3 storage functions (the quantized-weight
direction of App. A.2): decode and round-to-nearest-even encode against the
format's definition, against PyTorch's independent float8_e4m3fn conversion,
and the scaled perturb / update against invariants that a dropped term, a
wrong sign or a wrong scale would break."""
import numpy as np
import pytest
import torch

CODES = np.arange(256, dtype=np.uint8)
FINITE = np.array([c for c in CODES if (c & 0x7F) != 0x7F], dtype=np.uint8)


def _torch_decode(codes):
    return torch.from_numpy(np.asarray(codes, dtype=np.uint8)).view(torch.float8_e4m3fn) \
        .to(torch.float32).numpy().astype(np.float64)


def _torch_encode(values):
    t = torch.from_numpy(np.asarray(values, dtype=np.float32)).to(torch.float8_e4m3fn)
    return t.view(torch.uint8).numpy()


def test_decode_equals_torch_for_every_code(oracle):
    got = oracle.e4m3_codes_to_f64(CODES)
    want = _torch_decode(CODES)
    nan = np.isnan(want)
    assert np.array_equal(np.isnan(got), nan)
    assert nan.sum() == 2                                  # 0x7F and 0xFF
    assert np.array_equal(got[~nan], want[~nan])
    assert np.array_equal(np.signbit(got[~nan]), np.signbit(want[~nan]))   # -0 kept


def test_format_extremes():
    from oracle import oracle as O
    assert O.e4m3_to_double(0x7E) == 448.0                # largest finite
    assert O.e4m3_to_double(0x01) == 2.0 ** -9            # smallest subnormal
    assert O.e4m3_to_double(0x07) == 7 * 2.0 ** -9        # largest subnormal
    assert O.e4m3_to_double(0x08) == 2.0 ** -6            # smallest normal
    assert O.e4m3_to_double(0x38) == 1.0


def test_every_finite_code_round_trips(oracle):
    vals = oracle.e4m3_codes_to_f64(FINITE)
    back = np.array([oracle.e4m3_from_double(v) for v in vals], dtype=np.uint8)
    assert np.array_equal(back, FINITE)


def test_positive_codes_are_strictly_increasing(oracle):
    vals = oracle.e4m3_codes_to_f64(np.arange(0, 0x7F, dtype=np.uint8))
    assert np.all(np.diff(vals) > 0)


def test_midpoints_round_to_the_even_code(oracle):
    # Between consecutive finite codes a < b: the midpoint goes to the code with
    # the even mantissa bit, points just inside go to the nearer code.
    for sign in (0x00, 0x80):
        for a in range(0, 0x7E):
            ca, cb = sign | a, sign | (a + 1)
            va, vb = oracle.e4m3_to_double(ca), oracle.e4m3_to_double(cb)
            mid = 0.5 * (va + vb)
            want = ca if (a & 1) == 0 else cb
            assert oracle.e4m3_from_double(mid) == want, (hex(ca), mid)
            assert oracle.e4m3_from_double(mid - 1e-3 * (vb - va)) == ca
            assert oracle.e4m3_from_double(mid + 1e-3 * (vb - va)) == cb


def test_encode_equals_torch_within_range(oracle):
    # torch rounds float32 to float8_e4m3fn to nearest, ties to even; inside the
    # finite range it must agree code for code (outside, torch gives NaN where
    # the oracle saturates).
    rng = np.random.default_rng(3)
    vals = np.concatenate([
        rng.uniform(-448, 448, 20000), rng.standard_normal(20000) * 2.0,
        rng.standard_normal(20000) * 0.01, rng.uniform(-2.0**-6, 2.0**-6, 5000),
        0.5 * (oracle.e4m3_codes_to_f64(FINITE[:-1]) + oracle.e4m3_codes_to_f64(FINITE[1:]))])
    vals = vals[np.isfinite(vals) & (np.abs(vals) <= 448)].astype(np.float32)
    got = np.array([oracle.e4m3_from_double(float(v)) for v in vals], dtype=np.uint8)
    want = _torch_encode(vals)
    # -0 and +0 may differ in sign only for inputs that are zero
    assert np.array_equal(got, want), np.nonzero(got != want)[0][:5]


def test_saturation_and_nan(oracle):
    for x, want in ((448.0, 0x7E), (449.0, 0x7E), (463.99, 0x7E), (464.0, 0x7E), (1e30, 0x7E),
                    (float("inf"), 0x7E), (-500.0, 0xFE), (float("-inf"), 0xFE)):
        assert oracle.e4m3_from_double(x) == want, x
    assert oracle.e4m3_from_double(float("nan")) & 0x7F == 0x7F


def _finite_codes(n, seed):
    rng = np.random.default_rng(seed)
    return rng.choice(FINITE, size=n)


def _same_values(a, b):
    """Codes with equal values (+0 and -0 are equal: IEEE -0 + +0 is +0)."""
    return np.array_equal(np.where(a == 0x80, 0, a), np.where(b == 0x80, 0, b))


def test_zero_sigma_leaves_every_code_unchanged(oracle):
    codes = np.tile(FINITE, 4)
    g = np.arange(codes.size, dtype=np.uint64)
    for s in (1.0, 0.02 / 448, 3.0):
        assert _same_values(oracle.perturb(codes, g, 5, 0.0, "e4m3", s), codes)
        assert _same_values(oracle.update(codes, g, [5], [0.0], "e4m3", s), codes)


def test_scaled_step_is_invariant_under_a_power_of_two(oracle):
    # (2s d + 2 sigma eps) / (2s) = (s d + sigma eps) / s exactly: doubling the
    # segment scale together with sigma (or the coefficients) changes nothing,
    # while doubling only sigma does.
    codes = _finite_codes(4096, 1)
    g = np.arange(2**34 - 2048, 2**34 + 2048, dtype=np.uint64)
    s, sigma = 0.1 / 448, 1e-3
    a = oracle.perturb(codes, g, 77, sigma, "e4m3", s)
    b = oracle.perturb(codes, g, 77, 2 * sigma, "e4m3", 2 * s)
    assert np.array_equal(a, b)
    assert not np.array_equal(a, oracle.perturb(codes, g, 77, 2 * sigma, "e4m3", s))
    c = oracle.update(codes, g, [3, 4], [1e-3, -2e-3], "e4m3", s)
    d = oracle.update(codes, g, [3, 4], [2e-3, -4e-3], "e4m3", 2 * s)
    assert np.array_equal(c, d)


def test_update_agrees_with_the_perturb_it_generalises(oracle):
    codes = _finite_codes(4096, 2)
    g = np.arange(8, 8 + codes.size, dtype=np.uint64)
    s = 0.05 / 448
    # one seed with coefficient c is a perturb by c
    assert np.array_equal(oracle.update(codes, g, [9], [3e-4], "e4m3", s),
                          oracle.perturb(codes, g, 9, 3e-4, "e4m3", s))
    # a seed listed twice adds twice; +c and -c of one seed cancel exactly
    assert np.array_equal(oracle.update(codes, g, [9, 9], [3e-4, 3e-4], "e4m3", s),
                          oracle.perturb(codes, g, 9, 6e-4, "e4m3", s))
    assert _same_values(oracle.update(codes, g, [9, 9], [3e-4, -3e-4], "e4m3", s), codes)


def test_perturb_moves_by_the_noise_within_half_a_step(oracle):
    # |stored value - (value + sigma eps)| <= half the E4M3 spacing there
    # (ties included), over many codes: the result is the nearest grid point.
    codes = _finite_codes(20000, 4)
    codes = codes[np.abs(oracle.e4m3_codes_to_f64(codes)) < 64]
    g = np.arange(codes.size, dtype=np.uint64) * 3 + 16
    s, sigma = 0.02 / 448, 1e-4           # sigma / s = 2.24 code units: no saturation
    out = oracle.perturb(codes, g, 123, sigma, "e4m3", s)
    exact = oracle.e4m3_codes_to_f64(codes) + sigma * oracle.noise_at(123, g) / s
    got = oracle.e4m3_codes_to_f64(out)
    a = np.maximum(np.abs(exact), 2.0 ** -6)
    spacing = 2.0 ** (np.floor(np.log2(a)) - 3)
    assert np.all(np.abs(got - exact) <= 0.5 * spacing * (1 + 1e-12))
    assert np.count_nonzero(out != codes) > codes.size // 4
