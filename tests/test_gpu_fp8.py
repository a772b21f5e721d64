"""FP8 E4M3 storage (App. A.2's quantized-weight direction; the step is
unchanged, only the storage grid is new): every device entry point on plans
whose segments hold E4M3 codes with one scale each, element by element against
the oracle, on ragged segments with 64-bit global indices. Codes must agree
within one E4M3 step (both sides round to nearest even, the GPU from an fp32
value and the oracle from a double one), or, where the value and the noise
term cancel, within the carried noise tolerance plus one step; NaN stays NaN
and +0 equals -0."""
import numpy as np
import pytest
import torch

from parity import noise_abs_tol

pytestmark = pytest.mark.gpu

NUMELS = [1, 15, 16, 17, 4099, 16384, 16385, 50021]
BASES = [8, 2**33 + 64, 2**34 - 4096, 2**36, 2**40 + 8, 2**50, 2**61, 2**62 - 2**20]


def e4m3_order(codes):
    c = np.asarray(codes, dtype=np.uint8).astype(np.int64)
    mag = c & 0x7F
    return np.where(c & 0x80, -mag, mag)


def e4m3_values(codes):
    return torch.from_numpy(np.ascontiguousarray(codes, dtype=np.uint8)) \
        .view(torch.float8_e4m3fn).to(torch.float32).numpy().astype(np.float64)


def assert_e4m3_close(got, want, what, abs_tol=0.0):
    """Within one E4M3 step, or within abs_tol (code units) plus one step."""
    got = np.asarray(got, dtype=np.uint8)
    want = np.asarray(want, dtype=np.uint8)
    g, w = e4m3_values(got), e4m3_values(want)
    nan_g, nan_w = np.isnan(g), np.isnan(w)
    assert np.array_equal(nan_g, nan_w), f"{what}: NaN pattern differs"
    ok = ~nan_g
    d = np.abs(e4m3_order(got) - e4m3_order(want))
    d = np.where((g == 0) & (w == 0), 0, d)               # +0 and -0
    a = np.maximum(np.maximum(np.abs(g), np.abs(w)), 2.0**-6)
    step = 2.0 ** (np.floor(np.log2(a)) - 3)
    near = np.abs(g - w) <= abs_tol + step
    bad = np.nonzero(ok & (d > 1) & ~near)[0]
    assert bad.size == 0, (f"{what}: {bad.size} of {got.size} codes more than one step apart; "
                           f"first at {bad[:5]}: got {got[bad[:5]]} want {want[bad[:5]]}")


def make_fp8(seed, numels=NUMELS, specials=True):
    """E4M3 codes of N(0, 0.02^2) weights with a per-tensor scale amax / 448,
    as uint8 CUDA tensors, plus the scales; the first tensors get the format's
    special codes (zeros, subnormals, the largest values, NaN) mixed in."""
    rng = np.random.default_rng(seed)
    codes, scales = [], []
    special = np.array([0x00, 0x80, 0x01, 0x81, 0x07, 0x08, 0x7E, 0xFE, 0x7D, 0x7F, 0x38],
                       dtype=np.uint8)
    for k, n in enumerate(numels):
        w = 0.02 * rng.standard_normal(n)
        s = np.float32(max(np.abs(w).max(), 1e-3) / 448)
        c = torch.from_numpy((w / s).astype(np.float32)).to(torch.float8_e4m3fn) \
            .view(torch.uint8).numpy().copy()
        if specials and n >= 64:
            pos = rng.choice(n, size=special.size, replace=False)
            c[pos] = special
        codes.append(torch.from_numpy(c).cuda())
        scales.append(float(s))
    return codes, scales


def host(t):
    return t.cpu().numpy().copy()


def build(es, codes, scales, bases=BASES):
    plan = es.plan_from_tensors(codes, bases[:len(codes)], scales=scales)
    g = [np.arange(b, b + t.numel(), dtype=np.uint64) for b, t in zip(bases, codes)]
    return plan, g


def test_perturb_restore_match_oracle(es, oracle):
    codes, scales = make_fp8(1)
    plan, g = build(es, codes, scales)
    seed, sigma = 2**41 + 3, 1e-3
    before = [host(t) for t in codes]
    es.es_perturb(plan, seed, sigma)
    torch.cuda.synchronize()
    mid = [host(t) for t in codes]
    for k in range(len(codes)):
        tol = noise_abs_tol([oracle.noise_at(seed, g[k])], [sigma]) / scales[k]
        assert_e4m3_close(mid[k], oracle.perturb(before[k], g[k], seed, sigma, "e4m3", scales[k]),
                          f"perturb seg {k}", tol)
        assert np.count_nonzero(mid[k] != before[k]) > 0 or codes[k].numel() < 64
    es.es_restore(plan, seed, sigma)
    torch.cuda.synchronize()
    for k in range(len(codes)):
        tol = noise_abs_tol([oracle.noise_at(seed, g[k])], [sigma]) / scales[k]
        assert_e4m3_close(host(codes[k]), oracle.restore(mid[k], g[k], seed, sigma, "e4m3",
                                                         scales[k]), f"restore seg {k}", tol)
    plan.close()


def test_zero_sigma_leaves_codes_unchanged(es):
    codes, scales = make_fp8(2)
    plan, _ = build(es, codes, scales)
    before = [host(t) for t in codes]
    es.es_perturb(plan, 5, 0.0)
    torch.cuda.synchronize()
    for a, t in zip(before, codes):
        b = host(t)
        same = (a == b) | ((a & 0x7F) == 0) & ((b & 0x7F) == 0) | \
            ((a & 0x7F) == 0x7F) & ((b & 0x7F) == 0x7F)
        assert np.all(same)
    plan.close()


@pytest.mark.parametrize("nseeds", [1, 3, 30, 128])
def test_update_matches_oracle(es, oracle, nseeds):
    codes, scales = make_fp8(3 + nseeds)
    plan, g = build(es, codes, scales)
    rng = np.random.default_rng(nseeds)
    seeds = rng.integers(0, 2**63, size=nseeds, dtype=np.uint64)
    coeffs = (1e-3 * rng.standard_normal(nseeds)).astype(np.float32)
    before = [host(t) for t in codes]
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    for k in range(len(codes)):
        tol = noise_abs_tol([oracle.noise_at(int(s), g[k]) for s in seeds], coeffs) / scales[k]
        assert_e4m3_close(host(codes[k]),
                          oracle.update(before[k], g[k], seeds, coeffs, "e4m3", scales[k]),
                          f"update N={nseeds} seg {k}", tol)
    plan.close()


def test_fused_calls_are_bit_identical_to_the_separate_ones(es, oracle):
    a, scales = make_fp8(7)
    b = [t.clone() for t in a]
    plan_a, g = build(es, a, scales)
    plan_b, _ = build(es, b, scales)
    for p in (plan_a, plan_b):
        es.es_perturb(p, 11, 1e-3)
    es.es_restore(plan_a, 11, 1e-3)
    es.es_perturb(plan_a, 12, 7e-4)
    es.es_restore_perturb(plan_b, 11, 1e-3, 12, 7e-4)
    es.es_restore(plan_a, 12, 7e-4)
    es.es_perturb(plan_a, 12, -7e-4)
    es.es_restore_perturb(plan_b, 12, 7e-4, 12, -7e-4)          # antithetic flip
    seeds = np.arange(500, 516, dtype=np.uint64)
    coeffs = np.linspace(-2e-3, 2e-3, 16).astype(np.float32)
    es.es_update(plan_a, seeds, coeffs)
    es.es_perturb(plan_a, 13, 1e-3)
    es.es_update_perturb(plan_b, seeds, coeffs, 13, 1e-3)
    counts = [3, 1, 2, 6]
    rs = np.arange(900, 912, dtype=np.uint64)
    rc = np.linspace(-1e-3, 1e-3, 12).astype(np.float32)
    off = 0
    for c in counts:
        es.es_update(plan_a, rs[off:off + c], rc[off:off + c])
        off += c
    es.es_replay(plan_b, rs, rc, counts)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(x, y)
    plan_a.close()
    plan_b.close()


def test_saturation_at_the_largest_value(es, oracle):
    # Codes near +-448 pushed outwards by a large sigma saturate to +-448 on
    # both sides; pushed inwards they round normally.
    n = 4096
    c = np.where(np.arange(n) % 2 == 0, 0x7E, 0xFE).astype(np.uint8)
    c[::3] = 0x7C
    t = torch.from_numpy(c).cuda()
    plan, g = build(es, [t], [1.0], [1024])
    es.es_perturb(plan, 77, 60.0)
    torch.cuda.synchronize()
    want = oracle.perturb(c, g[0], 77, 60.0, "e4m3", 1.0)
    tol = noise_abs_tol([oracle.noise_at(77, g[0])], [60.0])
    assert_e4m3_close(host(t), want, "saturation", tol)
    assert np.count_nonzero((host(t) & 0x7F) == 0x7E) > n // 4
    plan.close()


def test_scaled_plan_argument_errors(es):
    t = torch.zeros(64, dtype=torch.uint8, device="cuda")
    seg = es.segments_from_tensors([t])
    for bad in (0.0, -1.0, float("nan"), float("inf"), 1e-45):
        with pytest.raises(es.EsError) as ei:
            es.es_plan_create_scaled(seg, [bad], es.ES_FP8_E4M3)
        assert ei.value.status == es.ES_ERR_INVALID_ARG
    with pytest.raises(es.EsError):
        es.es_plan_create_scaled(seg, [1.0], es.ES_BF16)
    p = es.es_plan_create(seg, es.ES_FP8_E4M3)                  # scale 1
    p.close()
