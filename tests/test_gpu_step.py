"""GPU parity of perturb / restore / fused update through the C ABI, element by
element against the oracle, on multi-segment plans with ragged tails, gaps in
the index space and 64-bit indices, in bf16 and fp32 storage."""
import numpy as np
import pytest
import torch

from parity import (assert_bf16_within_ulp, assert_f32_close, bf16_order, bf16_values,
                    noise_abs_tol)

pytestmark = pytest.mark.gpu

RAGGED = [1, 7, 8, 9, 8191, 8192, 8193, 20000, 100003, 4096 * 3 + 5]


def make_params(dtype, numels, seed=0):
    rng = np.random.default_rng(seed)
    tensors = []
    for n in numels:
        v = torch.from_numpy((0.02 * rng.standard_normal(n)).astype(np.float32))
        tensors.append((v.to(torch.bfloat16) if dtype == "bf16" else v).cuda())
    return tensors


def host_values(t):
    c = t.detach().cpu()
    if c.dtype == torch.bfloat16:
        return c.view(torch.int16).numpy().view(np.uint16).copy()
    return c.numpy().copy()


def indices(plan_segs):
    return [np.arange(s.index_base, s.index_base + s.numel, dtype=np.uint64) for s in plan_segs]


def compare(dtype, got, want, what, abs_tol=0.0):
    if dtype == "bf16":
        assert_bf16_within_ulp(got, want, what, abs_tol=abs_tol)
    else:
        assert_f32_close(got, want, what, abs_tol)


def ulp32(x):
    return np.spacing(np.abs(np.asarray(x, dtype=np.float32))).astype(np.float64)


def build_plan(es, tensors, bases=None):
    segs = es.segments_from_tensors(tensors, bases)
    plan = es.plan_from_tensors(tensors, [s.index_base for s in segs])
    return plan, segs


def _sparse64(n):
    bases = [2**35 + k * 2**21 for k in range(n)]
    bases[8] = 2**34 - 40      # 100003 elements straddle g = 2^34 (block j = 2^32)
    bases[-1] = 2**61
    return bases


BASE_LAYOUTS = {
    "packed": None,
    # gaps, indices past 2^32 blocks (g >= 2^34) and one segment straddling g = 2^34
    "sparse64": lambda numels: _sparse64(len(numels)),
}


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("layout", list(BASE_LAYOUTS))
def test_perturb_then_restore_match_oracle(es, oracle, dtype, layout):
    tensors = make_params(dtype, RAGGED, seed=1)
    bases = BASE_LAYOUTS[layout](RAGGED) if BASE_LAYOUTS[layout] else None
    plan, segs = build_plan(es, tensors, bases)
    before = [host_values(t) for t in tensors]
    g = indices(segs)
    seed, sigma = 2**40 + 17, 1e-3
    es.es_perturb(plan, seed, sigma)
    torch.cuda.synchronize()
    perturbed = [host_values(t) for t in tensors]
    eps = [oracle.noise_at(seed, gk) for gk in g]
    for k in range(len(tensors)):
        want = oracle.perturb(before[k], g[k], seed, sigma, dtype)
        compare(dtype, perturbed[k], want, f"perturb seg {k} ({layout})",
                noise_abs_tol([eps[k]], [sigma]))
    es.es_restore(plan, seed, sigma)
    torch.cuda.synchronize()
    for k in range(len(tensors)):
        got = host_values(tensors[k])
        want = oracle.restore(perturbed[k], g[k], seed, sigma, dtype)   # step by step
        compare(dtype, got, want, f"restore seg {k} ({layout})", noise_abs_tol([eps[k]], [sigma]))
        if dtype == "f32":     # the round trip returns theta within one rounding
            bound = 2 * ulp32(np.maximum(np.abs(before[k]), sigma * np.abs(eps[k])))
            assert np.all(np.abs(got.astype(np.float64) - before[k]) <= bound), f"round trip {k}"
    plan.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_restore_perturb_is_bit_identical_to_the_two_calls(es, oracle, dtype):
    a = make_params(dtype, RAGGED, seed=7)
    b = [t.clone() for t in a]
    plan_a, segs = build_plan(es, a, _sparse64(len(RAGGED)))
    plan_b, _ = build_plan(es, b, _sparse64(len(RAGGED)))
    s1, s2, sig1, sig2 = 11, 2**45 + 3, 1e-3, 7e-4
    for p in (plan_a, plan_b):
        es.es_perturb(p, s1, sig1)
    torch.cuda.synchronize()
    mid = [host_values(t) for t in a]
    es.es_restore(plan_a, s1, sig1)
    torch.cuda.synchronize()
    restored = [host_values(t) for t in a]
    es.es_perturb(plan_a, s2, sig2)
    es.es_restore_perturb(plan_b, s1, sig1, s2, sig2)
    torch.cuda.synchronize()
    iv = torch.int16 if dtype == "bf16" else torch.int32
    for x, y in zip(a, b):
        assert torch.equal(x.view(iv), y.view(iv))
    # and against the oracle, step by step (each step from the GPU's input)
    g = indices(segs)
    for k in range(len(a)):
        tol1 = noise_abs_tol([oracle.noise_at(s1, g[k])], [sig1])
        compare(dtype, restored[k], oracle.restore(mid[k], g[k], s1, sig1, dtype),
                f"restore step seg {k}", tol1)
        tol2 = noise_abs_tol([oracle.noise_at(s2, g[k])], [sig2])
        compare(dtype, host_values(b[k]), oracle.perturb(restored[k], g[k], s2, sig2, dtype),
                f"perturb step seg {k}", tol2)
    with pytest.raises(es.EsError) as ei:
        es.es_restore_perturb(plan_b, 1, float("nan"), 2, 1e-3)
    assert ei.value.status == es.ES_ERR_NONFINITE
    plan_a.close()
    plan_b.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
@pytest.mark.parametrize("nseeds", [1, 2, 3, 8, 30, 129, 256, 1024])
def test_update_matches_oracle(es, oracle, dtype, nseeds):
    numels = [9, 8193, 20000, 4096 * 3 + 5]
    tensors = make_params(dtype, numels, seed=2)
    plan, segs = build_plan(es, tensors, [8, 2**34 - 1024, 2**36, 2**50])
    before = [host_values(t) for t in tensors]
    rng = np.random.default_rng(nseeds)
    seeds = rng.integers(0, 2**63, size=nseeds, dtype=np.uint64)
    coeffs = (1e-3 * rng.standard_normal(nseeds)).astype(np.float32)
    if nseeds > 2:
        coeffs[1] = 0.0          # a zero coefficient is skipped without changing the result
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    g = indices(segs)
    for k in range(len(tensors)):
        want = oracle.update(before[k], g[k], seeds, coeffs, dtype)
        tol = noise_abs_tol([oracle.noise_at(int(s), g[k]) for s in seeds], coeffs)
        compare(dtype, host_values(tensors[k]), want, f"update N={nseeds} seg {k}", tol)
    plan.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_update_is_deterministic_and_launch_independent(es, dtype):
    tensors = make_params(dtype, [100003, 77], seed=3)
    copies = [t.clone() for t in tensors]
    plan_a, _ = build_plan(es, tensors)
    plan_b, _ = build_plan(es, copies)
    seeds, coeffs = np.arange(1, 17, dtype=np.uint64), np.linspace(-1e-3, 1e-3, 16, dtype=np.float32)
    es.es_update(plan_a, seeds, coeffs)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        es.es_update(plan_b, seeds, coeffs, stream=s)
    torch.cuda.synchronize()
    for a, b in zip(tensors, copies):
        assert torch.equal(a.view(torch.int16 if dtype == "bf16" else torch.int32),
                           b.view(torch.int16 if dtype == "bf16" else torch.int32))


def test_all_zero_coefficients_leave_theta_bit_identical(es):
    tensors = make_params("bf16", [8192, 5], seed=4)
    ref = [t.clone() for t in tensors]
    plan, _ = build_plan(es, tensors)
    es.es_update(plan, np.arange(8, dtype=np.uint64), np.zeros(8, np.float32))
    torch.cuda.synchronize()
    assert all(torch.equal(a.view(torch.int16), b.view(torch.int16)) for a, b in zip(tensors, ref))


def test_step_argument_errors(es):
    t = make_params("bf16", [64], seed=5)[0]
    plan, _ = build_plan(es, [t])
    with pytest.raises(es.EsError) as ei:
        es.es_perturb(plan, 1, float("nan"))
    assert ei.value.status == es.ES_ERR_NONFINITE
    with pytest.raises(es.EsError) as ei:
        es.es_restore(plan, 1, float("inf"))
    assert ei.value.status == es.ES_ERR_NONFINITE
    with pytest.raises(es.EsError) as ei:
        n = es.ES_MAX_SEEDS + 1
        es.es_update(plan, np.arange(n, dtype=np.uint64), np.ones(n, np.float32))
    assert ei.value.status == es.ES_ERR_TOO_MANY_SEEDS
    with pytest.raises(es.EsError) as ei:
        es.es_update(plan, [1, 2], np.array([1.0, np.nan], np.float32))
    assert ei.value.status == es.ES_ERR_NONFINITE
    with pytest.raises(es.EsError) as ei:
        es.es_update(plan, [], [])
    assert ei.value.status == es.ES_ERR_INVALID_ARG
    # misaligned segment: data pointer one bf16 element into the tensor
    with pytest.raises(es.EsError) as ei:
        es.es_plan_create([es.Segment(t.data_ptr() + 2, 8, 0)], es.ES_BF16)
    assert ei.value.status == es.ES_ERR_ALIGNMENT
    # two segments sharing memory
    with pytest.raises(es.EsError) as ei:
        es.es_plan_create([es.Segment(t.data_ptr(), 32, 0), es.Segment(t.data_ptr() + 32, 32, 64)],
                          es.ES_BF16)
    assert ei.value.status == es.ES_ERR_OVERLAP
    plan.close()


def test_max_population_update(es, oracle):
    t = make_params("f32", [4099], seed=6)[0]
    plan, segs = build_plan(es, [t])
    before = host_values(t)
    seeds = np.arange(10**6, 10**6 + es.ES_MAX_SEEDS, dtype=np.uint64)
    coeffs = np.full(es.ES_MAX_SEEDS, 1e-4, np.float32)
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    g = indices(segs)[0]
    want = oracle.update(before, g, seeds, coeffs, "f32")
    tol = noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs)
    assert_f32_close(host_values(t), want, f"N={es.ES_MAX_SEEDS}", tol)
    plan.close()


def _int_view(t):
    return t.view(torch.int16 if t.dtype == torch.bfloat16 else torch.int32)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_replay_is_bit_identical_to_sequential_updates(es, dtype):
    numels = [9, 8193, 20000, 4096 * 3 + 5]
    a = make_params(dtype, numels, seed=8)
    b = [t.clone() for t in a]
    bases = [8, 2**34 - 1024, 2**36, 2**50]
    plan_a, _ = build_plan(es, a, bases)
    plan_b, _ = build_plan(es, b, bases)
    rng = np.random.default_rng(9)
    # 300 generations of 1..8 seeds (over 256 generations and 1024 seeds: several
    # passes), some all-zero generations and zero coefficients
    counts = rng.integers(1, 9, size=300)
    total = int(counts.sum())
    seeds = rng.integers(0, 2**63, size=total, dtype=np.uint64)
    coeffs = (1e-3 * rng.standard_normal(total)).astype(np.float32)
    coeffs[rng.random(total) < 0.1] = 0.0
    off = 0
    for g, c in enumerate(counts):
        if g % 37 == 5:
            coeffs[off:off + c] = 0.0
        es.es_update(plan_a, seeds[off:off + c], coeffs[off:off + c])
        off += c
    es.es_replay(plan_b, seeds, coeffs, counts)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


def test_replay_of_many_small_generations_is_bit_identical(es):
    # 600 generations of 1..3 seeds: they are fused, so the limit of 256
    # generations per pass is reached; a few larger generations in between
    # take passes of their own.
    numels = [8193, 4096 * 3 + 5]
    a = make_params("bf16", numels, seed=18)
    b = [t.clone() for t in a]
    plan_a, _ = build_plan(es, a)
    plan_b, _ = build_plan(es, b)
    rng = np.random.default_rng(19)
    counts = rng.integers(1, 4, size=600)
    counts[[100, 101, 400]] = [5, 12, 4]
    total = int(counts.sum())
    seeds = rng.integers(0, 2**63, size=total, dtype=np.uint64)
    coeffs = (1e-3 * rng.standard_normal(total)).astype(np.float32)
    off = 0
    for c in counts:
        es.es_update(plan_a, seeds[off:off + c], coeffs[off:off + c])
        off += c
    es.es_replay(plan_b, seeds, coeffs, counts)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_update_perturb_is_bit_identical_to_the_two_calls(es, oracle, dtype):
    a = make_params(dtype, RAGGED, seed=10)
    b = [t.clone() for t in a]
    plan_a, segs = build_plan(es, a, _sparse64(len(RAGGED)))
    plan_b, _ = build_plan(es, b, _sparse64(len(RAGGED)))
    before = [host_values(t) for t in a]
    seeds = np.arange(500, 516, dtype=np.uint64)
    coeffs = np.linspace(-2e-3, 2e-3, 16).astype(np.float32)
    es.es_update(plan_a, seeds, coeffs)
    torch.cuda.synchronize()
    updated = [host_values(t) for t in a]
    es.es_perturb(plan_a, 2**40 + 1, 9e-4)
    es.es_update_perturb(plan_b, seeds, coeffs, 2**40 + 1, 9e-4)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    # against the oracle, step by step (each step from the GPU's input)
    g = indices(segs)
    for k in (0, 5, 8):
        tol = noise_abs_tol([oracle.noise_at(int(s), g[k]) for s in seeds], coeffs)
        compare(dtype, updated[k], oracle.update(before[k], g[k], seeds, coeffs, dtype),
                f"update step seg {k}", tol)
        tol = noise_abs_tol([oracle.noise_at(2**40 + 1, g[k])], [9e-4])
        compare(dtype, host_values(b[k]), oracle.perturb(updated[k], g[k], 2**40 + 1, 9e-4, dtype),
                f"perturb step seg {k}", tol)
    # all-zero coefficients: only the perturb
    es.es_update_perturb(plan_b, seeds, np.zeros(16, np.float32), 77, 1e-3)
    es.es_perturb(plan_a, 77, 1e-3)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_antithetic_restore_perturb_reuses_one_seed(es, dtype):
    # restore (+sigma eps_i) then perturb (-sigma eps_i): the same noise twice
    a = make_params(dtype, RAGGED, seed=12)
    b = [t.clone() for t in a]
    plan_a, _ = build_plan(es, a, _sparse64(len(RAGGED)))
    plan_b, _ = build_plan(es, b, _sparse64(len(RAGGED)))
    for p in (plan_a, plan_b):
        es.es_perturb(p, 31, 5e-2)
    es.es_restore(plan_a, 31, 5e-2)
    es.es_perturb(plan_a, 31, -5e-2)
    es.es_restore_perturb(plan_b, 31, 5e-2, 31, -5e-2)
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


def _sample(segs, rng, per_seg=2048, edge=64):
    """Indices into each segment: its first and last `edge` elements plus
    about `per_seg` random ones (all of a short segment)."""
    out = []
    for s in segs:
        n = s.numel
        if n <= per_seg + 2 * edge:
            out.append(np.arange(n))
            continue
        idx = np.concatenate([np.arange(edge), np.arange(n - edge, n),
                              rng.integers(edge, n - edge, size=per_seg)])
        out.append(np.unique(idx))
    return out


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_replay_matches_oracle_generation_by_generation(es, oracle, dtype):
    # The seed log of a run is replayed from the base parameters (App. D.2-D.4):
    # 400 logged generations. The first 300 have 1..3 seeds, so they share
    # passes over theta and pass the 256-generation limit of one pass; the
    # last 100 have 1..8 seeds, so generations of 4 or more get passes of their
    # own through the single-generation kernel. Some generations and some
    # coefficients are zero. The oracle applies the same generations one by one
    # in double precision, rounding to storage after each, from the same start.
    numels = [9, 8193, 20000, 4096 * 3 + 5]
    tensors = make_params(dtype, numels, seed=40)
    plan, segs = build_plan(es, tensors, [8, 2**34 - 1024, 2**36, 2**50])
    rng = np.random.default_rng(41)
    counts = np.concatenate([rng.integers(1, 4, size=300), rng.integers(1, 9, size=100)])
    total = int(counts.sum())
    seeds = rng.integers(0, 2**63, size=total, dtype=np.uint64)
    coeffs = (1e-3 * rng.standard_normal(total)).astype(np.float32)
    coeffs[rng.random(total) < 0.05] = 0.0
    ends = np.cumsum(counts)
    starts = ends - counts
    for gen in (7, 250, 333):
        coeffs[starts[gen]:ends[gen]] = 0.0
    pick = _sample(segs, rng)
    g = indices(segs)
    state = [host_values(t)[ix] for t, ix in zip(tensors, pick)]
    gidx = [gk[ix] for gk, ix in zip(g, pick)]
    es.es_replay(plan, seeds, coeffs, counts)
    torch.cuda.synchronize()

    def values(x):
        return bf16_values(x) if dtype == "bf16" else np.asarray(x, dtype=np.float64)

    tol = [0.0] * len(segs)
    peak = [np.abs(values(x)) for x in state]
    for a, b in zip(starts, ends):
        for k in range(len(segs)):
            state[k] = oracle.update(state[k], gidx[k], seeds[a:b], coeffs[a:b], dtype)
            tol[k] = tol[k] + noise_abs_tol(
                [oracle.noise_at(int(sd), gidx[k]) for sd in seeds[a:b]], coeffs[a:b])
            peak[k] = np.maximum(peak[k], np.abs(values(state[k])))
    # Each generation rounds once on both sides: the GPU from an fp32 sum, the
    # oracle from a double one. Where the exact value lies within the fp32 sum's
    # error of a rounding tie, the two round to neighbouring values one unit in
    # the last place apart, and later generations carry that absolute
    # difference even after |theta| has shrunk. So the replay is held to the
    # step's unit: two units in the last place of the largest |theta| the
    # element took along the oracle's trajectory (bf16), or the per-call
    # relative bound 1e-5 of that magnitude (fp32), plus the carried noise
    # tolerance; and for bf16 at most 0.1 % of the elements may differ by more
    # than one such unit.
    for k in range(len(segs)):
        got = values(host_values(tensors[k])[pick[k]])
        want = values(state[k])
        err = np.abs(got - want)
        if dtype == "bf16":
            unit = 2.0 ** (np.floor(np.log2(np.maximum(peak[k], 2.0**-126))) - 7)
            bad = err > 2 * unit + tol[k]
            far = err > unit + tol[k]
            assert np.count_nonzero(far) <= max(1, got.size // 1000), f"replay seg {k}"
        else:
            bad = err > 1e-5 * peak[k] + tol[k]
        assert not np.any(bad), (f"replay seg {k}: {np.count_nonzero(bad)} elements; first "
                                 f"got {got[bad][:3]} want {want[bad][:3]}")
    plan.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_antithetic_flip_matches_oracle(es, oracle, dtype):
    # The flip of an antithetic pair, es_restore_perturb(s, sigma, s, -sigma),
    # takes theta + sigma eps_s to theta - sigma eps_s in one pass with the
    # noise generated once: restore, then perturb with -sigma (§3), each
    # rounded to storage. Against the oracle's two steps from the GPU's input,
    # over several flips and seeds, on ragged 64-bit layouts.
    tensors = make_params(dtype, RAGGED, seed=42)
    plan, segs = build_plan(es, tensors, _sparse64(len(RAGGED)))
    g = indices(segs)
    for seed, sigma in ((31, 5e-2), (2**41 + 9, 1e-3), (2**63 + 5, 2.5e-4)):
        es.es_perturb(plan, seed, sigma)
        torch.cuda.synchronize()
        before = [host_values(t) for t in tensors]
        es.es_restore_perturb(plan, seed, sigma, seed, -sigma)
        torch.cuda.synchronize()
        # Two roundings (restore, then perturb), and the intermediate is not
        # observable: where the GPU and the oracle round the intermediate to
        # neighbouring values, that one-ulp difference at the intermediate's
        # magnitude is carried into the result, and the second rounding can add
        # one ulp at the result's. bf16 is held to that sum (plus the carried
        # noise tolerance), with at most 0.1 % of the elements beyond one ulp of
        # the larger magnitude; fp32 to the per-call relative bound of it. The
        # fused flip is also bit-identical to the two separate calls, each
        # checked one step at a time elsewhere.
        for k in range(len(tensors)):
            eps = oracle.noise_at(seed, g[k])
            mid = oracle.restore(before[k], g[k], seed, sigma, dtype)
            want = oracle.perturb(mid, g[k], seed, -sigma, dtype)
            got = host_values(tensors[k])
            tol = noise_abs_tol([eps, eps], [sigma, sigma])
            if dtype == "bf16":
                g_v, w_v, m_v = bf16_values(got), bf16_values(want), bf16_values(mid)

                def ulp(x):
                    return 2.0 ** (np.floor(np.log2(np.maximum(np.abs(x), 2.0**-126))) - 7)

                err = np.abs(g_v - w_v)
                bound = ulp(m_v) + ulp(w_v) + tol
                assert np.all(err <= bound), f"flip seed {seed} seg {k}"
                far = err > np.maximum(ulp(m_v), ulp(w_v)) + tol
                assert np.count_nonzero(far) <= max(1, got.size // 1000), f"flip seed {seed} seg {k}"
            else:
                m_v = np.abs(np.asarray(mid, dtype=np.float64))
                err = np.abs(got.astype(np.float64) - np.asarray(want, dtype=np.float64))
                assert np.all(err <= 1e-5 * np.maximum(m_v, np.abs(want)) + tol), \
                    f"flip seed {seed} seg {k}"
        es.es_restore(plan, seed, -sigma)
    plan.close()


def test_replay_argument_errors(es):
    t = make_params("bf16", [64], seed=13)[0]
    plan, _ = build_plan(es, [t])
    for counts, status in (([0], es.ES_ERR_INVALID_ARG), ([es.ES_MAX_SEEDS + 1], es.ES_ERR_TOO_MANY_SEEDS)):
        n = sum(counts)
        with pytest.raises(es.EsError) as ei:
            es.es_replay(plan, np.arange(n, dtype=np.uint64), np.ones(n, np.float32), counts)
        assert ei.value.status == status
    with pytest.raises(es.EsError) as ei:
        es.es_replay(plan, [1, 2], np.array([1.0, np.inf], np.float32), [2])
    assert ei.value.status == es.ES_ERR_NONFINITE
    with pytest.raises(es.EsError) as ei:
        es.es_update_perturb(plan, [1], [1.0], 2, float("nan"))
    assert ei.value.status == es.ES_ERR_NONFINITE
    plan.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_results_do_not_depend_on_the_work_distribution(es, dtype):
    # The same tensors (same index bases) in plans that list them in different
    # orders give different tile-to-CTA assignments; every element must come
    # out bit-identical all the same.
    numels = [100003, 7, 8192 * 5 + 3, 2560, 65536, 9]
    a = make_params(dtype, numels, seed=14)
    b = [t.clone() for t in a]
    bases = [s.index_base for s in es.segments_from_tensors(a)]
    plan_a = es.plan_from_tensors(a, bases)
    order = [3, 0, 5, 2, 4, 1]
    plan_b = es.plan_from_tensors([b[k] for k in order], [bases[k] for k in order])
    seeds = np.arange(40, 52, dtype=np.uint64)
    coeffs = np.linspace(-1e-3, 1e-3, 12).astype(np.float32)
    for p in (plan_a, plan_b):
        es.es_perturb(p, 5, 1e-3)
        es.es_restore_perturb(p, 5, 1e-3, 6, 1e-3)
        es.es_update_perturb(p, seeds, coeffs, 7, 1e-3)
        es.es_replay(p, seeds, coeffs, [5, 7])
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


def test_many_tiny_segments(es, oracle):
    # 2000 segments of 1..40 elements with gaps in index space: thousands of
    # ragged one-tile segments, each CTA walking far through the table.
    rng = np.random.default_rng(15)
    numels = [int(n) for n in rng.integers(1, 41, size=2000)]
    tensors = make_params("bf16", numels, seed=16)
    bases, pos = [], 0
    for n in numels:
        bases.append(pos)
        pos += (n + 7) // 8 * 8 + 8 * int(rng.integers(0, 3))
    plan, segs = build_plan(es, tensors, bases)
    before = [host_values(t) for t in tensors]
    seeds = np.array([3, 4, 5], dtype=np.uint64)
    coeffs = np.array([1e-3, -2e-3, 5e-4], dtype=np.float32)
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    g = np.concatenate(indices(segs))
    got = np.concatenate([host_values(t) for t in tensors])
    want = oracle.update(np.concatenate(before), g, seeds, coeffs, "bf16")
    tol = noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs)
    compare("bf16", got, want, "2000 tiny segments", tol)
    plan.close()


def test_segment_larger_than_2_to_32_elements(es, oracle):
    # One 8.6 GB bf16 segment: element offsets inside it pass 2^32, and its
    # global indices cross a 2^34 boundary (index base chosen so).
    n = 2**32 + 8200
    t = torch.empty(n, dtype=torch.bfloat16, device="cuda")
    t.normal_(0.0, 0.02, generator=torch.Generator(device="cuda").manual_seed(3))
    base = 2**34 - 8 * 1000
    plan = es.es_plan_create([es.Segment(t.data_ptr(), n, base)], es.ES_BF16, [t])
    offs = np.unique(np.concatenate([np.arange(0, 64), np.arange(8000 - 64, 8000 + 64),
                                     np.arange(2**32 - 64, 2**32 + 64), np.arange(n - 64, n),
                                     np.random.default_rng(4).integers(0, n, 20000)])).astype(np.int64)
    idx = torch.from_numpy(offs).cuda()
    g = (np.uint64(base) + offs.astype(np.uint64))
    before = t.index_select(0, idx).view(torch.int16).cpu().numpy().view(np.uint16)
    es.es_perturb(plan, 77, 1e-3)
    torch.cuda.synchronize()
    got = t.index_select(0, idx).view(torch.int16).cpu().numpy().view(np.uint16)
    tol = noise_abs_tol([oracle.noise_at(77, g)], [1e-3])
    compare("bf16", got, oracle.perturb(before, g, 77, 1e-3, "bf16"), "2^32+ segment perturb", tol)
    seeds, coeffs = np.array([5, 6], np.uint64), np.array([1e-3, -1e-3], np.float32)
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    after = t.index_select(0, idx).view(torch.int16).cpu().numpy().view(np.uint16)
    tol = noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs)
    compare("bf16", after, oracle.update(got, g, seeds, coeffs, "bf16"), "2^32+ segment update", tol)
    plan.close()
    del t
    torch.cuda.empty_cache()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_special_values(es, oracle, dtype):
    # inf stays inf, NaN stays NaN, signed zeros, subnormals and the largest
    # finite values go through the same rounding as on the oracle.
    fmax = 3.3895313892515355e38 if dtype == "bf16" else float(np.finfo(np.float32).max)
    vals = np.array([np.inf, -np.inf, np.nan, 0.0, -0.0, 1e-40, -1e-40, 1e-45, fmax, -fmax,
                     1.0, -2.0, 3e38, 6e-39] * 16, dtype=np.float32)
    t = torch.from_numpy(vals.copy())
    t = (t.to(torch.bfloat16) if dtype == "bf16" else t).cuda()
    plan, segs = build_plan(es, [t])
    before = host_values(t)
    g = indices(segs)[0]
    es.es_perturb(plan, 9, 0.5)
    torch.cuda.synchronize()
    got = host_values(t)
    want = oracle.perturb(before, g, 9, 0.5, dtype)
    if dtype == "bf16":
        gv = (got.astype(np.uint32) << 16).view(np.float32)
        wv = (want.astype(np.uint32) << 16).view(np.float32)
    else:
        gv, wv = got, want
    nan = np.isnan(wv)
    assert np.array_equal(np.isnan(gv), nan)
    inf = np.isinf(wv)
    assert np.array_equal(gv[inf], wv[inf])
    fin = ~nan & ~inf
    tol = noise_abs_tol([oracle.noise_at(9, g)], [0.5])[fin]
    compare(dtype, got[fin], want[fin], f"special values {dtype}", tol)
    plan.close()


def test_generation_captured_in_a_cuda_graph_replays_bit_identically(es):
    # The device entry points make no host synchronisation and allocate
    # nothing per call, so a generation can be captured once and replayed; the
    # host-side arguments (seeds, coefficients) are fixed at capture.
    a = make_params("bf16", [100003, 8192 + 7], seed=17)
    b = [t.clone() for t in a]
    plan_a, _ = build_plan(es, a)
    plan_b, _ = build_plan(es, b)
    seeds = np.arange(60, 68, dtype=np.uint64)
    coeffs = np.linspace(-1e-3, 1e-3, 8).astype(np.float32)

    def generation(plan, stream=None):
        es.es_perturb(plan, int(seeds[0]), 1e-3, stream)
        for i in range(1, 8):
            es.es_restore_perturb(plan, int(seeds[i - 1]), 1e-3, int(seeds[i]), 1e-3, stream)
        es.es_restore(plan, int(seeds[7]), 1e-3, stream)
        es.es_update(plan, seeds, coeffs, stream)

    for _ in range(3):
        generation(plan_a)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        generation(plan_b, s)
    for _ in range(3):
        g.replay()
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    plan_a.close()
    plan_b.close()


def test_host_buffers_are_refused_before_any_launch(es):
    # Page-locked host tensors: device-accessible through unified addressing,
    # so nothing could fault even if a launch happened; the library must still
    # refuse them (parameters belong in device memory) and leave them untouched.
    host = torch.zeros(4096, dtype=torch.float32).pin_memory()
    bits = torch.zeros(64, dtype=torch.int32).pin_memory()
    seg = [es.Segment(int(host.data_ptr()), host.numel(), 0)]
    for call in (lambda: es.es_plan_create(seg, es.ES_FP32),
                 lambda: es.es_perturb_noalloc(seg, es.ES_FP32, 1, 1e-3),
                 lambda: es.es_noise_fill(1, 0, host.numel(), host),
                 lambda: es.es_noise_bits(1, 0, 16, bits)):
        with pytest.raises(es.EsError) as err:
            call()
        assert err.value.status == es.ES_ERR_INVALID_ARG
        assert "not device memory" in es.es_last_error()
    torch.cuda.synchronize()
    assert not host.any() and not bits.any()
    with pytest.raises(ValueError):
        es.plan_from_tensors([host])


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_zero_sigma_moves_only_the_sign_of_negative_zeros(es, oracle, dtype):
    # theta + 0 * eps: finite non-zero values, infinities and NaN stay as they
    # are; -0 becomes the IEEE sum -0 + (0 * eps), whose sign follows eps, and
    # the oracle takes the same decision in double.
    rng = np.random.default_rng(12)
    vals = np.concatenate([0.02 * rng.standard_normal(8192 + 37), [0.0, -0.0] * 64,
                           [np.inf, -np.inf, np.nan] * 8]).astype(np.float32)
    t = torch.from_numpy(vals.copy())
    t = (t.to(torch.bfloat16) if dtype == "bf16" else t).cuda()
    plan, segs = build_plan(es, [t])
    g = indices(segs)[0]
    for call, oracle_call in ((es.es_perturb, oracle.perturb), (es.es_restore, oracle.restore)):
        before = host_values(t)
        call(plan, 3, 0.0)
        torch.cuda.synchronize()
        got, want = host_values(t), oracle_call(before, g, 3, 0.0, dtype)
        bits = got.view(np.uint16 if dtype == "bf16" else np.uint32)
        wbits = want.view(np.uint16 if dtype == "bf16" else np.uint32)
        if dtype == "bf16":
            nan = np.isnan((want.astype(np.uint32) << 16).view(np.float32))
        else:
            nan = np.isnan(want)
        assert np.array_equal(bits[~nan], wbits[~nan])
        assert np.array_equal(bits[~nan & (vals != 0)], host_bits(before, dtype)[~nan & (vals != 0)])
        assert np.all(np.isnan((bits.astype(np.uint32) << 16).view(np.float32) if dtype == "bf16"
                               else got)[nan])
    plan.close()


def host_bits(v, dtype):
    return v.view(np.uint16 if dtype == "bf16" else np.uint32)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_zero_coefficients_are_skipped_and_repeated_seeds_add(es, oracle, dtype):
    a = make_params(dtype, RAGGED[:6], seed=13)
    b = [x.clone() for x in a]
    plan_a, segs = build_plan(es, a)
    plan_b, _ = build_plan(es, b, [s.index_base for s in segs])
    es.es_update(plan_a, [11, 12, 13, 14], np.array([2e-4, 0.0, -1e-4, 0.0], np.float32))
    es.es_update(plan_b, [11, 13], np.array([2e-4, -1e-4], np.float32))
    torch.cuda.synchronize()
    for x, y in zip(a, b):
        assert torch.equal(_int_view(x), _int_view(y))
    # the same seed twice contributes twice
    before = [host_values(x) for x in a]
    seeds = np.array([21, 21, 22], dtype=np.uint64)
    coeffs = np.array([1e-4, 3e-4, -2e-4], np.float32)
    es.es_update(plan_a, seeds, coeffs)
    torch.cuda.synchronize()
    for x, s, h in zip(a, segs, before):
        g = indices([s])[0]
        tol = noise_abs_tol([oracle.noise_at(int(k), g) for k in seeds], coeffs)
        compare(dtype, host_values(x), oracle.update(h, g, seeds, coeffs, dtype), "repeated seed", tol)
    plan_a.close()
    plan_b.close()


def test_two_plans_on_two_streams_equal_the_sequential_result(es):
    # Launches on two streams with no synchronisation between them (distinct
    # plans over distinct tensors) give bit-identically what the same calls
    # give one after the other on one stream.
    a = make_params("bf16", RAGGED, seed=20)
    b = make_params("bf16", RAGGED[::-1], seed=21)
    a_ref = [t.clone() for t in a]
    b_ref = [t.clone() for t in b]
    plans = [build_plan(es, ts)[0] for ts in (a, b, a_ref, b_ref)]
    seeds = np.arange(40, 48, dtype=np.uint64)
    coeffs = np.linspace(-2e-4, 3e-4, 8).astype(np.float32)

    def generation(plan, stream):
        for s in seeds:
            es.es_perturb(plan, int(s), 1e-3, stream)
            es.es_restore(plan, int(s), 1e-3, stream)
        es.es_update(plan, seeds, coeffs, stream)

    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    torch.cuda.synchronize()
    for _ in range(3):
        generation(plans[0], s1.cuda_stream)
        generation(plans[1], s2.cuda_stream)
    torch.cuda.synchronize()
    for _ in range(3):
        generation(plans[2], None)
        generation(plans[3], None)
    torch.cuda.synchronize()
    for x, y in zip(a + b, a_ref + b_ref):
        assert torch.equal(_int_view(x), _int_view(y))
    for p in plans:
        p.close()


def _near_one_elements(oracle, seed, nblocks, threshold):
    """Elements (ascending) of the Box-Muller pairs whose radius word is at least
    `threshold`, within Philox blocks 0 .. nblocks - 1 of `seed` (the oracle's
    words)."""
    w = oracle.noise_blocks(seed, 0, nblocks)
    b0 = np.nonzero(w[:, 0] >= threshold)[0].astype(np.uint64)
    b2 = np.nonzero(w[:, 2] >= threshold)[0].astype(np.uint64)
    return np.unique(np.concatenate([4 * b0, 4 * b0 + 1, 4 * b2 + 2, 4 * b2 + 3]))


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_near_one_radius_inputs_match_oracle(es, oracle, dtype):
    # Radius inputs within 2^-10 of 1 (raw word >= 0xFFC00000, one pair in
    # 1024) take the series of -2 ln u on a branch of their own in every
    # kernel. From theta = 0 each call's output is its rounded noise term, so
    # these elements are compared with the oracle directly: all near-one pairs
    # of 2^21 blocks per seed, and in particular those within 2^-20 of 1
    # (word >= 0xFFFFF000), where the hardware log2 alone would miss the
    # tolerance several times over.
    nblocks = 1 << 21
    n = 4 * nblocks
    tdt = torch.bfloat16 if dtype == "bf16" else torch.float32
    theta = torch.zeros(n, dtype=tdt, device="cuda")
    plan, segs = build_plan(es, [theta], [0])
    seeds = [3, 2**33 + 9, 77, 2**60 + 1, 12345, 2**40 + 5]
    near = {s: _near_one_elements(oracle, s, nblocks, 0xFFC00000) for s in seeds}
    sharp = sum(_near_one_elements(oracle, s, nblocks, 0xFFFFF000).size for s in seeds)
    assert sharp >= 8 and all(v.size > 6000 for v in near.values())
    zeros = lambda m: np.zeros(m, dtype=np.uint16 if dtype == "bf16" else np.float32)
    sigma = 1e-3

    def gather(sel):
        return host_values(theta[torch.from_numpy(sel.astype(np.int64)).cuda()])

    for k, s in enumerate(seeds):
        sel = near[s]
        eps = oracle.noise_at(s, sel)
        # one-seed pass
        theta.zero_()
        es.es_perturb(plan, s, sigma)
        torch.cuda.synchronize()
        compare(dtype, gather(sel), oracle.perturb(zeros(sel.size), sel, s, sigma, dtype),
                f"es_perturb, seed {s}", noise_abs_tol([eps], [sigma]))
        # two-seed pass: restore of s, perturb of the next seed (its near-one
        # elements too)
        s2 = seeds[(k + 1) % len(seeds)]
        sel2 = np.union1d(sel, near[s2])
        theta.zero_()
        es.es_restore_perturb(plan, s, sigma, s2, sigma)
        torch.cuda.synchronize()
        mid = oracle.restore(zeros(sel2.size), sel2, s, sigma, dtype)
        compare(dtype, gather(sel2), oracle.perturb(mid, sel2, s2, sigma, dtype),
                f"es_restore_perturb, seeds {s}, {s2}",
                noise_abs_tol([oracle.noise_at(s, sel2), oracle.noise_at(s2, sel2)],
                              [sigma, sigma]))
        # update over two seeds, then the fused update + next perturb
        coeffs = np.array([2.5e-4, -1.5e-4], dtype=np.float32)
        theta.zero_()
        es.es_update(plan, np.array([s, s2], dtype=np.uint64), coeffs)
        torch.cuda.synchronize()
        tol = noise_abs_tol([oracle.noise_at(s, sel2), oracle.noise_at(s2, sel2)], coeffs)
        compare(dtype, gather(sel2),
                oracle.update(zeros(sel2.size), sel2, [s, s2], coeffs, dtype),
                f"es_update, seeds {s}, {s2}", tol)
        theta.zero_()
        es.es_update_perturb(plan, np.array([s2], dtype=np.uint64), coeffs[:1], s, sigma)
        torch.cuda.synchronize()
        upd = oracle.update(zeros(sel2.size), sel2, [s2], coeffs[:1], dtype)
        compare(dtype, gather(sel2), oracle.perturb(upd, sel2, s, sigma, dtype),
                f"es_update_perturb, seeds {s2} then {s}",
                noise_abs_tol([oracle.noise_at(s2, sel2), oracle.noise_at(s, sel2)],
                              [coeffs[0], sigma]))
    plan.close()


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_tiles_meeting_a_high_counter_word_boundary(es, oracle, dtype):
    # Inside a tile whose blocks share the high counter word, the kernels take
    # round 0's Philox product of a thread's later blocks from its first one's
    # by 64-bit additions, which is exact only while the low counter word does
    # not wrap. Here three whole tiles end exactly at block 2^32 (their last
    # low word is 2^32 - 1) and three more start there, plus a ragged tail;
    # every call is checked on every element: against the oracle one step at a
    # time, and the fused calls bit for bit against the separate ones.
    tile = 256 * 4 * (8 if dtype == "bf16" else 4)
    n = 6 * tile + 5
    a = make_params(dtype, [n], seed=21)
    b = [t.clone() for t in a]
    base = [2**34 - 3 * tile]
    plan_a, segs = build_plan(es, a, base)
    plan_b, _ = build_plan(es, b, base)
    g = indices(segs)[0]
    iv = torch.int16 if dtype == "bf16" else torch.int32
    s1, s2, sig = 2**40 + 3, 77, 1e-3

    before = host_values(a[0])
    for p in (plan_a, plan_b):
        es.es_perturb(p, s1, sig)
    torch.cuda.synchronize()
    got = host_values(a[0])
    compare(dtype, got, oracle.perturb(before, g, s1, sig, dtype), "perturb",
            noise_abs_tol([oracle.noise_at(s1, g)], [sig]))
    # fused restore + perturb against the two separate calls, each checked
    es.es_restore_perturb(plan_a, s1, sig, s2, sig)
    es.es_restore(plan_b, s1, sig)
    torch.cuda.synchronize()
    mid = host_values(b[0])
    compare(dtype, mid, oracle.restore(got, g, s1, sig, dtype), "restore",
            noise_abs_tol([oracle.noise_at(s1, g)], [sig]))
    es.es_perturb(plan_b, s2, sig)
    torch.cuda.synchronize()
    assert torch.equal(a[0].view(iv), b[0].view(iv))
    compare(dtype, host_values(b[0]), oracle.perturb(mid, g, s2, sig, dtype), "perturb 2",
            noise_abs_tol([oracle.noise_at(s2, g)], [sig]))
    # the antithetic flip against the separate restore and perturb with -sigma
    es.es_restore_perturb(plan_a, s2, sig, s2, -sig)
    es.es_restore(plan_b, s2, sig)
    es.es_perturb(plan_b, s2, -sig)
    torch.cuda.synchronize()
    assert torch.equal(a[0].view(iv), b[0].view(iv))
    # the update (and its fused perturb) on the same tiles
    seeds = np.array([5, 2**33 + 1, 99], dtype=np.uint64)
    coeffs = np.array([1e-3, -2e-3, 5e-4], dtype=np.float32)
    before = host_values(a[0])
    es.es_update_perturb(plan_a, seeds, coeffs, s1, sig)
    es.es_update(plan_b, seeds, coeffs)
    torch.cuda.synchronize()
    upd = host_values(b[0])
    compare(dtype, upd, oracle.update(before, g, seeds, coeffs, dtype), "update",
            noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs))
    es.es_perturb(plan_b, s1, sig)
    torch.cuda.synchronize()
    assert torch.equal(a[0].view(iv), b[0].view(iv))
    plan_a.close()
    plan_b.close()
