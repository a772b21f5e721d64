"""GPU parity on the workloads, through the C ABI, against the oracle.

  toy        1,048,576 fp32, N = 8: every element of every call, and the whole
             generation run free on both sides
  quadratic  65,536 fp32, 32 antithetic pairs, 200 generations with cosine sigma
             0.05 -> 0.005: every generation's update checked step by step on
             sampled coordinates, rewards checked against the oracle's own f
  qwen4b     4,022,458,880 bf16 parameters in 326 tensors, N = 16
  qwen27b    22,695,777,280 bf16 parameters in 579 tensors, N = 30
  sweep      the 4B set with N in {1, 2, 4, 8, 16, 32, 64, 128}
At full size the oracle checks, for every call, the first and last 64 elements
of every tensor plus about 10^6 random elements, in the launch configuration
the benchmark times.
"""
import gc

import numpy as np
import pytest
import torch

from paper_2608_17310_gb300 import inputs as I
from parity import assert_bf16_within_ulp, assert_f32_close, noise_abs_tol

pytestmark = pytest.mark.gpu


def _bits16(t):
    return t.view(torch.int16).cpu().numpy().view(np.uint16)


class Sampled:
    """Fixed sample of elements of a parameter set, gathered on the device."""

    def __init__(self, tensors, segs, n_random, seed):
        self.tensors = tensors
        offs = [I.sample_offsets(t.numel(), n_random, seed + k) for k, t in enumerate(tensors)]
        self.dev_offs = [torch.from_numpy(o).cuda() for o in offs]
        self.g = np.concatenate([np.uint64(s.index_base) + o.astype(np.uint64)
                                 for s, o in zip(segs, offs)])

    def gather(self):
        parts = [t.index_select(0, o) for t, o in zip(self.tensors, self.dev_offs)]
        flat = torch.cat(parts)
        return _bits16(flat) if flat.dtype == torch.bfloat16 else flat.cpu().numpy()


def _release():
    gc.collect()
    torch.cuda.empty_cache()


# ---------------------------------------------------------------------------------------------
# toy
# ---------------------------------------------------------------------------------------------

@pytest.mark.parametrize("mode", [0, 1])
def test_toy_generation(es, oracle, mode):
    wl = I.WORKLOADS["toy"]
    theta0 = I.toy_theta()
    t = torch.from_numpy(theta0.copy()).cuda()
    plan = es.plan_from_tensors([t])
    g = np.arange(theta0.size, dtype=np.uint64)
    seeds = np.arange(1, wl.population + 1, dtype=np.uint64)
    sigma = float(np.float32(wl.sigma))
    eps = [oracle.noise_at(int(s), g) for s in seeds]
    state = theta0.copy()
    for i, s in enumerate(seeds):
        es.es_perturb(plan, int(s), sigma)
        torch.cuda.synchronize()
        p = t.cpu().numpy()
        tol = noise_abs_tol([eps[i]], [sigma])
        assert_f32_close(p, oracle.perturb(state, g, int(s), sigma), f"toy perturb {i}", tol)
        es.es_restore(plan, int(s), sigma)
        torch.cuda.synchronize()
        state = t.cpu().numpy()
        assert_f32_close(state, oracle.restore(p, g, int(s), sigma), f"toy restore {i}", tol)
    rewards = I.rewards("uniform", wl.population, seed=1)
    rhat = es.es_normalize_rewards(rewards)
    coeffs = es.es_update_coeffs(rhat, wl.alpha, sigma, mode)
    assert np.array_equal(coeffs, oracle.update_coeffs(oracle.zscore(rewards), wl.alpha, sigma, mode))
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    got = t.cpu().numpy()
    tol_u = noise_abs_tol(eps, coeffs)
    assert_f32_close(got, oracle.update(state, g, seeds, coeffs), "toy update", tol_u)
    # the whole generation run free on the oracle from theta_0
    free = theta0.copy()
    for s in seeds:
        free = oracle.restore(oracle.perturb(free, g, int(s), sigma), g, int(s), sigma)
    free = oracle.update(free, g, seeds, coeffs)
    drift = 2 * np.spacing(np.abs(theta0)).astype(np.float64) * wl.population
    assert_f32_close(got, free, "toy free-running", tol_u + drift)
    plan.close()


# ---------------------------------------------------------------------------------------------
# quadratic sanity loop
# ---------------------------------------------------------------------------------------------

def _quadratic_run(es, oracle, mode, generations, check_every=1):
    wl = I.WORKLOADS["quadratic"]
    theta0, star = I.quadratic_problem()
    d = theta0.size
    t = torch.from_numpy(theta0.copy()).cuda()
    star_d = torch.from_numpy(star).cuda().double()
    plan = es.plan_from_tensors([t])
    g_all = np.arange(d, dtype=np.uint64)
    rng = np.random.default_rng(5)
    sample = np.unique(np.concatenate([np.arange(64), np.arange(d - 64, d),
                                       rng.integers(0, d, 1024)])).astype(np.int64)
    g = g_all[sample]
    npairs, T = wl.population, 200

    def f():
        return -float((t.double() - star_d).pow(2).sum().item())

    losses = [-f()]
    for gen in range(generations):
        sigma = float(np.float32(es.es_sigma_cosine(0.05, 0.005, gen, T)))
        seeds = I.population_seeds(npairs, generation=gen, first=1000)
        r_pos, r_neg = np.empty(npairs), np.empty(npairs)
        check = gen % check_every == 0
        for i, s in enumerate(seeds):
            for sign, out in ((1.0, r_pos), (-1.0, r_neg)):
                es.es_perturb(plan, int(s), sign * sigma)
                out[i] = f()
                if check and i == 0 and gen in (0, generations - 1):
                    # the reward computed on the GPU matches the oracle's own f
                    want = oracle.quadratic_reward(t.cpu().numpy(), star)
                    assert abs(out[i] - want) <= 1e-6 * abs(want)
                es.es_restore(plan, int(s), sign * sigma)
        rhat = es.es_normalize_rewards(np.concatenate([r_pos, r_neg]))
        coeffs = es.es_fold_antithetic(rhat[:npairs], rhat[npairs:], wl.alpha, sigma, mode)
        if check:
            before = t.cpu().numpy()[sample]
            o_rhat = oracle.zscore(np.concatenate([r_pos, r_neg]))
            o_coeffs = oracle.fold_antithetic(o_rhat[:npairs], o_rhat[npairs:], wl.alpha, sigma, mode)
            assert np.array_equal(coeffs, o_coeffs)
        es.es_update(plan, seeds, coeffs)
        if check:
            torch.cuda.synchronize()
            after = t.cpu().numpy()[sample]
            tol = noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs)
            assert_f32_close(after, oracle.update(before, g, seeds, coeffs), f"gen {gen}", tol)
        losses.append(-f())
    plan.close()
    return np.array(losses)


def test_quadratic_loop_paper_scale(es, oracle):
    losses = _quadratic_run(es, oracle, 0, 200, check_every=1)
    # the paper-scale update lowers ||theta - theta*||^2 over the run
    assert losses[-1] < losses[0] * 0.995
    assert losses[100] < losses[0]


def test_quadratic_loop_canonical_scale(es, oracle):
    # canonical alpha/(G sigma): parity for the first 40 generations
    losses = _quadratic_run(es, oracle, 1, 40, check_every=1)
    assert np.all(np.isfinite(losses))


# ---------------------------------------------------------------------------------------------
# LLM-shaped sets at full size
# ---------------------------------------------------------------------------------------------

def _llm_generation(es, oracle, workload, n_random, check_members, reward_kind=None):
    wl = I.WORKLOADS[workload]
    specs = I.shapes_for(workload)
    params = I.init_params_torch(specs, torch.bfloat16, "cuda", seed=0)
    segs = es.segments_from_tensors(params)
    plan = es.plan_from_tensors(params, [s.index_base for s in segs])
    smp = Sampled(params, segs, n_random, seed=17)
    n = wl.population
    sigma = float(np.float32(wl.sigma))
    seeds = I.population_seeds(n, generation=0)
    for i, s in enumerate(seeds):
        check = i in check_members
        if check:
            before = smp.gather()
        es.es_perturb(plan, int(s), sigma)
        if check:
            torch.cuda.synchronize()
            pert = smp.gather()
            tol = noise_abs_tol([oracle.noise_at(int(s), smp.g)], [sigma])
            assert_bf16_within_ulp(pert, oracle.perturb(before, smp.g, int(s), sigma, "bf16"),
                                   f"{workload} perturb {i}", abs_tol=tol)
        es.es_restore(plan, int(s), sigma)
        if check:
            torch.cuda.synchronize()
            assert_bf16_within_ulp(smp.gather(), oracle.restore(pert, smp.g, int(s), sigma, "bf16"),
                                   f"{workload} restore {i}", abs_tol=tol)
    rewards = I.rewards(reward_kind or wl.rewards, n, seed=3)
    coeffs = es.es_update_coeffs(es.es_normalize_rewards(rewards), wl.alpha, sigma, es.ES_SCALE_PAPER)
    before = smp.gather()
    es.es_update(plan, seeds, coeffs)
    torch.cuda.synchronize()
    tol = noise_abs_tol([oracle.noise_at(int(s), smp.g) for s in seeds], coeffs)
    assert_bf16_within_ulp(smp.gather(), oracle.update(before, smp.g, seeds, coeffs, "bf16"),
                           f"{workload} update", abs_tol=tol)
    plan.close()
    del params, smp, plan, segs
    _release()


def test_qwen4b_generation_full_size(es, oracle):
    # 326 tensors x (3000 random + 128 edge) elements: about 10^6 sampled indices
    _llm_generation(es, oracle, "qwen4b", n_random=3000, check_members=set(range(16)))


def test_qwen27b_generation_full_size(es, oracle):
    # 579 tensors x (1700 random + 128 edge) elements: about 10^6 sampled indices
    _llm_generation(es, oracle, "qwen27b", n_random=1700, check_members={0, 1, 14, 29})


def test_population_sweep_on_qwen4b(es, oracle):
    specs = I.qwen4b_shapes()
    params = I.init_params_torch(specs, torch.bfloat16, "cuda", seed=0)
    segs = es.segments_from_tensors(params)
    plan = es.plan_from_tensors(params, [s.index_base for s in segs])
    smp = Sampled(params, segs, 60, seed=23)
    for n in (1, 2, 4, 8, 16, 32, 64, 128):
        seeds = I.population_seeds(n, generation=n, first=7)
        rhat = I.rewards("normal", n, seed=n)      # N(0, 1) rewards used directly as Rhat
        coeffs = es.es_update_coeffs(rhat, 5e-4, 1e-3, es.ES_SCALE_PAPER)
        before = smp.gather()
        es.es_update(plan, seeds, coeffs)
        torch.cuda.synchronize()
        tol = noise_abs_tol([oracle.noise_at(int(s), smp.g) for s in seeds], coeffs)
        assert_bf16_within_ulp(smp.gather(), oracle.update(before, smp.g, seeds, coeffs, "bf16"),
                               f"sweep N={n}", abs_tol=tol)
    plan.close()
    del params, smp, plan, segs
    _release()


def test_all_equal_rewards_leave_the_4b_set_bit_identical(es):
    # Bernoulli rewards that all come out equal (p ~ 0.3% at N = 16): no update.
    params = I.init_params_torch(I.qwen4b_shapes()[:20], torch.bfloat16, "cuda", seed=1)
    ref = [p.clone() for p in params]
    plan = es.plan_from_tensors(params)
    rhat = es.es_normalize_rewards(np.zeros(16))
    coeffs = es.es_update_coeffs(rhat, 5e-4, 1e-3, es.ES_SCALE_PAPER)
    es.es_update(plan, I.population_seeds(16), coeffs)
    torch.cuda.synchronize()
    assert all(torch.equal(a.view(torch.int16), b.view(torch.int16)) for a, b in zip(params, ref))
    plan.close()
    del params, ref, plan
    _release()


def test_bench_step_on_the_27b_set_equals_the_oracle_checked_separate_calls(es, oracle):
    # The benchmarked generation exactly as bench.py times it: its flat
    # single-allocation layout, its plan and its fused loop (bench.start_loop,
    # then bench.run_step: es_restore_perturb x 29, es_restore,
    # es_update_perturb). A twin copy of the set runs the same generation as
    # separate calls, each checked against the oracle on sampled elements from
    # the state before it; at the end all 22.7e9 parameters of the two copies
    # must be bit-identical.
    import bench
    wl = I.WORKLOADS["qwen27b"]
    specs = I.shapes_for("qwen27b")
    n = wl.population
    flat, params = I.init_params_flat(specs, torch.bfloat16, "cuda", seed=0)
    twin_flat = flat.clone()
    offs = I.flat_offsets(specs)
    twin = [twin_flat[o:o + s.numel] for s, o in zip(specs, offs)]
    plan = es.plan_from_tensors(params)
    segs = es.segments_from_tensors(twin)
    twin_plan = es.plan_from_tensors(twin, [s.index_base for s in segs])
    smp = Sampled(twin, segs, 30, seed=41)
    stream = torch.cuda.current_stream().cuda_stream

    def sigma_at(t):
        return float(np.float32(es.es_sigma_cosine(wl.sigma, bench.SIGMA_FINAL["qwen27b"], t,
                                                  bench.SCHEDULE_T)))

    sigma, sigma_next = sigma_at(0), sigma_at(1)
    bench.start_loop(es, plan, wl, 0, n, sigma, stream, True)
    launches = bench.run_step(es, plan, wl, 0, n, sigma, sigma_next, stream, None, True)
    assert launches == n + 1

    seeds, rewards = bench.generation_inputs(wl, 0, n)
    coeffs = es.es_update_coeffs(es.es_normalize_rewards(rewards, 1e-8), wl.alpha, sigma,
                                 es.ES_SCALE_PAPER)
    next_seed = int(bench.generation_inputs(wl, 1, n)[0][0])

    def checked(call, oracle_call, seed_list, coeff_list, what):
        before = smp.gather()
        call()
        torch.cuda.synchronize()
        want = oracle_call(before)
        tol = noise_abs_tol([oracle.noise_at(int(s), smp.g) for s in seed_list], coeff_list)
        assert_bf16_within_ulp(smp.gather(), want, what, abs_tol=tol)

    for i, s in enumerate(seeds):
        s = int(s)
        checked(lambda: es.es_perturb(twin_plan, s, sigma),
                lambda b: oracle.perturb(b, smp.g, s, sigma, "bf16"), [s], [sigma], f"perturb {i}")
        checked(lambda: es.es_restore(twin_plan, s, sigma),
                lambda b: oracle.restore(b, smp.g, s, sigma, "bf16"), [s], [sigma], f"restore {i}")
    checked(lambda: es.es_update(twin_plan, seeds, coeffs),
            lambda b: oracle.update(b, smp.g, seeds, coeffs, "bf16"), seeds, coeffs, "update")
    checked(lambda: es.es_perturb(twin_plan, next_seed, sigma_next),
            lambda b: oracle.perturb(b, smp.g, next_seed, sigma_next, "bf16"), [next_seed],
            [sigma_next], "next perturb")
    assert torch.equal(flat.view(torch.int16), twin_flat.view(torch.int16))
    plan.close()
    twin_plan.close()
    del flat, twin_flat, params, twin, smp, plan, twin_plan
    _release()
