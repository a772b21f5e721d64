"""The e2e leg of bench.py computes exactly the generation it times: its
grouped schedule (copy in, the first passes group by group, middle passes on
the whole plan, last pass per group plan, copy out, and with pipelining the
next step's copy in right after each group's copy out) leaves, after three
generations, the host buffer and the device buffer bit-identical to the
whole-plan loop that the device-timed leg runs."""
import numpy as np
import pytest
import torch

from paper_2608_17310_gb300 import inputs as I

pytestmark = pytest.mark.gpu


@pytest.mark.parametrize("fused,population,pipelined",
                         [(True, None, True), (True, None, False), (False, None, True),
                          (True, 1, True)])
def test_e2e_leg_equals_the_device_loop(es, fused, population, pipelined):
    import bench
    name = "qwen4b_4layer"
    wl = I.WORKLOADS[name]
    specs = I.shapes_for(name)
    n = population or wl.population
    flat, params = I.init_params_flat(specs, torch.bfloat16, "cuda", seed=0)
    twin_flat = flat.clone()
    offs = I.flat_offsets(specs)
    twin = [twin_flat[o:o + s.numel] for s, o in zip(specs, offs)]
    plan = es.plan_from_tensors(params)
    twin_plan = es.plan_from_tensors(twin)
    sh = torch.cuda.current_stream().cuda_stream

    def sigma_at(t):
        return float(np.float32(es.es_sigma_cosine(wl.sigma, bench.SIGMA_FINAL[name], t,
                                                  bench.SCHEDULE_T)))

    bench.start_loop(es, plan, wl, 0, n, sigma_at(0), sh, fused)
    bench.start_loop(es, twin_plan, wl, 0, n, sigma_at(0), sh, fused)
    loop = bench.E2ELoop(torch, es, plan, flat, params, wl, n, 2, sigma_at, sh, fused)
    for t in range(3):
        # pipelined: each step issues the next step's copies to the device
        loop.step(t, copy_next=pipelined and t < 2)
        bench.run_step(es, twin_plan, wl, t, n, sigma_at(t), sigma_at(t + 1), sh, None, fused)
    torch.cuda.synchronize()
    want = twin_flat.view(torch.int16)
    assert torch.equal(flat.view(torch.int16), want)
    assert torch.equal(loop.host.view(torch.int16), want.cpu())
    loop.close()
    plan.close()
    twin_plan.close()
