"""es_perturb_noalloc: the perturb/restore pass for callers that cannot
allocate device memory (a process whose device memory belongs to its own pool
allocator, or a loop that must not call into the allocator). It must give the
same parameters as the plan-based es_perturb / es_restore, call after call.

Kept in a file that is collected last, so a run that stops at the first
failure has run every other test before this one.
"""
import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

NUMELS = [7, 2560, 8193, 20000, 100003]


def _params(dtype, seed):
    rng = np.random.default_rng(seed)
    out = []
    for n in NUMELS:
        v = torch.from_numpy((0.02 * rng.standard_normal(n)).astype(np.float32))
        out.append((v.to(torch.bfloat16) if dtype == "bf16" else v).cuda())
    return out


def _bits(t):
    return t.view(torch.int16) if t.dtype == torch.bfloat16 else t.view(torch.int32)


@pytest.mark.parametrize("dtype", ["bf16", "f32"])
def test_noalloc_matches_plan_entry_points_on_two_calls_in_a_row(es, dtype):
    # Both paths run the same kernel on the same segments, so the parameters
    # must agree bit for bit after every call.
    a = _params(dtype, 11)
    b = [t.clone() for t in a]
    plan = es.plan_from_tensors(a)
    bases = [s.index_base for s in es.segments_from_tensors(a)]
    segs_b = es.segments_from_tensors(b, bases)
    code = es.ES_BF16 if dtype == "bf16" else es.ES_FP32
    seed, sigma = 2**33 + 5, 1e-3
    # call 1: perturb; call 2: restore (-sigma) of the same seed
    for k, (plan_call, scale) in enumerate([(es.es_perturb, sigma), (es.es_restore, -sigma)]):
        plan_call(plan, seed, sigma)
        es.es_perturb_noalloc(segs_b, code, seed, scale)
        torch.cuda.synchronize()
        for j, (x, y) in enumerate(zip(a, b)):
            assert torch.equal(_bits(x), _bits(y)), f"call {k + 1} segment {j}"
    plan.close()


def test_noalloc_allocates_no_device_memory(es):
    # The reason the entry point exists: after the first call on the device,
    # calls (including one that fills the whole static table) leave the device's
    # free memory and torch's reserved pool exactly as they were.
    a = _params("bf16", 5)
    segs = es.segments_from_tensors(a)
    n = es.ES_STATIC_MAX_SEGMENTS
    flat = torch.zeros(8 * n, dtype=torch.bfloat16, device="cuda")
    full = es.segments_from_tensors([flat[8 * k:8 * k + 8] for k in range(n)])
    es.es_perturb_noalloc(segs, es.ES_BF16, 3, 1e-3)
    es.es_perturb_noalloc(full, es.ES_BF16, 3, 1e-3)
    torch.cuda.synchronize()
    free0, reserved0 = torch.cuda.mem_get_info()[0], torch.cuda.memory_reserved()
    for k in range(40):
        es.es_perturb_noalloc(segs, es.ES_BF16, 100 + k, 1e-3)
        es.es_perturb_noalloc(full, es.ES_BF16, 100 + k, -1e-3)
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] == free0
    assert torch.cuda.memory_reserved() == reserved0


def test_noalloc_refuses_a_capturing_stream(es):
    # The segment table is copied from the call's stack; a graph could not
    # replay that copy. A call on a capturing stream is refused before anything
    # is copied or launched, so the capture stays valid and records nothing.
    a = _params("bf16", 7)
    before = [t.clone() for t in a]
    segs = es.segments_from_tensors(a)
    side = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    counter = torch.zeros(1, device="cuda")
    refused = None
    with torch.cuda.graph(graph, stream=side):
        counter.add_(1)
        try:
            es.es_perturb_noalloc(segs, es.ES_BF16, 9, 1e-3, side.cuda_stream)
        except es.EsError as e:
            refused = e
    assert refused is not None and refused.status == es.ES_ERR_INVALID_ARG
    assert "captur" in str(refused)
    graph.replay()
    torch.cuda.synchronize()
    assert counter.item() == 1.0
    for x, y in zip(a, before):
        assert torch.equal(_bits(x), _bits(y))


def test_noalloc_rejects_more_segments_than_its_static_table(es):
    # Rejected before any device work: the pointers are never dereferenced.
    n = es.ES_STATIC_MAX_SEGMENTS + 1
    segs = [es.Segment(0x100000 + 16 * k, 1, 8 * k) for k in range(n)]
    with pytest.raises(es.EsError) as ei:
        es.es_perturb_noalloc(segs, es.ES_BF16, 1, 1e-3)
    assert ei.value.status == es.ES_ERR_INVALID_ARG
    assert "ES_STATIC_MAX_SEGMENTS" in str(ei.value)


def test_noalloc_at_its_segment_limit_matches_the_plan(es):
    # Exactly ES_STATIC_MAX_SEGMENTS ragged segments (1 .. 600 elements, 16-byte
    # aligned views of one buffer): the whole static table is in use.
    n = es.ES_STATIC_MAX_SEGMENTS
    rng = np.random.default_rng(31)
    sizes = rng.integers(1, 601, size=n)
    offs = np.concatenate([[0], np.cumsum((sizes + 7) // 8 * 8)])
    flat = torch.from_numpy((0.02 * rng.standard_normal(int(offs[-1]))).astype(np.float32))
    flat = flat.to(torch.bfloat16).cuda()
    twin = flat.clone()
    a = [flat[int(o):int(o) + int(m)] for o, m in zip(offs[:-1], sizes)]
    b = [twin[int(o):int(o) + int(m)] for o, m in zip(offs[:-1], sizes)]
    plan = es.plan_from_tensors(a)
    segs_b = es.segments_from_tensors(b, [s.index_base for s in es.segments_from_tensors(a)])
    for seed, sigma in ((2**40 + 3, 1e-3), (2**40 + 3, -1e-3), (77, 5e-4)):
        es.es_perturb(plan, seed, sigma)
        es.es_perturb_noalloc(segs_b, es.ES_BF16, seed, sigma)
        torch.cuda.synchronize()
        assert torch.equal(flat.view(torch.int16), twin.view(torch.int16))
    plan.close()
