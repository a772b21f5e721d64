"""The generator's uniform mapping + Box-Muller transform, checked on the GPU
over its whole input domain: each word enters only through its top 23 bits, so
every radius input and every angle input is evaluated and compared with the
oracle's exact pair. This proves |delta eps| <= 1e-5 * max(1, |eps|) for the
fast hardware-function path for every possible Philox output."""
import numpy as np
import pytest
import torch

from parity import EPS_TOL, assert_eps_close

pytestmark = pytest.mark.gpu

M = 1 << 23                  # distinct 23-bit inputs
R_MAX = np.sqrt(-2.0 * np.log(2.0**-24))


def _run(es, words):
    w = torch.from_numpy(words.view(np.int32).copy()).cuda()
    out = torch.empty(words.size, dtype=torch.float32, device="cuda")
    es.es_box_muller(w, words.size // 2, out)
    torch.cuda.synchronize()
    return out.cpu().numpy().astype(np.float64)


def _pairs(a_words, b_words):
    w = np.empty(2 * a_words.size, dtype=np.uint32)
    w[0::2] = a_words
    w[1::2] = b_words
    return w


def test_every_radius_input(es, oracle):
    m = np.arange(M, dtype=np.uint32)
    rng = np.random.default_rng(0)
    low = rng.integers(0, 512, size=M, dtype=np.uint32)          # ignored low bits
    # angle input next to 1/2: cos(2 pi u_b) = -1 to 1e-13, so eps0 carries the radius
    words = _pairs((m << 9) | low, np.full(M, (1 << 22) << 9, dtype=np.uint32))
    got = _run(es, words)
    want = oracle.box_muller(words)
    assert_eps_close(got, want, "radius sweep")
    radius_err = np.max(np.abs(got[0::2] - want[0::2]))
    assert radius_err < 2e-6, radius_err


def test_every_angle_input(es, oracle):
    m = np.arange(M, dtype=np.uint32)
    for a in (0, 1 << 22, M - 1):     # largest radius, r = 1.18, smallest radius
        words = _pairs(np.full(M, a << 9, dtype=np.uint32), m << 9)
        got = _run(es, words)
        want = oracle.box_muller(words)
        assert_eps_close(got, want, f"angle sweep (radius input {a})")
        if a == 0:
            # angle error scaled by the largest radius, plus the radius error:
            # together with the radius sweep this bounds every (radius, angle) pair
            angle_err = np.max(np.abs(got - want))
            assert angle_err + 2e-6 <= EPS_TOL, angle_err


def test_random_pairs(es, oracle):
    rng = np.random.default_rng(1)
    words = rng.integers(0, 2**32, size=1 << 23, dtype=np.uint64).astype(np.uint32)
    got = _run(es, words)
    assert_eps_close(got, oracle.box_muller(words), "random pairs")
    assert np.max(np.abs(got)) <= R_MAX * (1 + 1e-6)


def test_box_muller_argument_errors(es):
    buf = torch.empty(16, dtype=torch.int32, device="cuda")
    out = torch.empty(16, dtype=torch.float32, device="cuda")
    with pytest.raises(es.EsError) as ei:
        es.es_box_muller(buf.data_ptr() + 4, 2, out)
    assert ei.value.status == es.ES_ERR_ALIGNMENT
    with pytest.raises(es.EsError) as ei:
        es.es_box_muller(0, 2, out)
    assert ei.value.status == es.ES_ERR_INVALID_ARG
