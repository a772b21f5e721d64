"""GPU parity of the noise generator through the C ABI: raw Philox words
bit-exact, Gaussians within 1e-5 * max(1, |eps|) of the oracle, including
ragged ranges, unaligned bases and 64-bit index ranges."""
import numpy as np
import pytest
import torch

from parity import assert_eps_close

pytestmark = pytest.mark.gpu


def _bits(es, seed, block_base, nblocks):
    out = torch.empty(4 * nblocks, dtype=torch.int32, device="cuda")
    es.es_noise_bits(seed, block_base, nblocks, out)
    torch.cuda.synchronize()
    return out.cpu().numpy().view(np.uint32).reshape(nblocks, 4)


def _fill(es, seed, base, n):
    out = torch.full((max(n, 1) + 8,), float("nan"), dtype=torch.float32, device="cuda")
    es.es_noise_fill(seed, base, n, out)
    torch.cuda.synchronize()
    host = out.cpu().numpy()
    assert np.all(np.isnan(host[n:])), "noise_fill wrote past the end of its range"
    return host[:n]


@pytest.mark.parametrize("seed,block_base,nblocks", [
    (0, 0, 1), (1, 0, 4096), (12345, 2**32 - 3, 7), (2**64 - 1, 2**62 - 9, 9),
    (7, 123456789, 1000), (2**63 + 11, 2**40, 333)])
def test_philox_words_bit_exact(es, oracle, seed, block_base, nblocks):
    got = _bits(es, seed, block_base, nblocks)
    want = np.array([oracle.noise_block(seed, block_base + t) for t in range(nblocks)],
                    dtype=np.uint32)
    assert np.array_equal(got, want)


def test_noise_fill_small_ragged_ranges(es, oracle):
    for base in (0, 1, 2, 3, 5, 8, 4 * 2**32 - 3, 2**64 - 40):
        for n in list(range(1, 34)):
            got = _fill(es, 99, base, n)
            assert_eps_close(got, oracle.noise_fill(99, base, n), f"base={base} n={n}")


def test_noise_fill_large_range_spans_many_ctas(es, oracle):
    n = 1_000_003
    got = _fill(es, 2026, 17, n)
    assert_eps_close(got, oracle.noise_fill(2026, 17, n), "n=1e6+3")


def test_noise_fill_zero_length_is_a_no_op(es):
    out = torch.full((8,), 3.0, device="cuda")
    es.es_noise_fill(1, 0, 0, out)
    torch.cuda.synchronize()
    assert torch.all(out == 3.0)


def test_noise_entry_point_argument_errors(es):
    buf = torch.empty(64, dtype=torch.float32, device="cuda")
    with pytest.raises(es.EsError) as ei:
        es.es_noise_fill(1, 0, 4, buf.data_ptr() + 2)       # not 4-byte aligned
    assert ei.value.status == es.ES_ERR_ALIGNMENT
    with pytest.raises(es.EsError) as ei:
        es.es_noise_bits(1, 0, 2, buf.data_ptr() + 4)       # not 16-byte aligned
    assert ei.value.status == es.ES_ERR_ALIGNMENT
    with pytest.raises(es.EsError) as ei:
        es.es_noise_fill(1, 2**64 - 2, 4, buf)               # index range past 2^64
    assert ei.value.status == es.ES_ERR_INVALID_ARG
    with pytest.raises(es.EsError) as ei:
        es.es_noise_fill(1, 0, 4, 0)                         # NULL
    assert ei.value.status == es.ES_ERR_INVALID_ARG


def test_noise_is_bit_identical_across_calls_and_streams(es):
    a = torch.empty(1 << 20, device="cuda")
    b = torch.empty(1 << 20, device="cuda")
    es.es_noise_fill(5, 64, a.numel(), a)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        es.es_noise_fill(5, 64, b.numel(), b, stream=s)
    torch.cuda.synchronize()
    assert torch.equal(a.view(torch.int32), b.view(torch.int32))


def test_noise_fill_aligned_path_equals_box_muller_of_the_words(es):
    # With an aligned output and index base, whole Philox blocks take the
    # 16-byte store path (packed transform); they must equal, bit for bit,
    # es_box_muller (scalar transform) applied to the same es_noise_bits words.
    # Ranges: plain, crossing the 2^32-block boundary, far out, ragged tails.
    seed = 424242
    for block_base, nb, extra in ((0, 4096 + 3, 0), (2**32 - 700, 1500, 3), (2**40 + 12, 999, 2)):
        words = torch.empty(4 * nb, dtype=torch.int32, device="cuda")
        es.es_noise_bits(seed, block_base, nb, words)
        bm = torch.empty(4 * nb, dtype=torch.float32, device="cuda")
        es.es_box_muller(words, 2 * nb, bm)
        torch.cuda.synchronize()
        got = _fill(es, seed, 4 * block_base, 4 * nb + extra)
        assert np.array_equal(got[:4 * nb].view(np.uint32), bm.cpu().numpy().view(np.uint32))


def test_noise_fill_large_aligned_range_matches_oracle(es, oracle):
    # 1,000,002 Gaussians from g = 2^34 - 16384: the aligned path across the
    # j = 2^32 block boundary, then a 2-element tail.
    base, n = 2**34 - 16384, 1_000_002
    got = _fill(es, 77, base, n)
    assert_eps_close(got, oracle.noise_fill(77, base, n), "aligned n=1e6+2")
