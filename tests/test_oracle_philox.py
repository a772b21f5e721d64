"""Pins for the oracle's counter-based generator (Philox4x32-10, SC'11).

The oracle's Philox is checked bit for bit against PyTorch's host Philox engine
(``ATen/core/PhiloxRNGEngine.h``), an independent implementation of the same
published algorithm: engine(seed, subsequence, offset) uses
key = (seed_lo, seed_hi) and counter = (offset_lo, offset_hi, subseq_lo,
subseq_hi), so the oracle's noise block j of a seed is the engine's block at
subsequence 0, offset j.
"""
import os
import shutil
import subprocess

import numpy as np
import pytest

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def torch_engine(tmp_path_factory):
    gxx = shutil.which("g++")
    if gxx is None:
        pytest.skip("g++ not available")
    try:
        import torch.utils.cpp_extension as ce
        incs = ce.include_paths()
    except Exception as exc:  # pragma: no cover - depends on the image
        pytest.skip(f"torch headers unavailable: {exc}")
    exe = str(tmp_path_factory.mktemp("philox") / "pdump")
    cmd = [gxx, "-O1", "-std=c++17"] + [f"-I{p}" for p in incs] + [
        os.path.join(HERE, "philox_torch_engine_dump.cpp"), "-o", exe]
    subprocess.run(cmd, check=True, capture_output=True)

    def run(triples):
        text = "".join(f"{s} {q} {o}\n" for s, q, o in triples)
        out = subprocess.run([exe], input=text, capture_output=True, text=True, check=True)
        return np.array([[int(w) for w in line.split()] for line in out.stdout.splitlines()],
                        dtype=np.uint64).astype(np.uint32)
    return run


def _cases():
    rng = np.random.default_rng(20260817)
    cases = [(0, 0, 0), (1, 0, 0), (0, 0, 1), (2**64 - 1, 0, 0), (0, 0, 2**32 - 1),
             (0, 0, 2**32), (0, 0, 2**32 + 1), (12345, 0, 2**62), (2**32, 0, 7),
             (2**32 - 1, 0, 2**33 + 5)]
    for _ in range(300):
        seed = int(rng.integers(0, 2**63)) * 2 + int(rng.integers(0, 2))
        off = int(rng.integers(0, 2**40))
        cases.append((seed, 0, off))
    return cases


def test_noise_block_matches_torch_engine(oracle, torch_engine):
    cases = _cases()
    ref = torch_engine(cases)
    got = np.array([oracle.noise_block(s, o) for s, _, o in cases], dtype=np.uint32)
    assert np.array_equal(got, ref)


def test_raw_block_all_counter_words_match_torch_engine(oracle, torch_engine):
    # Non-zero upper counter words exercise the x2/x3 lanes of every round.
    rng = np.random.default_rng(7)
    cases = []
    for _ in range(200):
        cases.append((int(rng.integers(0, 2**63)), int(rng.integers(0, 2**63)),
                      int(rng.integers(0, 2**63))))
    ref = torch_engine(cases)
    for (seed, sub, off), want in zip(cases, ref):
        ctr = [off & 0xFFFFFFFF, off >> 32, sub & 0xFFFFFFFF, sub >> 32]
        key = [seed & 0xFFFFFFFF, seed >> 32]
        assert np.array_equal(oracle.philox4x32_10(ctr, key), want)


def test_uniform_mapping_closed_form(oracle):
    # u = (2 m + 1) / 2^24 with m = x >> 9: open interval, low 9 bits ignored.
    assert oracle.uniform(0) == 2.0**-24
    assert oracle.uniform(0x1FF) == 2.0**-24
    assert oracle.uniform(0x200) == 3 * 2.0**-24
    assert oracle.uniform(0xFFFFFFFF) == 1.0 - 2.0**-24
    assert oracle.uniform(0x80000000) == 0.5 + 2.0**-24
    # symmetric about 1/2: u(m) + u(2^23 - 1 - m) == 1
    for m in (0, 1, 12345, 2**22, 2**23 - 1):
        assert oracle.uniform(m << 9) + oracle.uniform((2**23 - 1 - m) << 9) == 1.0


def test_philox_output_bits_are_uniform(oracle):
    # Every output bit of a block is a fair coin (binomial, 6-sigma band) and the
    # four words are distinct streams.
    n = 20000
    words = np.array([oracle.noise_block(99, j) for j in range(n)], dtype=np.uint32)
    bits = ((words[:, :, None] >> np.arange(32, dtype=np.uint32)) & 1).astype(np.int64)
    ones = bits.sum(axis=0)
    assert np.all(np.abs(ones - n / 2) < 6 * np.sqrt(n) / 2)
    assert len(np.unique(words.ravel())) > 4 * n - 10


def test_noise_blocks_is_noise_block_over_a_range(oracle):
    # the bulk form (used to find inputs with given raw words) gives each
    # block's words, across the 2^32-block boundary of the counter's low word
    for seed, j0 in ((5, 0), (2**40 + 3, 2**32 - 3)):
        w = oracle.noise_blocks(seed, j0, 7)
        for k in range(7):
            assert np.array_equal(w[k], oracle.noise_block(seed, j0 + k))
