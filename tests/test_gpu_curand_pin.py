"""A second independent pin of the generator, on the GPU: cuRAND's device
Philox4_32_10 (curand_init(seed, subsequence, 4 j) then curand4) gives block j
at counter (j_lo, j_hi, subsequence_lo, subsequence_hi) under key
(seed_lo, seed_hi). Both the oracle's words and the library's es_noise_bits
must equal it bit for bit."""
import os
import shutil
import subprocess

import numpy as np
import pytest
import torch

pytestmark = pytest.mark.gpu

HERE = os.path.dirname(os.path.abspath(__file__))


@pytest.fixture(scope="module")
def curand_dump(tmp_path_factory):
    nvcc = shutil.which("nvcc") or "/usr/local/cuda/bin/nvcc"
    if not os.path.exists(nvcc):
        pytest.skip("nvcc not available")
    exe = str(tmp_path_factory.mktemp("curand") / "cdump")
    subprocess.run([nvcc, "-gencode", "arch=compute_103a,code=sm_103a", "-O2",
                    os.path.join(HERE, "curand_philox_dump.cu"), "-o", exe],
                   check=True, capture_output=True)

    def run(triples):
        text = "".join(f"{s} {q} {b}\n" for s, q, b in triples)
        out = subprocess.run([exe], input=text, capture_output=True, text=True, check=True)
        return np.array([[int(w) for w in line.split()] for line in out.stdout.splitlines()],
                        dtype=np.uint64).astype(np.uint32)
    return run


def _cases():
    rng = np.random.default_rng(31)
    cases = [(0, 0, 0), (1, 0, 0), (2**64 - 1, 0, 0), (0, 0, 2**32 - 1), (0, 0, 2**32),
             (7, 0, 2**34 - 1), (7, 0, 2**34), (2**32, 0, 5), (12345, 0, 2**61 + 3)]
    for _ in range(400):
        cases.append((int(rng.integers(0, 2**63)) * 2 + int(rng.integers(0, 2)), 0,
                      int(rng.integers(0, 2**36))))
    return cases


def test_oracle_blocks_equal_curand(oracle, curand_dump):
    cases = _cases()
    want = curand_dump(cases)
    got = np.array([oracle.noise_block(s, b) for s, _, b in cases], dtype=np.uint32)
    assert np.array_equal(got, want)


def test_oracle_raw_rounds_equal_curand_with_subsequence(oracle, curand_dump):
    rng = np.random.default_rng(32)
    cases = [(int(rng.integers(0, 2**63)), int(rng.integers(0, 2**63)),
              int(rng.integers(0, 2**61))) for _ in range(200)]
    want = curand_dump(cases)
    for (seed, sub, b), w in zip(cases, want):
        ctr = [b & 0xFFFFFFFF, b >> 32, sub & 0xFFFFFFFF, sub >> 32]
        assert np.array_equal(oracle.philox4x32_10(ctr, [seed & 0xFFFFFFFF, seed >> 32]), w)


def test_library_noise_bits_equal_curand(es, curand_dump):
    # Runs of 1024 consecutive blocks, covering the tile path and the 2^32-block
    # boundary of the counter's low word.
    for seed, base in ((3, 0), (2**40 + 9, 2**32 - 512), (99, 2**34 - 300)):
        n = 1024
        out = torch.empty(4 * n, dtype=torch.int32, device="cuda")
        es.es_noise_bits(seed, base, n, out)
        torch.cuda.synchronize()
        got = out.cpu().numpy().view(np.uint32).reshape(n, 4)
        want = curand_dump([(seed, 0, base + t) for t in range(n)])
        assert np.array_equal(got, want), (seed, base)
