"""The C ABI used from plain C, with no Python in the path: tests/abi_c_consumer.c
allocates device memory with the CUDA runtime, calls es_plan_create,
es_perturb, es_restore, es_update and es_noise_fill directly, and prints every
intermediate state. Each state is checked against the oracle from the state
before it, and a host pointer must be refused."""
import subprocess

import numpy as np
import pytest
import torch

from paper_2608_17310_gb300 import inputs as I
from parity import assert_bf16_within_ulp, build_c_consumer, noise_abs_tol

pytestmark = pytest.mark.gpu


def test_plain_c_program_matches_the_oracle(es, oracle, tmp_path):
    exe = build_c_consumer(tmp_path)
    n = 3 * 8192 + 37                       # several tiles and a ragged tail
    theta = torch.from_numpy(I.normal_f32(n, 4, 0.02)).to(torch.bfloat16) \
        .view(torch.int16).numpy().view(np.uint16)
    text = f"{n}\n" + " ".join(str(int(v)) for v in theta) + "\n"
    r = subprocess.run([exe], input=text, capture_output=True, text=True, timeout=120)
    assert r.returncode == 0, r.stderr
    out = {}
    for line in r.stdout.splitlines():
        tag, *vals = line.split()
        out[tag] = vals
    assert set(out) == {"P", "R", "U", "E"}
    P = np.array(out["P"], dtype=np.uint64).astype(np.uint16)
    R = np.array(out["R"], dtype=np.uint64).astype(np.uint16)
    U = np.array(out["U"], dtype=np.uint64).astype(np.uint16)
    E = np.array(out["E"], dtype=np.float64)
    g = np.arange(n, dtype=np.uint64)
    sigma = float(np.float32(1e-3))
    eps11 = oracle.noise_at(11, g)
    tol = noise_abs_tol([eps11], [sigma])
    assert_bf16_within_ulp(P, oracle.perturb(theta, g, 11, sigma, "bf16"), "C perturb", abs_tol=tol)
    assert_bf16_within_ulp(R, oracle.restore(P, g, 11, sigma, "bf16"), "C restore", abs_tol=tol)
    seeds = np.array([3, 5, 7], dtype=np.uint64)
    coeffs = np.array([1e-4, -2e-4, 5e-5], dtype=np.float32)
    tol_u = noise_abs_tol([oracle.noise_at(int(s), g) for s in seeds], coeffs)
    assert_bf16_within_ulp(U, oracle.update(R, g, seeds, coeffs, "bf16"), "C update", abs_tol=tol_u)
    assert np.all(np.abs(E - eps11) <= 1e-5 * np.maximum(1.0, np.abs(eps11)))
