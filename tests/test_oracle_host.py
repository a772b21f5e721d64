"""Pins for the oracle's host-side generation control: population z-score (§3),
cosine sigma decay (§3.1), update coefficients (§3, App. C.1) and the
invalid-reward rule of App. D.5 / D.6."""
import math

import numpy as np
import pytest


def test_zscore_matches_numpy_population_std(oracle):
    rng = np.random.default_rng(0)
    for n in (2, 3, 8, 16, 30, 64, 128):
        R = rng.standard_normal(n) * 3 + 1
        want = (R - R.mean()) / (R.std(ddof=0) + 1e-8)
        assert np.allclose(oracle.zscore(R, 1e-8), want, rtol=1e-12, atol=1e-12)


def test_zscore_moments_and_affine_invariance(oracle):
    rng = np.random.default_rng(1)
    R = rng.uniform(size=30)
    z = oracle.zscore(R, 0.0)
    assert abs(z.mean()) < 1e-12 and abs(np.mean(z**2) - 1) < 1e-12
    assert np.allclose(oracle.zscore(7.5 * R - 3.0, 0.0), z, rtol=1e-10, atol=1e-12)
    # a negative scale flips the sign
    assert np.allclose(oracle.zscore(-2.0 * R, 0.0), -z, rtol=1e-10, atol=1e-12)


def test_zscore_degenerate_batches_give_no_update(oracle):
    assert np.all(oracle.zscore(np.full(16, 0.3)) == 0)           # all equal
    assert np.all(oracle.zscore(np.ones(8)) == 0)
    assert np.all(oracle.zscore([float("nan")] * 4) == 0)           # all invalid
    assert np.all(oracle.zscore([float("inf"), float("nan")]) == 0)
    assert np.all(oracle.zscore([5.0]) == 0)                         # G = 1


def test_zscore_invalid_rewards_get_the_batch_minimum(oracle):
    R = np.array([0.2, float("nan"), 0.9, float("-inf"), 0.5])
    Rp = np.array([0.2, 0.2, 0.9, 0.2, 0.5])
    assert np.allclose(oracle.zscore(R), oracle.zscore(Rp), rtol=0, atol=0)


def test_sigma_cosine_closed_forms(oracle):
    s0, sT, T = 1e-3, 2.5e-4, 100
    assert oracle.sigma_cosine(s0, sT, 0, T) == s0
    assert oracle.sigma_cosine(s0, sT, T, T) == sT
    assert math.isclose(oracle.sigma_cosine(s0, sT, T // 2, T), (s0 + sT) / 2, rel_tol=1e-15)
    vals = [oracle.sigma_cosine(s0, sT, t, T) for t in range(T + 1)]
    assert all(a >= b for a, b in zip(vals, vals[1:]))
    # symmetric about the midpoint: sigma_t + sigma_{T-t} = sigma_0 + sigma_T
    for t in range(T + 1):
        assert math.isclose(vals[t] + vals[T - t], s0 + sT, rel_tol=1e-14)
    # test-time schedule decays to zero (§3.1, AHD setting)
    assert oracle.sigma_cosine(1e-3, 0.0, 50, 50) == 0.0
    # quarter point: (1 + cos(pi/4)) / 2
    assert math.isclose(oracle.sigma_cosine(1.0, 0.0, 25, 100), (1 + math.sqrt(0.5)) / 2, rel_tol=1e-15)
    # clamping and degenerate T
    assert oracle.sigma_cosine(s0, sT, -3, T) == s0
    assert oracle.sigma_cosine(s0, sT, T + 9, T) == sT
    assert oracle.sigma_cosine(s0, sT, 0, 0) == s0


def test_update_coeff_modes(oracle):
    rhat = np.array([1.0, -0.5, 0.0, 2.0])
    alpha, sigma = 5e-4, 1e-3
    paper = oracle.update_coeffs(rhat, alpha, sigma, 0)
    canon = oracle.update_coeffs(rhat, alpha, sigma, 1)
    assert np.array_equal(paper, (alpha * rhat / 4).astype(np.float32))
    assert np.allclose(canon.astype(np.float64), alpha * rhat / (4 * sigma), rtol=1e-7)
    with pytest.raises(ValueError):
        oracle.update_coeffs(rhat, alpha, sigma, 2)


def test_quadratic_reward_matches_numpy(oracle):
    rng = np.random.default_rng(3)
    a = rng.standard_normal(1000).astype(np.float32)
    b = rng.standard_normal(1000).astype(np.float32)
    want = -np.sum((a.astype(np.float64) - b.astype(np.float64)) ** 2)
    assert math.isclose(oracle.quadratic_reward(a, b), want, rel_tol=1e-13)
