"""Pins for the oracle's sampler updates and probe drift (no GPU).

DDPM (Eqs. 2-3): with the true noise, the mean of Eq. 3 is the posterior mean of the forward
process of Eq. 1,  mu~(x_t, x_0) = sqrt(ab_{t-1}) beta_t / (1 - ab_t) x_0
+ sqrt(alpha_t) (1 - ab_{t-1}) / (1 - ab_t) x_t  (ab = alpha_bar) -- an identity independent of
how Eq. 3 is written.  DDIM: with the true noise the deterministic step (eta = 0) lands exactly
on the forward marginal sqrt(ab_prev) x_0 + sqrt(1 - ab_prev) eps, and at eta = 1 its mean is
the same posterior mean.  The drift is pinned by closed forms.
"""
import math

import numpy as np
import pytest

import oracle


def _schedule(T=1000):
    betas = np.linspace(1e-4, 0.02, T)      # a standard linear DDPM schedule
    alphas = 1.0 - betas
    return alphas, np.cumprod(alphas)


@pytest.mark.parametrize("t", [1, 10, 250, 500, 999])
def test_ddpm_mean_is_the_forward_posterior_mean(t):
    alphas, ab = _schedule()
    rng = np.random.default_rng(t)
    x0 = rng.standard_normal(64)
    eps = rng.standard_normal(64)
    xt = math.sqrt(ab[t]) * x0 + math.sqrt(1 - ab[t]) * eps
    a, b, c = oracle.ddpm_coefficients(alphas[t], ab[t])
    beta = 1 - alphas[t]
    post = (math.sqrt(ab[t - 1]) * beta / (1 - ab[t])) * x0 + \
           (math.sqrt(alphas[t]) * (1 - ab[t - 1]) / (1 - ab[t])) * xt
    np.testing.assert_allclose(a * xt + b * eps, post, rtol=1e-9, atol=1e-9)
    assert c == pytest.approx(math.sqrt(beta), rel=1e-15)


def test_ddpm_trivial_step():
    # alpha_t = 1: no noise was added at this step, so the mean is x_t and the deviation 0.
    a, b, c = oracle.ddpm_coefficients(1.0, 0.5)
    assert (a, b, c) == (1.0, 0.0, 0.0)


@pytest.mark.parametrize("t,s", [(999, 979), (500, 480), (40, 20), (20, 0)])
def test_ddim_deterministic_step_is_exact_on_the_forward_marginal(t, s):
    _, ab = _schedule()
    rng = np.random.default_rng(t)
    x0 = rng.standard_normal(64)
    eps = rng.standard_normal(64)
    xt = math.sqrt(ab[t]) * x0 + math.sqrt(1 - ab[t]) * eps
    a, b, c = oracle.ddim_coefficients(ab[t], ab[s], 0.0)
    assert c == 0.0
    np.testing.assert_allclose(a * xt + b * eps, math.sqrt(ab[s]) * x0 + math.sqrt(1 - ab[s]) * eps,
                               rtol=1e-10, atol=1e-10)


@pytest.mark.parametrize("t", [2, 100, 700, 999])
def test_ddim_eta_one_mean_is_the_ddpm_posterior_mean(t):
    alphas, ab = _schedule()
    rng = np.random.default_rng(t + 1)
    x0 = rng.standard_normal(32)
    eps = rng.standard_normal(32)
    xt = math.sqrt(ab[t]) * x0 + math.sqrt(1 - ab[t]) * eps
    a, b, _ = oracle.ddim_coefficients(ab[t], ab[t - 1], 1.0)
    da, db, _ = oracle.ddpm_coefficients(alphas[t], ab[t])
    np.testing.assert_allclose(a * xt + b * eps, da * xt + db * eps, rtol=1e-9, atol=1e-9)


def test_sampler_coefficients_reject_bad_schedules():
    for args in [(0.0, 0.5), (1.2, 0.5), (0.9, 1.0), (0.9, 0.0)]:
        with pytest.raises(oracle.OracleError):
            oracle.ddpm_coefficients(*args)
    for args in [(0.5, 0.4, 0.0), (1.0, 1.0, 0.0), (0.5, 0.6, -1.0), (0.1, 0.9, 5.0)]:
        with pytest.raises(oracle.OracleError):
            oracle.ddim_coefficients(*args)


def test_update_on_linear_data_with_noise():
    rng = np.random.default_rng(3)
    n = 301
    p0 = rng.integers(-8, 9, n).astype(np.float64)
    p1 = rng.integers(-8, 9, n).astype(np.float64)
    s = [0.5, 0.75]
    t = 0.25
    V = [(p0 + p1 * sj).astype(np.float32) for sj in s]
    x = rng.integers(-50, 50, n).astype(np.float32)
    z = rng.integers(-4, 5, n).astype(np.float32)
    W = oracle.lagrange(s, t)                  # exact for a line: v_hat = p0 + p1 t
    a, b, c = 0.5, -2.0, 0.25
    got, bound = oracle.update(V, W, x, a, b, c, z)
    np.testing.assert_allclose(got, a * x + b * (p0 + p1 * t) + c * z, atol=1e-12)
    got0, _ = oracle.update(V, W, x, a, b)      # no noise term
    np.testing.assert_allclose(got0, a * x + b * (p0 + p1 * t), atol=1e-12)
    assert np.all(bound >= np.abs(a * x))


def test_drift_closed_forms():
    prev = np.array([1, -2, 3, -4, 5], dtype=np.float32)
    assert list(oracle.drift(prev, prev)) == [0.0, 15.0, 0.0]
    cur = prev + np.float32(0.5)
    np.testing.assert_allclose(oracle.drift(cur, prev), [2.5, 15.0, 2.5 / 15.0])
    assert oracle.drift(np.ones(3, np.float32), np.zeros(3, np.float32))[2] == math.inf
    assert list(oracle.drift(np.zeros(3, np.float32), np.zeros(3, np.float32))) == [0, 0, 0]
    # a NaN in either tensor poisons the ratio instead of reading as "no change"
    nan3 = np.array([0.0, np.nan, 0.0], np.float32)
    assert math.isnan(oracle.drift(np.zeros(3, np.float32), nan3)[2])
    assert math.isnan(oracle.drift(nan3, np.zeros(3, np.float32))[2])
    assert math.isnan(oracle.drift(nan3, np.ones(3, np.float32))[2])
    # scale invariance: scaling both tensors leaves the ratio unchanged
    rng = np.random.default_rng(0)
    a = rng.standard_normal(999).astype(np.float32)
    b = rng.standard_normal(999).astype(np.float32)
    np.testing.assert_allclose(oracle.drift(4 * a, 4 * b)[2], oracle.drift(a, b)[2], rtol=1e-12)
    # bf16 storage decodes exactly: 1.0 (0x3F80) against 1.5 (0x3FC0)
    bits = lambda v: np.array(v, dtype=np.uint16)
    np.testing.assert_allclose(oracle.drift(bits([0x3FC0] * 4), bits([0x3F80] * 4)),
                               [2.0, 4.0, 0.5])
