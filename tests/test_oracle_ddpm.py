"""Pins of the oracle's stochastic steps (eta > 0; eta = 1 is DDPM, Table 2).

The draws z_i are fixed before sampling and passed in (the reading in the
design notes), so the stochastic sampler is a deterministic recursion given
them and the Picard iteration applies unchanged. These tests check the oracle
against facts that do not come from its own formulas: the textbook DDPM
posterior q(x_{t-1} | x_t, x0), a scalar second implementation written in that
posterior form, the closed form of the single-Gaussian case, and the sample
statistics of exact DDPM sampling of a Gaussian.
"""
import numpy as np
import pytest

import workload as W
from oracle.ddim import ddim_step, step_coefficients, serial_ddim, ddim_sigma
from oracle.gmm import make_eps_fn
from oracle.picard import run_picard
from scalar_picard import scalar_cached_picard


def _posterior_step(x, eps, a_t, a_prev, z):
    """Ho et al.'s posterior mean and variance for x_{t-1} given x_t and x0_hat."""
    beta = 1.0 - a_t / a_prev
    alpha = 1.0 - beta
    x0 = (x - np.sqrt(1.0 - a_t) * eps) / np.sqrt(a_t)
    mean = (np.sqrt(a_prev) * beta / (1.0 - a_t)) * x0 + (np.sqrt(alpha) * (1.0 - a_prev) / (1.0 - a_t)) * x
    var = (1.0 - a_prev) / (1.0 - a_t) * beta
    return mean + np.sqrt(var) * z


def test_eta1_full_schedule_is_the_ddpm_posterior():
    a = W.alphas_cumprod(1000)                 # tau_i = 999 - i: every training step
    rng = np.random.default_rng(0)
    for i in (0, 1, 10, 500, 900, 998, 999):
        x, eps, z = rng.standard_normal((3, 64))
        got = ddim_step(x, eps, a[i], a[i + 1], eta=1.0, z=z)
        want = _posterior_step(x, eps, a[i], a[i + 1], z)
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
    # the last step (to alpha-bar 1) adds no noise
    assert ddim_sigma(a[999], a[1000], 1.0) == 0.0


@pytest.mark.parametrize("eta", [0.0, 0.3, 1.0])
def test_step_coefficients_reproduce_the_step(eta):
    a = W.alphas_cumprod(50)
    c, e, s = step_coefficients(a, eta)
    rng = np.random.default_rng(1)
    for i in range(50):
        x, eps, z = rng.standard_normal((3, 16))
        want = ddim_step(x, eps, a[i], a[i + 1], eta, z)
        np.testing.assert_allclose(c[i] * x + e[i] * eps + s[i] * z, want, rtol=1e-12, atol=1e-13)
    if eta == 0.0:
        assert np.all(s == 0.0)


def _tiny_noisy(T=12, B=2, D=16, K=3, seed=0):
    rng = np.random.default_rng(seed)
    a = W.alphas_cumprod(T)
    return a, rng.standard_normal((B, D)), rng.standard_normal((K, D)), rng.standard_normal((B, T, D))


@pytest.mark.parametrize("P", [1, 3, 7, 12])
def test_tol0_noisy_picard_equals_serial(P):
    a, x0, mu, z = _tiny_noisy()
    fn = make_eps_fn(a, mu, 0.5)
    serial = serial_ddim(a, x0, fn, eta=1.0, noise=z)[:, -1]
    r = run_picard(a, x0, fn, P, 0.0, 0.0, use_cache=False, eta=1.0, noise=z)
    np.testing.assert_allclose(r.x_final, serial, rtol=1e-10, atol=1e-10)


def test_eta0_ignores_the_draws():
    a, x0, mu, z = _tiny_noisy()
    fn = make_eps_fn(a, mu, 0.5)
    r0 = run_picard(a, x0, fn, 4, 1e-3, 0.05)
    r1 = run_picard(a, x0, fn, 4, 1e-3, 0.05, eta=0.0, noise=z)
    assert np.array_equal(r0.x_final, r1.x_final)


@pytest.mark.parametrize("T,P,thresh,tol,seed", [(4, 2, 0.05, 1e-3, 0), (6, 3, 0.2, 1e-2, 2),
                                                 (5, 5, 1e9, 0.0, 3), (6, 2, 0.0, 0.05, 4)])
def test_scalar_ddpm_posterior_form_agrees(T, P, thresh, tol, seed):
    rng = np.random.default_rng(seed)
    B, D, K = 2, 4, 2
    a = W.alphas_cumprod(T)
    x0 = rng.standard_normal((B, D))
    mu = rng.standard_normal((K, D))
    z = rng.standard_normal((B, T, D))
    r = run_picard(a, x0, make_eps_fn(a, mu, 0.5), P, tol, thresh, eta=1.0, noise=z)
    finals, log = scalar_cached_picard(list(a), x0.tolist(), mu.tolist(), 0.5, P, tol, thresh,
                                       noise=z.tolist())
    assert [m for m, _, _ in log] == [rec.miss_bt for rec in r.records]
    assert [s for _, s, _ in log] == [rec.stride for rec in r.records]
    np.testing.assert_allclose(np.array(finals), r.x_final, rtol=1e-11, atol=1e-11)


def test_single_gaussian_closed_form_with_noise():
    """K = 1: eps* is affine in x (Tweedie), so DDPM is x_{i+1} = A_i x_i + b_i with
    A_i = c_i + e_i g_i, b_i = -e_i g_i sqrt(a_i) mu + sigma_i z_i, g = sqrt(1-a)/v;
    x_T = (prod A) x_0 + sum_i (prod_{j>i} A_j) b_i, evaluated with suffix products."""
    T, D, s = 40, 32, 0.5
    rng = np.random.default_rng(5)
    a = W.alphas_cumprod(T)
    x0 = rng.standard_normal((1, D))
    mu = rng.standard_normal((1, D))
    z = rng.standard_normal((1, T, D))
    got = serial_ddim(a, x0, make_eps_fn(a, mu, s), eta=1.0, noise=z)[0, -1]
    c, e, sig = step_coefficients(a, 1.0)
    ai = a[:-1]
    v = ai * s * s + 1.0 - ai
    g = np.sqrt(1.0 - ai) / v
    A = c + e * g
    suffix = np.append(np.cumprod(A[::-1])[::-1][1:], 1.0)      # prod_{j>i} A_j
    b = -(e * g * np.sqrt(ai))[:, None] * mu[0][None, :] + sig[:, None] * z[0]
    want = np.prod(A) * x0[0] + np.sum(suffix[:, None] * b, axis=0)
    np.testing.assert_allclose(got, want, rtol=1e-10, atol=1e-10)


def test_ddpm_samples_a_gaussian_with_the_right_variance():
    """Exact-posterior DDPM over the full 1000-step schedule samples the data
    distribution: for a single Gaussian N(mu, s^2 I) the standardised outputs
    (x_T - mu) / s of independent coordinates have mean 0 and variance 1. A
    wrong noise scale (or a missing noise term) moves the variance well off 1."""
    T, D, s = 1000, 8192, 0.5
    rng = np.random.default_rng(7)
    a = W.alphas_cumprod(T)
    x0 = rng.standard_normal((1, D))
    mu = rng.standard_normal((1, D))
    z = rng.standard_normal((1, T, D))
    out = serial_ddim(a, x0, make_eps_fn(a, mu, s), eta=1.0, noise=z)[0, -1]
    u = (out - mu[0]) / s
    assert abs(u.mean()) < 0.05
    assert abs(u.std() - 1.0) < 0.04
