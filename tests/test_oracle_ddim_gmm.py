"""Pins for the oracle's DDIM step and mixture denoiser (CPU only).

Each check ties the oracle to mathematics it does not itself contain:
closed-form trajectories, Tweedie's formula against a brute-force log-density,
and invariances that a transposed operand or wrong index would break.
"""
import numpy as np
import pytest

import workload as W
from oracle.ddim import ddim_step, drift_coefficients, serial_ddim
from oracle.gmm import gmm_eps, gmm_eps_row, log_density, make_eps_fn


def _sigma(a):
    return np.sqrt((1.0 - a) / a)


def test_schedule_generator():
    """Linear-beta schedule: alpha-bar_0 = 1 - 1e-4, product form, DDIM spacing."""
    full = W.train_alphas_cumprod()
    assert full[0] == pytest.approx(1 - 1e-4, rel=1e-15)
    betas = np.linspace(1e-4, 0.02, 1000)
    assert full[999] == pytest.approx(np.prod(1 - betas), rel=1e-12)
    assert list(W.ddim_timesteps(16)[:3]) == [930, 868, 806]
    assert W.ddim_timesteps(100)[0] == 990 and W.ddim_timesteps(100)[-1] == 0
    a = W.alphas_cumprod(100)
    assert len(a) == 101 and a[-1] == 1.0
    assert np.all(np.diff(a) > 0)          # noise decreases along sampling order


def test_point_mass_ddim_is_exact():
    """A point-mass prior (std 0, K = 1): the exact eps makes DDIM follow the
    closed form x_i = sqrt(a_i) mu + sqrt(1 - a_i) eps0 at every step, and land on mu."""
    rng = np.random.default_rng(3)
    D = 7
    mu = rng.standard_normal((1, D))
    a = W.alphas_cumprod(25)
    x0 = rng.standard_normal((1, D))
    traj = serial_ddim(a, x0, make_eps_fn(a, mu, std=0.0))
    eps0 = (x0[0] - np.sqrt(a[0]) * mu[0]) / np.sqrt(1 - a[0])
    for i in range(len(a)):
        want = np.sqrt(a[i]) * mu[0] + np.sqrt(1 - a[i]) * eps0
        np.testing.assert_allclose(traj[0, i], want, rtol=1e-11, atol=1e-11)
    np.testing.assert_allclose(traj[0, -1], mu[0], rtol=1e-11, atol=1e-11)


@pytest.mark.parametrize("T", [4, 16, 100])
def test_single_gaussian_ddim_closed_form(T):
    """K = 1, std s: in y = x / sqrt(a), sigma = sqrt((1-a)/a), DDIM reads
    y_{i+1} = y_i + (sigma_{i+1} - sigma_i) eps and the exact eps is
    sigma (y - mu) / (s^2 + sigma^2), so y - mu is scaled per step by
    1 + (sigma_{i+1} - sigma_i) sigma_i / (s^2 + sigma_i^2)."""
    rng = np.random.default_rng(T)
    D, s = 5, 0.5
    mu = rng.standard_normal((1, D))
    a = W.alphas_cumprod(T)
    x0 = rng.standard_normal((1, D))
    traj = serial_ddim(a, x0, make_eps_fn(a, mu, std=s))
    sig = _sigma(a)
    y = x0[0] / np.sqrt(a[0])
    for i in range(T):
        y = mu[0] + (y - mu[0]) * (1 + (sig[i + 1] - sig[i]) * sig[i] / (s * s + sig[i] ** 2))
        np.testing.assert_allclose(traj[0, i + 1], np.sqrt(a[i + 1]) * y, rtol=1e-10, atol=1e-12)


def test_fine_ddim_approaches_exact_ode():
    """With 1000 steps DDIM approaches the exact probability-flow ODE solution
    of a Gaussian prior, (y - mu) proportional to sqrt(s^2 + sigma^2)."""
    rng = np.random.default_rng(5)
    D, s = 4, 0.5
    mu = rng.standard_normal((1, D))
    a = W.alphas_cumprod(1000)
    x0 = rng.standard_normal((1, D))
    xT = serial_ddim(a, x0, make_eps_fn(a, mu, std=s))[0, -1]
    sig0 = _sigma(a[0])
    exact = mu[0] + (x0[0] / np.sqrt(a[0]) - mu[0]) * s / np.sqrt(s * s + sig0 * sig0)
    np.testing.assert_allclose(xT, exact, rtol=5e-3, atol=5e-3)


def test_drift_coefficients_reproduce_step():
    a = W.alphas_cumprod(16)
    c, e = drift_coefficients(a)
    rng = np.random.default_rng(0)
    for i in range(16):
        x, eps = rng.standard_normal(9), rng.standard_normal(9)
        np.testing.assert_allclose(c[i] * x + e[i] * eps, ddim_step(x, eps, a[i], a[i + 1]),
                                   rtol=1e-13, atol=1e-13)
    # last step lands on alpha-bar = 1: x_T = x0_pred, so c = 1/sqrt(a), e = -sqrt((1-a)/a)
    assert c[-1] == pytest.approx(1 / np.sqrt(a[-2]))
    assert e[-1] == pytest.approx(-np.sqrt((1 - a[-2]) / a[-2]))


@pytest.mark.parametrize("a", [1e-4, 0.05, 0.5, 0.97, 0.9999])
def test_tweedie_matches_finite_difference_of_log_density(a):
    """eps*(x) = -sqrt(1 - a) * grad log p_a(x) (Tweedie), with log p_a computed
    by brute force (log-sum-exp of Gaussian log-densities, normalisers included)."""
    rng = np.random.default_rng(11)
    K, D, s = 3, 6, 0.5
    mu = rng.standard_normal((K, D))
    x = np.sqrt(a) * mu[1] + np.sqrt(1 - a) * rng.standard_normal(D) * 0.7
    eps = gmm_eps_row(x, a, mu, s)
    h = 1e-5 * max(1.0, np.sqrt(a * s * s + 1 - a))
    for d in range(D):
        xp, xm = x.copy(), x.copy()
        xp[d] += h
        xm[d] -= h
        g = (log_density(xp, a, mu, s) - log_density(xm, a, mu, s)) / (2 * h)
        assert eps[d] == pytest.approx(-np.sqrt(1 - a) * g, rel=1e-6, abs=1e-8)


def test_single_component_is_gaussian_conditioning():
    rng = np.random.default_rng(2)
    D, s, a = 8, 0.5, 0.3
    mu = rng.standard_normal((1, D))
    x = rng.standard_normal(D)
    # E[eps | x] = Cov(eps, x) / Var(x) * (x - E x), Cov = sqrt(1-a), Var = a s^2 + 1 - a
    want = np.sqrt(1 - a) / (a * s * s + 1 - a) * (x - np.sqrt(a) * mu[0])
    np.testing.assert_allclose(gmm_eps_row(x, a, mu, s), want, rtol=1e-13)


def test_component_order_and_hard_assignment():
    rng = np.random.default_rng(4)
    K, D, s, a = 5, 64, 0.5, 0.9
    mu = rng.standard_normal((K, D)) * 3.0
    x = np.sqrt(a) * mu[2] + 0.1 * rng.standard_normal(D)
    e1 = gmm_eps_row(x, a, mu, s)
    perm = rng.permutation(K)
    np.testing.assert_allclose(gmm_eps_row(x, a, mu[perm], s), e1, rtol=1e-12, atol=1e-14)
    # well separated: responsibilities are one-hot on the nearest mean
    hard = np.sqrt(1 - a) / (a * s * s + 1 - a) * (x - np.sqrt(a) * mu[2])
    np.testing.assert_allclose(e1, hard, rtol=1e-10, atol=1e-12)
    # batch form equals row form
    rows = np.stack([x, -x])
    out = gmm_eps(rows, np.array([a, 0.1]), mu, s)
    np.testing.assert_allclose(out[1], gmm_eps_row(-x, 0.1, mu, s), rtol=1e-14)
