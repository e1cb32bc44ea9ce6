"""DDIM step (eta = 0, and the stochastic eta > 0 family that includes DDPM),
drift coefficients and serial sampling, fp64.

Sec. 2.1 (Eq. 1) writes the Picard update with a probability-flow-ODE drift
s_theta(x, u) that "combines the current latent x and the noise prediction
eps_theta(x, u) with coefficients determined by the noise schedule". For a DDIM
scheduler (Sec. 3.3) the discrete drift of step i is the DDIM update minus the
identity, so that x_{i+1} = x_i + s(x_i, i). Reading of the paper: the 1/T of
Eq. 1's continuous form is absorbed into the discrete step (the ParaDiGMS
discrete form).

Index convention: sampling index i = 0 is the noisiest state (Eq. 1 starts from
x_0, the initial noise); ``alphas[i]`` is alpha-bar at sampling index i and
``alphas[T] == 1``.

Stochastic samplers (eta > 0; eta = 1 over the full 1000-step schedule is DDPM,
Table 2): step i adds sigma_i z_i with z_i ~ N(0, I) drawn once per trajectory
and step before sampling and passed in, so that, given the draws, the sampler
is a deterministic recursion and the Picard drift of step i is
(c_i - 1) x + e_i eps + sigma_i z_i. The paper does not state this rule; it is
the reading written down in the design notes.
"""
from __future__ import annotations

import numpy as np


def ddim_sigma(a_i, a_next, eta):
    """Noise scale of the DDIM step from alpha-bar a_i to a_next:
    eta * sqrt((1 - a_next) / (1 - a_i)) * sqrt(1 - a_i / a_next)."""
    return eta * np.sqrt((1.0 - a_next) / (1.0 - a_i)) * np.sqrt(1.0 - a_i / a_next)


def ddim_step(x, eps, a_i, a_next, eta=0.0, z=None):
    """One DDIM step from alpha-bar a_i to a_next, written as the textbook
    two-stage update: predict x0, then re-noise to the next level with
    sqrt(1 - a_next - sigma^2) eps + sigma z (sigma = 0 for eta = 0)."""
    x0_pred = (x - np.sqrt(1.0 - a_i) * eps) / np.sqrt(a_i)
    sig = ddim_sigma(a_i, a_next, eta)
    out = np.sqrt(a_next) * x0_pred + np.sqrt(1.0 - a_next - sig * sig) * eps
    if eta != 0.0:
        out = out + sig * z
    return out


def step_coefficients(alphas, eta=0.0):
    """(c, e, sigma), fp64 [T], with
    ddim_step(x, eps, a_i, a_{i+1}, eta, z) == c_i x + e_i eps + sigma_i z."""
    a = np.asarray(alphas, dtype=np.float64)
    a_i, a_n = a[:-1], a[1:]
    sig = ddim_sigma(a_i, a_n, eta)
    c = np.sqrt(a_n / a_i)
    e = np.sqrt(1.0 - a_n - sig * sig) - np.sqrt(a_n) * np.sqrt(1.0 - a_i) / np.sqrt(a_i)
    return c, e, sig


def drift_coefficients(alphas):
    """(c, e), fp64 [T], with ddim_step(x, eps, a_i, a_{i+1}) == c_i x + e_i eps.

    The Picard drift of step i is then s_i(x, eps) = (c_i - 1) x + e_i eps.
    """
    c, e, _ = step_coefficients(alphas, 0.0)
    return c, e


def drift(x, eps, c_i, e_i, s_i=0.0, z=None):
    """s_theta at the current latent x (Sec. 2.2 last paragraph): (c-1) x + e eps,
    plus sigma z for a stochastic step."""
    d = (c_i - 1.0) * x + e_i * eps
    if z is not None:
        d = d + s_i * z
    return d


def serial_ddim(alphas, x_init, eps_fn, eta=0.0, noise=None):
    """Serial DDIM sampler, T network evaluations (Table 1 row "Serial").

    alphas : fp64 [T+1]; x_init : [B][D]; eps_fn(x_rows [n][D], idx [n]) -> [n][D];
    eta > 0 needs noise [B][T][D] (the draws z_i of every trajectory and step).
    Returns the full trajectory, fp64 [B][T+1][D].
    """
    a = np.asarray(alphas, dtype=np.float64)
    T = len(a) - 1
    x = np.asarray(x_init, dtype=np.float64)
    B = x.shape[0]
    if eta != 0.0 and noise is None:
        raise ValueError("eta > 0 needs the noise draws")
    traj = np.empty((B, T + 1, x.shape[1]), dtype=np.float64)
    traj[:, 0] = x
    for i in range(T):
        eps = eps_fn(x, np.full(B, i))
        z = None if eta == 0.0 else np.asarray(noise, dtype=np.float64)[:, i]
        x = ddim_step(x, eps, a[i], a[i + 1], eta, z)
        traj[:, i + 1] = x
    return traj
