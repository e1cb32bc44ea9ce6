"""DDIM (eta = 0) step, drift coefficients and serial DDIM, fp64.

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
"""
from __future__ import annotations

import numpy as np


def ddim_step(x, eps, a_i, a_next):
    """One DDIM (eta = 0) step from alpha-bar a_i to a_next, written as the
    textbook two-stage update: predict x0, then re-noise to the next level."""
    x0_pred = (x - np.sqrt(1.0 - a_i) * eps) / np.sqrt(a_i)
    return np.sqrt(a_next) * x0_pred + np.sqrt(1.0 - a_next) * eps


def drift_coefficients(alphas):
    """(c, e), fp64 [T], with ddim_step(x, eps, a_i, a_{i+1}) == c_i x + e_i eps.

    The Picard drift of step i is then s_i(x, eps) = (c_i - 1) x + e_i eps.
    """
    a = np.asarray(alphas, dtype=np.float64)
    a_i, a_n = a[:-1], a[1:]
    c = np.sqrt(a_n / a_i)
    e = np.sqrt(1.0 - a_n) - np.sqrt(a_n) * np.sqrt(1.0 - a_i) / np.sqrt(a_i)
    return c, e


def drift(x, eps, c_i, e_i):
    """s_theta at the current latent x (Sec. 2.2 last paragraph): (c-1) x + e eps."""
    return (c_i - 1.0) * x + e_i * eps


def serial_ddim(alphas, x_init, eps_fn):
    """Serial DDIM sampler, T network evaluations (Table 1 row "Serial").

    alphas : fp64 [T+1]; x_init : [B][D]; eps_fn(x_rows [n][D], idx [n]) -> [n][D].
    Returns the full trajectory, fp64 [B][T+1][D].
    """
    a = np.asarray(alphas, dtype=np.float64)
    T = len(a) - 1
    x = np.asarray(x_init, dtype=np.float64)
    B = x.shape[0]
    traj = np.empty((B, T + 1, x.shape[1]), dtype=np.float64)
    traj[:, 0] = x
    for i in range(T):
        eps = eps_fn(x, np.full(B, i))
        x = ddim_step(x, eps, a[i], a[i + 1])
        traj[:, i + 1] = x
    return traj
