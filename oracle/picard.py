"""Sliding-window Picard DDIM sampling with ParaAnya's output cache, fp64.

Follows Sec. 2.1 (Eq. 1, Eq. 2) and Sec. 2.2 (Eq. 3-7) in the paper's order.
Full-length arrays (every state 0..T, every cache entry 0..T-1) are used on
purpose: no rings, no index tricks, so the code can be read against the paper.

One Picard iteration k, per trajectory with window start t and
p = min(P, T - t) evaluation points t .. t+p-1:

1.  Cache distance (Eq. 4): for every evaluation point i that has a cache entry,
    delta_i = (1/D) * || x_i - xhat_i ||_1.
2.  Hit/miss (Eq. 5): a point entering the window for the first time has no
    entry and is a miss; otherwise hit iff delta_i < tau_cache (strict).
3.  All misses of all trajectories are evaluated in one batch, ordered by
    trajectory, then by ascending point index (the order is our reading; the
    paper only says the misses form one batched forward pass).
4.  Assembly (Eq. 6): eps_i = cached ehat_i for hits, fresh eps for misses.
5.  Cache update (Eq. 7), misses only: (xhat_i, ehat_i) <- (x_i, eps_i).
6.  Drift at the current latent (Sec. 2.2 last paragraph):
    d_i = (c_i - 1) x_i + e_i eps_i (+ sigma_i z_i for a stochastic step, with
    the draw z_i fixed before sampling).
7.  Picard update (Eq. 1, window form): x_{t+j+1} <- x_t + sum_{i=t}^{t+j} d_i.
8.  Convergence error (Eq. 2): err_j = (1/D) || x^{new}_{t+j+1} - x^{old}_{t+j+1} ||^2.
9.  Window advance: stride = min(p, 1 + number of leading j with err_j <= tau)
    (the ParaDiGMS rule; the paper only says the window advances once the
    leading states satisfy Eq. 2). New states entering at the tail take the
    value of the last computed state x_{t+p}. Done when t reaches T.

Readings where the paper is silent are listed in the design notes and in the
docstrings above; uncached sampling (``use_cache=False``) skips steps 1, 2 and 5
entirely -- a separate path, which the tau_cache = 0 pin compares against.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

from .ddim import drift, step_coefficients


@dataclass
class CacheAdaptation:
    """Online adaptation of tau_cache (the paper names it as future work in
    its conclusion and states no rule; this is the reading written down in the
    design notes). Per trajectory, after every iteration: with n_e of its
    window positions that had a cache entry and n_h hits among them,
      n_h / n_e <  target: tau <- min(tau * (1 + rate), tau_max), but only if
                           the window advanced beyond its first position
                           (stride > 1); with stride 1 tau holds;
      n_h / n_e >= target: tau <- max(tau / (1 + rate), tau_min);
    no entries (n_e = 0): tau holds. The next iteration's hit test (Eq. 5)
    uses the new tau. rate = 0 keeps tau_cache fixed."""

    rate: float
    target: float
    tau_min: float = 0.0
    tau_max: float = float("inf")

    def step(self, tau, n_e, n_h, stride):
        if n_e == 0:
            return tau
        up = 1.0 + self.rate
        if n_h / n_e < self.target:
            return min(tau * up, self.tau_max) if stride > 1 else tau
        return max(tau / up, self.tau_min)


@dataclass
class IterRecord:
    """What one Picard iteration decided, per trajectory and globally."""

    k: int
    t: List[int]                      # window start per trajectory (-1 if done)
    p: List[int]                      # evaluation points per trajectory (0 if done)
    delta: List[List[Optional[float]]]  # per point: None for first entry (or uncached)
    hit: List[List[bool]]
    miss_bt: List[tuple]              # canonical miss order (b, i)
    err: List[List[float]]            # Eq. 2 error per window position
    stride: List[int]
    tau: Optional[List[float]] = None  # tau_cache per trajectory used by this iteration's hit test


@dataclass
class PicardResult:
    x_final: np.ndarray               # [B][D], state T of every trajectory
    states: np.ndarray                # [B][T+1][D], final states
    iters: int                        # global Picard iterations
    iters_per_traj: List[int]
    nfe: int                          # sum over iterations of misses
    hits: int
    records: List[IterRecord] = field(default_factory=list)
    xhat: Optional[np.ndarray] = None     # [B][T][D] cached inputs (Eq. 3)
    ehat: Optional[np.ndarray] = None     # [B][T][D] cached outputs
    has_entry: Optional[np.ndarray] = None  # [B][T] entry exists


def run_picard(alphas, x_init, eps_fn, window, tol, cache_thresh,
               use_cache=True, max_iters=None, record=True, eta=0.0, noise=None,
               cache_store=None, adapt=None):
    """Cached (or uncached) sliding-window Picard sampling of B trajectories.

    alphas       : fp64 [T+1] sampling-order alpha-bar (alphas[T] == 1).
    x_init       : [B][D] initial noise (x_0 of Eq. 1).
    eps_fn       : eps_fn(x_rows [n][D] fp64, idx [n]) -> eps [n][D].
    window       : P, the number of active timesteps.
    tol          : tau of Eq. 2 (converged iff err <= tau).
    cache_thresh : tau_cache of Eq. 5 (hit iff delta < tau_cache).
    use_cache    : False gives the uncached sampler (every point evaluated).
    max_iters    : stop early after this many iterations (bounded samples).
    eta, noise   : stochastic steps (eta > 0): noise [B][T][D] holds the draws
                   z_i; the drift of step i gains sigma_i z_i (the same draw in
                   every iteration).
    cache_store  : how a cache entry is stored (step 5): None keeps the value,
                   oracle.storage.round_bf16 stores bfloat16 entries (states
                   and the fresh eps of a miss keep full precision).
    adapt        : a CacheAdaptation: tau_cache per trajectory, starting at
                   cache_thresh and adapted after every iteration; None keeps
                   cache_thresh fixed.
    """
    a = np.asarray(alphas, dtype=np.float64)
    T = len(a) - 1
    c, e, sig = step_coefficients(a, eta)
    Z = None
    if eta != 0.0:
        if noise is None:
            raise ValueError("eta > 0 needs the noise draws")
        Z = np.asarray(noise, dtype=np.float64)
    x0 = np.asarray(x_init, dtype=np.float64)
    B, D = x0.shape
    P = int(window)
    if P < 1 or T < 1:
        raise ValueError("window and T must be >= 1")

    X = np.zeros((B, T + 1, D))
    p0 = min(P, T)
    X[:, : p0 + 1] = x0[:, None, :]          # first window initialised to x_init
    Xhat = np.zeros((B, T, D))
    Ehat = np.zeros((B, T, D))
    has_entry = np.zeros((B, T), dtype=bool)

    t = np.zeros(B, dtype=np.int64)
    active = np.ones(B, dtype=bool)
    iters_per = [0] * B
    nfe = hits = 0
    tau = [float(cache_thresh)] * B
    records: List[IterRecord] = []
    k = 0
    while active.any():
        if max_iters is not None and k >= max_iters:
            break
        k += 1
        p = [int(min(P, T - t[b])) if active[b] else 0 for b in range(B)]
        tau_k = list(tau)

        # 1-2. cache distance (Eq. 4) and hit/miss partition (Eq. 5)
        deltas, hitflags = [], []
        for b in range(B):
            db, hb = [], []
            for j in range(p[b]):
                i = int(t[b]) + j
                if use_cache and has_entry[b, i]:
                    d_bi = float(np.sum(np.abs(X[b, i] - Xhat[b, i])) / D)
                    db.append(d_bi)
                    hb.append(d_bi < tau[b])
                else:
                    db.append(None)          # first entry (or no cache): miss
                    hb.append(False)
            deltas.append(db)
            hitflags.append(hb)

        # 3. one batched evaluation of every miss
        miss_bt = [(b, int(t[b]) + j) for b in range(B) for j in range(p[b])
                   if not hitflags[b][j]]
        if miss_bt:
            rows = np.stack([X[b, i] for b, i in miss_bt])
            fresh = eps_fn(rows, np.array([i for _, i in miss_bt]))
        fresh_of = {bt: r for r, bt in enumerate(miss_bt)}

        errs, strides = [], []
        for b in range(B):
            if not active[b]:
                errs.append([])
                strides.append(0)
                continue
            tb, pb = int(t[b]), p[b]
            # 4. assembly (Eq. 6)
            eps_w = np.empty((pb, D))
            for j in range(pb):
                i = tb + j
                if hitflags[b][j]:
                    eps_w[j] = Ehat[b, i]
                else:
                    eps_w[j] = fresh[fresh_of[(b, i)]]
            # 5. cache update for misses only (Eq. 7)
            if use_cache:
                for j in range(pb):
                    if not hitflags[b][j]:
                        i = tb + j
                        if cache_store is None:
                            Xhat[b, i] = X[b, i]
                            Ehat[b, i] = eps_w[j]
                        else:
                            Xhat[b, i] = cache_store(X[b, i])
                            Ehat[b, i] = cache_store(eps_w[j])
                        has_entry[b, i] = True
            # 6. drift at the current latents
            idx = np.arange(tb, tb + pb)
            d = drift(X[b, idx], eps_w, c[idx][:, None], e[idx][:, None],
                      sig[idx][:, None], None if Z is None else Z[b, idx])
            # 7. Picard update, window form of Eq. 1
            x_new = X[b, tb][None, :] + np.cumsum(d, axis=0)
            # 8. convergence error, Eq. 2
            err = np.sum((x_new - X[b, tb + 1: tb + pb + 1]) ** 2, axis=1) / D
            X[b, tb + 1: tb + pb + 1] = x_new
            # 9. window advance
            lead = 0
            while lead < pb and err[lead] <= tol:
                lead += 1
            stride = min(pb, 1 + lead)
            t_new = tb + stride
            p_new = min(P, T - t_new)
            if t_new + p_new > tb + pb:      # new tail states copy x_{t+p}
                X[b, tb + pb + 1: t_new + p_new + 1] = X[b, tb + pb]
            t[b] = t_new
            iters_per[b] += 1
            if t_new == T:
                active[b] = False
            errs.append([float(v) for v in err])
            strides.append(stride)
            if adapt is not None:   # tau_cache for the next iteration's hit test
                n_e = sum(1 for dv in deltas[b] if dv is not None)
                tau[b] = adapt.step(tau[b], n_e, sum(hitflags[b]), stride)

        n_miss = len(miss_bt)
        nfe += n_miss
        hits += sum(p) - n_miss
        if record:
            records.append(IterRecord(
                k=k,
                t=[int(t[b] - strides[b]) if p[b] else -1 for b in range(B)],
                p=p, delta=deltas, hit=hitflags, miss_bt=miss_bt,
                err=errs, stride=strides, tau=tau_k))

    return PicardResult(x_final=X[:, T].copy(), states=X, iters=k,
                        iters_per_traj=iters_per, nfe=nfe, hits=hits,
                        records=records, xhat=Xhat, ehat=Ehat,
                        has_entry=has_entry)
