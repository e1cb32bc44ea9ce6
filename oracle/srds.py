"""Parareal (SRDS-style) DDIM sampling with ParaAnya's output cache, fp64.

Sec. 2.1 names Parareal-based samplers (SRDS): a coarse solver initialises the
trajectory and fine solvers refine it. Sec. 2.2 (last paragraph on Parareal)
applies the cache to the network evaluations of both solvers and leaves the
Parareal update unchanged. The paper gives no more than that; the rest is the
published Parareal scheme written out, with these readings (listed in the
design notes):

* Blocks: s = ceil(sqrt(T)) steps per block, N = ceil(T / s) blocks; block n
  covers sampling indices [n s, min((n + 1) s, T)) and ends at index e_n.
* Fine solver F_n(u): the DDIM steps of block n, starting from u.
* Coarse solver G_n(u): one DDIM step from alpha-bar at n s straight to
  alpha-bar at e_n, with eps evaluated at (u, n s).
* Iteration 0: U_0 = x_init, U_{n+1} = G_n(U_n) in block order.
* Iteration k >= 1: first the fine sweep, F_n(U_n^{k-1}) for every block (the
  evaluations at step j of every block form one batch), then the correction in
  block order: U_0^k = x_init,
      U_{n+1}^k = G_n(U_n^k) + F_n(U_n^{k-1}) - G_n(U_n^{k-1}).
* Convergence (Eq. 2 applied to the block boundaries):
      err = max_{n >= 1} (1/D) ||U_n^k - U_n^{k-1}||^2 <= tol,
  or k = N, after which Parareal is exact (U_N is the serial fine solution). A
  converged trajectory is frozen: no further evaluations, U kept.
* Cache: one entry per (trajectory, sampling index), shared by the coarse and
  fine evaluations at that index. An evaluation with an entry whose distance
  (Eq. 4) to the current input is below tau_cache (strict, Eq. 5) reuses the
  cached eps; otherwise it is a miss, evaluated fresh, and the entry becomes
  (input, eps) (Eq. 7). Within one batch every row is tested against the cache
  as it was before the batch.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field
from typing import List

import numpy as np


def srds_blocks(T):
    """(s, N, starts, ends) of the block partition (s = ceil(sqrt(T)))."""
    s = int(math.ceil(math.sqrt(T)))
    N = (T + s - 1) // s
    starts = [n * s for n in range(N)]
    ends = [min((n + 1) * s, T) for n in range(N)]
    return s, N, starts, ends


def ddim_jump(x, eps, a_from, a_to):
    """One DDIM (eta = 0) step from alpha-bar a_from to a_to (any gap): predict
    x0, then re-noise to the target level."""
    x0 = (x - np.sqrt(1.0 - a_from) * eps) / np.sqrt(a_from)
    return np.sqrt(a_to) * x0 + np.sqrt(1.0 - a_to) * eps


@dataclass
class SrdsResult:
    x_final: np.ndarray                # [B][D], U_N of every trajectory
    iters: int                         # Parareal iterations after the coarse initialisation
    nfe: int
    hits: int
    iters_per_traj: List[int]
    boundaries: List[np.ndarray] = field(default_factory=list)  # U after init and each iteration, [B][N+1][D]
    errs: List[List[float]] = field(default_factory=list)       # per iteration, per trajectory (None if frozen)
    batches: List[list] = field(default_factory=list)           # per evaluation batch: (b, i, hit, delta)


def run_srds(alphas, x_init, eps_fn, tol, cache_thresh, use_cache=True, max_iters=None):
    """Cached Parareal DDIM for B trajectories.

    alphas : fp64 [T+1] sampling-order alpha-bar (alphas[T] == 1).
    x_init : [B][D]; eps_fn(x_rows [n][D], idx [n]) -> [n][D].
    tol, cache_thresh : tau (block-boundary error) and tau_cache.
    use_cache=False evaluates every network call (separate path).
    """
    a = np.asarray(alphas, dtype=np.float64)
    T = len(a) - 1
    x0 = np.asarray(x_init, dtype=np.float64)
    B, D = x0.shape
    s, N, starts, ends = srds_blocks(T)
    xhat = np.zeros((B, T, D))
    ehat = np.zeros((B, T, D))
    has = np.zeros((B, T), dtype=bool)
    stats = {"nfe": 0, "hits": 0}
    batches = []

    def evaluate(rows, bs, idx):
        """Cache test for every row against the cache as it stands, one batch of misses."""
        out = np.empty_like(rows)
        miss = []
        log = []
        for r, (b, i) in enumerate(zip(bs, idx)):
            hit = False
            delta = None
            if use_cache and has[b, i]:
                delta = float(np.sum(np.abs(rows[r] - xhat[b, i])) / D)
                hit = delta < cache_thresh
            log.append((int(b), int(i), hit, delta))
            if hit:
                out[r] = ehat[b, i]
            else:
                miss.append(r)
        if miss:
            fresh = eps_fn(rows[miss], np.asarray(idx)[miss])
            for k, r in enumerate(miss):
                out[r] = fresh[k]
                if use_cache:
                    b, i = bs[r], idx[r]
                    xhat[b, i] = rows[r]
                    ehat[b, i] = fresh[k]
                    has[b, i] = True
        stats["nfe"] += len(miss)
        stats["hits"] += len(rows) - len(miss)
        batches.append(log)
        return out

    U = np.empty((B, N + 1, D))
    U[:, 0] = x0
    G = np.empty((B, N, D))
    # iteration 0: coarse sweep
    for n in range(N):
        eps = evaluate(U[:, n].copy(), list(range(B)), [starts[n]] * B)
        G[:, n] = ddim_jump(U[:, n], eps, a[starts[n]], a[ends[n]])
        U[:, n + 1] = G[:, n]
    boundaries = [U.copy()]
    errs_log = []
    active = np.ones(B, dtype=bool)
    iters_per = [0] * B
    k = 0
    limit = N if max_iters is None else min(N, max_iters)
    while active.any() and k < limit:
        k += 1
        act = [b for b in range(B) if active[b]]
        # fine sweep from the previous boundaries
        Y = U[act, :N].copy()                          # [A][N][D]
        for j in range(s):
            rows, bs, idx, where = [], [], [], []
            for ai, b in enumerate(act):
                for n in range(N):
                    i = starts[n] + j
                    if i < ends[n]:
                        rows.append(Y[ai, n])
                        bs.append(b)
                        idx.append(i)
                        where.append((ai, n))
            if not rows:
                continue
            eps = evaluate(np.stack(rows), bs, idx)
            for r, (ai, n) in enumerate(where):
                i = idx[r]
                Y[ai, n] = ddim_jump(Y[ai, n], eps[r], a[i], a[i + 1])
        F = Y
        # correction sweep in block order
        Unew = U.copy()
        for n in range(N):
            eps = evaluate(Unew[act, n].copy(), act, [starts[n]] * len(act))
            g_new = ddim_jump(Unew[act, n], eps, a[starts[n]], a[ends[n]])
            Unew[act, n + 1] = g_new + F[:, n] - G[act, n]
            G[act, n] = g_new
        err_k = [None] * B
        for b in act:
            e = float(np.max(np.sum((Unew[b, 1:] - U[b, 1:]) ** 2, axis=1) / D))
            err_k[b] = e
            iters_per[b] += 1
            if e <= tol:
                active[b] = False
        U = Unew
        boundaries.append(U.copy())
        errs_log.append(err_k)
    return SrdsResult(x_final=U[:, N].copy(), iters=k, nfe=stats["nfe"], hits=stats["hits"],
                      iters_per_traj=iters_per, boundaries=boundaries, errs=errs_log, batches=batches)
