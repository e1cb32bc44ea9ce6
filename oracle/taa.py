"""Sliding-window Picard DDIM with triangular Anderson mixing (ParaTAA-style),
with ParaAnya's output cache, fp64 -- TEST INFRASTRUCTURE (see the package
docstring: only tests, smoke() and bench.py's CPU legs use it).

Sec. 2.1 names ParaTAA among the Picard-family samplers that ParaAnya plugs
into, and Sec. 2.2 says the cache changes only which network evaluations run:
the sampler's own update, convergence test and window advance stay as they
are. The paper states no formula for ParaTAA's update. Reading (written down in
the design notes): the Picard map of Eq. 1 followed by Anderson mixing with a
history of depth m (m = 0 or 1), whose coefficient for each window position is
a least-squares fit over that position and the earlier ones -- lower
triangular in time, so that a timestep is mixed only with information from
itself and the timesteps it depends on.

One iteration k, per trajectory with window start t and p positions, state
s = t + j + 1 for window position j (j = 0 .. p-1):

1-6. Cache distance, hit/miss, one batched evaluation of the misses, assembly,
     cache update and drift: exactly as in ``oracle.picard`` (Eq. 3-7).
7.   Picard map (Eq. 1, window form): G_s = x_t + sum_{i <= j} d_{t+i}.
8.   Residual at the current iterate: R_s = G_s - X_s.
9.   Anderson mixing (m = 1). A state that was in the previous iteration's
     window has a history (G'_s, R'_s) from that iteration: states
     t+1 .. min(t+p, e) with e the previous frontier. With dG_s = G_s - G'_s and
     dR_s = R_s - R'_s, position j's coefficient is the least-squares fit over
     the positions j' <= j that have a history:
         gamma_j = sum_{j'<=j} <dR_{s'}, R_{s'}> / sum_{j'<=j} <dR_{s'}, dR_{s'}>
     (0 when the denominator is 0), and the next iterate is
         X_s <- G_s - gamma_j dG_s        (history positions j >= 1)
         X_s <- G_s                        (position 0, positions without a history).
     Position 0 is never mixed: its Picard value depends only on the converged
     window start x_t, so it is already exact -- the fact the stride rule
     relies on when it accepts position 0 whatever its error.
     With m = 0 every position takes X_s <- G_s: plain Picard.
     (G_s, R_s) become the history of state s for the next iteration.
10.  Convergence error (Eq. 2) of the new iterate against the old one, the
     stride rule and the window advance: as in ``oracle.picard``; the Eq. 4
     distances of the next iteration are taken at the new iterate.
"""
from __future__ import annotations

from typing import List, Optional

import numpy as np

from .ddim import drift, step_coefficients
from .picard import IterRecord, PicardResult


def run_taa(alphas, x_init, eps_fn, window, tol, cache_thresh, depth=1,
            use_cache=True, record=True, eta=0.0, noise=None, gammas=None, adapt=None):
    """Cached (or uncached) sliding-window Picard sampling with triangular
    Anderson mixing of history depth ``depth`` (0 or 1), for B trajectories.

    Arguments as ``oracle.picard.run_picard`` (``adapt``: tau_cache adapted per
    trajectory after every iteration, oracle.picard.CacheAdaptation); ``gammas``, if a list, receives
    per iteration the list over trajectories of the mixing coefficients of the
    window positions (0.0 where a position has no history).
    """
    if depth not in (0, 1):
        raise ValueError("depth must be 0 or 1")
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
    X[:, : p0 + 1] = x0[:, None, :]
    Xhat = np.zeros((B, T, D))
    Ehat = np.zeros((B, T, D))
    has_entry = np.zeros((B, T), dtype=bool)
    # Anderson history per state s = 1..T: the previous iteration's G_s and R_s
    Gh = np.zeros((B, T + 1, D))
    Rh = np.zeros((B, T + 1, D))
    has_hist = np.zeros((B, T + 1), dtype=bool)

    t = np.zeros(B, dtype=np.int64)
    active = np.ones(B, dtype=bool)
    iters_per = [0] * B
    nfe = hits = 0
    tau = [float(cache_thresh)] * B
    records: List[IterRecord] = []
    k = 0
    while active.any():
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
                    db.append(None)
                    hb.append(False)
            deltas.append(db)
            hitflags.append(hb)

        # 3. one batched evaluation of every miss
        miss_bt = [(b, int(t[b]) + j) for b in range(B) for j in range(p[b]) if not hitflags[b][j]]
        if miss_bt:
            rows = np.stack([X[b, i] for b, i in miss_bt])
            fresh = eps_fn(rows, np.array([i for _, i in miss_bt]))
        fresh_of = {bt: r for r, bt in enumerate(miss_bt)}

        errs, strides, gam_k = [], [], []
        for b in range(B):
            if not active[b]:
                errs.append([])
                strides.append(0)
                gam_k.append([])
                continue
            tb, pb = int(t[b]), p[b]
            # 4. assembly (Eq. 6)
            eps_w = np.empty((pb, D))
            for j in range(pb):
                i = tb + j
                eps_w[j] = Ehat[b, i] if hitflags[b][j] else fresh[fresh_of[(b, i)]]
            # 5. cache update for misses only (Eq. 7)
            if use_cache:
                for j in range(pb):
                    if not hitflags[b][j]:
                        i = tb + j
                        Xhat[b, i] = X[b, i]
                        Ehat[b, i] = eps_w[j]
                        has_entry[b, i] = True
            # 6. drift at the current latents
            idx = np.arange(tb, tb + pb)
            d = drift(X[b, idx], eps_w, c[idx][:, None], e[idx][:, None],
                      sig[idx][:, None], None if Z is None else Z[b, idx])
            # 7. Picard map, window form of Eq. 1
            G = X[b, tb][None, :] + np.cumsum(d, axis=0)
            s_idx = np.arange(tb + 1, tb + pb + 1)
            X_old = X[b, s_idx].copy()
            # 8. residual at the current iterate
            R = G - X_old
            # 9. triangular Anderson mixing
            gam = np.zeros(pb)
            X_new = G.copy()
            if depth == 1:
                hist = has_hist[b, s_idx]
                dG = G - Gh[b, s_idx]
                dR = R - Rh[b, s_idx]
                num = np.where(hist, np.sum(dR * R, axis=1), 0.0)
                den = np.where(hist, np.sum(dR * dR, axis=1), 0.0)
                num_c, den_c = np.cumsum(num), np.cumsum(den)
                for j in range(1, pb):
                    if hist[j] and den_c[j] > 0.0:
                        gam[j] = num_c[j] / den_c[j]
                X_new = G - gam[:, None] * dG
                Gh[b, s_idx] = G
                Rh[b, s_idx] = R
                has_hist[b, s_idx] = True
            # 10. convergence error (Eq. 2), window advance
            err = np.sum((X_new - X_old) ** 2, axis=1) / D
            X[b, s_idx] = X_new
            lead = 0
            while lead < pb and err[lead] <= tol:
                lead += 1
            stride = min(pb, 1 + lead)
            t_new = tb + stride
            p_new = min(P, T - t_new)
            if t_new + p_new > tb + pb:
                X[b, tb + pb + 1: t_new + p_new + 1] = X[b, tb + pb]
            t[b] = t_new
            iters_per[b] += 1
            if t_new == T:
                active[b] = False
            errs.append([float(v) for v in err])
            strides.append(stride)
            gam_k.append([float(v) for v in gam])
            if adapt is not None:   # tau_cache for the next iteration's hit test
                n_e = sum(1 for dv in deltas[b] if dv is not None)
                tau[b] = adapt.step(tau[b], n_e, sum(hitflags[b]), stride)

        n_miss = len(miss_bt)
        nfe += n_miss
        hits += sum(p) - n_miss
        if gammas is not None:
            gammas.append(gam_k)
        if record:
            records.append(IterRecord(
                k=k, t=[int(t[b] - strides[b]) if p[b] else -1 for b in range(B)],
                p=p, delta=deltas, hit=hitflags, miss_bt=miss_bt, err=errs, stride=strides, tau=tau_k))

    return PicardResult(x_final=X[:, T].copy(), states=X, iters=k, iters_per_traj=iters_per,
                        nfe=nfe, hits=hits, records=records, xhat=Xhat, ehat=Ehat,
                        has_entry=has_entry)
