"""A second, independent statement of the triangular Anderson (depth 1) cached
Picard sampler, in scalar pure Python, to pin ``oracle.taa`` on tiny cases
(T <= 8, D <= 6): plain floats and lists, dicts keyed by absolute state index,
explicit loops for every inner product and prefix sum. Shares no code with
``oracle/``; it reuses only this directory's scalar DDIM step and mixture
posterior (``scalar_picard``).
"""
from scalar_picard import _ddim, _eps


def scalar_cached_taa(alphas, x_init, means, std, P, tol, thresh):
    """Returns (final states per trajectory, per-iteration (misses, strides,
    gammas per trajectory))."""
    T = len(alphas) - 1
    B = len(x_init)
    D = len(x_init[0])
    states = []
    for b in range(B):
        st = {}
        for i in range(0, min(P, T) + 1):
            st[i] = list(x_init[b])
        states.append(st)
    cache = [dict() for _ in range(B)]          # i -> (xhat, ehat)
    hist = [dict() for _ in range(B)]           # state s -> (G, R) of the previous iteration
    start = [0] * B
    log = []
    while any(s < T for s in start):
        plan, misses = [], []
        for b in range(B):
            if start[b] >= T:
                plan.append([])
                continue
            row = []
            for j in range(min(P, T - start[b])):
                i = start[b] + j
                hit = False
                if i in cache[b]:
                    dist = sum(abs(u - w) for u, w in zip(states[b][i], cache[b][i][0])) / D
                    hit = dist < thresh
                row.append(hit)
                if not hit:
                    misses.append((b, i))
            plan.append(row)
        fresh = {(b, i): _eps(states[b][i], alphas[i], means, std) for (b, i) in misses}
        strides, gams = [], []
        for b in range(B):
            if start[b] >= T:
                strides.append(0)
                gams.append([])
                continue
            t = start[b]
            p = len(plan[b])
            eps_of = {}
            for j in range(p):
                i = t + j
                if plan[b][j]:
                    eps_of[i] = cache[b][i][1]
                else:
                    eps_of[i] = fresh[(b, i)]
                    cache[b][i] = (list(states[b][i]), eps_of[i])
            # the Picard map from the fixed start state, step by step
            G = {}
            run = list(states[b][t])
            for j in range(p):
                i = t + j
                stepped = _ddim(states[b][i], eps_of[i], alphas[i], alphas[i + 1])
                run = [r + (s_ - x_) for r, s_, x_ in zip(run, stepped, states[b][i])]
                G[i + 1] = run
            # mixing: prefix sums over the window positions that have a history
            num_c = den_c = 0.0
            new, gam_b = {}, []
            for j in range(p):
                s = t + j + 1
                g = G[s]
                r = [gv - xv for gv, xv in zip(g, states[b][s])]
                gamma = 0.0
                if s in hist[b]:
                    gp, rp = hist[b][s]
                    dr = [u - w for u, w in zip(r, rp)]
                    num_c += sum(u * w for u, w in zip(dr, r))
                    den_c += sum(u * u for u in dr)
                    if den_c > 0.0 and j > 0:   # the first window state is exact: not mixed
                        gamma = num_c / den_c
                    new[s] = [gv - gamma * (gv - gpv) for gv, gpv in zip(g, gp)]
                else:
                    new[s] = list(g)
                hist[b][s] = (g, r)
                gam_b.append(gamma)
            errs = [sum((u - w) ** 2 for u, w in zip(new[t + j + 1], states[b][t + j + 1])) / D for j in range(p)]
            for s, v in new.items():
                states[b][s] = v
            lead = 0
            while lead < p and errs[lead] <= tol:
                lead += 1
            stride = min(p, lead + 1)
            nt = t + stride
            npp = min(P, T - nt)
            for i in range(t + p + 1, nt + npp + 1):
                states[b][i] = list(states[b][t + p])
            start[b] = nt
            strides.append(stride)
            gams.append(gam_b)
        log.append((misses, strides, gams))
    return [states[b][T] for b in range(B)], log
