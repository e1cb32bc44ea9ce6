"""A second, independent statement of cached Picard DDIM, in scalar pure Python.

Used only to pin the vectorised fp64 oracle on tiny cases (T <= 6, D <= 6):
plain Python floats and lists, explicit loops over coordinates, its own DDIM
step (predict x0 then re-noise), its own mixture posterior, its own window
bookkeeping (a dict of states keyed by absolute index). It shares no code with
``oracle/``.
"""
import math


def _ddim(x, eps, a, an):
    out = []
    for xd, ed in zip(x, eps):
        x0 = (xd - math.sqrt(1.0 - a) * ed) / math.sqrt(a)
        out.append(math.sqrt(an) * x0 + math.sqrt(1.0 - an) * ed)
    return out


def _ddpm(x, eps, a, an, z):
    """Ancestral DDPM step in the posterior form q(x_{t-1} | x_t, x0): the
    mean (sqrt(an) beta / (1 - a)) x0 + (sqrt(alpha) (1 - an) / (1 - a)) x and
    the variance (1 - an) / (1 - a) * beta, with beta = 1 - a / an."""
    beta = 1.0 - a / an
    alpha = 1.0 - beta
    var = (1.0 - an) / (1.0 - a) * beta
    out = []
    for xd, ed, zd in zip(x, eps, z):
        x0 = (xd - math.sqrt(1.0 - a) * ed) / math.sqrt(a)
        mean = math.sqrt(an) * beta / (1.0 - a) * x0 + math.sqrt(alpha) * (1.0 - an) / (1.0 - a) * xd
        out.append(mean + math.sqrt(var) * zd)
    return out


def _eps(x, a, means, std):
    K = len(means)
    v = a * std * std + 1.0 - a
    logits = []
    for mu in means:
        sq = 0.0
        for xd, md in zip(x, mu):
            diff = xd - math.sqrt(a) * md
            sq += diff * diff
        logits.append(math.log(1.0 / K) - sq / (2.0 * v))
    top = max(logits)
    ws = [math.exp(l - top) for l in logits]
    tot = sum(ws)
    out = []
    for d in range(len(x)):
        m = sum(ws[k] / tot * means[k][d] for k in range(K))
        out.append(math.sqrt(1.0 - a) / v * (x[d] - math.sqrt(a) * m))
    return out


def scalar_cached_picard(alphas, x_init, means, std, P, tol, thresh, noise=None, adapt=None, taus=None):
    """Returns (final states per trajectory, per-iteration (misses, strides, distances)).

    noise: None for DDIM; else the draws noise[b][i] of every trajectory and
    step, and every step is an ancestral DDPM step (eta = 1).
    adapt: None, or (rate, target, lo, hi): each trajectory's threshold moves
    after every iteration -- up by the factor 1 + rate when fewer than
    target of its points with an entry hit and its window moved by more than
    one point, down by that factor when at least target of them hit, never
    outside [lo, hi], unchanged when no point had an entry. taus, if a list,
    receives every iteration's thresholds."""
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
    start = [0] * B
    log = []
    thr_b = [thresh] * B
    while any(s < T for s in start):
        if taus is not None:
            taus.append(list(thr_b))
        # decide hits and misses, trajectory by trajectory, point by point
        plan = []
        misses = []
        dists = []
        for b in range(B):
            if start[b] >= T:
                plan.append([])
                dists.append([])
                continue
            p = min(P, T - start[b])
            row = []
            drow = []
            for j in range(p):
                i = start[b] + j
                hit = False
                dist = None
                if i in cache[b]:
                    xh = cache[b][i][0]
                    dist = sum(abs(u - w) for u, w in zip(states[b][i], xh)) / D
                    hit = dist < thr_b[b]
                row.append(hit)
                drow.append(dist)
                if not hit:
                    misses.append((b, i))
            plan.append(row)
            dists.append(drow)
        fresh = {}
        for (b, i) in misses:
            fresh[(b, i)] = _eps(states[b][i], alphas[i], means, std)
        strides = []
        for b in range(B):
            if start[b] >= T:
                strides.append(0)
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
            # sequential recomputation of the window from the fixed start state
            new = {}
            run = list(states[b][t])
            for j in range(p):
                i = t + j
                if noise is None:
                    stepped = _ddim(states[b][i], eps_of[i], alphas[i], alphas[i + 1])
                else:
                    stepped = _ddpm(states[b][i], eps_of[i], alphas[i], alphas[i + 1], noise[b][i])
                drift = [s_ - x_ for s_, x_ in zip(stepped, states[b][i])]
                run = [r + d for r, d in zip(run, drift)]
                new[i + 1] = run
            errs = []
            for j in range(p):
                i = t + j + 1
                errs.append(sum((u - w) ** 2 for u, w in zip(new[i], states[b][i])) / D)
            for i, v in new.items():
                states[b][i] = v
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
            if adapt is not None:
                rate, target, lo, hi = adapt
                had = [dv for dv in dists[b] if dv is not None]
                if had:
                    n_hit = sum(1 for h in plan[b] if h)
                    if n_hit / len(had) < target:
                        if stride > 1:
                            thr_b[b] = min(thr_b[b] * (1.0 + rate), hi)
                    else:
                        thr_b[b] = max(thr_b[b] / (1.0 + rate), lo)
        log.append((misses, strides, dists))
    finals = [states[b][T] for b in range(B)]
    return finals, log
