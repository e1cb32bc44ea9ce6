"""Decision-margin guard for generated inputs.

The GPU keeps fp32 states while the oracle runs in fp64, so a cache distance
(Eq. 4) or a convergence error (Eq. 2) that lies very close to its threshold
could be decided differently by the two. Inputs are therefore rejected when any
decision the oracle actually took lies within ``rel`` (relative) of its
threshold: every delta of a point that had a cache entry (it decides hit or
miss, against the tau_cache of that iteration and trajectory when tau_cache
adapts), and every err_j that the stride depends on (the leading run up to and
including the first err_j > tau, excluding the last window position, whose
error never changes the stride).
"""
from __future__ import annotations

import math


def decision_margins(result, tol, cache_thresh):
    """(min relative |delta - tau_cache| / tau_cache, min relative |err - tau| / tau).

    A margin is +inf when the threshold is 0 (no finite value can sit on the
    other side by rounding: delta >= 0 is never < 0) or no decision was taken.
    """
    m_delta = math.inf
    m_err = math.inf
    for rec in result.records:
        for b, deltas in enumerate(rec.delta):
            thr = rec.tau[b] if rec.tau is not None else cache_thresh   # adapted per iteration
            if thr > 0:
                for d in deltas:
                    if d is not None:
                        m_delta = min(m_delta, abs(d - thr) / thr)
            errs = rec.err[b]
            p = len(errs)
            if tol > 0 and p > 1:
                for j in range(p - 1):
                    m_err = min(m_err, abs(errs[j] - tol) / tol)
                    if errs[j] > tol:
                        break
    return m_delta, m_err


def margins_ok(result, tol, cache_thresh, rel=1e-6):
    md, me = decision_margins(result, tol, cache_thresh)
    return md > rel and me > rel
