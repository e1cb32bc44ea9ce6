"""Pins for the oracle's cached Picard sampler (CPU only).

* tol = 0, no cache: Picard reproduces serial DDIM for every window size,
  including window = T and window = 1 (Sec. 2.1; Eq. 1 is a fixed-point
  iteration whose fixed point is the serial trajectory).
* tau_cache = 0: strict "<" in Eq. 5 never hits, so the cached sampler is the
  uncached one bit for bit (separate code path in the oracle).
* tau_cache huge: every point is evaluated exactly once, NFE = B * T.
* Counting: NFE = sum of misses, hits + misses = sum of window sizes,
  stride >= 1, iterations <= T; first entries are misses (Sec. 2.2).
* The cache invariant ehat = eps_theta(xhat) holds for every entry (Sec. 2.2).
* Threshold edges: a delta equal to tau_cache is a miss, an err equal to tau
  counts as converged (Eq. 5 strict, Eq. 2 non-strict).
* Batched trajectories are independent and misses come out trajectory-major.
* A separate scalar pure-Python implementation agrees on tiny cases.
"""
import numpy as np
import pytest

import workload as W
from oracle import run_picard, serial_ddim
from oracle.gmm import make_eps_fn
from oracle.guard import decision_margins, margins_ok
from scalar_picard import scalar_cached_picard


def _small(T=12, P=5, B=2, D=6, K=3, seed=0):
    a = W.alphas_cumprod(T)
    rng = np.random.default_rng(100 + seed)
    x0 = rng.standard_normal((B, D))
    mu = rng.standard_normal((K, D))
    return a, x0, mu, make_eps_fn(a, mu, 0.5)


@pytest.mark.parametrize("P", [1, 3, 7, 12])
def test_tol0_uncached_equals_serial(P):
    a, x0, mu, f = _small(T=12, P=P)
    ser = serial_ddim(a, x0, f)
    r = run_picard(a, x0, f, P, tol=0.0, cache_thresh=0.0, use_cache=False)
    np.testing.assert_allclose(r.states, ser, rtol=1e-11, atol=1e-11)
    assert r.iters <= 12
    if P == 1:
        assert r.iters == 12 and r.nfe == 2 * 12


def test_tol0_window_T_sd_schedule():
    a, x0, mu, f = _small(T=40, P=40, B=1, D=10, K=4)
    ser = serial_ddim(a, x0, f)
    r = run_picard(a, x0, f, 40, tol=0.0, cache_thresh=0.0, use_cache=False)
    np.testing.assert_allclose(r.x_final, ser[:, -1], rtol=1e-11, atol=1e-11)


def test_cache_thresh_zero_equals_uncached():
    a, x0, mu, f = _small(T=20, P=8, B=3)
    rc = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=0.0, use_cache=True)
    ru = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=0.0, use_cache=False)
    assert rc.hits == 0 and rc.nfe == ru.nfe and rc.iters == ru.iters
    assert np.array_equal(rc.states, ru.states)
    assert [r.miss_bt for r in rc.records] == [r.miss_bt for r in ru.records]


def test_huge_threshold_evaluates_each_point_once():
    a, x0, mu, f = _small(T=20, P=8, B=3)
    r = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=1e30)
    assert r.nfe == 3 * 20
    seen = [bt for rec in r.records for bt in rec.miss_bt]
    assert len(seen) == len(set(seen)) == 60


def test_counting_invariants_and_first_entry():
    a, x0, mu, f = _small(T=30, P=10, B=2, D=8, K=4, seed=1)
    r = run_picard(a, x0, f, 10, tol=1e-3, cache_thresh=0.05)
    assert r.nfe == sum(len(rec.miss_bt) for rec in r.records)
    assert r.nfe + r.hits == sum(sum(rec.p) for rec in r.records)
    assert r.iters <= 30
    entered = [set(), set()]
    for rec in r.records:
        for b in range(2):
            if rec.p[b] == 0:
                continue
            assert rec.stride[b] >= 1
            for j in range(rec.p[b]):
                i = rec.t[b] + j
                if i not in entered[b]:
                    assert rec.delta[b][j] is None and not rec.hit[b][j]
                    entered[b].add(i)
                else:
                    assert rec.delta[b][j] is not None
        # canonical order: trajectory-major, ascending point index
        assert rec.miss_bt == sorted(rec.miss_bt)
    assert r.hits > 0


def test_cache_invariant():
    a, x0, mu, f = _small(T=30, P=10, B=2, D=8, K=4, seed=2)
    r = run_picard(a, x0, f, 10, tol=1e-3, cache_thresh=0.08)
    for b in range(2):
        for i in range(30):
            if r.has_entry[b, i]:
                fresh = f(r.xhat[b, i][None], np.array([i]))[0]
                np.testing.assert_array_equal(r.ehat[b, i], fresh)
    assert r.has_entry.all()


def test_threshold_edges_strict_and_nonstrict():
    a, x0, mu, f = _small(T=24, P=8, B=1, D=8, K=4, seed=3)
    base = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=0.05)
    # pick a recorded delta; with tau_cache equal to it the point must miss,
    # with the next float above it must hit (only the first decision is compared)
    for k, rec in enumerate(base.records):
        ds = [d for d in rec.delta[0] if d is not None]
        if ds:
            d0 = ds[0]
            j0 = rec.delta[0].index(d0)
            break
    eq = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=d0, max_iters=k + 1)
    up = run_picard(a, x0, f, 8, tol=1e-3, cache_thresh=np.nextafter(d0, np.inf),
                    max_iters=k + 1)
    assert eq.records[k].delta[0][j0] == d0 and not eq.records[k].hit[0][j0]
    assert up.records[k].hit[0][j0]
    # err equal to tau converges (Eq. 2 uses <=)
    rec0 = base.records[0]
    e0 = rec0.err[0][0]
    r_eq = run_picard(a, x0, f, 8, tol=e0, cache_thresh=0.05, max_iters=1)
    r_dn = run_picard(a, x0, f, 8, tol=np.nextafter(e0, 0), cache_thresh=0.05, max_iters=1)
    assert r_eq.records[0].err[0][0] == e0
    assert r_eq.records[0].stride[0] >= 2
    assert r_dn.records[0].stride[0] == 1


def test_batched_equals_separate():
    a, x0, mu, f = _small(T=18, P=6, B=3, seed=4)
    rb = run_picard(a, x0, f, 6, tol=1e-3, cache_thresh=0.05)
    for b in range(3):
        rs = run_picard(a, x0[b:b + 1], f, 6, tol=1e-3, cache_thresh=0.05)
        np.testing.assert_array_equal(rs.states[0], rb.states[b])
        assert rs.iters == rb.iters_per_traj[b]
        mine = [[(0, i) for (bb, i) in rec.miss_bt if bb == b] for rec in rb.records]
        mine = [m for m, rec in zip(mine, rb.records) if rec.p[b] > 0]
        assert mine == [rec.miss_bt for rec in rs.records]


@pytest.mark.parametrize("T,P,thresh,tol,seed", [
    (4, 2, 0.05, 1e-3, 0), (5, 2, 0.5, 1e-2, 1), (6, 3, 0.2, 1e-2, 2),
    (4, 4, 1e9, 0.0, 3), (6, 2, 0.0, 0.05, 4)])
def test_scalar_brute_force_agrees(T, P, thresh, tol, seed):
    rng = np.random.default_rng(seed)
    B, D, K = 2, 4, 2
    a = W.alphas_cumprod(T)
    x0 = rng.standard_normal((B, D))
    mu = rng.standard_normal((K, D))
    r = run_picard(a, x0, make_eps_fn(a, mu, 0.5), P, tol, thresh)
    finals, log = scalar_cached_picard(list(a), x0.tolist(), mu.tolist(), 0.5, P, tol, thresh)
    assert [m for m, _, _ in log] == [rec.miss_bt for rec in r.records]
    assert [s for _, s, _ in log] == [rec.stride for rec in r.records]
    for (_, _, dists), rec in zip(log, r.records):
        for db_s, db_o in zip(dists, rec.delta):
            assert len(db_s) == len(db_o)
            for u, v in zip(db_s, db_o):
                assert (u is None) == (v is None)
                if u is not None:
                    assert v == pytest.approx(u, rel=1e-12, abs=1e-15)
    np.testing.assert_allclose(np.array(finals), r.x_final, rtol=1e-12, atol=1e-12)


def test_guard_reports_margins():
    w = W.TINY
    a, x0, mu = W.inputs(w)
    r = run_picard(a, x0, make_eps_fn(a, mu, w.gmm_std), w.window, w.tol, w.cache_thresh)
    md, me = decision_margins(r, w.tol, w.cache_thresh)
    assert 0 < md < np.inf and 0 < me < np.inf
    assert margins_ok(r, w.tol, w.cache_thresh)
    assert not margins_ok(r, w.tol, w.cache_thresh, rel=1.0)


# ---- online adaptation of tau_cache (CacheAdaptation) -----------------------

from oracle.picard import CacheAdaptation  # noqa: E402

ADAPT_W = W.Workload("adapt", T=40, window=16, batch=2, latent_shape=(2, 4, 4), K=3, tol=1e-3,
                     cache_thresh=0.02, seed=6)


def _adapt_run(w, adapt, thr=None):
    a, x0, mu = W.inputs(w)
    return run_picard(a, x0, make_eps_fn(a, mu, w.gmm_std), w.window, w.tol,
                      w.cache_thresh if thr is None else thr, adapt=adapt)


def test_adaptation_with_rate_zero_is_fixed_tau():
    fixed = _adapt_run(ADAPT_W, None)
    off = _adapt_run(ADAPT_W, CacheAdaptation(rate=0.0, target=0.5))
    assert np.array_equal(fixed.states, off.states)
    assert [r.miss_bt for r in fixed.records] == [r.miss_bt for r in off.records]
    assert all(t == ADAPT_W.cache_thresh for r in off.records for t in r.tau)


def test_adaptation_limits():
    """tau_cache 0 stays 0 (uncached); a floor of +inf-like size hits every
    point with an entry (NFE = B * T); tau never leaves [tau_min, tau_max]."""
    zero = _adapt_run(ADAPT_W, CacheAdaptation(rate=0.5, target=1.0), thr=0.0)
    assert zero.hits == 0 and all(t == 0.0 for r in zero.records for t in r.tau)
    always = _adapt_run(ADAPT_W, CacheAdaptation(rate=0.5, target=0.0, tau_min=1e30), thr=1e30)
    assert always.nfe == ADAPT_W.batch * ADAPT_W.T
    bounded = _adapt_run(ADAPT_W, CacheAdaptation(rate=0.5, target=0.9, tau_min=0.01, tau_max=0.04))
    taus = [t for r in bounded.records for t in r.tau]
    assert min(taus[ADAPT_W.batch:]) >= 0.01 and max(taus) <= 0.04
    assert len(set(taus)) > 1   # it did move


def test_adaptation_raises_reuse_toward_the_target():
    """Starting where the fixed threshold gives no hits, a high target raises
    tau and the run reuses more cache entries than the fixed run."""
    fixed = _adapt_run(ADAPT_W, None, thr=0.005)
    adapt = _adapt_run(ADAPT_W, CacheAdaptation(rate=1.0, target=0.9), thr=0.005)
    assert adapt.hits > fixed.hits


@pytest.mark.parametrize("rate,target,lo,hi,thr,seed", [(0.5, 0.8, 0.0, 1.0, 0.02, 0), (1.0, 0.3, 0.005, 0.2, 0.05, 1),
                                                        (0.25, 1.0, 0.0, 0.5, 0.01, 2)])
def test_adaptation_scalar_second_implementation_agrees(rate, target, lo, hi, thr, seed):
    w = W.Workload("adapt scalar", T=8, window=4, batch=2, latent_shape=(1, 2, 3), K=3, tol=1e-3,
                   cache_thresh=thr, seed=seed)
    a, x0, mu = W.inputs(w)
    r = run_picard(a, x0, make_eps_fn(a, mu, w.gmm_std), w.window, w.tol, thr,
                   adapt=CacheAdaptation(rate=rate, target=target, tau_min=lo, tau_max=hi))
    taus = []
    finals, log = scalar_cached_picard(list(a), x0.astype(np.float64).tolist(), mu.astype(np.float64).tolist(),
                                       0.5, w.window, w.tol, thr, adapt=(rate, target, lo, hi), taus=taus)
    assert len(log) == r.iters
    for rec, (misses, strides, _), tk in zip(r.records, log, taus):
        assert rec.miss_bt == misses and rec.stride == strides
        assert rec.tau == tk
    assert np.abs(np.array(finals) - r.x_final).max() <= 1e-12 * np.abs(r.x_final).max()
