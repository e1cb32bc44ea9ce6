"""Pins of the triangular Anderson (ParaTAA-style) cached Picard oracle,
``oracle.taa.run_taa``, against what the method and the mathematics fix:

* history depth 0 is the plain Picard update: identical to ``run_picard``
  (states, decisions, counters), with and without cache and stochastic steps;
* tol = 0 (no position is accepted before it stops changing) reproduces serial
  DDIM for windows 1, 3, 7 and T, with depth 1 mixing active in between;
* tau_cache = 0 equals the separate uncached path; an always-hit cache
  evaluates every timestep exactly once (NFE = B * T);
* the mixing coefficients are 0 where a position has no history, and every
  iteration's NFE + hits equals the window points it planned;
* a scalar pure-Python second implementation agrees on tiny cases (decisions
  exactly, coefficients and states to 1e-12).
Planted mistakes in the oracle's mixing (a sign, a dropped prefix sum, the
history of the wrong iteration, mixing positions without a history) each fail
one of these.
"""
import numpy as np
import pytest

import workload as W
from oracle import run_picard, serial_ddim
from oracle.gmm import make_eps_fn
from oracle.taa import run_taa
from scalar_taa import scalar_cached_taa


def _inputs(w):
    a, x0, mu = W.inputs(w)
    return a, x0, make_eps_fn(a, mu, w.gmm_std), mu


SMALL = W.Workload("taa small", T=24, window=8, batch=2, latent_shape=(2, 4, 4), K=3,
                   tol=1e-3, cache_thresh=0.05, seed=4)


@pytest.mark.parametrize("w", [SMALL, SMALL.with_(cache_thresh=0.0), SMALL.with_(eta=1.0, T=20),
                               W.TINY], ids=["cached", "uncached", "stochastic", "tiny"])
def test_depth_zero_is_picard(w):
    a, x0, f, _ = _inputs(w)
    kw = dict(eta=w.eta, noise=W.noise(w))
    p = run_picard(a, x0, f, w.window, w.tol, w.cache_thresh, **kw)
    q = run_taa(a, x0, f, w.window, w.tol, w.cache_thresh, depth=0, **kw)
    assert np.array_equal(p.states, q.states)
    assert (p.iters, p.nfe, p.hits) == (q.iters, q.nfe, q.hits)
    assert [r.stride for r in p.records] == [r.stride for r in q.records]
    assert [r.miss_bt for r in p.records] == [r.miss_bt for r in q.records]


@pytest.mark.parametrize("window", [1, 3, 7, 24])
def test_tol_zero_reproduces_serial_ddim(window):
    w = SMALL.with_(tol=0.0, cache_thresh=0.0)
    a, x0, f, _ = _inputs(w)
    gam = []
    r = run_taa(a, x0, f, window, 0.0, 0.0, depth=1, gammas=gam)
    ser = serial_ddim(a, x0, f)
    scale = np.abs(ser).max()
    assert np.abs(r.states - ser).max() <= 1e-12 * scale
    if window > 2:   # the mixing was active on the way (nonzero coefficients)
        assert any(abs(g) > 0.0 for it in gam for tr in it for g in tr)


def test_uncached_equals_cache_threshold_zero():
    w = SMALL
    a, x0, f, _ = _inputs(w)
    u = run_taa(a, x0, f, w.window, w.tol, 0.0, depth=1, use_cache=False)
    c = run_taa(a, x0, f, w.window, w.tol, 0.0, depth=1)
    assert np.array_equal(u.states, c.states) and u.nfe == c.nfe and c.hits == 0


def test_always_hit_evaluates_each_timestep_once():
    w = SMALL
    a, x0, f, _ = _inputs(w)
    r = run_taa(a, x0, f, w.window, w.tol, 1e30, depth=1)
    assert r.nfe == w.batch * w.T


def test_coefficients_only_where_a_history_exists_and_counts():
    w = SMALL
    a, x0, f, _ = _inputs(w)
    gam = []
    r = run_taa(a, x0, f, w.window, w.tol, w.cache_thresh, depth=1, gammas=gam)
    assert all(g == 0.0 for tr in gam[0] for g in tr)      # first iteration: nothing to mix with
    assert all(tr[0] == 0.0 for it in gam for tr in it if tr)  # the first window state is never mixed
    for rec, gk in zip(r.records, gam):
        assert sum(rec.p) == len(rec.miss_bt) + sum(h for hb in rec.hit for h in hb)
        for b in range(w.batch):
            assert len(gk[b]) == rec.p[b]
    assert r.nfe + r.hits == sum(sum(rec.p) for rec in r.records)


@pytest.mark.parametrize("T,P,thresh,tol,seed", [(6, 3, 0.3, 1e-4, 0), (8, 4, 0.05, 1e-3, 1),
                                                 (7, 7, 0.2, 1e-6, 2), (5, 2, 1e9, 1e-3, 3)])
def test_scalar_second_implementation_agrees(T, P, thresh, tol, seed):
    w = W.Workload("taa scalar", T=T, window=P, batch=2, latent_shape=(1, 2, 3), K=3, tol=tol,
                   cache_thresh=thresh, seed=seed)
    a, x0, f, mu = _inputs(w)
    gam = []
    r = run_taa(a, x0, f, P, tol, thresh, depth=1, gammas=gam)
    finals, log = scalar_cached_taa(list(a), x0.astype(np.float64).tolist(), mu.astype(np.float64).tolist(),
                                     0.5, P, tol, thresh)
    assert len(log) == r.iters
    for rec, (misses, strides, gams), gk in zip(r.records, log, gam):
        assert rec.miss_bt == misses
        assert [s for s in rec.stride] == strides
        for b in range(w.batch):
            assert np.allclose(gk[b], gams[b], rtol=1e-12, atol=1e-12)
    scale = np.abs(r.x_final).max()
    assert np.abs(np.array(finals) - r.x_final).max() <= 1e-12 * scale
