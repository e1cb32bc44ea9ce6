"""Pins of the Parareal (SRDS-style) oracle with the output cache.

Parareal has exact properties that do not come from its own formulas: with the
cache off it reproduces the serial fine solver after N iterations, and after k
iterations its first k block boundaries already equal the serial trajectory.
Together with the cache rule's counting invariants these tie every part of the
oracle (block partition, coarse jump, fine sweep, correction order, cache test
and update) to something else.
"""
import numpy as np
import pytest

import workload as W
from oracle.ddim import serial_ddim, ddim_step
from oracle.gmm import make_eps_fn
from oracle.srds import run_srds, srds_blocks, ddim_jump


def _case(T, B=2, D=24, K=3, seed=0):
    rng = np.random.default_rng(seed)
    a = W.alphas_cumprod(T)
    return a, rng.standard_normal((B, D)), rng.standard_normal((K, D))


@pytest.mark.parametrize("T", [1, 2, 5, 16, 30, 100])
def test_block_partition(T):
    s, N, starts, ends = srds_blocks(T)
    assert s * s >= T and (s - 1) * (s - 1) < T
    assert starts[0] == 0 and ends[-1] == T
    assert all(ends[n] == starts[n + 1] for n in range(N - 1))
    assert all(0 < ends[n] - starts[n] <= s for n in range(N))


def test_jump_of_one_step_is_the_ddim_step():
    a = W.alphas_cumprod(20)
    rng = np.random.default_rng(3)
    x, e = rng.standard_normal((2, 8))
    for i in range(20):
        np.testing.assert_allclose(ddim_jump(x, e, a[i], a[i + 1]), ddim_step(x, e, a[i], a[i + 1]),
                                   rtol=1e-14, atol=1e-14)


@pytest.mark.parametrize("T", [2, 5, 16, 30])
def test_uncached_parareal_is_exact_after_n_iterations(T):
    a, x0, mu = _case(T)
    fn = make_eps_fn(a, mu, 0.5)
    serial = serial_ddim(a, x0, fn)
    r = run_srds(a, x0, fn, 0.0, 0.0)
    s, N, starts, ends = srds_blocks(T)
    assert r.iters == N
    np.testing.assert_allclose(r.x_final, serial[:, -1], rtol=1e-11, atol=1e-11)


@pytest.mark.parametrize("T", [9, 16, 30])
def test_first_k_boundaries_exact_after_k_iterations(T):
    """The Parareal property: after iteration k the boundaries U_0..U_k equal
    the serial trajectory at the block starts."""
    a, x0, mu = _case(T, seed=1)
    fn = make_eps_fn(a, mu, 0.5)
    serial = serial_ddim(a, x0, fn)
    s, N, starts, ends = srds_blocks(T)
    bound_idx = starts + [T]
    r = run_srds(a, x0, fn, 0.0, 0.0)
    for k, U in enumerate(r.boundaries):          # k = 0 is the coarse initialisation
        for n in range(min(k, N) + 1):
            np.testing.assert_allclose(U[:, n], serial[:, bound_idx[n]], rtol=1e-11, atol=1e-11)
        if k == 0:  # the coarse jump over a block of s > 1 steps is not the fine solution
            assert not np.allclose(U[:, 1], serial[:, bound_idx[1]], rtol=1e-6, atol=1e-6)


def test_threshold_zero_equals_uncached_path():
    a, x0, mu = _case(16, seed=2)
    fn = make_eps_fn(a, mu, 0.5)
    r0 = run_srds(a, x0, fn, 1e-3, 0.0)
    ru = run_srds(a, x0, fn, 1e-3, 0.05, use_cache=False)
    assert np.array_equal(r0.x_final, ru.x_final)
    assert r0.nfe == ru.nfe and r0.hits == 0 and ru.hits == 0
    assert r0.iters == ru.iters


def test_counting_invariants_and_first_entries():
    a, x0, mu = _case(30, B=3, seed=4)
    fn = make_eps_fn(a, mu, 0.5)
    r = run_srds(a, x0, fn, 1e-4, 0.05)
    evals = sum(len(b) for b in r.batches)
    assert r.nfe + r.hits == evals
    assert r.nfe == sum(1 for b in r.batches for (_, _, hit, _) in b if not hit)
    seen = set()
    for batch in r.batches:
        for (b, i, hit, _) in batch:
            if (b, i) not in seen:
                assert not hit                 # first entry is a miss (Sec. 2.2)
            seen.add((b, i))


def test_huge_threshold_evaluates_each_index_once():
    T, B = 30, 2
    a, x0, mu = _case(T, B=B, seed=5)
    fn = make_eps_fn(a, mu, 0.5)
    r = run_srds(a, x0, fn, 0.0, 1e12, max_iters=3)
    assert r.nfe == B * T          # the init's block starts, then every other index once


def test_cache_saves_evaluations_and_stays_close():
    w = W.SD15.with_(latent_shape=(4, 16, 16))
    a, x0, mu = W.inputs(w)
    fn = make_eps_fn(a, mu, w.gmm_std)
    rc = run_srds(a, x0, fn, w.tol, w.cache_thresh)
    ru = run_srds(a, x0, fn, w.tol, w.cache_thresh, use_cache=False)
    assert rc.nfe < ru.nfe
    serial = serial_ddim(a, x0, fn)[:, -1]
    dev = np.abs(rc.x_final - serial).max() / np.abs(serial).max()
    assert dev < 0.05


def test_parareal_correction_converges_before_n_iterations():
    """With a coarse jump close to the fine steps, the Parareal correction
    converges to 1e-10 in well under N iterations; a sampler that only
    propagates fine solves (no G(new) - G(old) correction) needs all N."""
    w = W.SD15.with_(latent_shape=(4, 8, 8))
    a, x0, mu = W.inputs(w)
    fn = make_eps_fn(a, mu, w.gmm_std)
    s, N, starts, ends = srds_blocks(w.T)
    r = run_srds(a, x0, fn, 1e-10, 0.0)
    assert r.iters <= N // 2, r.iters
    serial = serial_ddim(a, x0, fn)[:, -1]
    assert np.abs(r.x_final - serial).max() / np.abs(serial).max() < 1e-6
