"""Pins for the oracle's bfloat16 cache-entry storage (CPU only).

* The rounding is the IEEE one: it agrees with torch's fp32 -> bfloat16
  conversion on random values, exact ties (both directions) and tiny and large
  magnitudes.
* tau_cache = 0 never hits, so how the entries are stored cannot matter: the
  bfloat16 run is the uncached sampler bit for bit (catches a rounding applied
  to the fresh eps or to the states).
* tau_cache huge: every timestep is evaluated once (NFE = B * T), every stored
  entry is a bfloat16 value, and the result moves away from the fp32-entry run
  by a small amount (nonzero: the hits really read rounded entries).
"""
import numpy as np
import pytest

import workload as W
from oracle import run_picard
from oracle.gmm import make_eps_fn
from oracle.storage import round_bf16


def test_round_bf16_matches_torch():
    torch = pytest.importorskip("torch")
    rng = np.random.default_rng(0)
    vals = [rng.standard_normal(20000) * 10.0 ** rng.integers(-6, 6, 20000)]
    # exact ties: low 16 bits 0x8000 under an even and an odd last kept bit (bit 16)
    n = 2000
    sign = rng.integers(0, 2, n, dtype=np.uint32) << np.uint32(31)
    expo = rng.integers(100, 150, n, dtype=np.uint32) << np.uint32(23)
    mant = rng.integers(0, 1 << 6, n, dtype=np.uint32) << np.uint32(17)      # kept bits above bit 16
    for lastbit in (0, 1):
        u = (sign | expo | mant | np.uint32(lastbit << 16) | np.uint32(0x8000)).astype(np.uint32)
        vals.append(u.view(np.float32).astype(np.float64))
    vals.append(np.array([0.0, -0.0, 1e-30, -1e-30, 3.0e38, -3.0e38, 1.0, -1.0]))
    x = np.concatenate(vals)
    ref = torch.from_numpy(x.astype(np.float32)).to(torch.bfloat16).to(torch.float64).numpy()
    got = round_bf16(x)
    assert np.array_equal(got, ref)
    assert np.array_equal(round_bf16(got), got)          # idempotent on bfloat16 values


def _case(T=16, P=6, B=2, shape=(4, 4, 4), K=3, seed=2):
    w = W.Workload("bf16", T=T, window=P, batch=B, latent_shape=shape, K=K, tol=1e-3,
                   cache_thresh=0.05, seed=seed)
    a, x0, mu = W.inputs(w)
    return w, a, x0, make_eps_fn(a, mu, w.gmm_std)


def test_threshold_zero_is_uncached_whatever_the_storage():
    w, a, x0, f = _case()
    u = run_picard(a, x0, f, w.window, w.tol, 0.0, use_cache=False)
    b = run_picard(a, x0, f, w.window, w.tol, 0.0, cache_store=round_bf16)
    assert np.array_equal(u.x_final, b.x_final) and u.nfe == b.nfe and b.hits == 0


def test_always_hit_reads_rounded_entries():
    w, a, x0, f = _case(T=20, P=5)
    full = run_picard(a, x0, f, w.window, w.tol, 1e30)
    half = run_picard(a, x0, f, w.window, w.tol, 1e30, cache_store=round_bf16)
    assert half.nfe == w.batch * w.T
    ent = half.has_entry
    assert np.array_equal(round_bf16(half.ehat[ent]), half.ehat[ent])
    assert np.array_equal(round_bf16(half.xhat[ent]), half.xhat[ent])
    rel = np.abs(half.x_final - full.x_final).max() / np.abs(full.x_final).max()
    assert 0.0 < rel < 1e-2, rel
