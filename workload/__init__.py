"""Seeded synthetic workloads for the cached Picard solver step.

This module only *generates inputs*. It holds none of the sampler's arithmetic
(no DDIM coefficients, no drift, no Picard update, no cache rule, no mixture
posterior): both the fp64 oracle under ``oracle/`` and the CUDA path consume the
arrays produced here, so neither side can disagree on an input.

What it produces, per workload:

* ``alphas_cumprod`` -- the sampling-order noise schedule, length T+1. The
  training schedule is the linear-beta DDPM schedule (beta from 1e-4 to 0.02 over
  1000 training steps); the paper only says "DDIM schedulers" on Stable Diffusion
  v1.5 (Sec. 3.2-3.3), so the subsampling is our reading: DDIM's uniform spacing
  tau_i = (1000 // T) * (T - 1 - i) for sampling index i = 0..T-1 (index 0 is the
  noisiest step, as in Eq. 1 where x_0 is the initial noise), and entry T is 1.0,
  the "previous" alpha-bar after the last training step.
* ``x_init`` -- initial noise N(0, 1), fp32, one row per trajectory.
* ``means`` -- Gaussian-mixture component means N(0, 1), fp32, [K][D]; the
  mixture has equal weights and isotropic component std ``gmm_std``.
* ``noise`` -- for stochastic steps (eta > 0) the draws z_i ~ N(0, 1) of every
  trajectory and step, fp32 [B][T][D], fixed before sampling.

The SD v1.5 latent shape 4x64x64 (512^2 images, Sec. 3.2) and the paper's
cache tolerance 0.05 (Sec. 3.3) set the shapes and thresholds; COCO prompts and
the trained UNet are replaced by seeded noise and the mixture denoiser.
"""
from __future__ import annotations

from dataclasses import dataclass, field, replace
from typing import Tuple

import numpy as np

TRAIN_STEPS = 1000
BETA_START = 1e-4
BETA_END = 0.02
GMM_STD = 0.5
MEANS_SEED_OFFSET = 1_000_000
NOISE_SEED_OFFSET = 2_000_000


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: solver sizes, thresholds and seeds."""

    name: str
    T: int                      # DDIM steps
    window: int                 # P, maximum evaluation points per Picard iteration
    batch: int                  # B, independent trajectories
    latent_shape: Tuple[int, ...]
    K: int                      # mixture components of the synthetic denoiser
    tol: float                  # Picard convergence tolerance tau (Eq. 2)
    cache_thresh: float         # tau_cache (Eq. 5)
    seed: int = 0               # trajectory b uses noise seed (seed + b)
    gmm_std: float = GMM_STD
    eta: float = 0.0            # stochastic steps (eta = 1: DDPM); 0 = DDIM
    sampler: str = "picard"     # "picard" (sliding window), "taa" (the same with triangular
                                # Anderson mixing of depth 1) or "srds" (Parareal blocks; window unused)
    extra: dict = field(default_factory=dict, compare=False)

    @property
    def D(self) -> int:
        return int(np.prod(self.latent_shape))

    def with_(self, **kw) -> "Workload":
        return replace(self, **kw)


# The five workloads, named by what they are.
TINY = Workload("tiny T16 P8 B1 4x8x8 K4", T=16, window=8, batch=1,
                latent_shape=(4, 8, 8), K=4, tol=1e-3, cache_thresh=0.05)
SD15 = Workload("SD-v1.5-shaped T100 P100 B1 4x64x64 K16", T=100, window=100, batch=1,
                latent_shape=(4, 64, 64), K=16, tol=1e-3, cache_thresh=0.05)
BATCHED = Workload("batched T100 P32 B8 4x64x64 K16", T=100, window=32, batch=8,
                   latent_shape=(4, 64, 64), K=16, tol=1e-3, cache_thresh=0.05)
LARGE = Workload("large T200 P64 B2 4x128x128 K64", T=200, window=64, batch=2,
                 latent_shape=(4, 128, 128), K=64, tol=5e-4, cache_thresh=0.05)
# Stochastic sampling (a next step beyond the DDIM workloads): DDPM, i.e. eta = 1
# over the full 1000-step schedule, window 64 (Table 2's best DDPM window).
DDPM = Workload("DDPM T1000 P64 B1 4x64x64 K16", T=1000, window=64, batch=1,
                latent_shape=(4, 64, 64), K=16, tol=1e-3, cache_thresh=0.05, eta=1.0)
# The same with a 128-point window, the longest window axis of Table 2.
DDPM128 = DDPM.with_(name="DDPM T1000 P128 B1 4x64x64 K16", window=128)
# Parareal (SRDS-style) sampling with the cache, on the SD-shaped and batched inputs.
SRDS = SD15.with_(name="SRDS T100 B1 4x64x64 K16", sampler="srds")
SRDS_BATCHED = BATCHED.with_(name="SRDS T100 B8 4x64x64 K16", sampler="srds")
# Triangular Anderson mixing (a ParaTAA-style update) on the SD-shaped and batched inputs.
SD15_TAA = SD15.with_(name="SD-v1.5-shaped T100 P100 B1 4x64x64 K16 TAA", sampler="taa")
BATCHED_TAA = BATCHED.with_(name="batched T100 P32 B8 4x64x64 K16 TAA", sampler="taa")
# Online adaptation of tau_cache on the SD-shaped inputs: tau starts at 0.02 and
# tracks a 50 % hit rate among points with an entry, by factors of 1.5, within
# [0, 0.2] (extra["adapt"] = (rate, target, tau_min, tau_max)).
SD15_ADAPT = SD15.with_(name="SD-v1.5-shaped T100 P100 B1 4x64x64 K16 adaptive tau_cache",
                        cache_thresh=0.02, extra={"adapt": (0.5, 0.5, 0.0, 0.2)})
SWEEP_THRESHOLDS = (0.0, 0.01, 0.02, 0.05, 0.1)


def sweep(base: Workload = SD15):
    """Cache-threshold sweep on the SD-v1.5-shaped workload (Table 3 analogue)."""
    return [base.with_(name=f"{base.name} cache{c:g}", cache_thresh=c)
            for c in SWEEP_THRESHOLDS]


ALL = {"tiny": TINY, "sd15": SD15, "batched": BATCHED, "large": LARGE, "ddpm": DDPM, "ddpm128": DDPM128,
       "srds": SRDS, "srds_batched": SRDS_BATCHED, "sd15_taa": SD15_TAA, "batched_taa": BATCHED_TAA, "sd15_adapt": SD15_ADAPT}


def train_alphas_cumprod() -> np.ndarray:
    """alpha-bar of the 1000-step linear-beta training schedule, fp64."""
    betas = np.linspace(BETA_START, BETA_END, TRAIN_STEPS, dtype=np.float64)
    return np.cumprod(1.0 - betas)


def ddim_timesteps(T: int) -> np.ndarray:
    """Training timestep used at sampling index i (uniform DDIM spacing)."""
    if not (1 <= T <= TRAIN_STEPS):
        raise ValueError(f"T must be in [1, {TRAIN_STEPS}], got {T}")
    step = TRAIN_STEPS // T
    return step * (T - 1 - np.arange(T, dtype=np.int64))


def alphas_cumprod(T: int) -> np.ndarray:
    """Sampling-order alpha-bar, length T+1: [0] noisiest, [T] = 1.0 (clean)."""
    a = train_alphas_cumprod()[ddim_timesteps(T)]
    return np.concatenate([a, [1.0]]).astype(np.float64)


def x_init(w: Workload) -> np.ndarray:
    """Initial noise, fp32 [B][D]; trajectory b draws from default_rng(seed + b)."""
    rows = [np.random.default_rng(w.seed + b).standard_normal(w.D).astype(np.float32)
            for b in range(w.batch)]
    return np.stack(rows, axis=0)


def means(w: Workload) -> np.ndarray:
    """Mixture means, fp32 [K][D], from default_rng(1_000_000 + seed)."""
    rng = np.random.default_rng(MEANS_SEED_OFFSET + w.seed)
    return rng.standard_normal((w.K, w.D)).astype(np.float32)


def noise(w: Workload) -> np.ndarray:
    """The draws z_i of stochastic steps, fp32 [B][T][D]; trajectory b draws
    from default_rng(2_000_000 + seed + b). None for eta = 0."""
    if w.eta == 0.0:
        return None
    rows = [np.random.default_rng(NOISE_SEED_OFFSET + w.seed + b).standard_normal((w.T, w.D)).astype(np.float32)
            for b in range(w.batch)]
    return np.stack(rows, axis=0)


def inputs(w: Workload):
    """(alphas_cumprod fp64 [T+1], x_init fp32 [B][D], means fp32 [K][D])."""
    return alphas_cumprod(w.T), x_init(w), means(w)
