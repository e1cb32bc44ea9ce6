"""fp64 CPU oracle for ParaAnya's cached Picard sampler -- TEST INFRASTRUCTURE.

This package is the plain, slow, obviously-correct statement of what the GPU
solver step computes. It exists to check the CUDA path and for nothing else:
only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline / reference
legs of ``bench.py`` may import it. The product path (``paper_2609_36522_gb300``)
never imports it, and this package never imports the product. The two share no
code; the only common module is ``workload`` (seeded input generation, which
holds none of the method's arithmetic).

Modules
-------
ddim    -- DDIM step (eta = 0, and eta > 0 with draws fixed before sampling),
           its drift coefficients, serial sampling (Eq. 1's drift s_theta,
           Sec. 2.1).
gmm     -- posterior-mean noise of an isotropic Gaussian mixture, the synthetic
           stand-in for the SD v1.5 UNet eps_theta.
picard  -- sliding-window Picard iteration (Eq. 1, Eq. 2) with ParaAnya's
           output cache (Eq. 3-7), for a batch of independent trajectories,
           optionally with tau_cache adapted online (CacheAdaptation).
taa     -- the same with triangular Anderson mixing of the iterates
           (a ParaTAA-style update, depth 0 or 1).
srds    -- Parareal (SRDS-style) DDIM sampling with the same cache on the
           coarse and fine evaluations (Sec. 2.1, Sec. 2.2).
guard   -- decision-margin guard used to reject generated inputs whose
           oracle distances / errors sit too close to a threshold.

Pins (what ties this oracle to something other than itself) live in
``tests/test_oracle_*.py``: closed forms (point-mass and single-Gaussian DDIM,
Tweedie's formula by finite differences of a brute-force log-density),
reductions to serial DDIM and to the uncached sampler, counting invariants
(NFE = sum of misses, NFE = B*T for an always-hit cache), and a second,
scalar pure-Python implementation for tiny T in ``tests/scalar_picard.py``.
Every function here carries a pin; none is "parity unpinned".
"""
from . import ddim, gmm, picard, guard, srds  # noqa: F401
from .picard import run_picard, PicardResult, CacheAdaptation  # noqa: F401
from .srds import run_srds, SrdsResult  # noqa: F401
from .ddim import serial_ddim, drift_coefficients  # noqa: F401
from .gmm import gmm_eps  # noqa: F401
