"""GB300-native cached Picard solver step (ParaAnya output cache on
sliding-window Picard DDIM sampling), as sm_103a CUDA kernels behind a C ABI.

    abi     -- ctypes binding, the C functions under their own names
    solver  -- Solver / GmmDenoiser: torch-allocated workspaces around the ABI
    build   -- nvcc build of lib/libparaanya.so
"""
from . import abi  # noqa: F401


def __getattr__(name):
    if name in ("Solver", "GmmDenoiser"):
        from . import solver
        return getattr(solver, name)
    raise AttributeError(name)
