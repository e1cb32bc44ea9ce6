"""The C ABI used from plain C: tests/c/abi_generation.c (gcc, no Python and no
torch in the process) runs cached-Picard generations through libparaanya.so
with cudaMalloc'd buffers, host x_init in and host x_T out, step by step and as
the device-driven loop (pa_loop_*); the results must
match the fp64 oracle exactly in NFE, iterations and hits and within 1e-5 in
the final latents."""
import os
import shutil
import subprocess

import numpy as np
import pytest

import workload as W
from gpu_harness import oracle_run

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
CUDA = os.environ.get("CUDA_HOME", "/usr/local/cuda")


def _build(tmp):
    from paper_2609_36522_gb300 import build as pa_build
    lib = pa_build.build()
    gcc = shutil.which("gcc")
    if gcc is None:
        pytest.skip("gcc not found")
    exe = os.path.join(tmp, "abi_generation")
    libdir = os.path.dirname(lib)
    cmd = [gcc, "-O2", "-Wall", os.path.join(ROOT, "tests", "c", "abi_generation.c"),
           "-I", os.path.join(ROOT, "include"), "-I", os.path.join(CUDA, "include"),
           "-L", libdir, "-lparaanya", "-L", os.path.join(CUDA, "lib64"), "-lcudart",
           f"-Wl,-rpath,{libdir}", f"-Wl,-rpath,{os.path.join(CUDA, 'lib64')}", "-o", exe]
    r = subprocess.run(cmd, capture_output=True, text=True)
    assert r.returncode == 0, r.stderr
    return exe


@pytest.mark.gpu
@pytest.mark.parametrize("w", [
    W.TINY,
    W.Workload("C batched", T=24, window=8, batch=3, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=21),
], ids=lambda w: w.name)
@pytest.mark.parametrize("mode", ["steps", "loop"])
def test_generation_from_c(w, mode, tmp_path):
    exe = _build(str(tmp_path))
    a, x0, mu = W.inputs(w)
    c, h, wd = w.latent_shape
    with open(tmp_path / "sizes.txt", "w") as f:
        f.write(f"{w.T} {w.window} {w.batch} {w.K} {c} {h} {wd} {w.tol!r} {w.cache_thresh!r} {w.gmm_std!r}\n")
    np.asarray(a, dtype=np.float64).tofile(tmp_path / "alphas.bin")
    np.ascontiguousarray(x0, dtype=np.float32).tofile(tmp_path / "x0.bin")
    np.ascontiguousarray(mu, dtype=np.float32).tofile(tmp_path / "mu.bin")
    r = subprocess.run([exe, str(tmp_path)] + (["loop"] if mode == "loop" else []), capture_output=True,
                       text=True, timeout=300)
    assert r.returncode == 0, r.stderr
    fields = r.stdout.split()
    nfe, iters, hits = int(fields[1]), int(fields[3]), int(fields[5])
    orc = oracle_run(w)
    assert (nfe, iters, hits) == (orc.nfe, orc.iters, orc.hits)
    xT = np.fromfile(tmp_path / "xT.bin", dtype=np.float32).reshape(w.batch, w.D)
    rel = np.abs(xT - orc.x_final).max(axis=1) / np.abs(orc.x_final).max(axis=1)
    assert rel.max() <= 1e-5, rel
