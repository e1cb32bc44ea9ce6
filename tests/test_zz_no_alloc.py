"""The allocation-free denoiser entry point, pa_gmm_eps_noalloc.

It serves callers that cannot allocate device memory when they run the
denoiser (plugins handed pre-allocated buffers by a host framework, real-time
loops that forbid cudaMalloc/cudaFree after start-up): its scratch is a fixed
4 MiB device array inside the library. This file is collected last on
purpose, so that a run stopping at the first failure has run every other test
first; it also passes when run on its own in a fresh process.
"""
import numpy as np
import pytest

import workload as W
from oracle.gmm import gmm_eps

pytestmark = pytest.mark.gpu

REL_TOL = 2e-6  # the mixture-denoiser tolerance of test_gpu_parity


@pytest.fixture(scope="module")
def lib():
    import torch
    from paper_2609_36522_gb300 import build as pa_build
    from paper_2609_36522_gb300 import abi
    assert torch.cuda.is_available()
    pa_build.build()
    return abi


def _rows(w, a, mu, n, seed):
    rng = np.random.default_rng(seed)
    idx = rng.integers(0, w.T, n).astype(np.int32)
    comp = rng.integers(0, w.K, n)
    x = (np.sqrt(a[idx])[:, None] * (mu[comp] + 0.5 * rng.standard_normal((n, w.D)))
         + np.sqrt(1 - a[idx])[:, None] * rng.standard_normal((n, w.D))).astype(np.float32)
    miss = np.stack([np.zeros(n, np.int32), idx], axis=1).astype(np.int32)
    return x, miss, idx


def test_noalloc_matches_handle_entry_point_on_two_calls(lib):
    import torch
    from paper_2609_36522_gb300.solver import GmmDenoiser
    abi = lib
    w = W.SD15
    a, _, mu = W.inputs(w)
    dev = torch.device("cuda")
    mu_d = torch.from_numpy(mu).to(dev)
    g = GmmDenoiser(mu_d, w.gmm_std, a, 100)
    stream = torch.cuda.current_stream()
    # two calls in a row; the second is smaller, so stale scratch of the first
    # must not leak into it
    for n, seed in ((100, 1), (37, 2)):
        x, miss, idx = _rows(w, a, mu, n, seed)
        xd = torch.from_numpy(x).to(dev)
        md = torch.from_numpy(miss).to(dev)
        nd = torch.tensor([n], dtype=torch.int32, device=dev)
        ref = torch.empty_like(xd)
        got = torch.full_like(xd, float("nan"))
        xfull = torch.zeros(100, w.D, dtype=torch.float32, device=dev)  # the handle's batch holds max_rows rows
        xfull[:n] = xd
        reff = torch.empty_like(xfull)
        g.eps(xfull.data_ptr(), md.data_ptr(), nd.data_ptr(), reff)
        ref.copy_(reff[:n])
        abi.pa_gmm_eps_noalloc(mu_d.data_ptr(), w.K, w.D, w.gmm_std, list(a), xd.data_ptr(),
                               md.data_ptr(), n, got.data_ptr(), stream.cuda_stream)
        torch.cuda.synchronize()
        r = ref.cpu().numpy().astype(np.float64)
        o = got.cpu().numpy().astype(np.float64)
        scale = np.abs(r).max(axis=1)
        assert np.isfinite(o).all()
        assert (np.abs(o - r).max(axis=1) / scale).max() <= REL_TOL
        want = gmm_eps(x.astype(np.float64), a[idx], mu.astype(np.float64), w.gmm_std)
        assert (np.abs(o - want).max(axis=1) / np.abs(want).max(axis=1)).max() <= REL_TOL
    g.close()


def test_noalloc_rejects_sizes_beyond_its_scratch(lib):
    import torch
    abi = lib
    # 4096 rows x 128 components need two sets of 4 MiB of int64 dot
    # accumulators, 8 MiB in all: twice the scratch
    K, D, n, T = 128, 256, 4096, 10
    a = W.alphas_cumprod(T)
    dev = torch.device("cuda")
    mu_d = torch.randn(K, D, device=dev)
    x = torch.zeros(n, D, device=dev)
    miss = torch.zeros(n, 2, dtype=torch.int32, device=dev)
    out = torch.zeros_like(x)
    with pytest.raises(abi.PaError) as e:
        abi.pa_gmm_eps_noalloc(mu_d.data_ptr(), K, D, 0.5, list(a), x.data_ptr(),
                               miss.data_ptr(), n, out.data_ptr(), 0)
    assert e.value.status == abi.PA_ERR_ARG
    assert "4 MiB" in str(e.value)


@pytest.mark.parametrize("shape,n", [((3, 7, 9), 11), ((4, 64, 64), 0), ((3, 7, 9), 0)],
                         ids=["odd D", "no rows", "no rows odd D"])
def test_noalloc_odd_rows_and_empty_batch(lib, shape, n):
    """D % 4 != 0 (rows staged by plain loads, scalar stores) against the
    handle entry point and the oracle; with no rows the call writes nothing,
    like the handle entry point."""
    import torch
    from paper_2609_36522_gb300.solver import GmmDenoiser
    abi = lib
    w = W.TINY.with_(T=30, latent_shape=shape, K=5, name="noalloc odd")
    a, _, mu = W.inputs(w)
    dev = torch.device("cuda")
    mu_d = torch.from_numpy(mu).to(dev)
    rows = max(n, 4)
    g = GmmDenoiser(mu_d, w.gmm_std, a, rows)
    x, miss, idx = _rows(w, a, mu, rows, 5)
    xd = torch.from_numpy(x).to(dev)
    md = torch.from_numpy(miss).to(dev)
    nd = torch.tensor([n], dtype=torch.int32, device=dev)
    stream = torch.cuda.current_stream()
    for _ in range(2):  # two calls in a row
        ref = torch.full_like(xd, float("nan"))
        got = torch.full_like(xd, float("nan"))
        g.eps(xd.data_ptr(), md.data_ptr(), nd.data_ptr(), ref)
        abi.pa_gmm_eps_noalloc(mu_d.data_ptr(), w.K, w.D, w.gmm_std, list(a), xd.data_ptr(),
                               md.data_ptr(), n, got.data_ptr(), stream.cuda_stream)
        torch.cuda.synchronize()
        r = ref.cpu().numpy().astype(np.float64)
        o = got.cpu().numpy().astype(np.float64)
        assert np.isnan(o[n:]).all() and np.isnan(r[n:]).all()   # rows past the count untouched
        if n:
            scale = np.abs(r[:n]).max(axis=1)
            assert np.isfinite(o[:n]).all()
            assert (np.abs(o[:n] - r[:n]).max(axis=1) / scale).max() <= REL_TOL
            want = gmm_eps(x[:n].astype(np.float64), a[idx[:n]], mu.astype(np.float64), w.gmm_std)
            assert (np.abs(o[:n] - want).max(axis=1) / np.abs(want).max(axis=1)).max() <= REL_TOL
    g.close()
