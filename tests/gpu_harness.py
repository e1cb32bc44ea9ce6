"""Drive the CUDA solver through the C ABI and the fp64 oracle on the same
seeded inputs, and collect what the parity tests compare."""
from __future__ import annotations

import numpy as np

import workload as W
from oracle import run_picard
from oracle.gmm import make_eps_fn, gmm_eps
from oracle.picard import CacheAdaptation
from oracle.taa import run_taa


def oracle_run(w: W.Workload, cache_thresh=None, use_cache=True, cache_store=None, anderson=0, adapt=None):
    """adapt: None or (rate, target, tau_min, tau_max) of the tau_cache adaptation."""
    a, x0, mu = W.inputs(w)
    thr = w.cache_thresh if cache_thresh is None else cache_thresh
    ad = None if adapt is None else CacheAdaptation(*adapt)
    if anderson:
        return run_taa(a, x0, make_eps_fn(a, mu, w.gmm_std), w.window, w.tol, thr, depth=anderson,
                       use_cache=use_cache, eta=w.eta, noise=W.noise(w), adapt=ad)
    return run_picard(a, x0, make_eps_fn(a, mu, w.gmm_std), w.window, w.tol, thr,
                      use_cache=use_cache, eta=w.eta, noise=W.noise(w), cache_store=cache_store, adapt=ad)


def gpu_run(w: W.Workload, cache_thresh=None, eps_source="gmm", update_kernel=None,
            mode="sync", x_init_host=False, gmm_form=None, cache_bits=None, reductions=False, anderson=None,
            adapt=None):
    """Run one generation on the GPU.

    eps_source: "gmm" (the CUDA mixture kernel) or "oracle" (fp64 mixture
    posterior evaluated on the host for the gathered batch, rounded to fp32).
    mode: "sync" (pa_step) or "async" (pa_step_async, device-side counts).
    reductions: keep every iteration's Eq. 2 / Eq. 4 reductions (sync mode).
    anderson: history depth of the triangular Anderson mixing (None: not set).
    adapt: None or (rate, target, tau_min, tau_max): tau_cache adapted online;
    every planned iteration's tau_cache per trajectory is kept (sync mode).
    """
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser

    a, x0, mu = W.inputs(w)
    thr = w.cache_thresh if cache_thresh is None else cache_thresh
    dev = torch.device("cuda")
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, thr, batch=w.batch)
    if update_kernel is not None:
        s.set_update_kernel(update_kernel)
    if cache_bits is not None:
        s.set_cache_precision(cache_bits)
    if anderson is not None:
        s.set_anderson(anderson)
    if adapt is not None:
        s.set_cache_adaptation(*adapt)
    max_rows = w.batch * s.window
    means = torch.from_numpy(mu).to(dev)
    g = GmmDenoiser(means, w.gmm_std, a, max_rows)
    if gmm_form is not None:
        g.set_form(gmm_form)
    eps_buf = torch.empty(max_rows, w.D, dtype=torch.float32, device=dev)
    noise_keep = None
    if w.eta != 0.0:
        z = torch.from_numpy(W.noise(w)).to(dev).reshape(-1)
        noise_keep = z
        from paper_2609_36522_gb300 import abi as _abi
        _abi.pa_set_noise(s.h, w.eta, z.data_ptr())
    x_init = torch.from_numpy(x0)
    if x_init_host:
        x_init = x_init.pin_memory()
    else:
        x_init = x_init.to(dev)
    s.init(x_init)
    misses = []
    batches = []
    reds = []
    taus = []
    if mode == "sync":
        while True:
            out = s.step()
            if out is None:
                break
            if adapt is not None:
                taus.append(s.cache_thresholds())
            n, bx, mb = out.n_miss, out.batch_x, out.miss_bt
            mbh = mb.cpu().numpy().copy()
            misses.append([tuple(int(v) for v in row) for row in mbh])
            if eps_source == "gmm":
                g.eps(out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps_buf)
            else:
                xb = bx.double().cpu().numpy()
                e = gmm_eps(xb, a[mbh[:, 1]], mu.astype(np.float64), w.gmm_std)
                eps_buf[:n].copy_(torch.from_numpy(e.astype(np.float32)))
            batches.append(n)
            s.submit_eps(eps_buf)
            if reductions:
                reds.append(s.last_reductions())
    else:
        if eps_source != "gmm":
            raise ValueError("async mode needs the device-side denoiser")
        for _ in range(w.T + 1):
            bx, mb, nm = s.step_async()
            g.eps(bx, mb, nm, eps_buf)
            s.submit_eps(eps_buf)
        s.poll()
    xT = s.result().cpu().numpy()
    res = dict(x_final=xT, nfe=s.nfe(), stats=s.stats(), log=s.iter_log(), misses=misses,
               batches=batches, gmm_launches=g.launches(), reductions=reds, taus=taus)
    s.close()
    g.close()
    return res


def compare(w, orc, gpu, check_misses=True):
    """Assert GPU == oracle: iteration log, miss lists, NFE exactly; latents 1e-5."""
    recs = orc.records
    log = gpu["log"]
    assert len(log) == orc.iters, (len(log), orc.iters)
    for k, rec in enumerate(recs):
        for b in range(w.batch):
            t, p, m, stride = (int(v) for v in log[k, b, :4])
            if rec.p[b] == 0:
                assert p == 0
                continue
            assert (t, p, stride) == (rec.t[b], rec.p[b], rec.stride[b]), (k, b)
            assert m == sum(1 for bb, _ in rec.miss_bt if bb == b), (k, b)
    if check_misses and gpu["misses"]:
        assert [list(r.miss_bt) for r in recs] == gpu["misses"]
    assert gpu["nfe"] == orc.nfe
    assert gpu["stats"]["iters"] == orc.iters
    assert gpu["stats"]["hits"] == orc.hits
    scale = np.abs(orc.x_final).max(axis=1)
    rel = np.abs(gpu["x_final"] - orc.x_final).max(axis=1) / scale
    return rel
