"""GPU parity: the CUDA solver (through the C ABI) against the fp64 oracle on
the same seeded inputs.

Bar (from the method's decisions and the fp32 state):
* iteration count, per-iteration window start / size / stride, per-trajectory
  miss counts, the canonical miss list (b, i) and NFE / hits: bit-exact;
* final latents: max_d |x_gpu - x_oracle| / max_d |x_oracle| <= 1e-5 per
  trajectory.
Inputs pass the decision-margin guard (no oracle distance or error within
1e-6 relative of its threshold) before they are compared.
"""
import numpy as np
import pytest

import workload as W
from oracle.guard import margins_ok, decision_margins
from oracle.gmm import gmm_eps
from gpu_harness import oracle_run, gpu_run, compare

pytestmark = pytest.mark.gpu

REL_TOL = 1e-5


@pytest.fixture(scope="module", autouse=True)
def _built():
    import torch
    from paper_2609_36522_gb300 import build as pa_build
    assert torch.cuda.is_available(), "GPU tests need a CUDA device"
    pa_build.build()


def _check(w, cache_thresh=None, **kw):
    thr = w.cache_thresh if cache_thresh is None else cache_thresh
    orc = oracle_run(w, cache_thresh=thr)
    assert margins_ok(orc, w.tol, thr, rel=1e-6), decision_margins(orc, w.tol, thr)
    gpu = gpu_run(w, cache_thresh=thr, **kw)
    rel = compare(w, orc, gpu)
    assert rel.max() <= REL_TOL, rel
    return orc, gpu


def test_tiny():
    _check(W.TINY)


def test_tiny_with_oracle_eps():
    """Solver kernels alone: eps of the gathered batch comes from the fp64 oracle."""
    _check(W.TINY, eps_source="oracle")


def test_sd15_full_size():
    orc, gpu = _check(W.SD15)
    assert gpu["stats"]["hits"] > 0
    assert gpu["stats"]["update_kernel"] == 2  # lean register update + planning kernel by default


def test_sd15_uncached_equals_oracle_uncached():
    w = W.SD15
    orc = oracle_run(w, cache_thresh=0.0, use_cache=False)
    gpu = gpu_run(w, cache_thresh=0.0)
    rel = compare(w, orc, gpu)
    assert rel.max() <= REL_TOL
    assert gpu["stats"]["hits"] == 0


@pytest.mark.parametrize("thr", W.SWEEP_THRESHOLDS)
def test_sd15_threshold_sweep(thr):
    _check(W.SD15, cache_thresh=thr)


def test_batched_eight_trajectories():
    _check(W.BATCHED)


def test_large_latent():
    _check(W.LARGE)


@pytest.mark.parametrize("w", [
    W.Workload("ragged odd D", T=12, window=5, batch=3, latent_shape=(3, 5, 7), K=3,
               tol=1e-3, cache_thresh=0.05, seed=3),
    W.Workload("ragged D%4==0", T=14, window=6, batch=2, latent_shape=(4, 5, 7), K=5,
               tol=1e-3, cache_thresh=0.05, seed=4),
    W.Workload("window 1", T=9, window=1, batch=2, latent_shape=(4, 4, 4), K=2,
               tol=1e-3, cache_thresh=0.05, seed=5),
    W.Workload("window T", T=20, window=20, batch=1, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=6),
    W.Workload("window > T", T=7, window=32, batch=2, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=7),
    W.Workload("T 1", T=1, window=4, batch=2, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=8),
    W.Workload("multi-chunk", T=30, window=12, batch=3, latent_shape=(4, 24, 24), K=8,
               tol=1e-3, cache_thresh=0.05, seed=9),
    W.Workload("tight tol", T=24, window=10, batch=2, latent_shape=(4, 16, 16), K=6,
               tol=1e-6, cache_thresh=0.02, seed=10),
    # more batch rows than one wave of planning CTAs (2 per SM): each CTA plans
    # once and copies every gridDim.y-th row
    W.Workload("4 x 100 pairs", T=100, window=100, batch=4, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=19),
    # past 512 pairs one CTA plans and a separate gather follows
    W.Workload("10 x 100 pairs", T=100, window=100, batch=10, latent_shape=(4, 8, 8), K=4,
               tol=1e-3, cache_thresh=0.05, seed=20),
    # more than 1024 (trajectory, position) pairs: one CTA plans, a separate gather follows
    W.Workload("9 x 128 pairs", T=200, window=128, batch=9, latent_shape=(4, 4, 4), K=4,
               tol=1e-3, cache_thresh=0.05, seed=13),
    W.Workload("64 trajectories", T=40, window=32, batch=64, latent_shape=(4, 4, 4), K=4,
               tol=1e-3, cache_thresh=0.05, seed=14),
    # a 1000-point window: tiled update kernel, one-CTA planner (2 x 1000 pairs)
    W.Workload("window 1000", T=1000, window=1000, batch=2, latent_shape=(4, 4, 4), K=3,
               tol=1e-3, cache_thresh=0.05, seed=16),
    # the largest problem the limits admit: 64 trajectories (the batch limit)
    # of the longest schedule, the window asked at its limit of 1024 and
    # clamped to T = 1000: 64,000 pairs, a 64,000-row denoiser batch
    W.Workload("64 x 1000", T=1000, window=1024, batch=64, latent_shape=(4, 4, 4), K=3,
               tol=1e-3, cache_thresh=0.05, seed=18),
], ids=lambda w: w.name)
def test_edge_shapes(w):
    _check(w)


def test_always_hit_cache_evaluates_each_timestep_once():
    w = W.Workload("always hit", T=24, window=8, batch=2, latent_shape=(4, 8, 8), K=4,
                   tol=1e-3, cache_thresh=1e30, seed=11)
    orc, gpu = _check(w)
    assert gpu["nfe"] == w.batch * w.T


def test_async_equals_sync_and_is_deterministic():
    w = W.BATCHED.with_(T=40)
    a = gpu_run(w, mode="sync")
    b = gpu_run(w, mode="async")
    c = gpu_run(w, mode="async")
    assert np.array_equal(a["x_final"], b["x_final"])
    assert np.array_equal(b["x_final"], c["x_final"])
    assert np.array_equal(a["log"], b["log"])
    assert a["nfe"] == b["nfe"]


@pytest.mark.parametrize("w,form", [
    (W.SD15, 2),
    (W.SD15, 0),
    (W.LARGE.with_(T=60), 1),
    (W.BATCHED.with_(T=40), 2),
    (W.BATCHED.with_(T=40), 0),
], ids=["sd15-cluster", "sd15-cuda-cores", "large-tensor-cores", "batched-cluster", "batched-cuda-cores"])
def test_graph_replay_equals_sync(w, form):
    """A whole generation captured as one CUDA graph (pa_init and every
    iteration's denoiser, update and planning kernels, chained by programmatic
    dependent launches with early triggers) and replayed twice gives the
    synchronous run's states and iteration log bit for bit: every kernel reads
    its predecessor's output only after its dependency wait."""
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    sync = gpu_run(w, gmm_form=form)
    n_iters = len(sync["log"])
    a, x0, mu = W.inputs(w)
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, stream=st)
        g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window, stream=st)
        g.set_form(form)
        eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")
        x_dev = torch.from_numpy(x0).cuda()
        s.init(x_dev)
        out = s.step_async()                       # eager warm-up of every launch path
        g.eps(*out, eps)
        s.submit_eps(eps)
        st.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=st):
            s.init(x_dev)
            for _ in range(n_iters):
                out = s.step_async()
                g.eps(*out, eps)
                s.submit_eps(eps)
        for _ in range(2):
            graph.replay()
            st.synchronize()
            assert s.poll() == 0
            assert np.array_equal(s.result().cpu().numpy(), sync["x_final"])
            assert np.array_equal(s.iter_log(), sync["log"])
    s.close()
    g.close()


@pytest.mark.parametrize("wname,chunk", [("sd15", 4), ("batched", 2), ("tiny", 6)])
def test_generate_equals_async_path(wname, chunk):
    """Solver.generate (captured chunks of iterations replayed until done,
    host x_init in and host x_T out) gives the asynchronous path's latents,
    log and counters bit for bit, on its first call (capture) and again on
    the second (replay only)."""
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    w = {"sd15": W.SD15, "batched": W.BATCHED.with_(T=40), "tiny": W.TINY}[wname]
    ref = gpu_run(w, mode="async")
    a, x0, mu = W.inputs(w)
    st = torch.cuda.Stream()
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, stream=st)
    g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window, stream=st)
    eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")

    def denoise(bx, mb, nm):
        g.eps(bx, mb, nm, eps)
        return eps

    x_host = torch.from_numpy(x0).pin_memory()
    for _ in range(2):
        out = torch.full((w.batch, w.D), float("nan"), dtype=torch.float32).pin_memory()
        s.generate(x_host, denoise, out=out, chunk=chunk)
        assert np.array_equal(out.numpy(), ref["x_final"])
        assert np.array_equal(s.iter_log(), ref["log"])
        assert s.stats()["nfe"] == ref["nfe"]
    # a setting changed after capture takes effect: the captured graph is dropped
    s.set_update_kernel(0)
    out = s.generate(x_host, denoise, chunk=chunk)
    assert s.stats()["update_kernel"] == 0
    assert np.array_equal(s.iter_log(), ref["log"])
    assert compare(w, oracle_run(w), dict(x_final=out.cpu().numpy(), nfe=s.nfe(), stats=s.stats(),
                                          log=s.iter_log(), misses=[])).max() <= REL_TOL
    s.close()
    g.close()


def test_host_x_init_equals_device_x_init():
    a = gpu_run(W.TINY)
    b = gpu_run(W.TINY, x_init_host=True)
    assert np.array_equal(a["x_final"], b["x_final"])


def _gmm_rows(w, n, seed=0):
    a, _, mu = W.inputs(w)
    rng = np.random.default_rng(seed)
    idx = np.linspace(0, w.T - 1, n).astype(np.int32)
    comp = rng.integers(0, w.K, n)
    x = (np.sqrt(a[idx])[:, None] * (mu[comp] + 0.5 * rng.standard_normal((n, w.D)))
         + np.sqrt(1 - a[idx])[:, None] * rng.standard_normal((n, w.D))).astype(np.float32)
    miss = np.stack([np.zeros(n, np.int32), idx], axis=1).astype(np.int32)
    return a, mu, idx, x, miss


@pytest.mark.parametrize("form", [2, 1, 0])
@pytest.mark.parametrize("wname,n,max_rows", [("sd15", 48, 48), ("sd15", 1, 100), ("sd15", 37, 100),
                                              ("sd15", 100, 100), ("batched", 256, 256),
                                              ("large", 48, 48), ("large", 1, 128), ("large", 70, 128),
                                              ("large", 128, 128), ("k32", 100, 100), ("k32", 300, 300),
                                              ("k32", 129, 200), ("tiny", 5, 8),
                                              ("k3 d64", 11, 16)])
def test_gmm_kernel_against_oracle(wname, n, max_rows, form):
    """The mixture denoiser alone, in one cluster kernel (form 2), with the dot
    products on the tensor cores (form 1) and on the CUDA cores (form 0), on
    rows spread over the whole schedule, with the device row count below the
    capacity and not a multiple of the cluster form's 8-row blocks, and over
    three calls in a row (the fixed-point accumulators and the tickets are
    reused). Rows past the count hold NaN: the cluster form copies them with
    the block and must keep them out of every counted row. With 64 components: one row, 70 rows (a ragged second 64-row
    block of the tensor-core form's row tiles is not reached; rows past 48
    are), and full 128-row tiles; exactly 32 components; 3 components over 64
    columns (4 columns per CTA of the cluster form)."""
    import torch
    from paper_2609_36522_gb300 import abi
    from paper_2609_36522_gb300.solver import GmmDenoiser
    w = {"k32": W.SD15.with_(K=32, name="k32"),
         "k3 d64": W.TINY.with_(K=3, latent_shape=(4, 4, 4), name="k3 d64")}.get(wname) or W.ALL[wname]
    a, mu, idx, x, miss = _gmm_rows(w, n)
    dev = torch.device("cuda")
    g = GmmDenoiser(torch.from_numpy(mu).to(dev), w.gmm_std, a, max_rows)
    assert g.form() == (1 if w.K > 16 else 2), "cluster form up to 16 components, tensor cores above"
    if form == 2 and w.K > 16:
        with pytest.raises(abi.PaError) as e:
            g.set_form(2)
        assert e.value.status == abi.PA_ERR_ARG
        g.close()
        return
    g.set_form(form)
    xd = torch.full((max_rows, w.D), float("nan"), dtype=torch.float32, device=dev)
    xd[:n] = torch.from_numpy(x).to(dev)
    md = torch.zeros(max_rows, 2, dtype=torch.int32, device=dev)
    md[:n] = torch.from_numpy(miss).to(dev)
    nd = torch.tensor([n], dtype=torch.int32, device=dev)
    outs = []
    for _ in range(3):
        out = torch.full_like(xd, float("nan"))
        g.eps(xd.data_ptr(), md.data_ptr(), nd.data_ptr(), out)
        outs.append(out)
    torch.cuda.synchronize()
    from paper_2609_36522_gb300 import abi
    abi.pa_gmm_check(g.h)
    got = outs[0][:n].cpu().numpy().astype(np.float64)
    want = gmm_eps(x.astype(np.float64), a[idx], mu.astype(np.float64), w.gmm_std)
    rel = np.abs(got - want).max(axis=1) / np.abs(want).max(axis=1)
    assert rel.max() <= 2e-6, rel.max()
    for o in outs[1:]:
        assert torch.equal(o[:n], outs[0][:n])       # bitwise reproducible
    assert torch.isnan(outs[0][n:]).all()            # rows past the count are not written
    g.close()


def test_gmm_in_cuda_graph():
    """The denoiser captured in a CUDA graph and replayed gives the eager
    result (bitwise), with a device row count that changes between replays."""
    import torch
    from paper_2609_36522_gb300.solver import GmmDenoiser
    w = W.SD15
    n = 100
    a, mu, idx, x, miss = _gmm_rows(w, n, seed=3)
    dev = torch.device("cuda")
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        g = GmmDenoiser(torch.from_numpy(mu).to(dev), w.gmm_std, a, n, stream=st)
        xd = torch.from_numpy(x).to(dev)
        md = torch.from_numpy(miss).to(dev)
        nd = torch.tensor([n], dtype=torch.int32, device=dev)
        want = torch.empty_like(xd)
        g.eps(xd.data_ptr(), md.data_ptr(), nd.data_ptr(), want)
        got = torch.empty_like(xd)
        st.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=st):
            g.eps(xd.data_ptr(), md.data_ptr(), nd.data_ptr(), got)
        for m in (n, 17, n):
            nd.fill_(m)
            got.fill_(float("nan"))
            graph.replay()
            st.synchronize()
            assert torch.equal(got[:m], want[:m])
            assert torch.isnan(got[m:]).all()
        from paper_2609_36522_gb300 import abi
        abi.pa_gmm_check(g.h)
        g.close()


@pytest.mark.parametrize("form", [1, 0])
def test_sd15_other_denoiser_forms(form):
    """Whole-pipeline parity with the denoiser's two-kernel forms (dot
    products on the tensor cores, the default only above 16 components, or
    on the CUDA cores) in place of the cluster form."""
    w = W.SD15
    assert compare(w, oracle_run(w), gpu_run(w, gmm_form=form)).max() <= REL_TOL


@pytest.mark.parametrize("kind", [0, 1] + list(range(100, 113)))
def test_update_kernels_agree(kind):
    """Plain-load and tile-parallel bulk-copy update kernels (every launch
    shape) take the same decisions and agree with the oracle; their states
    differ only by the rounding of the compensated prefix sums."""
    w = W.Workload("multi-strip", T=40, window=24, batch=3, latent_shape=(4, 20, 20), K=6,
                   tol=1e-3, cache_thresh=0.05, seed=12)
    orc = oracle_run(w)
    ref = gpu_run(w, update_kernel=0)
    got = gpu_run(w, update_kernel=kind)
    assert got["stats"]["update_kernel"] == (0 if kind == 0 else 1)
    assert compare(w, orc, got).max() <= REL_TOL
    assert np.array_equal(ref["log"], got["log"])
    scale = np.abs(ref["x_final"]).max()
    assert np.abs(ref["x_final"] - got["x_final"]).max() <= 1e-6 * scale


@pytest.mark.parametrize("window,eta", [(24, 0.0), (64, 0.0), (100, 0.0), (64, 1.0), (32, 0.5)])
def test_register_update_matches_staged(window, eta):
    """The register-resident update (launch shape 12) performs the staged
    segment kernel's arithmetic (4 columns per lane, 8 warps) in the same
    order: decisions and final latents bit-identical, on a ragged last strip."""
    w = W.Workload("reg-vs-staged", T=100, window=window, batch=2, latent_shape=(4, 20, 20), K=6,
                   tol=1e-3, cache_thresh=0.05, seed=5, eta=eta)
    orc = oracle_run(w)
    staged = gpu_run(w, update_kernel=110)
    reg = gpu_run(w, update_kernel=112)
    assert np.array_equal(staged["log"], reg["log"])
    assert np.array_equal(staged["x_final"], reg["x_final"])
    assert compare(w, orc, reg).max() <= REL_TOL


# ---- lean register update kernel (launch shapes 200 + n) ---------------------

LEAN_SHAPES = {0: None, 1: (16, 7), 2: (12, 9), 3: (8, 4), 4: (8, 8), 5: (8, 4), 6: (4, 8)}
_LEAN_REF = {}


@pytest.mark.parametrize("kind", [200, 201, 202, 203, 204, 205, 206, 210, 211, 212, 213, 214])
@pytest.mark.parametrize("T,window,eta", [(100, 24, 0.0), (100, 64, 0.0), (100, 100, 0.0), (100, 32, 1.0),
                                          (100, 64, 0.5), (150, 112, 0.0), (150, 113, 0.0)])
def test_lean_update(kind, T, window, eta):
    """The lean register update (every launch shape, plain and compensated
    sums) takes the oracle's decisions, agrees with the oracle within 1e-5 and
    with the plain-load kernel within 1e-5 of the latents' scale, on a ragged
    last strip; a shape that cannot hold the window (or, with stochastic
    steps, compensated sums or the by-window choice) falls back to the bulk
    forms, as do shapes 5 and 6 (three and four CTAs per SM) with draws.
    Windows of 112 and 113 points are the 16 x 7 shape's capacity and one
    past it."""
    w = W.Workload("lean", T=T, window=window, batch=2, latent_shape=(4, 20, 20), K=6,
                   tol=1e-3, cache_thresh=0.05, seed=5, eta=eta)
    if (T, window, eta) not in _LEAN_REF:  # the oracle and the plain-load run, once per case
        _LEAN_REF[(T, window, eta)] = (oracle_run(w), gpu_run(w, update_kernel=0))
    orc, ref = _LEAN_REF[(T, window, eta)]
    got = gpu_run(w, update_kernel=kind)
    P = min(window, T)
    shape = LEAN_SHAPES[kind % 10] or ((8, 4) if P <= 32 else (8, 8) if P <= 64 else (16, 7))
    # stochastic steps: compensated sums and the by-window choice keep the bulk forms
    fits = P <= shape[0] * shape[1] and not (eta != 0.0 and (kind >= 210 or kind in (200, 205, 206)))
    assert got["stats"]["update_kernel"] == (2 if fits else 1)
    assert compare(w, orc, got).max() <= REL_TOL
    assert np.array_equal(ref["log"], got["log"])
    scale = np.abs(ref["x_final"]).max()
    assert np.abs(ref["x_final"] - got["x_final"]).max() <= 1e-5 * scale


@pytest.mark.parametrize("kind,eta", [(200, 0.0), (204, 0.0), (201, 1.0), (204, 1.0)])
def test_lean_update_long_schedule(kind, eta):
    """A 1000-step schedule: every CTA stages 1000 coefficient sets (two per
    thread and more) before the plan is known; decisions exact, latents
    within 1e-5 of the oracle."""
    w = W.Workload("lean-long", T=1000, window=64, batch=1, latent_shape=(4, 16, 16), K=4,
                   tol=1e-3, cache_thresh=0.05, seed=3, eta=eta)
    orc = oracle_run(w)
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-6), decision_margins(orc, w.tol, w.cache_thresh)
    got = gpu_run(w, update_kernel=kind)
    assert got["stats"]["update_kernel"] == 2
    assert compare(w, orc, got).max() <= REL_TOL


# ---- fused solver step: update, grid barrier, decision, batch from registers --

FUSED_CASES = [
    W.SD15,
    W.TINY,
    W.SD15.with_(window=64, name="SD window 64"),
    W.SD15.with_(T=150, window=112, latent_shape=(4, 32, 32), name="window 112"),
    W.Workload("ragged strips B3", T=40, window=24, batch=3, latent_shape=(4, 20, 20), K=6,
               tol=1e-3, cache_thresh=0.05, seed=12),
    # every error below tol: the window slides by p and the next window is all
    # lazy tail states, which the warp holding the frontier state writes
    W.Workload("huge tol", T=40, window=16, batch=2, latent_shape=(4, 8, 8), K=4,
               tol=1e3, cache_thresh=0.05, seed=2),
    W.Workload("cache 0.1", T=60, window=60, batch=1, latent_shape=(4, 32, 32), K=8,
               tol=1e-3, cache_thresh=0.1, seed=4),
]


@pytest.mark.parametrize("w", FUSED_CASES, ids=lambda w: w.name)
def test_fused_step_equals_update_and_planning(w):
    """The fused step (one kernel per iteration) against the update kernel +
    planning kernel pair of the same launch shape: the same arithmetic, so the
    iteration log, the final states and every iteration's reductions are
    bitwise equal -- the Eq. 2 / Eq. 4 sums are exact whatever order the CTAs
    add their partials in --, and both take the oracle's decisions."""
    orc = oracle_run(w)
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-6), decision_margins(orc, w.tol, w.cache_thresh)
    fused = gpu_run(w, update_kernel=3, reductions=True)
    split = gpu_run(w, reductions=True)
    assert fused["stats"]["update_kernel"] == 3 and split["stats"]["update_kernel"] == 2
    assert compare(w, orc, fused).max() <= REL_TOL
    assert np.array_equal(fused["log"], split["log"])
    assert np.array_equal(fused["x_final"], split["x_final"])
    assert len(fused["reductions"]) == len(split["reductions"]) > 0
    for (ef, df), (es, dss) in zip(fused["reductions"], split["reductions"]):
        assert np.array_equal(ef, es) and np.array_equal(df, dss)


def test_fused_step_falls_back_beyond_one_wave():
    """The batched workload's grid (128 strips x 8 trajectories) is not
    resident in one wave: the update and planning kernels run instead."""
    orc, gpu = _check(W.BATCHED.with_(T=40), update_kernel=3)
    assert gpu["stats"]["update_kernel"] == 2


@pytest.mark.parametrize("window", [24, 64])
def test_fused_step_stochastic(window):
    """Stochastic steps through the fused step (8 x 4 and 16 x 7 shapes)
    against the oracle and against the register-resident bulk form."""
    w = W.Workload("fused eta", T=100, window=window, batch=1, latent_shape=(4, 32, 32), K=6,
                   tol=1e-3, cache_thresh=0.05, seed=5, eta=1.0)
    orc = oracle_run(w)
    fused = gpu_run(w, update_kernel=3)
    assert fused["stats"]["update_kernel"] == 3
    assert compare(w, orc, fused).max() <= REL_TOL
    bulk = gpu_run(w, update_kernel=112)
    assert np.array_equal(fused["log"], bulk["log"])


# ---- stochastic steps (eta > 0): DDPM over the full 1000-step schedule -------

@pytest.mark.parametrize("w", [W.DDPM, W.DDPM128], ids=["window 64", "window 128"])
def test_ddpm_full_schedule(w):
    """DDPM (eta = 1, T = 1000, window 64, and 128: past the lean kernel's
    112 positions, so the staged form runs): decisions, miss lists and NFE
    bit-exact, final latents within 1e-5 of the oracle."""
    orc = oracle_run(w)
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-6), decision_margins(orc, w.tol, w.cache_thresh)
    rel = compare(w, orc, gpu_run(w))
    assert rel.max() <= 1e-5, rel


@pytest.mark.parametrize("eta", [1.0, 0.5])
@pytest.mark.parametrize("kind", [0, 1])
def test_noisy_steps_small(eta, kind):
    """Stochastic steps on small cases through both update kernels."""
    w = W.TINY.with_(T=16, window=8, eta=eta)
    rel = compare(w, oracle_run(w), gpu_run(w, update_kernel=kind))
    assert rel.max() <= 1e-5, rel


@pytest.mark.parametrize("shape,window", [((3, 7, 9), 5), ((4, 32, 32), 40), ((4, 16, 16), 128)])
def test_noisy_steps_shapes(shape, window):
    """Ragged D (plain kernel), a window past T, and a 128-point window."""
    w = W.TINY.with_(T=100, window=window, latent_shape=shape, K=4, eta=1.0)
    rel = compare(w, oracle_run(w), gpu_run(w))
    assert rel.max() <= 1e-5, rel


def test_noisy_misaligned_draws_rejected():
    """Draws not 16-byte aligned are refused on the host (no kernel runs)."""
    import torch
    from paper_2609_36522_gb300 import abi
    from paper_2609_36522_gb300.solver import Solver
    w = W.TINY.with_(T=20, window=8, latent_shape=(4, 8, 8), eta=1.0)
    a, x0, mu = W.inputs(w)
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch)
    buf = torch.zeros(w.batch * w.T * w.D + 1, dtype=torch.float32, device="cuda")
    with pytest.raises(abi.PaError) as e:
        abi.pa_set_noise(s.h, 1.0, buf[1:].data_ptr())
    assert e.value.status == abi.PA_ERR_ARG
    with pytest.raises(abi.PaError) as e:
        abi.pa_set_noise(s.h, 1.5, buf.data_ptr())
    assert e.value.status == abi.PA_ERR_ARG
    s.close()


def test_eta_zero_restores_ddim():
    """pa_set_noise(eta = 0) gives the DDIM run bit for bit."""
    w = W.TINY.with_(T=30, window=10, latent_shape=(4, 16, 16))
    plain = gpu_run(w)
    again = gpu_run(w.with_(eta=0.0))
    assert np.array_equal(plain["x_final"], again["x_final"])


# ---- bfloat16 cache entries (a storage option, not from the paper) ----------

def bf16_tolerance(w, orc):
    """Where the GPU's fp32 value and the oracle's fp64 value of a cache entry
    element straddle a bfloat16 rounding boundary, the two store neighbouring
    bfloat16 values: one ulp apart, at most 2^(floor(log2 max|ehat|) - 7). A
    reuse of that element moves one drift by |e_i| times that ulp, which the
    window sum carries to the final state. Two such events at the largest DDIM
    coefficient, relative to the smallest max|x_T|."""
    from oracle.ddim import step_coefficients
    _, e, _ = step_coefficients(W.alphas_cumprod(w.T), w.eta)
    ulp = 2.0 ** (np.floor(np.log2(np.abs(orc.ehat[orc.has_entry]).max())) - 7)
    return 2.0 * np.abs(e).max() * ulp / np.abs(orc.x_final).max(axis=1).min()


@pytest.mark.parametrize("w", [
    W.SD15, W.BATCHED,
    W.Workload("multi-strip", T=40, window=24, batch=3, latent_shape=(4, 20, 20), K=6,
               tol=1e-3, cache_thresh=0.05, seed=16),
    W.Workload("window 64", T=100, window=64, batch=2, latent_shape=(4, 20, 20), K=6,
               tol=1e-3, cache_thresh=0.05, seed=16),
    W.Workload("ragged odd D", T=30, window=12, batch=2, latent_shape=(3, 5, 7), K=3,
               tol=1e-3, cache_thresh=0.05, seed=3),
    W.Workload("window 128", T=150, window=128, batch=1, latent_shape=(4, 16, 16), K=4,
               tol=1e-3, cache_thresh=0.05, seed=15),
    W.TINY.with_(T=60, window=16, latent_shape=(4, 8, 8), eta=1.0, seed=3, name="stochastic steps"),
], ids=lambda w: w.name)
def test_bf16_cache_entries(w):
    """Entries stored as bfloat16 on both sides: decisions, miss lists and NFE
    exact (inputs guarded at 1e-3 relative, since an entry element can round to
    a neighbouring bfloat16 value when the GPU's fp32 value and the oracle's
    fp64 value straddle a rounding boundary), final latents within the bound of
    bf16_tolerance (about 1.6e-3 at T = 100). The lean register form runs where
    it applies, the plain-load kernel elsewhere (odd D, window 128, stochastic
    steps)."""
    from oracle.storage import round_bf16
    orc = oracle_run(w, cache_store=round_bf16)
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-3), decision_margins(orc, w.tol, w.cache_thresh)
    gpu = gpu_run(w, cache_bits=16)
    rel = compare(w, orc, gpu)
    assert rel.max() <= bf16_tolerance(w, orc), (rel, bf16_tolerance(w, orc))


@pytest.mark.parametrize("kind", [112, 0])
def test_bf16_cache_entries_other_forms(kind):
    """The register-resident bulk form and the plain-load kernel with
    bfloat16 entries, on the SD-shaped workload."""
    from oracle.storage import round_bf16
    w = W.SD15
    orc = oracle_run(w, cache_store=round_bf16)
    gpu = gpu_run(w, cache_bits=16, update_kernel=kind)
    assert gpu["stats"]["update_kernel"] == (1 if kind == 112 else 0)
    assert compare(w, orc, gpu).max() <= bf16_tolerance(w, orc)


def test_bf16_cache_rejected_while_stepped():
    from paper_2609_36522_gb300 import abi
    import torch
    from paper_2609_36522_gb300.solver import Solver
    w = W.TINY
    a, x0, _ = W.inputs(w)
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch)
    s.init(torch.from_numpy(x0).cuda())
    s.step()
    with pytest.raises(abi.PaError) as e:
        s.set_cache_precision(16)
    assert e.value.status == abi.PA_ERR_STATE
    with pytest.raises(abi.PaError) as e:
        abi.pa_set_cache_precision(s.h, 8)
    assert e.value.status == abi.PA_ERR_ARG
    s.close()



# ---- triangular Anderson mixing (ParaTAA-style update, pa_set_anderson) ------

TAA_CASES = [
    W.SD15, W.BATCHED.with_(T=60), W.TINY,
    W.SD15.with_(T=150, window=112, latent_shape=(4, 32, 32), name="window 112"),
    W.Workload("ragged strips B3", T=40, window=24, batch=3, latent_shape=(4, 20, 20), K=6,
               tol=1e-3, cache_thresh=0.05, seed=12),
    W.Workload("tight tol", T=100, window=100, batch=1, latent_shape=(4, 16, 16), K=16,
               tol=1e-5, cache_thresh=0.0, seed=0),
    W.Workload("cache 0.1", T=60, window=60, batch=1, latent_shape=(4, 32, 32), K=8,
               tol=1e-3, cache_thresh=0.1, seed=4),
    W.Workload("stochastic P24", T=100, window=24, batch=1, latent_shape=(4, 32, 32), K=6,
               tol=1e-3, cache_thresh=0.05, seed=5, eta=1.0),
    W.Workload("stochastic P64", T=100, window=64, batch=1, latent_shape=(4, 32, 32), K=6,
               tol=1e-3, cache_thresh=0.05, seed=5, eta=1.0),
]


@pytest.mark.parametrize("w", TAA_CASES, ids=lambda w: w.name)
def test_anderson_against_oracle(w):
    """Depth-1 triangular Anderson mixing: iteration log, miss lists, NFE and
    hits bit-exact against oracle.taa, final latents within 1e-5."""
    orc = oracle_run(w, anderson=1)
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-6), decision_margins(orc, w.tol, w.cache_thresh)
    gpu = gpu_run(w, anderson=1)
    assert gpu["stats"]["update_kernel"] == 4
    rel = compare(w, orc, gpu)
    assert rel.max() <= REL_TOL, rel


def test_anderson_depth_zero_restores_picard():
    """Switching the mixing on and off again gives the Picard run bit for bit."""
    w = W.Workload("taa off", T=40, window=16, batch=2, latent_shape=(4, 16, 16), K=4,
                   tol=1e-3, cache_thresh=0.05, seed=3)
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    ref = gpu_run(w)
    a, x0, mu = W.inputs(w)
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch)
    s.set_anderson(1)
    s.set_anderson(0)
    g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window)
    eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")
    s.init(torch.from_numpy(x0).cuda())
    while (out := s.step()) is not None:
        g.eps(out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps)
        s.submit_eps(eps)
    assert np.array_equal(s.result().cpu().numpy(), ref["x_final"])
    assert s.stats()["update_kernel"] == 2
    s.close()
    g.close()


def test_anderson_rejects_unsupported_settings():
    """Odd D, windows beyond 112 points and bfloat16 entries are refused with
    PA_ERR_ARG; a workspace that is too small with PA_ERR_WORKSPACE."""
    import torch
    from paper_2609_36522_gb300 import abi
    from paper_2609_36522_gb300.solver import Solver
    a = W.alphas_cumprod(30)
    for shape, window in (((3, 5, 7), 8), ((4, 8, 8), 113)):
        s = Solver(30 if window < 30 else 150, window, shape, W.alphas_cumprod(30 if window < 30 else 150),
                   1e-3, 0.05)
        with pytest.raises(abi.PaError) as e:
            s.set_anderson(1)
        assert e.value.status == abi.PA_ERR_ARG
        s.close()
    s = Solver(30, 8, (4, 8, 8), a, 1e-3, 0.05)
    s.set_cache_precision(16)
    with pytest.raises(abi.PaError) as e:
        s.set_anderson(1)
    assert e.value.status == abi.PA_ERR_ARG
    s.set_cache_precision(32)
    need = abi.pa_anderson_workspace_bytes(30, 8, 256, 1)
    buf = torch.empty(need, dtype=torch.uint8, device="cuda")
    with pytest.raises(abi.PaError) as e:
        abi.pa_set_anderson(s.h, 1, buf.data_ptr(), need - 256)
    assert e.value.status == abi.PA_ERR_WORKSPACE
    abi.pa_set_anderson(s.h, 1, buf.data_ptr(), need)
    with pytest.raises(abi.PaError) as e:
        s.set_cache_precision(16)
    assert e.value.status == abi.PA_ERR_ARG
    s.close()


def test_anderson_graph_replay_equals_sync():
    """A mixed generation captured as one CUDA graph (three solver kernels
    and the denoiser's two per iteration, chained by dependent launches) and
    replayed twice gives the synchronous run bit for bit."""
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    w = W.SD15
    sync = gpu_run(w, anderson=1)
    n_iters = len(sync["log"])
    a, x0, mu = W.inputs(w)
    st = torch.cuda.Stream()
    with torch.cuda.stream(st):
        s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, stream=st)
        s.set_anderson(1)
        g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window, stream=st)
        eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")
        x_dev = torch.from_numpy(x0).cuda()
        s.init(x_dev)
        out = s.step_async()
        g.eps(*out, eps)
        s.submit_eps(eps)
        st.synchronize()
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=st):
            s.init(x_dev)
            for _ in range(n_iters):
                out = s.step_async()
                g.eps(*out, eps)
                s.submit_eps(eps)
        for _ in range(2):
            graph.replay()
            st.synchronize()
            assert s.poll() == 0
            assert np.array_equal(s.result().cpu().numpy(), sync["x_final"])
            assert np.array_equal(s.iter_log(), sync["log"])
    s.close()
    g.close()


# ---- online adaptation of tau_cache (pa_set_cache_adaptation) -----------------

ADAPT_CASES = [
    (W.SD15.with_(cache_thresh=0.02, name="SD tau0 0.02"), (0.5, 0.5, 0.0, 0.2), {}),
    (W.SD15.with_(cache_thresh=0.1, name="SD tau0 0.1"), (0.5, 0.3, 0.01, 0.2), {}),
    (W.BATCHED.with_(T=60, cache_thresh=0.05), (1.0, 0.6, 0.0, 1.0), {}),
    (W.TINY, (1.0, 0.9, 0.0, 1.0), {}),
    (W.SD15.with_(cache_thresh=0.02, name="SD fused"), (0.5, 0.5, 0.0, 0.2), {"update_kernel": 3}),
    (W.SD15.with_(cache_thresh=0.02, name="SD anderson"), (0.5, 0.5, 0.0, 0.2), {"anderson": 1}),
    # 1000 pairs: without adaptation one CTA would plan; adaptation keeps the
    # every-CTA planner, here with several batch rows per CTA
    (W.Workload("10 x 100 adaptive", T=100, window=100, batch=10, latent_shape=(4, 8, 8), K=4,
                tol=1e-3, cache_thresh=0.02, seed=21), (0.5, 0.5, 0.0, 0.2), {}),
]


@pytest.mark.parametrize("w,adapt,kw", ADAPT_CASES, ids=lambda v: v.name if isinstance(v, W.Workload) else "")
def test_cache_adaptation_against_oracle(w, adapt, kw):
    """tau_cache adapted online on the device: the same tau per trajectory and
    iteration as the oracle (fp64, bit for bit), the same decisions, miss lists,
    NFE and hits; final latents within 1e-5. Also through the fused step and
    with Anderson mixing."""
    orc = oracle_run(w, adapt=adapt, anderson=kw.get("anderson", 0))
    assert margins_ok(orc, w.tol, w.cache_thresh, rel=1e-6), decision_margins(orc, w.tol, w.cache_thresh)
    gpu = gpu_run(w, adapt=adapt, **kw)
    rel = compare(w, orc, gpu)
    assert rel.max() <= REL_TOL, rel
    assert [r.tau for r in orc.records] == gpu["taus"]
    assert len({t for r in orc.records for t in r.tau}) > 1   # tau did move


def test_cache_adaptation_rate_zero_is_fixed():
    """Rate 0 (adaptation off) gives the fixed-threshold run bit for bit."""
    w = W.SD15
    fixed = gpu_run(w)
    off = gpu_run(w, adapt=(0.0, 0.5, 0.0, 1.0))
    assert np.array_equal(fixed["x_final"], off["x_final"])
    assert np.array_equal(fixed["log"], off["log"])
    assert all(t == [w.cache_thresh] for t in off["taus"])


def test_cache_adaptation_rejects_bad_arguments():
    from paper_2609_36522_gb300 import abi
    from paper_2609_36522_gb300.solver import Solver
    w = W.TINY
    s = Solver(w.T, w.window, w.latent_shape, W.alphas_cumprod(w.T), w.tol, w.cache_thresh)
    for args in ((-0.1, 0.5, 0.0, 1.0), (0.5, 1.5, 0.0, 1.0), (0.5, 0.5, 0.2, 0.1), (float("nan"), 0.5, 0.0, 1.0)):
        with pytest.raises(abi.PaError) as e:
            s.set_cache_adaptation(*args)
        assert e.value.status == abi.PA_ERR_ARG
    s.close()
    big = Solver(200, 128, (4, 4, 4), W.alphas_cumprod(200), 1e-3, 0.05, batch=9)
    with pytest.raises(abi.PaError) as e:
        big.set_cache_adaptation(0.5, 0.5)
    assert e.value.status == abi.PA_ERR_ARG
    big.close()
