"""The device-driven generation loop (pa_loop_*): a CUDA graph whose
conditional WHILE node repeats two captured iterations until every trajectory
has reached T (Sec. 2.1's outer loop, Eq. 1 and 2, run by the GPU). Each case
compares the loop with the synchronous host-driven run of the same handle bit
for bit: final states, iteration log, NFE and hits."""
import numpy as np
import pytest

import workload as W
from paper_2609_36522_gb300 import abi

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_36522_gb300 import build as pa_build
    pa_build.build()


def _setup(w, anderson=0, adapt=None, eta=0.0):
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    a, x0, mu = W.inputs(w)
    st = torch.cuda.Stream()
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, stream=st)
    g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window, stream=st)
    eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")
    if anderson:
        s.set_anderson(anderson)
    if adapt:
        s.set_cache_adaptation(*adapt)
    if eta:
        gen = torch.Generator(device="cuda").manual_seed(7)
        s.set_noise(eta, torch.randn(w.batch * w.T * w.D, generator=gen, device="cuda"))
    torch.cuda.synchronize()

    def denoise(bx, mb, nm):
        g.eps(bx, mb, nm, eps)
        return eps

    return s, g, eps, torch.from_numpy(x0).cuda(), denoise


def _sync(s, x0, denoise):
    s.init(x0)
    while True:
        plan = s.step()
        if plan is None:
            break
        s.submit_eps(denoise(plan.batch_x_ptr, plan.miss_bt_ptr, s.n_miss_dev()))
    st = s.stats()
    return s.result().clone(), s.iter_log(), st["nfe"], st["hits"], st["iters"]


LOOP_CASES = [
    ("sd15", W.SD15, {}),
    ("sd15 body 2", W.SD15, {"chunk": 2}),
    ("large auto body", W.LARGE.with_(T=60), {"chunk": None}),
    ("batched body 6", W.BATCHED.with_(T=40), {"chunk": 6}),
    ("batched", W.BATCHED.with_(T=40), {}),
    ("large", W.LARGE.with_(T=60), {}),
    ("tiny", W.TINY, {}),
    ("sd15 anderson", W.SD15.with_(T=60), {"anderson": 1}),
    ("batched adaptive", W.BATCHED.with_(T=40), {"adapt": (0.5, 0.2, 0.0, 1.0)}),
    ("ddim eta 1", W.SD15.with_(T=50, window=24), {"eta": 1.0}),
    ("64 trajectories", W.Workload("64 trajectories", T=40, window=32, batch=64, latent_shape=(4, 4, 4), K=4,
                                   tol=1e-3, cache_thresh=0.05, seed=14), {"chunk": None}),
    ("9 x 128 pairs", W.Workload("9 x 128 pairs", T=200, window=128, batch=9, latent_shape=(4, 4, 4), K=4,
                                 tol=1e-3, cache_thresh=0.05, seed=13), {"chunk": None}),
    # more batch rows than one wave of planning CTAs: each CTA copies several rows
    ("4 x 100 pairs", W.Workload("4 x 100 pairs", T=100, window=100, batch=4, latent_shape=(4, 8, 8), K=4,
                                 tol=1e-3, cache_thresh=0.05, seed=19), {"chunk": None}),
    ("window past T, odd T", W.Workload("odd", T=37, window=64, batch=3, latent_shape=(4, 8, 8), K=4,
                                        tol=1e-3, cache_thresh=0.05, seed=15), {"chunk": 2}),
    ("ragged D", W.Workload("ragged", T=20, window=7, batch=2, latent_shape=(3, 7, 9), K=4,
                            tol=1e-3, cache_thresh=0.05, seed=16), {"chunk": 6}),
]


@pytest.mark.parametrize("name,w,kw", LOOP_CASES, ids=[c[0] for c in LOOP_CASES])
def test_loop_equals_host_driven_run(name, w, kw):
    """generate() through the device loop (bodies of 4 iterations unless
    stated), twice in a row and then after eager iterations (the launch
    starts over from x_init), gives the host-driven run's x_T, log, NFE and
    hits: iterations run past the end change nothing."""
    import torch
    kw = dict(kw)
    chunk = kw.pop("chunk", 4)
    s, g, eps, x0, denoise = _setup(w, **kw)
    want, log, nfe, hits, iters = _sync(s, x0, denoise)
    for _ in range(2):
        out = s.generate(x0, denoise, chunk=chunk)
        assert s.generate_path() == "device loop", s.__dict__.get("loop_error")
        assert s.last_chunk == (chunk or iters + (iters & 1))
        assert torch.equal(out, want)
        st = s.stats()
        assert np.array_equal(s.iter_log(), log)
        assert (st["nfe"], st["hits"], st["iters"]) == (nfe, hits, iters)
    # eager iterations first: the launch starts over from x_init
    s.init(x0)
    for _ in range(3):
        bx, mb, nm = s.step_async()
        s.submit_eps(denoise(bx, mb, nm))
    abi.pa_loop_launch(s.h, x0.data_ptr())
    stt, n = abi.pa_poll_result(s.h, out.data_ptr())
    assert stt == abi.PA_DONE and n == 0
    assert torch.equal(out, want)
    assert np.array_equal(s.iter_log(), log)
    s.close()
    g.close()


def test_loop_generations_in_flight():
    """generate(wait=False) keeps up to two generations queued; each output
    equals the host-driven run of its own x_init, and finish() checks the
    rest."""
    import torch
    w = W.BATCHED.with_(T=40)
    s, g, eps, x0, denoise = _setup(w)
    inits = [x0, x0.flip(0).contiguous(), (0.5 * x0).contiguous(), x0.roll(1, dims=1).contiguous()]
    wants = [_sync(s, xi, denoise)[0] for xi in inits]
    outs = [torch.empty(w.batch, w.D, dtype=torch.float32).pin_memory() for _ in inits]
    s.generate(inits[0], denoise, out=outs[0])  # the capture
    for xi, o in zip(inits, outs):
        o.fill_(float("nan"))
        s.generate(xi, denoise, out=o, wait=False)
    s.finish()
    for o, want in zip(outs, wants):
        assert torch.equal(o, want.cpu())
    # pinned host (the poll kernel writes it), device and pageable host (the copy engine) outputs
    for out in (torch.empty(w.batch, w.D, dtype=torch.float32).pin_memory(),
                torch.empty(w.batch, w.D, dtype=torch.float32, device="cuda"),
                torch.empty(w.batch, w.D, dtype=torch.float32)):
        out.fill_(float("nan"))
        assert torch.equal(s.generate(inits[1], denoise, out=out).cpu(), wants[1].cpu())
    s.close()
    g.close()


def test_loop_call_order_and_settings():
    """PA_ERR_STATE: pa_loop_capture_end with no capture, a launch with
    nothing captured, capture_begin before pa_init, after an odd number of
    iterations, with kernel timing enabled and while a capture is open, a
    setter during a capture, a body of one iteration (the capture is closed
    and the stream works after it), host stepping after a launch, a launch
    between pa_step_async and pa_submit_eps. Launches back to back each
    start over; a setter drops the loop."""
    import torch
    w = W.SD15.with_(T=40)
    s, g, eps, x0, denoise = _setup(w)

    def state_error(f, *a):
        with pytest.raises(abi.PaError) as e:
            f(*a)
        assert e.value.status == abi.PA_ERR_STATE

    state_error(abi.pa_loop_capture_end, s.h)
    state_error(abi.pa_loop_launch, s.h, x0.data_ptr())   # nothing captured
    state_error(abi.pa_loop_capture_begin, s.h)   # before pa_init
    s.init(x0)
    bx, mb, nm = s.step_async()
    s.submit_eps(denoise(bx, mb, nm))
    state_error(abi.pa_loop_capture_begin, s.h)   # odd iteration count
    s.init(x0)
    abi.pa_set_kernel_timing(s.h, 1)
    state_error(abi.pa_loop_capture_begin, s.h)
    abi.pa_set_kernel_timing(s.h, 0)
    abi.pa_loop_capture_begin(s.h)
    state_error(abi.pa_loop_capture_begin, s.h)
    state_error(abi.pa_set_update_kernel, s.h, 2)
    with torch.cuda.stream(s.stream):
        bx, mb, nm = s.step_async()
        s.submit_eps(denoise(bx, mb, nm))
    state_error(abi.pa_loop_capture_end, s.h)     # one iteration only: closed, nothing kept
    state_error(abi.pa_loop_launch, s.h, x0.data_ptr())
    want, log, nfe, hits, iters = _sync(s, x0, denoise)  # the stream and the handle still work
    out = s.generate(x0, denoise)
    assert torch.equal(out, want)
    state_error(s.step_async)                     # host stepping closed after a launch ...
    s.init(x0)                                    # ... until pa_init
    bx, mb, nm = s.step_async()
    state_error(abi.pa_loop_launch, s.h, x0.data_ptr())   # between pa_step_async and pa_submit_eps
    s.submit_eps(denoise(bx, mb, nm))
    abi.pa_loop_launch(s.h, x0.data_ptr())
    abi.pa_loop_launch(s.h, x0.data_ptr())        # back to back: each starts over
    stt, n = abi.pa_poll_result(s.h, out.data_ptr())
    assert stt == abi.PA_DONE and torch.equal(out, want)
    abi.pa_set_update_kernel(s.h, 2)              # drops the loop
    state_error(abi.pa_loop_launch, s.h, x0.data_ptr())
    s.close()
    g.close()


def test_loop_ends_on_a_device_error():
    """With the device-side wait limit at zero the staged update kernel's
    bounded waits (segment form) give up at once: the loop test sees the status and ends
    the loop (the launch returns); the poll reports PA_ERR_TIMEOUT, and after
    pa_init the handle reproduces the clean run through the loop."""
    import torch
    w = W.SD15.with_(T=30, window=30)
    s, g, eps, x0, denoise = _setup(w)
    s.set_update_kernel(101)  # the staged segment form: its row copies wait on mbarriers
    want = _sync(s, x0, denoise)[0]
    abi.pa_debug_set_wait_limit(s.h, 0)
    s.init(x0)
    for _ in range(2):
        bx, mb, nm = s.step_async()
        s.submit_eps(denoise(bx, mb, nm))
    s.init(x0)
    abi.pa_loop_capture_begin(s.h)
    with torch.cuda.stream(s.stream):
        for _ in range(2):
            bx, mb, nm = s.step_async()
            s.submit_eps(denoise(bx, mb, nm))
    abi.pa_loop_capture_end(s.h)
    abi.pa_loop_launch(s.h, x0.data_ptr())
    out = torch.empty_like(want)
    with pytest.raises(abi.PaError) as e:
        abi.pa_poll_result(s.h, out.data_ptr())
    assert e.value.status == abi.PA_ERR_TIMEOUT
    abi.pa_debug_set_wait_limit(s.h, 1 << 17)     # drops the loop
    s._drop_graphs()
    assert torch.equal(s.generate(x0, denoise), want)
    assert s.stats()["device_status"] == 0
    s.close()
    g.close()


def test_loop_capture_survives_other_cuda_work_and_reports_invalidation():
    """(a) Another CUDA graph destroyed while the loop is being captured (as a
    finalizer of an unrelated object may do) leaves the capture valid: it is
    relaxed, so the loop runs and gives the host-driven x_T. (b) A capture the
    caller invalidates (a synchronisation of the capturing stream) makes
    pa_loop_capture_end report PA_ERR_CUDA, keeping and destroying nothing;
    the handle then captures again and runs."""
    import torch
    w = W.SD15.with_(T=40)
    s, g, eps, x0, denoise = _setup(w)
    want = _sync(s, x0, denoise)[0]
    s.init(x0)
    bx, mb, nm = s.step_async()  # eager warm-up outside the capture
    s.submit_eps(denoise(bx, mb, nm))

    def other_graph():
        side = torch.cuda.Stream()
        buf = torch.zeros(1024, device="cuda")
        gr = torch.cuda.CUDAGraph()
        with torch.cuda.graph(gr, stream=side):
            buf.add_(1.0)
        return gr, buf

    gr, buf = other_graph()
    torch.cuda.synchronize()
    s.init(x0)
    abi.pa_loop_capture_begin(s.h)
    with torch.cuda.stream(s.stream):
        for k in range(4):
            bx, mb, nm = s.step_async()
            s.submit_eps(denoise(bx, mb, nm))
            if k == 1:
                del gr  # destroys that graph (and its executable) mid-capture
    abi.pa_loop_capture_end(s.h)
    abi.pa_loop_launch(s.h, x0.data_ptr())
    out = torch.empty_like(want)
    stt, n = abi.pa_poll_result(s.h, out.data_ptr())
    assert stt == abi.PA_DONE and torch.equal(out, want)
    # (b) invalidated by the caller
    s.init(x0)
    abi.pa_loop_capture_begin(s.h)
    with torch.cuda.stream(s.stream):
        bx, mb, nm = s.step_async()
        g.eps(bx, mb, nm, eps)
        with pytest.raises(RuntimeError):
            s.stream.synchronize()  # not allowed while capturing: the capture is invalidated
        with pytest.raises(abi.PaError):
            s.submit_eps(eps)  # its launches fail on the invalidated capture
    with pytest.raises(abi.PaError) as e:
        abi.pa_loop_capture_end(s.h)
    assert e.value.status == abi.PA_ERR_CUDA
    with pytest.raises(abi.PaError) as e:
        abi.pa_loop_launch(s.h, x0.data_ptr())  # nothing was kept
    assert e.value.status == abi.PA_ERR_STATE
    torch.cuda.synchronize()
    s._drop_graphs()
    assert torch.equal(s.generate(x0, denoise), want)
    s.close()
    g.close()
