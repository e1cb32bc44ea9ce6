"""GPU-side ABI behaviour: call order, restart, counters, device status."""
import numpy as np
import pytest

import workload as W
from paper_2609_36522_gb300 import abi

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    from paper_2609_36522_gb300 import build as pa_build
    pa_build.build()


def _solver(w=W.TINY, **kw):
    import torch
    from paper_2609_36522_gb300.solver import Solver, GmmDenoiser
    a, x0, mu = W.inputs(w)
    s = Solver(w.T, w.window, w.latent_shape, a, w.tol, w.cache_thresh, batch=w.batch, **kw)
    g = GmmDenoiser(torch.from_numpy(mu).cuda(), w.gmm_std, a, w.batch * s.window, **kw)
    eps = torch.empty(w.batch * s.window, w.D, dtype=torch.float32, device="cuda")
    x0d = torch.from_numpy(x0).cuda()
    torch.cuda.synchronize()
    return s, g, eps, x0d


def _run(s, g, eps):
    while True:
        out = s.step()
        if out is None:
            return
        n, bx, mb = out.n_miss, out.batch_x, out.miss_bt
        g.eps(out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps)
        s.submit_eps(eps)


def test_call_order_is_enforced():
    s, g, eps, x0 = _solver()
    with pytest.raises(abi.PaError) as e:
        s.submit_eps(eps)
    assert e.value.status == abi.PA_ERR_STATE
    with pytest.raises(abi.PaError) as e:
        abi.pa_step(s.h)
    assert e.value.status == abi.PA_ERR_STATE
    s.init(x0)
    with pytest.raises(abi.PaError) as e:
        s.result()
    assert e.value.status == abi.PA_ERR_STATE
    out = s.step()
    assert out is not None and out[0] == W.TINY.window
    with pytest.raises(abi.PaError) as e:
        abi.pa_step(s.h)                       # step twice without submitting
    assert e.value.status == abi.PA_ERR_STATE
    s.submit_eps(eps)
    with pytest.raises(abi.PaError) as e:
        s.submit_eps(eps)                      # submit twice
    assert e.value.status == abi.PA_ERR_STATE
    _run(s, g, eps)
    assert s.step() is None                    # PA_DONE is sticky
    s.result()
    st = s.stats()
    assert st["device_status"] == 0 and st["n_active"] == 0


def test_restart_reproduces_bits_and_counters():
    s, g, eps, x0 = _solver(W.BATCHED.with_(T=30))
    s.init(x0)
    _run(s, g, eps)
    first = s.result().cpu().numpy()
    n1, st1, log1 = s.nfe(), s.stats(), s.iter_log()
    s.init(x0)
    _run(s, g, eps)
    assert np.array_equal(first, s.result().cpu().numpy())
    assert s.nfe() == n1
    assert np.array_equal(log1, s.iter_log())
    assert s.stats()["iters"] == st1["iters"]


def test_launch_counter_and_reductions():
    s, g, eps, x0 = _solver()
    s.init(x0)
    _run(s, g, eps)
    st = s.stats()
    # the first plan with its batch (one kernel) + per iteration: the update
    # and the planning kernel (decision fused with the next gather), or the
    # fused step
    assert st["update_kernel"] == 2
    assert st["launches"] == 1 + 2 * st["iters"]
    s.set_update_kernel(3)
    s.init(x0)
    _run(s, g, eps)
    st2 = s.stats()
    assert st2["update_kernel"] == 3
    assert st2["launches"] - st["launches"] == 1 + st2["iters"]
    err, dl = s.last_reductions()
    assert np.isfinite(err).all() and np.isfinite(dl).all()


def test_nonblocking_stream():
    import torch
    st = torch.cuda.Stream()
    w = W.TINY
    s, g, eps, x0 = _solver(w, stream=st)
    with torch.cuda.stream(st):
        s.init(x0)
        while True:
            out = s.step()
            if out is None:
                break
            n, bx, mb = out.n_miss, out.batch_x, out.miss_bt
            abi.pa_gmm_eps(g.h, out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps.data_ptr())
            s.submit_eps(eps)
        a = s.result().cpu().numpy()
    st.synchronize()
    s2, g2, eps2, _ = _solver(w)
    s2.init(x0)
    _run(s2, g2, eps2)
    assert np.array_equal(a, s2.result().cpu().numpy())


@pytest.mark.parametrize("kind", [110, 101, 3])
def test_bounded_wait_reports_timeout_and_context_survives(kind):
    """Force every mbarrier wait of a bulk-copy update kernel (the staged
    segment form, the tiled pipeline), or the fused step's grid barrier, to
    give up at once: the kernel records a timeout (no hang, no fault), drains
    its copies, and the next synchronising call reports PA_ERR_TIMEOUT. After
    pa_init the same solver reproduces a clean run bit for bit."""
    w = W.SD15.with_(T=30, window=30)
    s, g, eps, x0 = _solver(w)
    s.set_update_kernel(kind)
    s.init(x0)
    _run(s, g, eps)
    clean = s.result().cpu().numpy()
    s.init(x0)
    out = s.step()
    g.eps(out.batch_x_ptr, out.miss_bt_ptr, s.n_miss_dev(), eps)
    abi.pa_debug_set_wait_limit(s.h, 0)
    s.submit_eps(eps)
    with pytest.raises(abi.PaError) as e:
        s.step()
    assert e.value.status == abi.PA_ERR_TIMEOUT
    abi.pa_debug_set_wait_limit(s.h, 1 << 17)
    s.init(x0)
    _run(s, g, eps)
    assert np.array_equal(clean, s.result().cpu().numpy())
    assert s.stats()["device_status"] == 0
    assert s.stats()["update_kernel"] == (3 if kind == 3 else 1)


def test_update_kernel_selector_rejects_unknown_shapes():
    """pa_set_update_kernel takes 0, 1, 2, 3, 100 + bulk shape, 200 + lean
    shape (0-6, 10-16) and 300 + fused shape (0-6); anything else is
    PA_ERR_ARG and leaves the choice as it was."""
    w = W.TINY
    s, g, eps, x0 = _solver(w)
    for kind in (3, 300, 306, 2, 0, 1, 100, 112, 200, 206, 210, 216):
        abi.pa_set_update_kernel(s.h, kind)
    for kind in (-1, 4, 99, 113, 199, 207, 209, 217, 299, 307, 310):
        with pytest.raises(abi.PaError) as e:
            abi.pa_set_update_kernel(s.h, kind)
        assert e.value.status == abi.PA_ERR_ARG
    s.init(x0)
    _run(s, g, eps)
    # the last accepted choice, 216, stays: shape 6 has no compensated form,
    # so the update falls back to the bulk forms
    assert s.stats()["update_kernel"] == 1


def test_result_buffer_is_checked():
    """Solver.result refuses an output buffer of the wrong size, type or
    layout before the library writes batch x D values into it."""
    import torch
    w = W.TINY
    s, g, eps, x0 = _solver(w)
    s.init(x0)
    _run(s, g, eps)
    for bad in (torch.empty(w.batch * w.D - 1, dtype=torch.float32, device="cuda"),
                torch.empty(w.batch, w.D, dtype=torch.float64, device="cuda"),
                torch.empty(w.batch, 2 * w.D, dtype=torch.float32, device="cuda")[:, ::2]):
        with pytest.raises(ValueError):
            s.result(bad)
    good = torch.empty(w.batch * w.D, dtype=torch.float32, device="cuda")
    assert torch.equal(s.result(good).view(w.batch, w.D), s.result())


def test_poll_result_is_poll_and_result_behind_one_sync():
    """pa_poll_result: PA_ERR_STATE before pa_init and between pa_step_async
    and pa_submit_eps; PA_OK with the active count while trajectories run;
    PA_DONE with x_out bit-equal to pa_result once they are done; and the
    generate() loop built on it gives the synchronous result."""
    import torch
    w = W.BATCHED.with_(T=30)
    st = torch.cuda.Stream()  # generate() captures a CUDA graph: not on the default stream
    s, g, eps, x0 = _solver(w, stream=st)
    out = torch.empty(w.batch, w.D, dtype=torch.float32, device="cuda")
    with pytest.raises(abi.PaError) as e:
        abi.pa_poll_result(s.h, out.data_ptr())
    assert e.value.status == abi.PA_ERR_STATE
    s.init(x0)
    bx, mb, nm = s.step_async()
    with pytest.raises(abi.PaError) as e:
        abi.pa_poll_result(s.h, out.data_ptr())
    assert e.value.status == abi.PA_ERR_STATE
    g.eps(bx, mb, nm, eps)
    s.submit_eps(eps)
    st, n = abi.pa_poll_result(s.h, out.data_ptr())
    assert st == abi.PA_OK and n == w.batch
    while True:
        bx, mb, nm = s.step_async()
        g.eps(bx, mb, nm, eps)
        s.submit_eps(eps)
        st, n = abi.pa_poll_result(s.h, out.data_ptr())
        if st == abi.PA_DONE:
            break
        assert n > 0
    assert n == 0
    assert torch.equal(out, s.result())
    host = torch.empty(w.batch, w.D, dtype=torch.float32).pin_memory()

    def denoise(bx, mb, nm):
        g.eps(bx, mb, nm, eps)
        return eps

    for _ in range(2):
        s.generate(x0, denoise, out=host)
        assert torch.equal(host, out.cpu())


def test_poll_begin_end_keeps_one_iteration_queued():
    """pa_poll_begin / pa_poll_end: PA_ERR_STATE before pa_init, with no poll
    pending, between pa_step_async and pa_submit_eps, for a third pending poll
    and inside a stream capture; two polls with no work between them report
    the same count; a loop that enqueues iteration k + 1 before it waits for
    the poll of iteration k sees the synchronous loop's active counts, ends
    with x_T bit-equal to pa_result, and the iteration it ran past the end
    changes neither the iteration log nor the NFE."""
    import torch
    w = W.BATCHED.with_(T=30)
    st = torch.cuda.Stream()
    s, g, eps, x0 = _solver(w, stream=st)
    out = torch.empty(w.batch, w.D, dtype=torch.float32, device="cuda")

    def state_error(f, *a):
        with pytest.raises(abi.PaError) as e:
            f(*a)
        assert e.value.status == abi.PA_ERR_STATE

    state_error(abi.pa_poll_begin, s.h, out.data_ptr())
    state_error(abi.pa_poll_end, s.h)
    # the synchronous loop's active counts, log and NFE
    s.init(x0)
    counts = []
    while True:
        bx, mb, nm = s.step_async()
        g.eps(bx, mb, nm, eps)
        s.submit_eps(eps)
        stt, n = abi.pa_poll_result(s.h, out.data_ptr())
        counts.append(n)
        if stt == abi.PA_DONE:
            break
    log, nfe, want = s.iter_log(), s.nfe(), out.clone()
    s.init(x0)
    bx, mb, nm = s.step_async()
    state_error(abi.pa_poll_begin, s.h, out.data_ptr())
    g.eps(bx, mb, nm, eps)
    s.submit_eps(eps)
    abi.pa_poll_begin(s.h, None)
    abi.pa_poll_begin(s.h, out.data_ptr())
    state_error(abi.pa_poll_begin, s.h, out.data_ptr())
    assert abi.pa_poll_end(s.h) == (abi.PA_OK, counts[0])
    assert abi.pa_poll_end(s.h) == (abi.PA_OK, counts[0])
    state_error(abi.pa_poll_end, s.h)
    with torch.cuda.stream(st):
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=st):
            state_error(abi.pa_poll_begin, s.h, out.data_ptr())
            out.zero_()  # something captured (never replayed)
    # pipelined: iteration k + 1 is enqueued before the poll of iteration k is read
    host = torch.full((w.batch, w.D), float("nan"), dtype=torch.float32).pin_memory()
    s.init(x0)
    seen = []
    for k in range(len(counts) + 1):
        bx, mb, nm = s.step_async()
        g.eps(bx, mb, nm, eps)
        s.submit_eps(eps)
        abi.pa_poll_begin(s.h, host.data_ptr())
        if k == 0:
            continue
        stt, n = abi.pa_poll_end(s.h)
        seen.append(n)
        if stt == abi.PA_DONE:
            assert abi.pa_poll_end(s.h) == (abi.PA_DONE, 0)
            break
    assert seen == counts
    assert torch.equal(host, want.cpu())
    assert torch.equal(s.result(), want)
    assert np.array_equal(s.iter_log(), log) and s.nfe() == nfe
