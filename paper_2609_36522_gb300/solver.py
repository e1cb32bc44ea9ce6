"""Thin torch-side handles over the C ABI.

PyTorch provides device memory (the workspaces are ``torch.uint8`` CUDA
tensors from the caching allocator) and the stream; every computation is a
kernel of libparaanya.so. Device outputs of the library are exposed as views
into the workspace, never copied.
"""
from __future__ import annotations

import gc
import numpy as np
import torch

from collections import namedtuple

from . import abi

# One planned iteration: M misses, views of the gathered batch and the miss
# list (both [M][...], empty when M == 0), and the raw device addresses (valid
# even when M == 0, for device-side denoisers that read M themselves).
Plan = namedtuple("Plan", "n_miss batch_x miss_bt batch_x_ptr miss_bt_ptr")


def _stream_ptr(stream):
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream), stream


class Solver:
    """Cached sliding-window Picard DDIM solver of ``batch`` trajectories."""

    def __init__(self, T, window, latent_shape, alphas_cumprod, tol, cache_thresh,
                 batch=1, stream=None, device="cuda"):
        if not torch.cuda.is_available():
            raise RuntimeError("Solver needs a CUDA device; there is no CPU implementation")
        self.T, self.batch = int(T), int(batch)
        self.window = min(int(window), self.T)
        self.latent_shape = tuple(int(v) for v in latent_shape)
        self.D = int(np.prod(self.latent_shape))
        self.stream_ptr, self.stream = _stream_ptr(stream)
        nbytes = abi.pa_workspace_bytes(self.T, int(window), self.D, self.batch)
        if nbytes == 0:
            raise abi.PaError("pa_workspace_bytes", abi.PA_ERR_ARG, "unsupported sizes")
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=device)
        self.h = abi.pa_create(self.T, int(window), self.latent_shape, list(alphas_cumprod),
                               tol, cache_thresh, self.batch, self.workspace.data_ptr(),
                               nbytes, self.stream_ptr)

    # -- views into the workspace -------------------------------------------
    def _view(self, ptr, n, dtype, shape):
        off = int(ptr) - self.workspace.data_ptr()
        nb = int(np.prod(shape)) * torch.tensor([], dtype=dtype).element_size()
        return self.workspace[off: off + nb].view(dtype).view(*shape)

    def set_noise(self, eta, noise=None):
        """Stochastic steps: noise is a CUDA float32 [batch][T][D] tensor of
        N(0, 1) draws (kept alive by this object); eta = 0 restores DDIM."""
        self._drop_graphs()
        if eta == 0.0:
            self._noise_keepalive = None
            abi.pa_set_noise(self.h, 0.0, None)
            return
        if (not isinstance(noise, torch.Tensor) or not noise.is_cuda or noise.dtype != torch.float32
                or not noise.is_contiguous() or noise.numel() != self.batch * self.T * self.D):
            raise ValueError("noise must be a contiguous CUDA float32 [batch][T][D] tensor")
        self._noise_keepalive = noise
        abi.pa_set_noise(self.h, eta, noise.data_ptr())

    def _x_init(self, x_init):
        x = x_init if isinstance(x_init, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(x_init))
        if x.dtype != torch.float32 or not x.is_contiguous() or x.numel() != self.batch * self.D:
            raise ValueError("x_init must be a contiguous float32 [batch][D] tensor")
        self._x_init_keepalive = x
        return x

    def init(self, x_init):
        """x_init: [batch][D] fp32 tensor (CUDA or CPU, contiguous)."""
        abi.pa_init(self.h, self._x_init(x_init).data_ptr())

    def step(self):
        """-> None when done, else a Plan (M, batch_x [M][D], miss_bt [M][2], raw pointers)."""
        st, n, bx, mb = abi.pa_step(self.h)
        if st == abi.PA_DONE:
            return None
        return Plan(n, self._view(bx, n, torch.float32, (n, self.D)),
                    self._view(mb, n, torch.int32, (n, 2)), bx, mb)

    def step_async(self):
        """-> (batch_x_ptr, miss_bt_ptr, n_miss_dev_ptr), no host synchronisation."""
        return abi.pa_step_async(self.h)

    def n_miss_dev(self):
        """Device address of the planned miss count (for device-side denoisers)."""
        return abi.pa_n_miss_dev(self.h)

    def submit_eps(self, eps):
        if isinstance(eps, torch.Tensor):
            if eps.dtype != torch.float32 or not eps.is_cuda or not eps.is_contiguous():
                raise ValueError("eps must be a contiguous CUDA float32 tensor")
            eps = eps.data_ptr()
        abi.pa_submit_eps(self.h, eps)

    def poll(self):
        st, n = abi.pa_poll(self.h)
        return n

    def _out(self, out):
        if out is None:
            return torch.empty(self.batch, self.D, dtype=torch.float32, device=self.workspace.device)
        if (not isinstance(out, torch.Tensor) or out.dtype != torch.float32 or not out.is_contiguous()
                or out.numel() != self.batch * self.D):
            raise ValueError("out must be a contiguous float32 tensor of batch x D elements")
        return out

    def result(self, out=None):
        """x_T [batch][D] into ``out`` (a contiguous float32 CUDA or host
        tensor of batch x D elements), else into a new CUDA tensor."""
        out = self._out(out)
        abi.pa_result(self.h, out.data_ptr())
        return out

    def poll_result(self, out):
        """pa_poll and pa_result behind one synchronisation: the number of
        trajectories still active; when it is 0, ``out`` holds x_T."""
        st, n = abi.pa_poll_result(self.h, out.data_ptr())
        return n

    def generate(self, x_init, denoise, out=None, chunk=None, wait=True):
        """One whole generation in one call: x_init [batch][D] (CUDA tensor or
        pinned host tensor) in, x_T out (into ``out``, a CUDA or pinned host
        tensor, else a new CUDA tensor).

        ``denoise(batch_x_ptr, miss_bt_ptr, n_miss_dev_ptr)`` enqueues eps_theta
        of the planned misses on this solver's stream, reading the miss count
        on the device (as ``GmmDenoiser.eps`` does), and returns the CUDA eps
        tensor it wrote; it must write the same buffer on every call, allocate
        nothing and be capturable in a CUDA graph.

        The first call per (denoiser, chunk) captures ``chunk`` (even)
        iterations as the body of a device-side loop
        (``pa_loop_capture_begin/_end``: a CUDA graph whose conditional WHILE
        node repeats the body until every trajectory has reached T;
        iterations after that, up to the end of the pass, do nothing). Each
        pass of the body costs a few microseconds of loop control and each
        iteration past the end a few more, so the best body holds the
        generation's iteration count: with ``chunk=None`` the first call per
        denoiser runs one host-driven generation of its x_init and takes its
        iteration count, rounded up to even, as the body (later generations
        that need more iterations simply take more passes). Each call then
        enqueues ``pa_loop_launch`` (x_init copied in, pa_init's kernel, one
        launch of the graph) and ``pa_poll_begin`` (x_T and the counters
        copied out): no host round trip inside a generation. With ``wait``
        the call returns after that poll; without it, it returns at once with
        at most two generations in flight (a third call first waits for the
        oldest and checks it), and ``finish()`` waits for the rest; ``out``
        and x_init must then stay untouched until then. The capture runs with
        the garbage collector paused (no finalizer's CUDA call lands in it).

        Where the loop cannot be built (a driver without conditional graph
        nodes, or a capture the runtime invalidated), ``chunk`` (even)
        iterations are captured as a CUDA graph and replayed with one
        ``pa_poll_result`` per replay instead (always waiting). The captured launches carry the solver's settings of the
        capture: the setters of this class drop them; a denoiser's own settings
        must stay as they were captured (or pass a new callable)."""
        if chunk is None:
            chunk = self._auto_chunk(x_init, denoise)
        if chunk < 2 or chunk % 2:
            raise ValueError("chunk must be a positive even number (iterations alternate two plan copies)")
        self.last_chunk = chunk
        out = self._out(out)
        key = (denoise, chunk)
        if self.__dict__.get("_loop_for") != key and self.__dict__.get("loop_error") is None:
            self._capture_loop(x_init, denoise, chunk)
        if self.__dict__.get("_loop_for") == key:
            pending = self.__dict__.setdefault("_pending", [])
            abi.pa_loop_launch(self.h, self._x_init(x_init).data_ptr())
            if len(pending) == 2:
                self._end_poll()
            abi.pa_poll_begin(self.h, out.data_ptr())
            pending.append((out, self._x_init_keepalive))
            if wait:
                self.finish()
            return out
        self.finish()
        graphs = self.__dict__.setdefault("_gen_graphs", {})
        self.init(x_init)
        gr = graphs.get(key)
        if gr is None:
            # one eager iteration first: launch-time set-up (kernel attributes)
            # happens outside the capture
            bx, mb, nm = self.step_async()
            self.submit_eps(denoise(bx, mb, nm))
            self.init(x_init)
            gr = torch.cuda.CUDAGraph()
            with torch.cuda.graph(gr, stream=self.stream):
                for _ in range(chunk):
                    bx, mb, nm = self.step_async()
                    self.submit_eps(denoise(bx, mb, nm))
            graphs[key] = gr
            self.init(x_init)  # the capture advanced the host state without running anything
        for _ in range(self.T // chunk + 2):
            with torch.cuda.stream(self.stream):  # replay() launches on the current stream
                gr.replay()
            if self.poll_result(out) == 0:  # one synchronisation: the counters and x_T together
                return out
        raise RuntimeError("generate: trajectories did not reach T within T iterations")

    def _auto_chunk(self, x_init, denoise):
        """The loop body for ``generate(chunk=None)``: the iteration count of
        one host-driven generation of x_init, rounded up to even (learned once
        per denoiser; 4 where the loop is not available)."""
        if self.__dict__.get("loop_error") is not None:
            return 4
        auto = self.__dict__.setdefault("_auto", {})
        if denoise not in auto:
            self.finish()
            self.init(x_init)
            while True:
                plan = self.step()
                if plan is None:
                    break
                self.submit_eps(denoise(plan.batch_x_ptr, plan.miss_bt_ptr, self.n_miss_dev()))
            n = int(self.stats()["iters"])
            auto[denoise] = max(2, n + (n & 1))
        return auto[denoise]

    def _capture_loop(self, x_init, denoise, chunk):
        self.finish()
        self.init(x_init)
        # one eager iteration first: launch-time set-up (kernel attributes)
        # happens outside the capture
        bx, mb, nm = self.step_async()
        self.submit_eps(denoise(bx, mb, nm))
        self.init(x_init)
        # no finalizer of unrelated objects (which may call into CUDA) runs
        # inside the capture: collect before it, pause the collector during it
        gc.collect()
        gc_was_on = gc.isenabled()
        gc.disable()
        try:
            abi.pa_loop_capture_begin(self.h)
            try:
                with torch.cuda.stream(self.stream):  # torch work of the denoiser lands in the body
                    for _ in range(chunk):
                        bx, mb, nm = self.step_async()
                        self.submit_eps(denoise(bx, mb, nm))
            except BaseException:
                try:
                    abi.pa_loop_capture_end(self.h)  # closes the capture; the body is incomplete
                except abi.PaError:
                    pass
                raise
            end_error = None
            try:
                abi.pa_loop_capture_end(self.h)
            except abi.PaError as e:
                end_error = e
        finally:
            if gc_was_on:
                gc.enable()
        if end_error is not None:
            if end_error.status != abi.PA_ERR_CUDA:
                raise end_error
            self.loop_error = str(end_error)  # refused or invalidated: replay and poll instead
            return
        self._loop_for = (denoise, chunk)

    def _end_poll(self):
        pending = self.__dict__.get("_pending", [])
        pending.pop(0)
        st, n = abi.pa_poll_end(self.h)
        if n != 0:
            raise RuntimeError(f"generate: {n} trajectories had not reached T when the device loop ended")

    def finish(self):
        """Wait for every generation still in flight (generate with wait=False) and check it."""
        while self.__dict__.get("_pending"):
            self._end_poll()

    def generate_path(self):
        """How generate runs: 'device loop' or, without conditional graph nodes, 'graph replay + poll'."""
        return "graph replay + poll" if self.__dict__.get("loop_error") else "device loop"

    def nfe(self):
        return abi.pa_nfe(self.h)

    def stats(self):
        return abi.pa_stats(self.h)

    def iter_log(self):
        return abi.pa_iter_log(self.h, self.T + 1, self.batch)

    def last_reductions(self):
        return abi.pa_last_reductions(self.h, self.batch, self.window)

    def set_update_kernel(self, kind):
        """Picard-update kernel: 0 plain loads, 1 bulk forms, 2 lean register
        form (the default), 3 fused step, 100 + n / 200 + n / 300 + n launch
        shapes of the bulk / lean / fused forms (a tuning aid;
        pa_set_update_kernel documents them)."""
        self._drop_graphs()
        abi.pa_set_update_kernel(self.h, kind)

    def set_cache_adaptation(self, rate, target, tau_min=0.0, tau_max=float("inf")):
        """Online adaptation of tau_cache per trajectory (rate 0: off); pa_init must follow."""
        self._drop_graphs()
        abi.pa_set_cache_adaptation(self.h, rate, target, tau_min, tau_max)

    def cache_thresholds(self):
        """tau_cache of the planned iteration's hit test, per trajectory."""
        return abi.pa_cache_thresholds(self.h, self.batch)

    def set_anderson(self, depth):
        """Triangular Anderson mixing of the iterates (ParaTAA-style update):
        depth 1 mixes with the previous iteration (its workspace is allocated
        here), 0 restores plain Picard. pa_init must follow."""
        self._drop_graphs()
        if depth == 0:
            abi.pa_set_anderson(self.h, 0, None, 0)
            self._taa_workspace = None
            return
        nbytes = abi.pa_anderson_workspace_bytes(self.T, self.window, self.D, self.batch)
        ws = torch.empty(nbytes, dtype=torch.uint8, device=self.workspace.device)
        abi.pa_set_anderson(self.h, depth, ws.data_ptr(), nbytes)
        self._taa_workspace = ws

    def set_cache_precision(self, bits):
        """16: bfloat16 cache entries, 32: fp32 (default). pa_init must follow."""
        self._drop_graphs()
        abi.pa_set_cache_precision(self.h, bits)

    def _drop_graphs(self):
        self.finish()
        self.__dict__.pop("_gen_graphs", None)
        self.__dict__.pop("_loop_for", None)  # the C setters drop the loop graph itself
        self.__dict__.pop("_auto", None)      # the settings may change the iteration count

    def close(self):
        try:
            if getattr(self, "h", None) is not None:
                self._drop_graphs()  # captured launches refer to this workspace
        finally:
            if getattr(self, "h", None) is not None:
                abi.pa_destroy(self.h)
                self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class GmmDenoiser:
    """Posterior-mean eps of an isotropic Gaussian mixture (synthetic eps_theta)."""

    def __init__(self, means, std, alphas_cumprod, max_rows, stream=None):
        if not isinstance(means, torch.Tensor) or not means.is_cuda or means.dtype != torch.float32:
            raise ValueError("means must be a CUDA float32 [K][D] tensor")
        self.means = means.contiguous()
        self.K, self.D = self.means.shape
        self.T = len(alphas_cumprod) - 1
        self.max_rows = int(max_rows)
        self.stream_ptr, self.stream = _stream_ptr(stream)
        nbytes = abi.pa_gmm_workspace_bytes(self.K, self.D, self.max_rows, self.T)
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=self.means.device)
        self.h = abi.pa_gmm_create(self.K, self.D, self.means.data_ptr(), std, list(alphas_cumprod),
                                   self.T, self.max_rows, self.workspace.data_ptr(), nbytes,
                                   self.stream_ptr)

    def eps(self, batch_x_ptr, miss_bt_ptr, n_rows_dev_ptr, out):
        abi.pa_gmm_eps(self.h, batch_x_ptr, miss_bt_ptr, n_rows_dev_ptr,
                       out.data_ptr() if isinstance(out, torch.Tensor) else out)

    def launches(self):
        return abi.pa_gmm_launches(self.h)

    def set_form(self, form):
        """1: dot products on the tensor cores; 0: on the CUDA cores."""
        abi.pa_gmm_set_form(self.h, form)

    def form(self):
        return abi.pa_gmm_form(self.h)

    def close(self):
        if getattr(self, "h", None) is not None:
            abi.pa_gmm_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


class SrdsSolver:
    """Cached Parareal (SRDS-style) DDIM sampler through the C ABI; the same
    denoiser interface as Solver (batch_x, miss_bt, device miss count)."""

    def __init__(self, T, latent_shape, alphas_cumprod, tol, cache_thresh, batch=1, stream=None):
        self.T, self.batch = int(T), int(batch)
        self.latent_shape = tuple(int(v) for v in latent_shape)
        self.D = int(np.prod(self.latent_shape))
        self.stream_ptr, self.stream = _stream_ptr(stream)
        nbytes = abi.pa_srds_workspace_bytes(self.T, self.D, self.batch)
        if nbytes == 0:
            raise ValueError("unsupported sizes for the Parareal sampler")
        dev = torch.device("cuda", torch.cuda.current_device())
        self.workspace = torch.empty(nbytes, dtype=torch.uint8, device=dev)
        self.h = abi.pa_srds_create(self.T, self.latent_shape, list(alphas_cumprod), tol, cache_thresh,
                                    self.batch, self.workspace.data_ptr(), nbytes, self.stream_ptr)
        st = abi.pa_srds_stats(self.h)
        self.blocks, self.block_steps = st["blocks"], st["block_steps"]
        self.max_rows = self.batch * self.blocks

    def init(self, x_init):
        x = x_init if isinstance(x_init, torch.Tensor) else torch.from_numpy(np.ascontiguousarray(x_init))
        if x.dtype != torch.float32 or not x.is_contiguous() or x.numel() != self.batch * self.D:
            raise ValueError("x_init must be a contiguous float32 [batch][D] tensor")
        self._x_init_keepalive = x
        abi.pa_srds_init(self.h, x.data_ptr())

    def _view(self, ptr, dtype, shape):
        off = int(ptr) - self.workspace.data_ptr()
        nb = int(np.prod(shape)) * torch.tensor([], dtype=dtype).element_size()
        return self.workspace[off: off + nb].view(dtype).view(*shape)

    def step(self):
        """-> None when done, else a Plan of the next evaluation stage."""
        st, n, bx, mb = abi.pa_srds_step(self.h)
        if st == abi.PA_DONE:
            return None
        return Plan(n, self._view(bx, torch.float32, (n, self.D)), self._view(mb, torch.int32, (n, 2)), bx, mb)

    def n_miss_dev(self):
        return abi.pa_srds_n_miss_dev(self.h)

    def step_async(self):
        """-> None when done, else (batch_x_ptr, miss_bt_ptr, n_miss_dev_ptr)."""
        st, bx, mb, nm = abi.pa_srds_step_async(self.h)
        if st == abi.PA_DONE:
            return None
        return bx, mb, nm

    def submit_eps(self, eps):
        if isinstance(eps, torch.Tensor):
            if eps.dtype != torch.float32 or not eps.is_cuda or not eps.is_contiguous():
                raise ValueError("eps must be a contiguous CUDA float32 tensor")
            eps = eps.data_ptr()
        abi.pa_srds_submit_eps(self.h, eps)

    def poll(self):
        st, n = abi.pa_srds_poll(self.h)
        return n

    def result(self, out=None):
        """x_T [batch][D] into ``out`` (a contiguous float32 CUDA or host
        tensor of batch x D elements), else into a new CUDA tensor."""
        if out is None:
            out = torch.empty(self.batch, self.D, dtype=torch.float32, device=self.workspace.device)
        elif (not isinstance(out, torch.Tensor) or out.dtype != torch.float32 or not out.is_contiguous()
              or out.numel() != self.batch * self.D):
            raise ValueError("out must be a contiguous float32 tensor of batch x D elements")
        abi.pa_srds_result(self.h, out.data_ptr())
        return out

    def generate(self, x_init, denoise, out=None):
        """One whole Parareal generation in one call: x_init in, x_T out (into
        ``out``, a CUDA or pinned host tensor, else a new CUDA tensor).
        ``denoise`` as for ``Solver.generate`` (enqueues on this sampler's
        stream, reads the miss count on the device, returns the eps buffer it
        always writes, capturable). The first call per denoiser captures every
        stage of every Parareal iteration as one CUDA graph of IF nodes
        (``pa_srds_loop_capture_begin/_end``; iterations after convergence
        are skipped on the device); each call then enqueues ``pa_srds_init``
        and ``pa_srds_loop_launch`` and reads x_T with ``pa_srds_result`` (one
        synchronisation). Where the driver refuses the conditional nodes, the
        stages are issued from Python with a ``pa_srds_poll`` every 4."""
        if self.__dict__.get("_loop_for") is not denoise and self.__dict__.get("loop_error") is None:
            self._capture(x_init, denoise)
        self.init(x_init)
        if self.__dict__.get("_loop_for") is denoise:
            abi.pa_srds_loop_launch(self.h)
        else:
            done = False
            while not done:
                for _ in range(4):
                    plan = self.step_async()
                    if plan is None:
                        done = True
                        break
                    self.submit_eps(denoise(*plan))
                if not done:
                    done = self.poll() == 0
        return self.result(out)

    def _capture(self, x_init, denoise):
        self.init(x_init)
        plan = self.step_async()  # one eager stage: launch-time set-up outside the capture
        self.submit_eps(denoise(*plan))
        self.init(x_init)
        gc.collect()  # no finalizer of unrelated objects runs inside the capture
        gc_was_on = gc.isenabled()
        gc.disable()
        try:
            abi.pa_srds_loop_capture_begin(self.h)
            try:
                with torch.cuda.stream(self.stream):
                    while True:
                        plan = self.step_async()
                        if plan is None:
                            break
                        self.submit_eps(denoise(*plan))
            except BaseException as exc:
                try:
                    abi.pa_srds_loop_capture_end(self.h)  # closes the capture if open; nothing is kept
                except abi.PaError:
                    pass
                if isinstance(exc, abi.PaError) and exc.status == abi.PA_ERR_CUDA:
                    self.loop_error = str(exc)  # the driver refused the graph: issue stages from Python
                    return
                raise
            try:
                abi.pa_srds_loop_capture_end(self.h)
            except abi.PaError as e:
                if e.status != abi.PA_ERR_CUDA:
                    raise
                self.loop_error = str(e)
                return
        finally:
            if gc_was_on:
                gc.enable()
        self._loop_for = denoise

    def generate_path(self):
        """'device graph' or, without conditional graph nodes, 'stages from Python'."""
        return "stages from Python" if self.__dict__.get("loop_error") else "device graph"

    def stats(self):
        return abi.pa_srds_stats(self.h)

    def errors(self):
        return abi.pa_srds_errors(self.h, self.blocks, self.batch)

    def close(self):
        if getattr(self, "h", None) is not None:
            abi.pa_srds_destroy(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
