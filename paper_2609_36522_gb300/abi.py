"""ctypes binding of libparaanya.so: the C functions under their own names.

Argument marshalling only -- every step of the solver runs in the library's
CUDA kernels. Functions returning a status raise ``PaError`` for a negative
status and return ``PA_DONE``/``PA_OK`` otherwise. Device pointers are plain
Python ints (e.g. ``tensor.data_ptr()``).

The library must have been built (``paper_2609_36522_gb300.build.build()`` or
``__graft_entry__.build()``); there is no fallback implementation.
"""
from __future__ import annotations

import ctypes as C
import os
import re

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "lib", "libparaanya.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "paraanya.h")

PA_OK, PA_DONE = 0, 1
PA_ERR_ARG, PA_ERR_STATE, PA_ERR_CUDA = -1, -2, -3
PA_ERR_WORKSPACE, PA_ERR_TIMEOUT, PA_ERR_DEVICE = -4, -5, -6


class PaError(RuntimeError):
    def __init__(self, fn, status, msg):
        super().__init__(f"{fn} -> {status_name(status)} ({status}): {msg}")
        self.status = status


class PaStats(C.Structure):
    _fields_ = [("iters", C.c_int64), ("nfe", C.c_int64), ("hits", C.c_int64),
                ("launches", C.c_int64), ("n_active", C.c_int32), ("n_miss", C.c_int32),
                ("device_status", C.c_int32), ("update_kernel", C.c_int32)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_}


class PaSrdsStats(C.Structure):
    _fields_ = [("iters", C.c_int64), ("nfe", C.c_int64), ("hits", C.c_int64),
                ("launches", C.c_int64), ("n_active", C.c_int32), ("n_miss", C.c_int32),
                ("device_status", C.c_int32), ("blocks", C.c_int32), ("block_steps", C.c_int32),
                ("reserved", C.c_int32)]

    def as_dict(self):
        return {k: getattr(self, k) for k, _ in self._fields_ if k != "reserved"}


_lib = None
VP = C.c_void_p
PVP = C.POINTER(C.c_void_p)

_PROTOS = {
    "pa_workspace_bytes": (C.c_size_t, [C.c_int, C.c_int, C.c_int64, C.c_int]),
    "pa_create": (C.c_int, [PVP, C.c_int, C.c_int, C.POINTER(C.c_int64), C.c_int,
                            C.POINTER(C.c_double), C.c_double, C.c_double, C.c_int,
                            VP, C.c_size_t, VP]),
    "pa_set_noise": (C.c_int, [VP, C.c_double, VP]),
    "pa_init": (C.c_int, [VP, VP]),
    "pa_step": (C.c_int, [VP, C.POINTER(C.c_int), PVP, PVP]),
    "pa_step_async": (C.c_int, [VP, PVP, PVP, PVP]),
    "pa_n_miss_dev": (C.c_void_p, [VP]),
    "pa_submit_eps": (C.c_int, [VP, VP]),
    "pa_poll": (C.c_int, [VP, C.POINTER(C.c_int)]),
    "pa_result": (C.c_int, [VP, VP]),
    "pa_poll_result": (C.c_int, [VP, VP, C.POINTER(C.c_int)]),
    "pa_poll_begin": (C.c_int, [VP, VP]),
    "pa_poll_end": (C.c_int, [VP, C.POINTER(C.c_int)]),
    "pa_loop_capture_begin": (C.c_int, [VP]),
    "pa_loop_capture_end": (C.c_int, [VP]),
    "pa_loop_launch": (C.c_int, [VP, VP]),
    "pa_nfe": (C.c_int64, [VP]),
    "pa_stats": (C.c_int, [VP, C.POINTER(PaStats)]),
    "pa_iter_log": (C.c_int, [VP, C.POINTER(C.c_int32), C.c_int, C.POINTER(C.c_int)]),
    "pa_last_reductions": (C.c_int, [VP, VP, VP]),
    "pa_set_update_kernel": (C.c_int, [VP, C.c_int]),
    "pa_set_cache_precision": (C.c_int, [VP, C.c_int]),
    "pa_anderson_workspace_bytes": (C.c_size_t, [C.c_int, C.c_int, C.c_int64, C.c_int]),
    "pa_set_cache_adaptation": (C.c_int, [VP, C.c_double, C.c_double, C.c_double, C.c_double]),
    "pa_cache_thresholds": (C.c_int, [VP, C.POINTER(C.c_double)]),
    "pa_set_anderson": (C.c_int, [VP, C.c_int, VP, C.c_size_t]),
    "pa_debug_set_wait_limit": (C.c_int, [VP, C.c_uint32]),
    "pa_set_kernel_timing": (C.c_int, [VP, C.c_int]),
    "pa_kernel_timing": (C.c_int, [VP, C.POINTER(C.c_double), C.POINTER(C.c_int64), C.c_int]),
    "pa_debug_gap": (C.c_int, [VP]),
    "pa_destroy": (None, [VP]),
    "pa_srds_workspace_bytes": (C.c_size_t, [C.c_int, C.c_int64, C.c_int]),
    "pa_srds_create": (C.c_int, [PVP, C.c_int, C.POINTER(C.c_int64), C.c_int, C.POINTER(C.c_double),
                                 C.c_double, C.c_double, C.c_int, VP, C.c_size_t, VP]),
    "pa_srds_init": (C.c_int, [VP, VP]),
    "pa_srds_step": (C.c_int, [VP, C.POINTER(C.c_int), PVP, PVP]),
    "pa_srds_step_async": (C.c_int, [VP, PVP, PVP, PVP]),
    "pa_srds_submit_eps": (C.c_int, [VP, VP]),
    "pa_srds_n_miss_dev": (VP, [VP]),
    "pa_srds_poll": (C.c_int, [VP, C.POINTER(C.c_int)]),
    "pa_srds_result": (C.c_int, [VP, VP]),
    "pa_srds_stats": (C.c_int, [VP, C.POINTER(PaSrdsStats)]),
    "pa_srds_errors": (C.c_int, [VP, VP]),
    "pa_srds_loop_capture_begin": (C.c_int, [VP]),
    "pa_srds_loop_capture_end": (C.c_int, [VP]),
    "pa_srds_loop_launch": (C.c_int, [VP]),
    "pa_srds_destroy": (None, [VP]),
    "pa_gmm_workspace_bytes": (C.c_size_t, [C.c_int, C.c_int64, C.c_int, C.c_int]),
    "pa_gmm_create": (C.c_int, [PVP, C.c_int, C.c_int64, VP, C.c_double,
                                C.POINTER(C.c_double), C.c_int, C.c_int, VP, C.c_size_t, VP]),
    "pa_gmm_eps": (C.c_int, [VP, VP, VP, VP, VP]),
    "pa_gmm_check": (C.c_int, [VP]),
    "pa_gmm_launches": (C.c_int64, [VP]),
    "pa_gmm_set_form": (C.c_int, [VP, C.c_int]),
    "pa_gmm_form": (C.c_int, [VP]),
    "pa_gmm_destroy": (None, [VP]),
    "pa_gmm_eps_noalloc": (C.c_int, [VP, C.c_int, C.c_int64, C.c_double, C.POINTER(C.c_double),
                                     C.c_int, VP, VP, C.c_int, VP, VP]),
    "pa_status_string": (C.c_char_p, [C.c_int]),
    "pa_last_error": (C.c_char_p, []),
}


def header_functions(path=HEADER):
    """Names of the functions include/paraanya.h declares."""
    text = open(path).read()
    return sorted(set(re.findall(r"^PA_API\s+[\w\s\*]+?\b(pa_\w+)\s*\(", text, re.M)))


def lib():
    """Load libparaanya.so (once). Raises if it has not been built."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise ImportError(f"{LIB_PATH} is missing: build it with "
                              "paper_2609_36522_gb300.build.build() (needs nvcc)")
        h = C.CDLL(LIB_PATH)
        for name, (res, args) in _PROTOS.items():
            f = getattr(h, name)
            f.restype = res
            f.argtypes = args
        _lib = h
    return _lib


def status_name(s):
    return lib().pa_status_string(int(s)).decode()


def last_error():
    return lib().pa_last_error().decode()


def _check(fn, status):
    if status < 0:
        raise PaError(fn, status, last_error())
    return status


def _dptr(x):
    return None if x is None else C.c_void_p(int(x))


# ---- the C functions ------------------------------------------------------

def pa_workspace_bytes(T, window, D, batch):
    return int(lib().pa_workspace_bytes(T, window, D, batch))


def pa_create(T, window, latent_shape, alphas_cumprod, tol, cache_thresh, batch,
              workspace_ptr, workspace_bytes, stream_ptr):
    shape = (C.c_int64 * len(latent_shape))(*[int(v) for v in latent_shape])
    alphas = (C.c_double * len(alphas_cumprod))(*[float(v) for v in alphas_cumprod])
    h = C.c_void_p()
    _check("pa_create", lib().pa_create(C.byref(h), T, window, shape, len(latent_shape), alphas,
                                        float(tol), float(cache_thresh), batch,
                                        _dptr(workspace_ptr), workspace_bytes, _dptr(stream_ptr)))
    return h


def pa_set_noise(h, eta, noise_ptr):
    return _check("pa_set_noise", lib().pa_set_noise(h, float(eta), _dptr(noise_ptr)))


def pa_init(h, x_init_ptr):
    return _check("pa_init", lib().pa_init(h, _dptr(x_init_ptr)))


def pa_step(h):
    """-> (status, n_miss, batch_x_ptr, miss_bt_ptr)."""
    n = C.c_int()
    bx, mb = C.c_void_p(), C.c_void_p()
    st = _check("pa_step", lib().pa_step(h, C.byref(n), C.byref(bx), C.byref(mb)))
    return st, n.value, bx.value, mb.value


def pa_step_async(h):
    """-> (batch_x_ptr, miss_bt_ptr, n_miss_dev_ptr)."""
    bx, mb, nm = C.c_void_p(), C.c_void_p(), C.c_void_p()
    _check("pa_step_async", lib().pa_step_async(h, C.byref(bx), C.byref(mb), C.byref(nm)))
    return bx.value, mb.value, nm.value


def pa_n_miss_dev(h):
    return lib().pa_n_miss_dev(h)


def pa_submit_eps(h, batch_eps_ptr):
    return _check("pa_submit_eps", lib().pa_submit_eps(h, _dptr(batch_eps_ptr)))


def pa_poll(h):
    """-> (status, n_active)."""
    n = C.c_int()
    st = _check("pa_poll", lib().pa_poll(h, C.byref(n)))
    return st, n.value


def pa_result(h, x_out_ptr):
    return _check("pa_result", lib().pa_result(h, _dptr(x_out_ptr)))


def pa_poll_result(h, x_out_ptr):
    """-> (status, n_active); x_out holds x_T when status is PA_DONE."""
    n = C.c_int()
    st = _check("pa_poll_result", lib().pa_poll_result(h, _dptr(x_out_ptr), C.byref(n)))
    return st, n.value


def pa_poll_begin(h, x_out_ptr):
    """Enqueue the copies of x_T (unless x_out_ptr is None) and the counters; no wait."""
    return _check("pa_poll_begin", lib().pa_poll_begin(h, _dptr(x_out_ptr)))


def pa_poll_end(h):
    """-> (status, n_active) of the oldest pending pa_poll_begin, after waiting for it."""
    n = C.c_int()
    st = _check("pa_poll_end", lib().pa_poll_end(h, C.byref(n)))
    return st, n.value


def pa_loop_capture_begin(h):
    return _check("pa_loop_capture_begin", lib().pa_loop_capture_begin(h))


def pa_loop_capture_end(h):
    return _check("pa_loop_capture_end", lib().pa_loop_capture_end(h))


def pa_loop_launch(h, x_init_ptr):
    return _check("pa_loop_launch", lib().pa_loop_launch(h, _dptr(x_init_ptr)))


def pa_srds_loop_capture_begin(h):
    return _check("pa_srds_loop_capture_begin", lib().pa_srds_loop_capture_begin(h))


def pa_srds_loop_capture_end(h):
    return _check("pa_srds_loop_capture_end", lib().pa_srds_loop_capture_end(h))


def pa_srds_loop_launch(h):
    return _check("pa_srds_loop_launch", lib().pa_srds_loop_launch(h))


def pa_nfe(h):
    v = int(lib().pa_nfe(h))
    if v < 0:
        raise PaError("pa_nfe", PA_ERR_STATE, last_error())
    return v


def pa_stats(h):
    s = PaStats()
    _check("pa_stats", lib().pa_stats(h, C.byref(s)))
    return s.as_dict()


LOG_FIELDS = 8   # t, p, misses, stride, e, hits at positions >= 1, positions with an entry, hits among them


def pa_iter_log(h, max_iters, batch):
    import numpy as np
    buf = (C.c_int32 * (max_iters * batch * LOG_FIELDS))()
    n = C.c_int()
    _check("pa_iter_log", lib().pa_iter_log(h, buf, max_iters, C.byref(n)))
    return np.frombuffer(buf, dtype=np.int32).reshape(max_iters, batch, LOG_FIELDS)[: n.value].copy()


def pa_last_reductions(h, batch, window):
    import numpy as np
    err = np.zeros((batch, window), dtype=np.float32)
    dl = np.zeros((batch, window), dtype=np.float32)
    _check("pa_last_reductions", lib().pa_last_reductions(
        h, err.ctypes.data_as(C.c_void_p), dl.ctypes.data_as(C.c_void_p)))
    return err, dl


def pa_set_update_kernel(h, kind):
    return _check("pa_set_update_kernel", lib().pa_set_update_kernel(h, int(kind)))


def pa_set_cache_precision(h, bits):
    return _check("pa_set_cache_precision", lib().pa_set_cache_precision(h, int(bits)))


def pa_set_cache_adaptation(h, rate, target, tau_min=0.0, tau_max=float("inf")):
    return _check("pa_set_cache_adaptation", lib().pa_set_cache_adaptation(h, float(rate), float(target),
                                                                             float(tau_min), float(tau_max)))


def pa_cache_thresholds(h, batch):
    buf = (C.c_double * batch)()
    _check("pa_cache_thresholds", lib().pa_cache_thresholds(h, buf))
    return [buf[b] for b in range(batch)]


def pa_anderson_workspace_bytes(T, window, D, batch):
    return int(lib().pa_anderson_workspace_bytes(T, window, D, batch))


def pa_set_anderson(h, depth, workspace_ptr, workspace_bytes):
    return _check("pa_set_anderson", lib().pa_set_anderson(h, int(depth), _dptr(workspace_ptr),
                                                             int(workspace_bytes)))


def pa_debug_set_wait_limit(h, polls):
    return _check("pa_debug_set_wait_limit", lib().pa_debug_set_wait_limit(h, int(polls)))


def pa_set_kernel_timing(h, enable):
    return _check("pa_set_kernel_timing", lib().pa_set_kernel_timing(h, int(bool(enable))))


def pa_kernel_timing(h, reset=True):
    """-> (total update-kernel ms, launches timed) since the last reset."""
    ms = C.c_double()
    n = C.c_int64()
    _check("pa_kernel_timing", lib().pa_kernel_timing(h, C.byref(ms), C.byref(n), int(bool(reset))))
    return ms.value, n.value


def pa_debug_gap(stream_ptr):
    return _check("pa_debug_gap", lib().pa_debug_gap(_dptr(stream_ptr)))


def pa_destroy(h):
    lib().pa_destroy(h)


def pa_gmm_workspace_bytes(K, D, max_rows, T):
    return int(lib().pa_gmm_workspace_bytes(K, D, max_rows, T))


def pa_gmm_create(K, D, means_ptr, std, alphas_cumprod, T, max_rows, workspace_ptr,
                  workspace_bytes, stream_ptr):
    alphas = (C.c_double * len(alphas_cumprod))(*[float(v) for v in alphas_cumprod])
    h = C.c_void_p()
    _check("pa_gmm_create", lib().pa_gmm_create(C.byref(h), K, D, _dptr(means_ptr), float(std),
                                                alphas, T, max_rows, _dptr(workspace_ptr),
                                                workspace_bytes, _dptr(stream_ptr)))
    return h


def pa_gmm_eps(g, batch_x_ptr, miss_bt_ptr, n_rows_dev_ptr, batch_eps_ptr):
    return _check("pa_gmm_eps", lib().pa_gmm_eps(g, _dptr(batch_x_ptr), _dptr(miss_bt_ptr),
                                                 _dptr(n_rows_dev_ptr), _dptr(batch_eps_ptr)))


def pa_gmm_check(g):
    return _check("pa_gmm_check", lib().pa_gmm_check(g))


def pa_gmm_launches(g):
    return int(lib().pa_gmm_launches(g))


def pa_gmm_set_form(g, form):
    return _check("pa_gmm_set_form", lib().pa_gmm_set_form(g, int(form)))


def pa_gmm_form(g):
    return int(lib().pa_gmm_form(g))


def pa_gmm_destroy(g):
    lib().pa_gmm_destroy(g)


def pa_gmm_eps_noalloc(means_ptr, K, D, std, alphas_cumprod, batch_x_ptr, miss_bt_ptr, n_rows,
                       batch_eps_ptr, stream_ptr):
    """Denoiser eps with the library's fixed device scratch (no allocation)."""
    alphas = (C.c_double * len(alphas_cumprod))(*[float(v) for v in alphas_cumprod])
    return _check("pa_gmm_eps_noalloc", lib().pa_gmm_eps_noalloc(
        _dptr(means_ptr), int(K), int(D), float(std), alphas, len(alphas_cumprod) - 1,
        _dptr(batch_x_ptr), _dptr(miss_bt_ptr), int(n_rows), _dptr(batch_eps_ptr), _dptr(stream_ptr)))


# ---- Parareal (SRDS-style) sampler -----------------------------------------

def pa_srds_workspace_bytes(T, D, batch):
    return int(lib().pa_srds_workspace_bytes(T, D, batch))


def pa_srds_create(T, latent_shape, alphas_cumprod, tol, cache_thresh, batch, workspace_ptr,
                   workspace_bytes, stream_ptr):
    shape = (C.c_int64 * len(latent_shape))(*[int(v) for v in latent_shape])
    alphas = (C.c_double * len(alphas_cumprod))(*[float(v) for v in alphas_cumprod])
    h = C.c_void_p()
    _check("pa_srds_create", lib().pa_srds_create(C.byref(h), T, shape, len(latent_shape), alphas, float(tol),
                                                  float(cache_thresh), batch, _dptr(workspace_ptr),
                                                  workspace_bytes, _dptr(stream_ptr)))
    return h


def pa_srds_init(h, x_ptr):
    return _check("pa_srds_init", lib().pa_srds_init(h, _dptr(x_ptr)))


def pa_srds_step(h):
    n = C.c_int(0)
    bx, mb = C.c_void_p(), C.c_void_p()
    st = _check("pa_srds_step", lib().pa_srds_step(h, C.byref(n), C.byref(bx), C.byref(mb)))
    return st, n.value, bx.value, mb.value


def pa_srds_step_async(h):
    bx, mb, nm = C.c_void_p(), C.c_void_p(), C.c_void_p()
    st = _check("pa_srds_step_async", lib().pa_srds_step_async(h, C.byref(bx), C.byref(mb), C.byref(nm)))
    return st, bx.value, mb.value, nm.value


def pa_srds_n_miss_dev(h):
    return lib().pa_srds_n_miss_dev(h)


def pa_srds_submit_eps(h, eps_ptr):
    return _check("pa_srds_submit_eps", lib().pa_srds_submit_eps(h, _dptr(eps_ptr)))


def pa_srds_poll(h):
    n = C.c_int(0)
    st = _check("pa_srds_poll", lib().pa_srds_poll(h, C.byref(n)))
    return st, n.value


def pa_srds_result(h, out_ptr):
    return _check("pa_srds_result", lib().pa_srds_result(h, _dptr(out_ptr)))


def pa_srds_stats(h):
    out = PaSrdsStats()
    _check("pa_srds_stats", lib().pa_srds_stats(h, C.byref(out)))
    return out.as_dict()


def pa_srds_errors(h, n_blocks, batch):
    import numpy as _np
    buf = _np.zeros((n_blocks, batch), dtype=_np.float32)
    _check("pa_srds_errors", lib().pa_srds_errors(h, buf.ctypes.data_as(C.c_void_p)))
    return buf


def pa_srds_destroy(h):
    lib().pa_srds_destroy(h)
