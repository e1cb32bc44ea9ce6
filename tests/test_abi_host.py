"""Host-only checks of the C ABI: the library builds, loads, exports every
function include/paraanya.h declares, and rejects bad arguments before it
touches a GPU. No kernel runs here."""
import ctypes as C

import pytest

from paper_2609_36522_gb300 import abi
from paper_2609_36522_gb300 import build as pa_build


@pytest.fixture(scope="module")
def lib():
    pa_build.build()
    return abi.lib()


def test_every_declared_function_is_exported(lib):
    names = abi.header_functions()
    assert len(names) >= 20
    exported = C.CDLL(abi.LIB_PATH)
    for n in names:
        assert hasattr(exported, n), n
    # and the binding covers exactly the declared functions
    assert sorted(abi._PROTOS) == names


def test_workspace_sizes(lib):
    b1 = abi.pa_workspace_bytes(100, 100, 16384, 1)
    # four window-sized fp32 arrays plus the batch buffer dominate
    assert b1 >= 4 * 100 * 16384 * 4
    assert b1 % 256 == 0
    assert abi.pa_workspace_bytes(100, 200, 16384, 1) == b1  # window clamps to T
    assert abi.pa_workspace_bytes(0, 8, 16, 1) == 0
    assert abi.pa_workspace_bytes(16, 0, 16, 1) == 0
    assert abi.pa_workspace_bytes(16, 2048, 16, 1) == 0
    assert abi.pa_workspace_bytes(16, 8, 16, 65) == 0
    assert abi.pa_gmm_workspace_bytes(16, 16384, 100, 100) > 0
    assert abi.pa_gmm_workspace_bytes(129, 16384, 100, 100) == 0


def test_status_strings(lib):
    assert abi.status_name(abi.PA_OK) == "PA_OK"
    assert abi.status_name(abi.PA_ERR_TIMEOUT) == "PA_ERR_TIMEOUT"
    assert abi.status_name(12345) == "PA_UNKNOWN"


def _create(**kw):
    args = dict(T=16, window=8, latent_shape=(4, 8, 8), alphas=[0.5] * 17, tol=1e-3,
                cache=0.05, batch=1, ws=0x1000, nbytes=1 << 30)
    args.update(kw)
    return abi.pa_create(args["T"], args["window"], args["latent_shape"], args["alphas"],
                         args["tol"], args["cache"], args["batch"], args["ws"], args["nbytes"], None)


@pytest.mark.parametrize("kw,status", [
    (dict(T=0, alphas=[0.5]), abi.PA_ERR_ARG),
    (dict(window=0), abi.PA_ERR_ARG),
    (dict(batch=0), abi.PA_ERR_ARG),
    (dict(latent_shape=(4, 0, 8)), abi.PA_ERR_ARG),
    (dict(alphas=[0.5] * 16 + [1.5]), abi.PA_ERR_ARG),
    (dict(alphas=[0.0] + [0.5] * 16), abi.PA_ERR_ARG),
    (dict(tol=-1.0), abi.PA_ERR_ARG),
    (dict(tol=float("inf")), abi.PA_ERR_ARG),
    (dict(cache=float("nan")), abi.PA_ERR_ARG),
    (dict(ws=0x1004), abi.PA_ERR_WORKSPACE),
    (dict(nbytes=1024), abi.PA_ERR_WORKSPACE),
    (dict(ws=0), abi.PA_ERR_WORKSPACE),
])
def test_create_rejects_bad_arguments(lib, kw, status):
    with pytest.raises(abi.PaError) as ei:
        _create(**kw)
    assert ei.value.status == status
    assert abi.last_error()


def test_null_handles_are_rejected(lib):
    L = abi.lib()
    n = C.c_int()
    assert L.pa_init(None, None) == abi.PA_ERR_ARG
    assert L.pa_step(None, C.byref(n), None, None) == abi.PA_ERR_ARG
    assert L.pa_submit_eps(None, None) == abi.PA_ERR_ARG
    assert L.pa_poll(None, None) == abi.PA_ERR_ARG
    assert L.pa_result(None, None) == abi.PA_ERR_ARG
    assert L.pa_poll_result(None, None, None) == abi.PA_ERR_ARG
    assert L.pa_poll_begin(None, None) == abi.PA_ERR_ARG
    assert L.pa_poll_end(None, None) == abi.PA_ERR_ARG
    assert L.pa_loop_capture_begin(None) == abi.PA_ERR_ARG
    assert L.pa_loop_capture_end(None) == abi.PA_ERR_ARG
    assert L.pa_loop_launch(None, None) == abi.PA_ERR_ARG
    assert L.pa_srds_loop_capture_begin(None) == abi.PA_ERR_ARG
    assert L.pa_srds_loop_capture_end(None) == abi.PA_ERR_ARG
    assert L.pa_srds_loop_launch(None) == abi.PA_ERR_ARG
    assert L.pa_nfe(None) == -1
    assert L.pa_n_miss_dev(None) is None
    assert L.pa_set_update_kernel(None, 0) == abi.PA_ERR_ARG
    assert L.pa_set_cache_precision(None, 16) == abi.PA_ERR_ARG
    L.pa_destroy(None)
    L.pa_gmm_destroy(None)
    assert L.pa_gmm_launches(None) == -1
    assert L.pa_gmm_form(None) == -1
    assert L.pa_gmm_set_form(None, 0) == abi.PA_ERR_ARG
    h = C.c_void_p()
    assert L.pa_gmm_create(C.byref(h), 0, 16, None, 0.5, None, 4, 4, None, 0, None) == abi.PA_ERR_ARG
