"""Host-side argument checks of the C ABI, called through ctypes without a
GPU: every entry point refuses NULL pointers, out-of-range sizes and
constants with BKT_EINVAL (and a message in bkt_last_error) before it makes
any CUDA call, so a bad call fails the same way on a machine with or without
a device.  The device-side checks (a label equal to the blank, a workspace
too small for the batch) are in the GPU tests."""
import ctypes
import math

import pytest

from paper_1708_05604_gb300 import binding as B


@pytest.fixture(scope="module")
def L():
    lib = B.lib()
    lib.bkt_last_error.restype = ctypes.c_char_p
    return lib


def _cfg(**kw):
    d = dict(n_layers=1, bidirectional=1, in_dim=4, hidden=32, n_classes=10, blank=0, gemm_precision=0)
    d.update(kw)
    return B.ModelCfg(*[d[k] for k in ("n_layers", "bidirectional", "in_dim", "hidden", "n_classes",
                                       "blank", "gemm_precision")])


def _einval(L, rc, words):
    assert rc == B.BKT_EINVAL
    msg = L.bkt_last_error().decode()
    assert words in msg, msg


def test_invalid_model_cfgs(L):
    assert L.bkt_param_count(ctypes.byref(_cfg())) > 0
    for bad in (dict(hidden=0), dict(n_classes=1), dict(blank=10), dict(blank=-1), dict(gemm_precision=7),
                dict(n_layers=0), dict(bidirectional=2), dict(in_dim=0)):
        assert L.bkt_param_count(ctypes.byref(_cfg(**bad))) == 0, bad
    out = ctypes.c_void_p()
    _einval(L, L.bkt_ctx_create(None, 100, 4, 4, ctypes.byref(out)), "invalid model cfg")
    _einval(L, L.bkt_ctx_create(ctypes.byref(_cfg(hidden=0)), 100, 4, 4, ctypes.byref(out)), "invalid model cfg")
    for cap in ((0, 4, 4), (100, 0, 4), (100, 4, -1)):
        _einval(L, L.bkt_ctx_create(ctypes.byref(_cfg()), *cap, ctypes.byref(out)), "capacity")
    _einval(L, L.bkt_ctx_create(ctypes.byref(_cfg()), 100, 4, 4, None), "out is NULL")
    assert not out.value


def test_steps_refuse_null_arguments(L):
    _einval(L, L.bkt_lstm_ctc_step(None, None, None, None, None, None), "NULL argument")
    _einval(L, L.bkt_lstm_ctc_step_static(None, None, None, None, None, None), "NULL argument")
    _einval(L, L.bkt_lstm_ctc_step_static(ctypes.byref(_cfg()), None, None, None, None, None), "NULL argument")


def test_update_rules_refuse_bad_arguments(L):
    n5, n0 = ctypes.c_int64(5), ctypes.c_int64(0)
    f = ctypes.c_float
    _einval(L, L.bkt_sgd_update(None, None, n5, f(0.1), None), "bad arguments")
    _einval(L, L.bkt_sgd_update(None, None, ctypes.c_int64(-1), f(0.1), None), "bad arguments")
    assert L.bkt_sgd_update(None, None, n0, f(0.1), None) == B.BKT_OK   # nothing to do
    _einval(L, L.bkt_adadelta_update(None, None, None, None, n5, f(0.95), f(1e-6), f(1.0), None), "bad arguments")
    for rho, eps, lr in ((1.0, 1e-6, 1.0), (-0.1, 1e-6, 1.0), (0.9, 0.0, 1.0), (0.9, 1e-6, -1.0),
                         (math.nan, 1e-6, 1.0)):
        _einval(L, L.bkt_adadelta_update(None, None, None, None, n0, f(rho), f(eps), f(lr), None), "rho")
    for n, k, beta in ((5, 2, 1e-6), (-1, 2, 1e-6), (0, 0, 1e-6), (0, 2, -1.0), (0, 2, math.nan)):
        _einval(L, L.bkt_average_models(None, None, ctypes.c_int64(n), ctypes.c_int32(k), f(beta), None),
                "bad arguments")


def test_ctx_queries_refuse_null(L):
    c, n = ctypes.c_int64(), ctypes.c_int32()
    _einval(L, L.bkt_ctx_sync_status(None), "NULL ctx")
    _einval(L, L.bkt_ctx_infeasible_count(None, ctypes.byref(c)), "NULL argument")
    _einval(L, L.bkt_ctx_set_wait_faults(None, 0, 0), "NULL ctx")
    _einval(L, L.bkt_ctx_set_timing(None, 1), "NULL ctx")
    _einval(L, L.bkt_ctx_kernel_times(None, None, 0, ctypes.byref(n)), "NULL argument")
    _einval(L, L.bkt_plan_get(None, None), "NULL argument")
    L.bkt_ctx_destroy(None)   # both accept NULL, as free() does
    L.bkt_plan_free(None)
