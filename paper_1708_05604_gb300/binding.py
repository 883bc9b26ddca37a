"""Thin ctypes binding of libbkt (include/bkt.h): argument marshalling only.

Every computation happens in the library (host C++ planner, CUDA kernels).
Device buffers are torch CUDA tensors passed as raw pointers; streams are
torch streams passed as their cudaStream_t handle.  If libbkt.so has not been
built, `lib()` raises: there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libbkt.so")

BKT_OK, BKT_EINVAL, BKT_ENOMEM, BKT_ECUDA, BKT_EDEVICE, BKT_ETIMEOUT = 0, 1, 2, 3, 4, 5
BKT_WITHHOLD_EXCHANGE, BKT_WITHHOLD_TMA = 1, 2
BKT_GEMM_FP32, BKT_GEMM_BF16 = 0, 1

# Every symbol include/bkt.h declares.
EXPORTS = ("bkt_plan_buckets", "bkt_plan_buckets_ordered", "bkt_plan_get", "bkt_plan_free", "bkt_param_count",
           "bkt_ctx_create", "bkt_ctx_destroy", "bkt_lstm_ctc_step", "bkt_lstm_ctc_step_static",
           "bkt_sgd_update", "bkt_adadelta_update", "bkt_average_models",
           "bkt_ctx_sync_status", "bkt_ctx_infeasible_count", "bkt_ctx_set_wait_faults",
           "bkt_ctx_set_timing", "bkt_ctx_kernel_times", "bkt_last_error")

i32p = ctypes.POINTER(ctypes.c_int32)
i64p = ctypes.POINTER(ctypes.c_int64)


class PlanView(ctypes.Structure):
    _fields_ = [("n_buckets", ctypes.c_int32), ("bounds", i32p), ("dp_cost", ctypes.c_int64),
                ("n_seqs", ctypes.c_int64), ("order", i32p), ("n_batches", ctypes.c_int32),
                ("batch_off", i32p), ("batch_bucket", i32p),
                ("padded_timesteps", ctypes.c_int64), ("unpadded_timesteps", ctypes.c_int64)]


class ModelCfg(ctypes.Structure):
    _fields_ = [("n_layers", ctypes.c_int32), ("bidirectional", ctypes.c_int32),
                ("in_dim", ctypes.c_int32), ("hidden", ctypes.c_int32),
                ("n_classes", ctypes.c_int32), ("blank", ctypes.c_int32),
                ("gemm_precision", ctypes.c_int32)]


class Batch(ctypes.Structure):
    _fields_ = [("n_seq", ctypes.c_int32), ("lengths", i32p), ("x_offsets", i64p),
                ("label_lengths", i32p), ("label_offsets", i64p),
                ("x", ctypes.c_void_p), ("labels", ctypes.c_void_p)]


class KernelTime(ctypes.Structure):
    _fields_ = [("name", ctypes.c_char_p), ("launches", ctypes.c_int64),
                ("total_ms", ctypes.c_double), ("flops", ctypes.c_double),
                ("bytes", ctypes.c_double), ("serial_steps", ctypes.c_int64)]


_lock = threading.Lock()
_lib = None


class BktError(RuntimeError):
    def __init__(self, rc: int, msg: str):
        super().__init__(f"libbkt status {rc}: {msg}")
        self.rc = rc


def lib() -> ctypes.CDLL:
    """The loaded library; raises if it was not built."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(f"{LIB_PATH} is missing: run __graft_entry__.build() first "
                               "(there is no CPU fallback)")
        L = ctypes.CDLL(LIB_PATH)
        vp = ctypes.c_void_p
        L.bkt_plan_buckets.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                       ctypes.c_uint64, ctypes.c_uint64, ctypes.POINTER(vp)]
        L.bkt_plan_buckets_ordered.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                               ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int32,
                                               ctypes.POINTER(vp)]
        L.bkt_plan_get.argtypes = [vp, ctypes.POINTER(PlanView)]
        L.bkt_plan_free.argtypes = [vp]
        L.bkt_plan_free.restype = None
        L.bkt_param_count.argtypes = [ctypes.POINTER(ModelCfg)]
        L.bkt_param_count.restype = ctypes.c_int64
        L.bkt_ctx_create.argtypes = [ctypes.POINTER(ModelCfg), ctypes.c_int64, ctypes.c_int32,
                                     ctypes.c_int32, ctypes.POINTER(vp)]
        L.bkt_ctx_destroy.argtypes = [vp]
        L.bkt_ctx_destroy.restype = None
        L.bkt_lstm_ctc_step.argtypes = [vp, ctypes.POINTER(Batch), vp, vp, vp, vp]
        L.bkt_lstm_ctc_step_static.argtypes = [ctypes.POINTER(ModelCfg), ctypes.POINTER(Batch), vp,
                                               vp, vp, vp]
        L.bkt_sgd_update.argtypes = [vp, vp, ctypes.c_int64, ctypes.c_float, vp]
        L.bkt_average_models.argtypes = [vp, vp, ctypes.c_int64, ctypes.c_int32, ctypes.c_float, vp]
        L.bkt_adadelta_update.argtypes = [vp, vp, vp, vp, ctypes.c_int64, ctypes.c_float,
                                          ctypes.c_float, ctypes.c_float, vp]
        L.bkt_ctx_sync_status.argtypes = [vp]
        L.bkt_ctx_infeasible_count.argtypes = [vp, i64p]
        L.bkt_ctx_set_wait_faults.argtypes = [vp, ctypes.c_int32, ctypes.c_int32]
        L.bkt_ctx_set_timing.argtypes = [vp, ctypes.c_int32]
        L.bkt_ctx_kernel_times.argtypes = [vp, ctypes.POINTER(KernelTime), ctypes.c_int32, i32p]
        L.bkt_last_error.argtypes = []
        L.bkt_last_error.restype = ctypes.c_char_p
        for name in ("bkt_plan_buckets", "bkt_plan_buckets_ordered", "bkt_plan_get", "bkt_ctx_create", "bkt_lstm_ctc_step",
                     "bkt_lstm_ctc_step_static",
                     "bkt_sgd_update", "bkt_adadelta_update", "bkt_average_models", "bkt_ctx_sync_status",
                     "bkt_ctx_infeasible_count", "bkt_ctx_set_wait_faults", "bkt_ctx_set_timing",
                     "bkt_ctx_kernel_times"):
            getattr(L, name).restype = ctypes.c_int
        _lib = L
        return L


def _check(rc: int):
    if rc != BKT_OK:
        raise BktError(rc, lib().bkt_last_error().decode())


def _i32(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int32)


def _i64(a) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=np.int64)


def _ptr(a: np.ndarray, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


def _stream_handle(stream) -> ctypes.c_void_p:
    if stream is None:
        import torch
        stream = torch.cuda.current_stream()
    if isinstance(stream, int):
        return ctypes.c_void_p(stream)
    return ctypes.c_void_p(stream.cuda_stream)


# ---------------------------------------------------------------------------
BATCH_ORDERS = {"ascending": 0, "descending": 1, "shuffle_buckets": 2, "shuffle_batches": 3}


def plan_buckets(lengths, n_buckets: int, batch: int, seed: int, epoch: int = 0,
                 batch_order: str = "ascending") -> dict:
    """bkt_plan_buckets_ordered + bkt_plan_get, copied into numpy arrays
    (batch_order: a key of BATCH_ORDERS; "ascending" is bkt_plan_buckets)."""
    L = _i32(lengths)
    h = ctypes.c_void_p()
    _check(lib().bkt_plan_buckets_ordered(_ptr(L, ctypes.c_int32), L.size, n_buckets, batch,
                                          ctypes.c_uint64(seed), ctypes.c_uint64(epoch),
                                          BATCH_ORDERS[batch_order], ctypes.byref(h)))
    try:
        v = PlanView()
        _check(lib().bkt_plan_get(h, ctypes.byref(v)))
        nb = v.n_batches
        arr = lambda p, n: np.ctypeslib.as_array(p, shape=(n,)).copy() if n else \
            np.zeros(0, np.int32)
        return {"bounds": arr(v.bounds, v.n_buckets), "dp_cost": int(v.dp_cost),
                "order": arr(v.order, int(v.n_seqs)), "batch_off": arr(v.batch_off, nb + 1),
                "batch_bucket": arr(v.batch_bucket, nb), "n_batches": nb,
                "padded_timesteps": int(v.padded_timesteps),
                "unpadded_timesteps": int(v.unpadded_timesteps)}
    finally:
        lib().bkt_plan_free(h)


def model_cfg(cfg: dict) -> ModelCfg:
    return ModelCfg(cfg["n_layers"], int(bool(cfg["bidirectional"])), cfg["in_dim"],
                    cfg["hidden"], cfg["n_classes"], cfg.get("blank", 0),
                    BKT_GEMM_BF16 if cfg.get("gemm_bf16") else BKT_GEMM_FP32)


def param_count(cfg: dict) -> int:
    c = model_cfg(cfg)
    return int(lib().bkt_param_count(ctypes.byref(c)))


def sgd_update(params, grads, lr: float, stream=None):
    """bkt_sgd_update on two CUDA fp32 tensors of equal size."""
    assert params.is_cuda and grads.is_cuda and params.numel() == grads.numel()
    _check(lib().bkt_sgd_update(ctypes.c_void_p(params.data_ptr()),
                                ctypes.c_void_p(grads.data_ptr()), params.numel(),
                                ctypes.c_float(lr), _stream_handle(stream)))


def adadelta_update(params, grads, eg2, edx2, rho: float = 0.95, eps: float = 1e-6,
                    lr: float = 1.0, stream=None):
    """bkt_adadelta_update on four CUDA fp32 tensors of equal size (eg2 and
    edx2 are the running averages, zero before the first update)."""
    n = params.numel()
    for t in (params, grads, eg2, edx2):
        assert t.is_cuda and t.numel() == n
    _check(lib().bkt_adadelta_update(ctypes.c_void_p(params.data_ptr()),
                                     ctypes.c_void_p(grads.data_ptr()),
                                     ctypes.c_void_p(eg2.data_ptr()),
                                     ctypes.c_void_p(edx2.data_ptr()), n, ctypes.c_float(rho),
                                     ctypes.c_float(eps), ctypes.c_float(lr),
                                     _stream_handle(stream)))


def average_models(summed, prev, n_models: int, beta: float = 1e-6, stream=None):
    """bkt_average_models on two CUDA fp32 tensors: `summed` (the element-wise
    sum of the n_models replicas' parameters) becomes eq. 3's
    summed / n_models - beta * prev, in place."""
    n = summed.numel()
    assert summed.is_cuda and prev.is_cuda and prev.numel() == n
    _check(lib().bkt_average_models(ctypes.c_void_p(summed.data_ptr()), ctypes.c_void_p(prev.data_ptr()), n,
                                    int(n_models), ctypes.c_float(beta), _stream_handle(stream)))


class Adadelta:
    """ADADELTA state for one flat parameter tensor (Section III.B step 4)."""

    def __init__(self, params, rho: float = 0.95, eps: float = 1e-6, lr: float = 1.0):
        import torch
        self.params, self.rho, self.eps, self.lr = params, rho, eps, lr
        self.eg2 = torch.zeros_like(params)
        self.edx2 = torch.zeros_like(params)

    def step(self, grads, stream=None):
        adadelta_update(self.params, grads, self.eg2, self.edx2, self.rho, self.eps, self.lr, stream)


def _batch(lengths, x_offsets, label_lengths, label_offsets, x_ptr: int, labels_ptr: int):
    """A bkt_batch plus the numpy arrays it points into (kept alive together)."""
    L, UL = _i32(lengths), _i32(label_lengths)
    XO, LO = _i64(x_offsets), _i64(label_offsets)
    b = Batch(L.size, _ptr(L, ctypes.c_int32), _ptr(XO, ctypes.c_int64),
              _ptr(UL, ctypes.c_int32), _ptr(LO, ctypes.c_int64),
              ctypes.c_void_p(x_ptr), ctypes.c_void_p(labels_ptr))
    return b, (L, UL, XO, LO)


def step_static(cfg: dict, dd: "DeviceDataset", seq_ids, params, grads, loss, stream=None):
    """bkt_lstm_ctc_step_static: the step with the library's fixed device
    scratch array instead of a ctx (for callers that cannot allocate)."""
    ids = np.asarray(seq_ids, dtype=np.int64)
    c = model_cfg(cfg)
    b, keep = _batch(dd.lengths[ids], dd.x_off[ids], dd.label_lengths[ids], dd.lab_off[ids],
                     dd.x.data_ptr(), dd.labels.data_ptr())
    _check(lib().bkt_lstm_ctc_step_static(ctypes.byref(c), ctypes.byref(b),
                                          ctypes.c_void_p(params.data_ptr()),
                                          ctypes.c_void_p(grads.data_ptr()),
                                          ctypes.c_void_p(loss.data_ptr()),
                                          _stream_handle(stream)))
    del keep


class DeviceDataset:
    """A synth.Dataset with x and labels resident on the GPU (torch tensors)
    and the per-sequence offsets on the host."""

    def __init__(self, ds, device="cuda"):
        import torch
        self.ds = ds
        self.x = torch.from_numpy(np.ascontiguousarray(ds.x, np.float32)).to(device)
        lab = ds.labels if ds.labels.size else np.zeros(1, np.int32)
        self.labels = torch.from_numpy(np.ascontiguousarray(lab, np.int32)).to(device)
        self.lengths = _i32(ds.lengths)
        self.label_lengths = _i32(ds.label_lengths)
        self.x_off = _i64(ds.x_off[:-1])
        self.lab_off = _i64(ds.lab_off[:-1])


class Ctx:
    """bkt_ctx: device workspace for batches up to the given sizes."""

    def __init__(self, cfg: dict, max_tokens: int, max_batch: int, max_label_len: int):
        self.cfg = cfg
        self._c = model_cfg(cfg)
        self.h = ctypes.c_void_p()
        _check(lib().bkt_ctx_create(ctypes.byref(self._c), int(max_tokens), int(max_batch),
                                    int(max_label_len), ctypes.byref(self.h)))
        self.n_params = param_count(cfg)

    def close(self):
        if self.h:
            lib().bkt_ctx_destroy(self.h)
            self.h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def step_raw(self, lengths, x_offsets, label_lengths, label_offsets, x_ptr: int,
                 labels_ptr: int, params, grads, loss, stream=None):
        """bkt_lstm_ctc_step with explicit host index arrays and device bases."""
        b, keep = _batch(lengths, x_offsets, label_lengths, label_offsets, x_ptr, labels_ptr)
        _check(lib().bkt_lstm_ctc_step(self.h, ctypes.byref(b),
                                       ctypes.c_void_p(params.data_ptr()),
                                       ctypes.c_void_p(grads.data_ptr()),
                                       ctypes.c_void_p(loss.data_ptr()), _stream_handle(stream)))

    def step(self, dd: DeviceDataset, seq_ids, params, grads, loss, stream=None):
        """One training step on dataset sequences `seq_ids` (batch order)."""
        ids = np.asarray(seq_ids, dtype=np.int64)
        self.step_raw(dd.lengths[ids], dd.x_off[ids], dd.label_lengths[ids], dd.lab_off[ids],
                      dd.x.data_ptr(), dd.labels.data_ptr(), params, grads, loss, stream)

    def sync_status(self):
        _check(lib().bkt_ctx_sync_status(self.h))

    def infeasible_count(self) -> int:
        """bkt_ctx_infeasible_count: sequences without a CTC alignment since
        the previous call (the counter is reset)."""
        n = ctypes.c_int64(0)
        _check(lib().bkt_ctx_infeasible_count(self.h, ctypes.byref(n)))
        return int(n.value)

    def set_wait_faults(self, poll_cap: int = 0, withhold: int = 0):
        """bkt_ctx_set_wait_faults: failure-detection hooks (0, 0 = off)."""
        _check(lib().bkt_ctx_set_wait_faults(self.h, int(poll_cap), int(withhold)))

    def set_timing(self, on: bool):
        _check(lib().bkt_ctx_set_timing(self.h, int(bool(on))))

    def kernel_times(self) -> list[tuple[str, int, float]]:
        """(name, launches, total ms) of every kernel timed since timing was
        switched on."""
        return [(k["name"], k["launches"], k["total_ms"]) for k in self.kernel_stats()]

    def kernel_stats(self) -> list[dict]:
        """bkt_ctx_kernel_times with the algorithmic work of each kernel:
        name, launches, total_ms, flops, bytes, serial_steps."""
        n = ctypes.c_int32(0)
        _check(lib().bkt_ctx_kernel_times(self.h, None, 0, ctypes.byref(n)))
        arr = (KernelTime * max(1, n.value))()
        _check(lib().bkt_ctx_kernel_times(self.h, arr, n.value, ctypes.byref(n)))
        return [{"name": arr[i].name.decode(), "launches": int(arr[i].launches),
                 "total_ms": float(arr[i].total_ms), "flops": float(arr[i].flops),
                 "bytes": float(arr[i].bytes), "serial_steps": int(arr[i].serial_steps)}
                for i in range(n.value)]
