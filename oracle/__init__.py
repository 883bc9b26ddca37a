"""Test infrastructure only: the fp64 CPU oracle of the bucketed LSTM-CTC step.

Only the tests, ``__graft_entry__.smoke()`` and the CPU-baseline leg of
``bench.py`` may import this package.  The product library never does, and the
two share no code.  The arithmetic lives in ``oracle.c`` (plain C, double
precision, single thread); this module compiles it with gcc on first use and
marshals numpy arrays to it.

Each function names the passage of the paper (arXiv 1708.05604) it follows:
  plan()              Section III.A (histogram, DYNAMICBUCKETING, bucket
                      assignment), Section III.B step 3 (shuffle), Section
                      IV.A (shorter buckets first).
  dynamic_bucketing() Section III.A, DYNAMICBUCKETING.
  ctc()               CTC loss and gradient, the paper's ref. [15].
  lstm_ctc_step()     The LSTM (ref. [1]) + CTC training step of Section IV.
  sgd()               theta <- theta - lr * g.
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None

OR_OK, OR_EINVAL, OR_ENOMEM = 0, 1, 2


def build(force: bool = False) -> str:
    """Compile oracle.c into liboracle.so (gcc, -O2, no fast-math)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-std=c99", "-fPIC", "-shared", "-fno-fast-math",
           "-ffp-contract=off", "-o", tmp, _SRC, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        i32p = ctypes.POINTER(ctypes.c_int32)
        i64p = ctypes.POINTER(ctypes.c_int64)
        f64p = ctypes.POINTER(ctypes.c_double)
        u64p = ctypes.POINTER(ctypes.c_uint64)
        lib.or_splitmix64.argtypes = [u64p]
        lib.or_splitmix64.restype = ctypes.c_uint64
        lib.or_histogram.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, i64p]
        lib.or_histogram.restype = ctypes.c_int
        lib.or_dynamic_bucketing.argtypes = [i64p, ctypes.c_int32, ctypes.c_int32, i32p, i64p]
        lib.or_dynamic_bucketing.restype = ctypes.c_int
        lib.or_plan.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                ctypes.c_uint64, ctypes.c_uint64, i32p, i64p, i32p,
                                i32p, i32p, i32p, i64p]
        lib.or_plan.restype = ctypes.c_int
        lib.or_plan_ordered.argtypes = [i32p, ctypes.c_int64, ctypes.c_int32, ctypes.c_int32,
                                        ctypes.c_uint64, ctypes.c_uint64, ctypes.c_int32, i32p,
                                        i64p, i32p, i32p, i32p, i32p, i64p]
        lib.or_plan_ordered.restype = ctypes.c_int
        lib.or_ctc.argtypes = [f64p, ctypes.c_int32, ctypes.c_int32, ctypes.c_int32,
                               i32p, ctypes.c_int32, f64p]
        lib.or_ctc.restype = ctypes.c_double
        lib.or_param_count.argtypes = [ctypes.c_int32] * 5
        lib.or_param_count.restype = ctypes.c_int64
        lib.or_lstm_ctc_step.argtypes = [ctypes.c_int32] * 7 + [
            i32p, f64p, i32p, i32p, f64p, f64p, f64p]
        lib.or_lstm_ctc_step.restype = ctypes.c_int
        lib.or_sgd.argtypes = [f64p, f64p, ctypes.c_int64, ctypes.c_double]
        lib.or_sgd.restype = None
        lib.or_adadelta.argtypes = [f64p, f64p, f64p, f64p, ctypes.c_int64, ctypes.c_double,
                                    ctypes.c_double, ctypes.c_double]
        lib.or_adadelta.restype = None
        lib.or_average_models.argtypes = [f64p, ctypes.c_int32, f64p, ctypes.c_int64, ctypes.c_double, f64p]
        lib.or_average_models.restype = ctypes.c_int
        _lib = lib
        return lib


def _p(a: np.ndarray, ct):
    return a.ctypes.data_as(ctypes.POINTER(ct))


class OracleError(RuntimeError):
    def __init__(self, rc: int, what: str):
        super().__init__(f"oracle {what} failed with status {rc}")
        self.rc = rc


def splitmix64_stream(state: int, count: int) -> list[int]:
    """`count` SplitMix64 outputs starting from `state` (the oracle's copy)."""
    lib = _load()
    s = ctypes.c_uint64(state & 0xFFFFFFFFFFFFFFFF)
    return [int(lib.or_splitmix64(ctypes.byref(s))) for _ in range(count)]


def histogram(lengths, lmax: int | None = None) -> np.ndarray:
    lib = _load()
    L = np.ascontiguousarray(lengths, dtype=np.int32)
    lmax = int(L.max()) if lmax is None else int(lmax)
    f = np.zeros(lmax + 1, dtype=np.int64)
    rc = lib.or_histogram(_p(L, ctypes.c_int32), L.size, lmax, _p(f, ctypes.c_int64))
    if rc:
        raise OracleError(rc, "histogram")
    return f


def dynamic_bucketing(f, Q: int):
    """Returns (bests[Q] as int32 array, optimal cost)."""
    lib = _load()
    f = np.ascontiguousarray(f, dtype=np.int64)
    bests = np.zeros(Q, dtype=np.int32)
    cost = ctypes.c_int64(0)
    rc = lib.or_dynamic_bucketing(_p(f, ctypes.c_int64), f.size, Q,
                                  _p(bests, ctypes.c_int32), ctypes.byref(cost))
    if rc:
        raise OracleError(rc, "dynamic_bucketing")
    return bests, int(cost.value)


PLAN_ORDERS = {"ascending": 0, "descending": 1, "shuffle_buckets": 2, "shuffle_batches": 3}


def plan(lengths, n_buckets: int, batch: int, seed: int, epoch: int = 0,
         batch_order: str = "ascending") -> dict:
    """The epoch plan: bounds, dp cost, emission order and mini-batches
    (or_plan for "ascending", or_plan_ordered otherwise)."""
    lib = _load()
    L = np.ascontiguousarray(lengths, dtype=np.int32)
    n = L.size
    bounds = np.zeros(max(n_buckets, 1), dtype=np.int32)
    order = np.zeros(n, dtype=np.int32)
    boff = np.zeros(n + 1, dtype=np.int32)
    bbuck = np.zeros(max(n, 1), dtype=np.int32)
    nb = ctypes.c_int32(0)
    cost = ctypes.c_int64(0)
    padded = ctypes.c_int64(0)
    tail = (_p(bounds, ctypes.c_int32), ctypes.byref(cost), _p(order, ctypes.c_int32),
            _p(boff, ctypes.c_int32), _p(bbuck, ctypes.c_int32), ctypes.byref(nb),
            ctypes.byref(padded))
    if batch_order == "ascending":
        rc = lib.or_plan(_p(L, ctypes.c_int32), n, n_buckets, batch, ctypes.c_uint64(seed),
                         ctypes.c_uint64(epoch), *tail)
    else:
        rc = lib.or_plan_ordered(_p(L, ctypes.c_int32), n, n_buckets, batch,
                                 ctypes.c_uint64(seed), ctypes.c_uint64(epoch),
                                 PLAN_ORDERS[batch_order], *tail)
    if rc:
        raise OracleError(rc, "plan")
    k = nb.value
    return {"bounds": bounds[:n_buckets].copy(), "dp_cost": int(cost.value),
            "order": order, "batch_off": boff[:k + 1].copy(),
            "batch_bucket": bbuck[:k].copy(), "n_batches": k,
            "padded_timesteps": int(padded.value)}


def ctc(logp, labels, blank: int = 0, grad: bool = True):
    """(-ln p, d(-ln p)/d logits) for one sequence; logp is [T x C] log-softmax."""
    lib = _load()
    lp = np.ascontiguousarray(logp, dtype=np.float64)
    T, C = lp.shape
    lab = np.ascontiguousarray(labels, dtype=np.int32)
    g = np.zeros((T, C), dtype=np.float64) if grad else None
    loss = lib.or_ctc(_p(lp, ctypes.c_double), T, C, blank, _p(lab, ctypes.c_int32),
                      lab.size, _p(g, ctypes.c_double) if grad else None)
    return float(loss), g


def param_count(n_layers: int, bidirectional: bool, in_dim: int, hidden: int,
                n_classes: int) -> int:
    return int(_load().or_param_count(n_layers, int(bool(bidirectional)), in_dim,
                                      hidden, n_classes))


def lstm_ctc_step(cfg: dict, lengths, x, label_lengths, labels, params):
    """fp64 training step over one mini-batch.

    cfg: n_layers, bidirectional, in_dim, hidden, n_classes, blank.
    x: [sum L x in_dim] rows of the sequences one after another; labels
    likewise.  Returns (per-sequence losses [n] float64, grads [P] float64),
    grads = d(sum of losses)/d params over the sequences with an alignment.
    """
    lib = _load()
    L = np.ascontiguousarray(lengths, dtype=np.int32)
    UL = np.ascontiguousarray(label_lengths, dtype=np.int32)
    X = np.ascontiguousarray(x, dtype=np.float64).reshape(-1)
    lab = np.ascontiguousarray(labels, dtype=np.int32)
    if lab.size == 0:
        lab = np.zeros(1, dtype=np.int32)
    prm = np.ascontiguousarray(params, dtype=np.float64)
    P = param_count(cfg["n_layers"], cfg["bidirectional"], cfg["in_dim"],
                    cfg["hidden"], cfg["n_classes"])
    if prm.size != P:
        raise ValueError(f"params has {prm.size} entries, expected {P}")
    if X.size != int(L.sum()) * cfg["in_dim"]:
        raise ValueError("x does not hold sum(lengths) rows")
    grads = np.zeros(P, dtype=np.float64)
    loss = np.zeros(max(L.size, 1), dtype=np.float64)
    rc = lib.or_lstm_ctc_step(cfg["n_layers"], int(bool(cfg["bidirectional"])),
                              cfg["in_dim"], cfg["hidden"], cfg["n_classes"],
                              cfg.get("blank", 0), L.size, _p(L, ctypes.c_int32),
                              _p(X, ctypes.c_double), _p(UL, ctypes.c_int32),
                              _p(lab, ctypes.c_int32), _p(prm, ctypes.c_double),
                              _p(grads, ctypes.c_double), _p(loss, ctypes.c_double))
    if rc:
        raise OracleError(rc, "lstm_ctc_step")
    return loss[:L.size].copy(), grads


def sgd(params, grads, lr: float) -> np.ndarray:
    lib = _load()
    p = np.array(params, dtype=np.float64, copy=True)
    g = np.ascontiguousarray(grads, dtype=np.float64)
    lib.or_sgd(_p(p, ctypes.c_double), _p(g, ctypes.c_double), p.size, lr)
    return p


def adadelta(params, grads, eg2, edx2, rho: float = 0.95, eps: float = 1e-6,
             lr: float = 1.0):
    """One ADADELTA update; returns new (params, eg2, edx2) as float64."""
    lib = _load()
    p = np.array(params, dtype=np.float64, copy=True)
    g = np.ascontiguousarray(grads, dtype=np.float64)
    a = np.array(eg2, dtype=np.float64, copy=True)
    b = np.array(edx2, dtype=np.float64, copy=True)
    lib.or_adadelta(_p(p, ctypes.c_double), _p(g, ctypes.c_double), _p(a, ctypes.c_double),
                    _p(b, ctypes.c_double), p.size, rho, eps, lr)
    return p, a, b


def average_models(models, prev, beta: float = 1e-6) -> np.ndarray:
    """Eq. 3 (Section III.B step 5, alpha = 1): the mean of the K models'
    parameters (rows of `models`) minus beta times the previous epoch's
    parameters `prev`, in float64."""
    lib = _load()
    M = np.ascontiguousarray(np.atleast_2d(np.asarray(models, dtype=np.float64)))
    p = np.ascontiguousarray(prev, dtype=np.float64)
    if M.shape[1] != p.size:
        raise ValueError("models and prev differ in length")
    out = np.zeros(p.size, dtype=np.float64)
    rc = lib.or_average_models(_p(M, ctypes.c_double), M.shape[0], _p(p, ctypes.c_double), p.size,
                               float(beta), _p(out, ctypes.c_double))
    if rc != 0:
        raise ValueError(f"or_average_models failed ({rc})")
    return out
