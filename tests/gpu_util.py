"""Helpers shared by the GPU parity tests: run one step through the C ABI and
through the oracle on the same seeded inputs, and compare per parameter
block."""
from __future__ import annotations

import numpy as np

import oracle
from paper_1708_05604_gb300 import binding, synth

FP32_TOL = 1e-4   # per-tensor relative Frobenius error and per-sequence loss, fp32 path
BF16_TOL = 2e-2   # the same with bf16 GEMM operands


def param_blocks(cfg: dict):
    """(name, start, stop) of every block of the flat parameter layout."""
    H, C = cfg["hidden"], cfg["n_classes"]
    dirs = 2 if cfg["bidirectional"] else 1
    out, off = [], 0
    for layer in range(cfg["n_layers"]):
        D = cfg["in_dim"] if layer == 0 else dirs * H
        for d in range(dirs):
            for nm, n in (("W_ih", 4 * H * D), ("W_hh", 4 * H * H), ("b", 4 * H)):
                out.append((f"l{layer}d{d}.{nm}", off, off + n))
                off += n
    out.append(("W_out", off, off + C * dirs * H))
    off += C * dirs * H
    out.append(("b_out", off, off + C))
    return out


def rel_err(a, b) -> float:
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    nb = np.linalg.norm(b)
    if nb == 0:
        return float(np.linalg.norm(a))
    return float(np.linalg.norm(a - b) / nb)


def gpu_step(cfg: dict, ds: synth.Dataset, params_np: np.ndarray, seq_ids=None, ctx=None,
             dd=None):
    """One step through bkt_lstm_ctc_step; returns (loss [b], grads [P])."""
    import torch
    if seq_ids is None:
        seq_ids = np.arange(ds.n)
    ids = np.asarray(seq_ids)
    if dd is None:
        dd = binding.DeviceDataset(ds)
    if ctx is None:
        ctx = binding.Ctx(cfg, max_tokens=int(ds.lengths[ids].sum()), max_batch=ids.size,
                          max_label_len=max(1, int(ds.label_lengths[ids].max())))
    params = torch.from_numpy(np.ascontiguousarray(params_np, np.float32)).cuda()
    grads = torch.full_like(params, float("nan"))
    loss = torch.full((ids.size,), float("nan"), dtype=torch.float32, device="cuda")
    ctx.step(dd, ids, params, grads, loss)
    ctx.sync_status()
    torch.cuda.synchronize()
    return loss.cpu().numpy().astype(np.float64), grads.cpu().numpy().astype(np.float64)


def oracle_step(cfg: dict, ds: synth.Dataset, params_np: np.ndarray, seq_ids=None):
    sub = ds if seq_ids is None else ds.subset(seq_ids)
    return oracle.lstm_ctc_step(cfg, sub.lengths, sub.x.astype(np.float64), sub.label_lengths,
                                sub.labels, np.asarray(params_np, np.float64))


def _seq_step(args):
    """One sequence through the oracle (worker of oracle_step_parallel)."""
    cfg, L, x, U, lab, params = args
    return oracle.lstm_ctc_step(cfg, np.array([L]), x, np.array([U]), lab, params)


_POOL = None


def oracle_step_parallel(cfg: dict, ds: synth.Dataset, params_np: np.ndarray, seq_ids, workers=None):
    """The oracle's step over `seq_ids`, one sequence per task in a process
    pool: the batch loss vector and the gradient, which the oracle defines as
    the sum of the sequences' gradients (summed here in fp64, in batch
    order).  The pool is started with the spawn method, so no worker is
    forked from a process that has touched the GPU."""
    import multiprocessing as mp
    import os
    global _POOL
    ids = [int(i) for i in seq_ids]
    prm = np.asarray(params_np, np.float64)
    tasks = [(cfg, int(ds.lengths[i]), ds.seq_x(i).astype(np.float64), int(ds.label_lengths[i]),
              ds.seq_labels(i), prm) for i in ids]
    # longest first, so the pool ends with short tasks
    order = sorted(range(len(ids)), key=lambda k: -int(ds.lengths[ids[k]]))
    if _POOL is None:
        n = workers or max(1, min(16, os.cpu_count() or 1))
        _POOL = mp.get_context("spawn").Pool(n)
    res = _POOL.map(_seq_step, [tasks[k] for k in order], chunksize=1)
    loss = np.zeros(len(ids))
    grad = np.zeros(prm.size)
    by_pos = {k: r for k, r in zip(order, res)}
    for k in range(len(ids)):
        lk, gk = by_pos[k]
        loss[k] = lk[0]
        grad += gk
    return loss, grad


def gate_blocks(cfg: dict):
    """(name, start, stop) of every gate row block (i, f, g, o) of every
    W_ih, W_hh and b block."""
    H = cfg["hidden"]
    out = []
    for name, a, b in param_blocks(cfg):
        if name.split(".")[-1] in ("W_ih", "W_hh", "b"):
            rows = (b - a) // (4 * H)   # columns per gate row (1 for b)
            for q, gname in enumerate("ifgo"):
                out.append((f"{name}[{gname}]", a + q * H * rows, a + (q + 1) * H * rows))
    return out


def compare(cfg, loss_g, grads_g, loss_o, grads_o, tol):
    """Asserts parity; returns the worst relative error seen.
      - per-sequence loss: relative error <= tol (the same +inf where the
        sequence has no alignment);
      - every parameter block and every gate row block of W_ih, W_hh and b:
        relative Frobenius error <= tol;
      - element by element in every parameter block:
        max |g - g*| <= tol * max |g*| over the block."""
    worst = 0.0
    fin = np.isfinite(loss_o)
    assert np.array_equal(np.isfinite(loss_g), fin), (loss_g, loss_o)
    assert np.all(loss_g[~fin] == loss_o[~fin])
    if fin.any():
        le = np.abs(loss_g[fin] - loss_o[fin]) / np.maximum(np.abs(loss_o[fin]), 1e-30)
        assert le.max() <= tol, f"loss rel err {le.max():.3e} > {tol}"
        worst = max(worst, float(le.max()))
    for name, a, b in param_blocks(cfg) + gate_blocks(cfg):
        e = rel_err(grads_g[a:b], grads_o[a:b])
        assert e <= tol, f"{name}: rel Frobenius err {e:.3e} > {tol}"
        worst = max(worst, e)
    for name, a, b in param_blocks(cfg):
        ref = np.abs(grads_o[a:b]).max()
        dev = np.abs(grads_g[a:b] - grads_o[a:b]).max()
        assert dev <= tol * ref, f"{name}: max element err {dev:.3e} > {tol} * {ref:.3e}"
        if ref > 0:
            worst = max(worst, float(dev / ref))
    return worst
