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


def compare(cfg, loss_g, grads_g, loss_o, grads_o, tol):
    """Asserts parity; returns the worst relative error seen."""
    worst = 0.0
    fin = np.isfinite(loss_o)
    assert np.array_equal(np.isfinite(loss_g), fin), (loss_g, loss_o)
    assert np.all(loss_g[~fin] == loss_o[~fin])
    if fin.any():
        le = np.abs(loss_g[fin] - loss_o[fin]) / np.maximum(np.abs(loss_o[fin]), 1e-30)
        assert le.max() <= tol, f"loss rel err {le.max():.3e} > {tol}"
        worst = max(worst, float(le.max()))
    for name, a, b in param_blocks(cfg):
        e = rel_err(grads_g[a:b], grads_o[a:b])
        assert e <= tol, f"{name}: rel Frobenius err {e:.3e} > {tol}"
        worst = max(worst, e)
    return worst
