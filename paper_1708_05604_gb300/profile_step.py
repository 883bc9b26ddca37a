"""Runs the training step on one mini-batch of a synthetic workload and prints
per-kernel CUDA-event times (per launch and per recurrent time step).

  python -m paper_1708_05604_gb300.profile_step [--workload NAME] [--buckets Q]
         [--batch K] [--rows M] [--repeat R]

The batch is batch K of the epoch-0 plan with Q buckets (its first M
sequences with --rows); the step runs R times on it (the first run includes
one-time set-up).  Useful on its own and as the
target of an ncu capture of a single kernel.
"""
from __future__ import annotations

import argparse
import os
import sys

import numpy as np


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="lstm1_bi_h128")
    ap.add_argument("--buckets", type=int, default=4)
    ap.add_argument("--batch", type=int, default=8)
    ap.add_argument("--rows", type=int, default=0, help="keep the batch's first M sequences")
    ap.add_argument("--repeat", type=int, default=3)
    ap.add_argument("--seed", type=int, default=0)
    a = ap.parse_args(argv)

    import torch

    from . import binding, build, synth

    build.build()
    w = synth.WORKLOADS[a.workload]
    ds = synth.make_workload(w, seed=a.seed)
    plan = binding.plan_buckets(ds.lengths, a.buckets, w.batch, a.seed, 0)
    k = min(a.batch, plan["n_batches"] - 1)
    ids = plan["order"][plan["batch_off"][k]:plan["batch_off"][k + 1]]
    if a.rows > 0:
        ids = ids[:a.rows]
    cfg = w.model_cfg()
    dd = binding.DeviceDataset(ds)
    ctx = binding.Ctx(cfg, int(ds.lengths[ids].sum()), len(ids), int(ds.label_lengths.max()))
    p = torch.from_numpy(synth.draw_params(np.random.default_rng(a.seed + 1),
                                           binding.param_count(cfg))).cuda()
    g = torch.zeros_like(p)
    loss = torch.zeros(len(ids), device="cuda")
    ctx.step(dd, ids, p, g, loss)  # set-up run
    torch.cuda.synchronize()
    ctx.set_timing(True)
    for _ in range(a.repeat):
        ctx.step(dd, ids, p, g, loss)
    torch.cuda.synchronize()
    ctx.sync_status()
    T = int(ds.lengths[ids].max())
    n_tok = int(ds.lengths[ids].sum())
    print(f"workload {w.name}  batch {k} of {plan['n_batches']}: {len(ids)} sequences, "
          f"{n_tok} tokens, longest {T}")
    total = 0.0
    for name, c, ms in ctx.kernel_times():
        per = ms / a.repeat
        total += per
        print(f"  {name:16s} {c // a.repeat:4d}/step {per:9.3f} ms/step {per / T * 1e3:8.3f} us/time step")
    print(f"  {'all kernels':16s}      {total:9.3f} ms/step")
    ctx.close()


if __name__ == "__main__":
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    main()
