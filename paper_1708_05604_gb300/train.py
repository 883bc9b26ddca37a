"""Multi-epoch training with per-epoch rebucketing and reshuffling.

Section III.B step 3 rebuilds the buckets and reshuffles them every epoch;
step 4 trains with ADADELTA (ref. [21]); Section IV.A holds out 5% of the
sequences for validation and feeds shorter buckets first; Fig. 3 plots the
validation loss against wall-clock time for several bucket counts Q and
Fig. 4 the epoch time against Q.  This driver runs that loop on one GPU on
a synthetic workload and reports, per epoch, the training time, the mean
training loss and the mean validation loss per sequence.

  python -m paper_1708_05604_gb300.train --workload lstm1_bi_h128 \\
      --buckets 1,2,3,4,6 --epochs 3 [--optimizer adadelta|sgd]
      [--batch-order ascending|descending|shuffle_buckets|shuffle_batches]
      [--checkpoint PATH] [--resume PATH] [--log-jsonl FILE] [--kernel-times]

With --checkpoint the parameters and the optimizer state are stored after
every epoch (`checkpoint.py`); --resume continues such a run from the epoch
after its checkpoint with the same mini-batches an uninterrupted run would
draw.  --log-jsonl appends each epoch's record to a JSON-lines file;
--kernel-times adds the library's per-kernel CUDA-event times to it (the
per-launch events add a little to the epoch they time).

Data-parallel training (Section III.B steps 3-5): launched with torchrun on
N GPUs, every epoch the training sequences are reshuffled into N portions,
each replica trains its portion from the same starting parameters, and the
replicas' parameters are combined by eq. 3 (an NCCL all-reduce of the flat
parameter buffer, then bkt_average_models):

  torchrun --nproc-per-node N -m paper_1708_05604_gb300.train --replicas ...

Every step runs in the library (bkt_plan_buckets_ordered, bkt_lstm_ctc_step,
bkt_adadelta_update / bkt_sgd_update, bkt_average_models); this module only
sequences the calls.
"""
from __future__ import annotations

import argparse
import json
import sys
import time

import numpy as np


def split_validation(n: int, frac: float, seed: int):
    """(train ids, validation ids): a seeded random `frac` of 0..n-1 held out
    (at least one sequence when frac > 0), both sorted ascending."""
    k = int(round(n * frac))
    if frac > 0:
        k = max(1, min(k, n - 1))
    perm = np.random.default_rng(seed).permutation(n)
    return np.sort(perm[k:]).astype(np.int64), np.sort(perm[:k]).astype(np.int64)


def epoch_batches(lengths, train_ids, n_buckets: int, batch: int, seed: int, epoch: int,
                  batch_order: str = "ascending"):
    """The epoch's mini-batches as arrays of dataset ids: the plan is made on
    the training sequences alone (their lengths in train_ids order)."""
    from . import binding
    lengths = np.asarray(lengths)
    plan = binding.plan_buckets(lengths[train_ids], n_buckets, batch, seed, epoch, batch_order)
    order, off = plan["order"], plan["batch_off"]
    return [train_ids[order[off[k]:off[k + 1]]] for k in range(plan["n_batches"])], plan


def data_portions(train_ids, world: int, seed: int, epoch: int):
    """Section III.B step 3: every epoch the training sequences are
    reshuffled (a permutation seeded by (seed, epoch)) and cut into `world`
    contiguous portions of near-equal size; portion r is replica r's data."""
    ids = np.asarray(train_ids, dtype=np.int64)
    perm = np.random.default_rng([int(seed), int(epoch), 0x5EED]).permutation(ids)
    return [np.sort(p) for p in np.array_split(perm, world)]


def data_parallel_epoch(params_start, portion, train_portion, all_reduce_sum, average, world: int):
    """Section III.B steps 4-5 on one replica: train this replica's portion
    from params_start (`train_portion(portion)` returns the replica's
    parameters after the epoch, a new buffer), sum the replicas' parameters
    in place (`all_reduce_sum`, the one exchange of the loop), then eq. 3:
    `average(summed, params_start, world)` leaves mean - beta * params_start.
    Every replica ends the epoch with the same parameters."""
    local = train_portion(portion)
    all_reduce_sum(local)
    average(local, params_start, world)
    return local


def validation_batches(lengths, val_ids, batch: int):
    """Held-out sequences sorted by length (longest first), cut into batches."""
    lengths = np.asarray(lengths)
    o = val_ids[np.argsort(-lengths[val_ids], kind="stable")]
    return [o[i:i + batch] for i in range(0, o.size, batch)]


def run_identity(workload: str, n_buckets: int, optimizer: str, batch_order: str, seed: int,
                 val_frac: float, lr, n_seqs, max_len, n_params: int) -> dict:
    """What a checkpoint must agree on for a run to resume from it: the data,
    the plan's inputs, the update rule and the parameter count."""
    return {"workload": workload, "n_buckets": int(n_buckets), "optimizer": optimizer,
            "batch_order": batch_order, "seed": int(seed), "val_frac": float(val_frac),
            "lr": None if lr is None else float(lr), "n_seqs": n_seqs, "max_len": max_len,
            "n_params": int(n_params)}


def resume_point(meta: dict, identity: dict, epochs: int):
    """(first epoch to run, per-epoch records so far, wall seconds so far,
    initial validation loss) of a run resumed from a checkpoint's meta;
    ValueError when the checkpoint is of another run or already past
    `epochs`."""
    from . import checkpoint
    checkpoint.check_compatible(meta, identity)
    start = int(meta["epoch_next"])
    if start > epochs:
        raise ValueError(f"checkpoint is after epoch {start - 1}; asked for {epochs} epochs in all")
    return start, list(meta["epochs"]), float(meta["wall_s"]), meta["val_loss_initial"]


def train(workload: str, n_buckets: int, epochs: int, optimizer: str = "adadelta",
          batch_order: str = "ascending", seed: int = 0, val_frac: float = 0.05,
          lr: float | None = None, n_seqs: int | None = None, max_len: int | None = None,
          params0=None, device: str = "cuda", log=None, checkpoint_path: str | None = None,
          resume: str | None = None, kernel_times: bool = False) -> dict:
    """Trains up to epoch `epochs` (counting from 0, so `epochs` epochs in
    all, fewer when resumed); returns the per-epoch record and final params.
    checkpoint_path: store parameters and optimizer state after every epoch;
    resume: continue the run stored there (same workload, Q, seed, order,
    update rule); kernel_times: per-kernel CUDA-event ms in each record."""
    import torch

    from . import binding, build, checkpoint, synth

    build.build()
    w = synth.WORKLOADS[workload]
    cfg = w.model_cfg()
    ds = synth.make_workload(w, seed=seed, n_seqs=n_seqs, max_len=max_len)
    train_ids, val_ids = split_validation(ds.n, val_frac, seed + 17)
    P = binding.param_count(cfg)
    ident = run_identity(workload, n_buckets, optimizer, batch_order, seed, val_frac, lr,
                         n_seqs, max_len, P)
    start, saved = 0, None
    if resume:
        meta, saved = checkpoint.load(resume)
        start, done, wall0, v_init = resume_point(meta, ident, epochs)
        params0 = saved["params"]
    elif params0 is None:
        params0 = synth.draw_params(np.random.default_rng(seed + 1), P)
    dev = torch.device(device)
    params = torch.from_numpy(np.ascontiguousarray(params0, np.float32)).to(dev)
    grads = torch.zeros_like(params)
    dd = binding.DeviceDataset(ds, device=dev)
    cap = int(np.sort(ds.lengths)[-w.batch:].sum())
    ctx = binding.Ctx(cfg, cap, w.batch, max(1, int(ds.label_lengths.max())))
    loss = torch.zeros(ds.n, dtype=torch.float32, device=dev)
    if optimizer == "adadelta":
        opt = binding.Adadelta(params, lr=1.0 if lr is None else lr)
        update = opt.step
        if saved is not None:
            opt.eg2.copy_(torch.from_numpy(saved["eg2"]))
            opt.edx2.copy_(torch.from_numpy(saved["edx2"]))
    elif optimizer == "sgd":
        step_lr = 1e-3 if lr is None else lr
        update = lambda g, stream=None: binding.sgd_update(params, g, step_lr, stream)
    else:
        raise ValueError(f"unknown optimizer {optimizer!r}")
    stream = torch.cuda.current_stream(dev)
    vbatches = validation_batches(ds.lengths, val_ids, w.batch)

    def validate():
        total = 0.0
        for ids in vbatches:
            lv = torch.zeros(ids.size, dtype=torch.float32, device=dev)
            ctx.step(dd, ids, params, grads, lv, stream)
            total += float(lv.double().sum())
        return total / max(1, val_ids.size)

    def store(e_next):
        arrays = {"params": params.cpu().numpy()}
        if optimizer == "adadelta":
            arrays["eg2"], arrays["edx2"] = opt.eg2.cpu().numpy(), opt.edx2.cpu().numpy()
        checkpoint.save(checkpoint_path, arrays,
                        {**ident, "epoch_next": e_next, "epochs": record["epochs"], "wall_s": wall,
                         "val_loss_initial": record["val_loss_initial"]})

    record = {"workload": workload, "n_buckets": n_buckets, "optimizer": optimizer,
              "batch_order": batch_order, "n_train": int(train_ids.size),
              "n_val": int(val_ids.size), "epochs": []}
    if resume:
        record["epochs"], wall, record["val_loss_initial"] = done, wall0, v_init
        record["resumed_at_epoch"] = start
    else:
        wall = 0.0
        v0 = validate()
        ctx.sync_status()
        record["val_loss_initial"] = v0
    for e in range(start, epochs):
        batches, plan = epoch_batches(ds.lengths, train_ids, n_buckets, w.batch, seed, e,
                                      batch_order)
        torch.cuda.synchronize(dev)
        t0 = time.perf_counter()
        ev0, ev1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
        if kernel_times:
            ctx.set_timing(True)
        ev0.record(stream)
        pos = 0
        for ids in batches:
            lv = loss[pos:pos + ids.size]
            ctx.step(dd, ids, params, grads, lv, stream)
            update(grads, stream)
            pos += ids.size
        ev1.record(stream)
        torch.cuda.synchronize(dev)
        host_s = time.perf_counter() - t0
        ms = ev0.elapsed_time(ev1)
        kms = None
        if kernel_times:
            kms = {k["name"]: round(k["total_ms"], 4) for k in ctx.kernel_stats()}
            ctx.set_timing(False)
        ctx.sync_status()
        wall += host_s
        tl = float(loss[:pos].double().sum()) / max(1, pos)
        vl = validate()
        rec = {"epoch": e, "epoch_ms": ms, "host_s": host_s, "wall_s": wall,
               "train_loss": tl, "val_loss": vl, "n_batches": plan["n_batches"],
               "padded_efficiency": plan["unpadded_timesteps"] / plan["padded_timesteps"],
               "timesteps": int(plan["unpadded_timesteps"]),
               "timesteps_per_s": plan["unpadded_timesteps"] / (ms / 1e3) if ms > 0 else None}
        if kms is not None:
            rec["kernel_ms"] = kms
        record["epochs"].append(rec)
        if checkpoint_path:
            store(e + 1)
        if log:
            log(rec)
    record["params"] = params.cpu().numpy()
    return record


def train_replicas(workload: str, n_buckets: int, epochs: int, seed: int = 0, beta: float = 1e-6,
                   lr: float | None = None, n_seqs: int | None = None, max_len: int | None = None,
                   log=None) -> dict:
    """Data-parallel training on the GPUs of a torchrun launch (one process
    per GPU, NCCL): per epoch, data portions, a local ADADELTA epoch of the
    replica's portion (bucketed within the portion), then eq. 3."""
    import torch
    import torch.distributed as dist

    from . import binding, build, synth

    world, rank = dist.get_world_size(), dist.get_rank()
    build.build()
    w = synth.WORKLOADS[workload]
    cfg = w.model_cfg()
    ds = synth.make_workload(w, seed=seed, n_seqs=n_seqs, max_len=max_len)
    train_ids, _ = split_validation(ds.n, 0.05, seed + 17)
    P = binding.param_count(cfg)
    dev = torch.device("cuda", torch.cuda.current_device())
    params = torch.from_numpy(synth.draw_params(np.random.default_rng(seed + 1), P)).to(dev)
    dd = binding.DeviceDataset(ds, device=dev)
    cap = int(np.sort(ds.lengths)[-w.batch:].sum())
    ctx = binding.Ctx(cfg, cap, w.batch, max(1, int(ds.label_lengths.max())))
    grads = torch.zeros_like(params)
    loss = torch.zeros(ds.n, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    record = {"workload": workload, "replicas": world, "n_buckets": n_buckets, "epochs": []}
    for e in range(epochs):
        portion = data_portions(train_ids, world, seed, e)[rank]

        def train_portion(ids_portion):
            local = params.clone()
            opt = binding.Adadelta(local, lr=1.0 if lr is None else lr)
            batches, _ = epoch_batches(ds.lengths, ids_portion, n_buckets, w.batch, seed + 1000 * rank, e)
            pos = 0
            for ids in batches:
                ctx.step(dd, ids, local, grads, loss[pos:pos + ids.size], stream)
                opt.step(grads, stream)
                pos += ids.size
            return local

        t0 = time.perf_counter()
        params = data_parallel_epoch(params, portion, train_portion,
                                     lambda t: dist.all_reduce(t, op=dist.ReduceOp.SUM),
                                     lambda v, prev, k: binding.average_models(v, prev, k, beta, stream), world)
        torch.cuda.synchronize(dev)
        ctx.sync_status()
        rec = {"epoch": e, "wall_s": time.perf_counter() - t0, "portion": int(portion.size)}
        record["epochs"].append(rec)
        if log and rank == 0:
            log(rec)
    record["params"] = params.cpu().numpy()
    ctx.close()
    return record


def main(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="lstm1_bi_h128")
    ap.add_argument("--buckets", default="1,2,3,4,6")
    ap.add_argument("--epochs", type=int, default=3)
    ap.add_argument("--optimizer", default="adadelta", choices=["adadelta", "sgd"])
    ap.add_argument("--batch-order", default="ascending",
                    choices=["ascending", "descending", "shuffle_buckets", "shuffle_batches"])
    ap.add_argument("--lr", type=float, default=None)
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--replicas", action="store_true",
                    help="data-parallel replicas with eq.-3 averaging (launch with torchrun)")
    ap.add_argument("--beta", type=float, default=1e-6)
    ap.add_argument("--checkpoint", default=None,
                    help="store parameters and optimizer state after every epoch (PATH.bin, PATH.json; "
                         "with several bucket counts, PATH.qQ)")
    ap.add_argument("--resume", default=None, help="continue the run stored at this checkpoint path")
    ap.add_argument("--log-jsonl", default=None, help="append every epoch's record to this file")
    ap.add_argument("--kernel-times", action="store_true", help="per-kernel CUDA-event ms in each record")
    a = ap.parse_args(argv)
    if a.replicas:
        import os

        import torch
        import torch.distributed as dist
        torch.cuda.set_device(int(os.environ.get("LOCAL_RANK", "0")))
        dist.init_process_group("nccl")
        for Q in [int(q) for q in a.buckets.split(",") if q]:
            r = train_replicas(a.workload, Q, a.epochs, a.seed, a.beta, a.lr)
            r.pop("params")
            if dist.get_rank() == 0:
                print(json.dumps(r), flush=True)
        dist.destroy_process_group()
        return 0
    from .checkpoint import JsonlLog
    qs = [int(q) for q in a.buckets.split(",") if q]
    if a.resume and len(qs) != 1:
        ap.error("--resume continues one run: give one bucket count")

    def ck(path, Q):
        return None if path is None else (path if len(qs) == 1 else f"{path}.q{Q}")

    for Q in qs:
        log = JsonlLog(a.log_jsonl, workload=a.workload, n_buckets=Q) if a.log_jsonl else None
        r = train(a.workload, Q, a.epochs, a.optimizer, a.batch_order, a.seed, lr=a.lr, log=log,
                  checkpoint_path=ck(a.checkpoint, Q), resume=a.resume, kernel_times=a.kernel_times)
        r.pop("params")
        print(json.dumps(r), flush=True)
    return 0


if __name__ == "__main__":
    sys.exit(main())
