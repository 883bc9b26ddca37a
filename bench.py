#!/usr/bin/env python3
"""Benchmark of the bucketed LSTM-CTC training step on GB300.

One "step" = one training epoch over the synthetic workload: plan the
buckets (bkt_plan_buckets: histogram, dynamic program, per-epoch reshuffle),
then for every mini-batch one bkt_lstm_ctc_step (packed layout, LSTM forward,
output + log-softmax, CTC, BPTT, weight gradients) and one bkt_sgd_update
(or, with --optimizer adadelta, the paper's update rule bkt_adadelta_update).
The metric is unpadded timesteps per second (sum of sequence lengths
processed / time).  Inputs are resident in HBM when the timed region starts;
L2 is flushed (a 256 MiB write) between timed steps, outside their events.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

--impl reference times the fp64 CPU oracle (test infrastructure) on bounded
samples of the same workload.  Under torchrun each rank runs an independent
replica of the workload (no collective on the data path) and rank 0 prints
the whole-job line.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "lstm1_bi_h128"
DEFAULT_BUCKETS = 4
LR = 1e-3


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--buckets", type=int, default=DEFAULT_BUCKETS)
    ap.add_argument("--compare-buckets", default="1",
                    help="extra bucket counts timed briefly for epoch time vs Q ('' = none)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--optimizer", default="sgd", choices=["sgd", "adadelta"])
    ap.add_argument("--cpu-baseline-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    return ap.parse_args()


# ---------------------------------------------------------------------------
class Clocks:
    """nvidia-smi sampling during the timed region."""
    Q = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.p = None

    def __enter__(self):
        try:
            self.p = subprocess.Popen(
                ["nvidia-smi", "-i", str(self.gpu), f"--query-gpu={self.Q}", "--format=csv,noheader,nounits",
                 "-lms", "200"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
        except OSError:
            self.p = None
        return self

    def __exit__(self, *a):
        self.out = ""
        if self.p is not None:
            self.p.terminate()
            try:
                self.out, _ = self.p.communicate(timeout=5)
            except subprocess.TimeoutExpired:
                self.p.kill()
                self.out, _ = self.p.communicate()

    def summary(self):
        sm, mx, reasons = [], None, set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in (self.out or "").splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                sm.append(float(f[1]))
                mx = float(f[2])
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not sm:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"], "samples": 0}
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": mx, "reasons": sorted(reasons),
                "samples": len(sm)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0,
            "sm_max_mhz": 2070.0}, "fallback"


# ---------------------------------------------------------------------------
def dist_init(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(world, v: float) -> float:
    if world <= 1:
        return v
    import torch
    import torch.distributed as dist
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    t = torch.tensor([v], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
def roofline_for(name, launches, total_ms, work, peaks, peak_src, clocks):
    """Achieved algorithmic rate of one kernel vs its bound."""
    avg_s = total_ms / 1e3 / max(1, launches)
    w = work.get(name)
    if w is None:
        return None
    kind, per_launch = w
    if kind == "hbm":
        ach = per_launch / avg_s / 1e9
        peak = peaks["hbm_gbs"]
        return {"kernel": name, "bound": "hbm", "achieved": ach, "peak": peak, "unit": "GB/s",
                "frac": ach / peak, "traffic": None, "peak_source": f"hbm_gbs of {peak_src}",
                "algorithmic_bytes_per_launch": per_launch, "avg_launch_ms": avg_s * 1e3}
    # fp32 FMA pipe of the whole GPU at the SM clock seen under load
    sm_mhz = clocks.get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
    n_sm = w[2] if len(w) > 2 else 152
    peak = n_sm * 128 * 2 * sm_mhz * 1e6 / 1e12
    ach = per_launch / avg_s / 1e12
    return {"kernel": name, "bound": "alu", "achieved": ach, "peak": peak, "unit": "TFLOP/s",
            "frac": ach / peak, "traffic": None,
            "peak_source": f"{n_sm} SMs x 128 fp32 FMA/clk x 2 x {sm_mhz:.0f} MHz (sampled median)",
            "algorithmic_flops_per_launch": per_launch, "avg_launch_ms": avg_s * 1e3}


def recorded_traffic(kernel: str, workload: str, buckets: int):
    """DRAM bytes per launch of `kernel` from the ncu record committed under
    profiles/ for this workload, or None when there is none or the kernel's
    source has changed since it was taken (sha256 of the source file)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}.json")
    try:
        rec = json.load(open(path))
        if rec.get("kernel") != kernel or int(rec.get("buckets", -1)) != buckets:
            return None, None
        src = open(os.path.join(ROOT, rec["source"]), "rb").read()
        if hashlib.sha256(src).hexdigest() != rec.get("source_sha256"):
            return None, None
        return float(rec["dram_bytes_per_launch"]), os.path.relpath(path, ROOT)
    except (OSError, ValueError, KeyError):
        return None, None


def kernel_work(cfg, plan, ds):
    """Algorithmic work per launch of the main kernels, averaged over the
    epoch's batches: name -> (kind, per-launch amount)."""
    H, C = cfg["hidden"], cfg["n_classes"]
    dirs = 2 if cfg["bidirectional"] else 1
    Lc = cfg["n_layers"]
    n_tok, n_b = 0, plan["n_batches"]
    ext_cells = 0
    for k in range(n_b):
        ids = plan["order"][plan["batch_off"][k]:plan["batch_off"][k + 1]]
        L = ds.lengths[ids]
        n_tok += int(L.sum())
        ext_cells += int((L * (2 * ds.label_lengths[ids] + 1)).sum())
    tok_pb = n_tok / n_b
    cells_pb = ext_cells / n_b
    # recurrent kernels: W_hh matvec, 8 H^2 flops per token and direction
    # (forward), twice that counted once per direction in the backward
    rec = 8.0 * H * H * tok_pb * dirs
    work = {
        "lstm_fwd": ("alu", rec),
        "lstm_bwd": ("alu", rec),
        # CTC tables: each cell written once (fp32), emissions read once per cell
        "ctc_tables": ("hbm", 2 * 4.0 * cells_pb * 2),
        # posterior: alpha + beta read, logp row read + dlogit row written
        "ctc_grad": ("hbm", 4.0 * (2 * cells_pb + 2 * C * tok_pb)),
        "proj_narrow": ("hbm", 4.0 * tok_pb * (cfg["in_dim"] + 4 * H * dirs)),
        "layout_gather": ("hbm", 4.0 * tok_pb * (2 * cfg["in_dim"] + 4)),
    }
    return work, tok_pb


# ---------------------------------------------------------------------------
def run_native(args, world, rank, local):
    import torch

    from paper_1708_05604_gb300 import binding, build, synth

    build.build()
    binding.lib()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    w = synth.WORKLOADS[args.workload]
    cfg = w.model_cfg()
    ds = synth.make_workload(w, seed=args.seed)
    P = binding.param_count(cfg)
    params0 = synth.draw_params(np.random.default_rng(args.seed + 1), P)
    dd = binding.DeviceDataset(ds, device=dev)
    max_batch = w.batch
    # capacity: the B longest sequences
    max_tokens = int(np.sort(ds.lengths)[-max_batch:].sum())
    ctx = binding.Ctx(cfg, max_tokens, max_batch, int(ds.label_lengths.max()))
    params = torch.from_numpy(params0).to(dev)
    grads = torch.zeros_like(params)
    loss = torch.zeros(ds.n, dtype=torch.float32, device=dev)
    stream = torch.cuda.current_stream(dev)
    flush = torch.empty(256 * 1024 * 1024 // 4, dtype=torch.float32, device=dev)
    unpadded = int(ds.lengths.sum())

    opt = binding.Adadelta(params) if args.optimizer == "adadelta" else None

    def epoch(e, Q, dataset=dd, loss_buf=loss):
        plan = binding.plan_buckets(ds.lengths, Q, w.batch, seed=args.seed, epoch=e)
        order, off = plan["order"], plan["batch_off"]
        for k in range(plan["n_batches"]):
            ids = order[off[k]:off[k + 1]]
            lv = loss_buf[off[k]:off[k + 1]]
            ctx.step(dataset, ids, params, grads, lv, stream)
            if opt is None:
                binding.sgd_update(params, grads, LR, stream)
            else:
                opt.step(grads, stream)
        return plan

    def timed(Q, steps, warmup, e0=0, with_timer=False, clocks=None):
        for i in range(warmup):
            epoch(e0 + i, Q)
        torch.cuda.synchronize(dev)
        barrier(world)
        torch.cuda.synchronize(dev)
        if with_timer:
            ctx.set_timing(True)
        evs = []
        plans = []
        cm = clocks if clocks is not None else _Null()
        with cm:
            for i in range(steps):
                flush.zero_()
                a = torch.cuda.Event(enable_timing=True)
                b = torch.cuda.Event(enable_timing=True)
                a.record(stream)
                plans.append(epoch(e0 + warmup + i, Q))
                b.record(stream)
                evs.append((a, b))
            torch.cuda.synchronize(dev)
        barrier(world)
        torch.cuda.synchronize(dev)
        ms = [a.elapsed_time(b) for a, b in evs]
        ktimes = ctx.kernel_times() if with_timer else []
        if with_timer:
            ctx.set_timing(False)
        ctx.sync_status()
        return ms, plans, ktimes

    clocks = Clocks(local if not os.environ.get("CUDA_VISIBLE_DEVICES") else 0)
    ms, plans, _ = timed(args.buckets, args.steps, args.warmup, clocks=clocks)
    # per-kernel durations come from separate epochs: the per-launch event
    # records they need would otherwise sit inside the timed epochs
    timer_steps = max(3, args.steps // 2)
    _, tplans, ktimes = timed(args.buckets, timer_steps, 0, e0=args.warmup, with_timer=True)
    ms_step = sum(ms) / len(ms)
    ms_max = max_over_ranks(world, ms_step)
    value = world * unpadded / (ms_max / 1e3)
    pe = [p["unpadded_timesteps"] / p["padded_timesteps"] for p in plans]
    clk = clocks.summary()

    # epoch time vs bucket count (short runs)
    by_q = {str(args.buckets): {"ms_per_epoch": ms_step, "padded_efficiency": float(np.mean(pe)),
                                "dp_cost": plans[0]["dp_cost"], "n_batches": plans[0]["n_batches"]}}
    for qs in [q for q in args.compare_buckets.split(",") if q.strip()]:
        q = int(qs)
        if q == args.buckets:
            continue
        m2, p2, _ = timed(q, max(2, args.steps // 3), 1, e0=1000)
        by_q[str(q)] = {"ms_per_epoch": sum(m2) / len(m2),
                        "padded_efficiency": float(np.mean([p["unpadded_timesteps"] / p["padded_timesteps"]
                                                            for p in p2])),
                        "dp_cost": p2[0]["dp_cost"], "n_batches": p2[0]["n_batches"]}

    # kernel launches in the timed region and the dominant kernel's roofline
    per_epoch = sum(n for _, n, _ in ktimes) / timer_steps + plans[0]["n_batches"]
    launches = round(per_epoch * args.steps)
    peaks, peak_src = measured_peaks()
    work, tok_pb = kernel_work(cfg, plans[0], ds)
    ktimes_sorted = sorted(ktimes, key=lambda t: -t[2])
    total_k = sum(t for _, _, t in ktimes) or 1.0
    roof = None
    for name, n, t in ktimes_sorted:
        roof = roofline_for(name, n, t, work, peaks, peak_src, clk)
        if roof:
            roof["share_of_kernel_time"] = t / total_k
            tb, tsrc = recorded_traffic(name, w.name, args.buckets)
            roof["traffic"] = tb
            roof["traffic_source"] = tsrc
            break
    kernel_table = [{"kernel": nm, "launches": n, "total_ms": round(t, 3),
                     "share": round(t / total_k, 4)} for nm, n, t in ktimes_sorted]

    # end to end through the public API with host buffers
    e2e = None
    if not args.no_e2e:
        x_host = torch.from_numpy(np.ascontiguousarray(ds.x, np.float32)).pin_memory()
        lab_host = torch.from_numpy(np.ascontiguousarray(dd.labels.cpu().numpy())).pin_memory()
        loss_host = torch.empty(ds.n, dtype=torch.float32).pin_memory()
        x_dev = torch.empty_like(dd.x)
        lab_dev = torch.empty_like(dd.labels)
        dd2 = binding.DeviceDataset.__new__(binding.DeviceDataset)
        dd2.__dict__.update(dd.__dict__)
        dd2.x, dd2.labels = x_dev, lab_dev
        e2e_ms = []
        for i in range(args.warmup + max(2, args.steps // 2)):
            flush.zero_()
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            x_dev.copy_(x_host, non_blocking=True)
            lab_dev.copy_(lab_host, non_blocking=True)
            epoch(5000 + i, args.buckets, dataset=dd2)
            loss_host.copy_(loss, non_blocking=True)
            torch.cuda.synchronize(dev)
            if i >= args.warmup:
                e2e_ms.append((time.perf_counter() - t0) * 1e3)
        e_ms = max_over_ranks(world, sum(e2e_ms) / len(e2e_ms))
        e2e = {"value": world * unpadded / (e_ms / 1e3), "unit": "timesteps/s",
               "ms_per_step": e_ms,
               "h2d_bytes_per_step": int(x_host.numel() * 4 + lab_host.numel() * 4),
               "d2h_bytes_per_step": int(loss_host.numel() * 4)}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, w, ds, params0, plans[0], args.cpu_baseline_seconds)

    line = {
        "metric": "unpadded timesteps/sec (LSTM+CTC fwd+bwd+SGD epoch, 1 GPU)",
        "optimizer": args.optimizer,
        "value": value, "unit": "timesteps/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32" if not w.gemm_bf16 else "bf16+f32",
        "data": "synthetic (seeded; stands in for the paper's handwriting set)",
        "config": {"workload": w.name, "layers": w.n_layers, "bidirectional": w.bidirectional,
                   "hidden": w.hidden, "n_seqs": w.n_seqs, "batch": w.batch,
                   "buckets": args.buckets, "unpadded_timesteps_per_epoch": unpadded,
                   "step": "one epoch: plan + every batch's fwd/bwd/CTC + SGD",
                   "l2": "flushed between timed steps (256 MiB write, outside the events)",
                   "parallelism": "replicas" if world > 1 else "1 GPU"},
        "padded_efficiency": float(np.mean(pe)),
        "epoch_time_vs_buckets": by_q,
        "clocks": clk,
        "gpu_launches": int(launches),
        "roofline": roof,
        "kernels": kernel_table,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    ctx.close()


class _Null:
    def __enter__(self):
        return self

    def __exit__(self, *a):
        pass


# ---------------------------------------------------------------------------
def oracle_sample(w, ds, params0, plan, budget_s, start=0):
    """Runs the oracle one sequence at a time through the epoch order until
    `budget_s` seconds have passed; returns (timesteps, seconds, sequences)."""
    import oracle
    cfg = w.model_cfg()
    prm = params0.astype(np.float64)
    order = plan["order"]
    t0 = time.perf_counter()
    steps = 0
    n = 0
    i = start
    while True:
        sid = int(order[i % order.size])
        sub = ds.subset([sid])
        oracle.lstm_ctc_step(cfg, sub.lengths, sub.x.astype(np.float64), sub.label_lengths,
                             sub.labels, prm)
        steps += int(sub.lengths[0])
        n += 1
        i += 1
        el = time.perf_counter() - t0
        if el >= budget_s:
            return steps, el, n, i


def cpu_baseline(args, w, ds, params0, plan, budget_s):
    steps, el, n, _ = oracle_sample(w, ds, params0, plan, budget_s)
    return {"value": steps / el, "unit": "timesteps/s", "cores": 1, "kind": "oracle",
            "sample": f"{n} sequences ({steps} timesteps) of the epoch's bucketed order, "
                      f"one at a time, {el:.1f} s, fp64 single-threaded C"}


def run_reference(args, world, rank):
    """The oracle, timed on bounded samples of the same workload."""
    import oracle
    from paper_1708_05604_gb300 import synth
    if rank != 0:
        return
    oracle.build()
    w = synth.WORKLOADS[args.workload]
    ds = synth.make_workload(w, seed=args.seed)
    cfg = w.model_cfg()
    P = oracle.param_count(cfg["n_layers"], cfg["bidirectional"], cfg["in_dim"], cfg["hidden"],
                           cfg["n_classes"])
    params0 = synth.draw_params(np.random.default_rng(args.seed + 1), P)
    plan = oracle.plan(ds.lengths, args.buckets, w.batch, seed=args.seed, epoch=0)
    per_step = max(1.0, 150.0 / (args.steps + args.warmup))
    pos = 0
    for _ in range(args.warmup):
        _, _, _, pos = oracle_sample(w, ds, params0, plan, per_step, pos)
    tot_steps, tot_s, tot_n = 0, 0.0, 0
    for _ in range(args.steps):
        s, el, n, pos = oracle_sample(w, ds, params0, plan, per_step, pos)
        tot_steps += s
        tot_s += el
        tot_n += n
    value = tot_steps / tot_s
    line = {"impl": "reference",
            "metric": "unpadded timesteps/sec (LSTM+CTC fwd+bwd+SGD epoch, 1 GPU)",
            "value": value, "unit": "timesteps/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": tot_s / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic (seeded; stands in for the paper's handwriting set)",
            "config": {"workload": w.name, "buckets": args.buckets,
                       "step": f"bounded sample: sequences of the epoch order for {per_step:.1f} s"},
            "cpu_baseline": {"value": value, "unit": "timesteps/s", "cores": 1, "kind": "oracle",
                             "sample": f"{tot_n} sequences, {tot_steps} timesteps over {args.steps} steps"},
            "e2e": {"value": value, "unit": "timesteps/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    world, rank, local = dist_init(args)
    if args.impl == "reference":
        run_reference(args, world, rank)
    else:
        run_native(args, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
