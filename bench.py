#!/usr/bin/env python3
"""Benchmark of the bucketed LSTM-CTC training step on GB300.

One "step" = one training epoch over the synthetic workload: plan the
buckets (bkt_plan_buckets: histogram, dynamic program, per-epoch reshuffle),
then for every mini-batch one bkt_lstm_ctc_step (packed layout, LSTM forward,
output + log-softmax, CTC, BPTT, weight gradients) and one bkt_sgd_update
(or, with --optimizer adadelta, the paper's update rule bkt_adadelta_update).
The metric is unpadded timesteps per second (sum of sequence lengths
processed / time), plus the epoch time against the bucket count (the
quantity of the paper's Fig. 4).  Inputs are resident in HBM when the timed
region starts; L2 is flushed (a 256 MiB write) between timed steps, outside
their events.

The default workload is the full-epoch sweep: a 3-layer bidirectional LSTM
(H = 256, bf16 tensor-core contractions, fp32 recurrence) with 81-class CTC
over 32,768 sequences of bimodal length (lognormal medians 150 and 900,
sigma 0.5, clipped to [20, 3000]), batch 128, timed at Q = 8 buckets with
single epochs at Q = 1, 2, 4, 16 and 32.  Every kernel's achieved rate
against its roofline comes from the library's per-launch work accounting
(bkt_ctx_kernel_times), measured in separate epochs.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

--impl reference times the fp64 CPU oracle (test infrastructure) on bounded
samples of the same workload.  Under torchrun each rank runs a replica of the workload
and the replicas' parameters are combined at the end of every epoch by the
paper's eq. 3 (an NCCL all-reduce, then bkt_average_models: the one
exchange of the data-parallel method); rank 0 prints the whole-job line.
"""
from __future__ import annotations

import argparse
import json
import math
import os
import statistics
import subprocess
import sys
import time

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

DEFAULT_WORKLOAD = "lstm3_bi_h256_bf16_bimodal"
DEFAULT_BUCKETS = 8
DEFAULT_COMPARE = "1,2,4,16,32"
LR = 1e-3
METRIC = "unpadded timesteps/sec (LSTM+CTC fwd+bwd, 1 GPU) and epoch time vs bucket count"


def parse(argv=None):
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", default="native", choices=["native", "reference"])
    ap.add_argument("--workload", default=DEFAULT_WORKLOAD)
    ap.add_argument("--buckets", type=int, default=DEFAULT_BUCKETS)
    ap.add_argument("--compare-buckets", default=DEFAULT_COMPARE,
                    help="extra bucket counts timed briefly for epoch time vs Q ('' = none)")
    ap.add_argument("--seed", type=int, default=0)
    ap.add_argument("--optimizer", default="sgd", choices=["sgd", "adadelta"])
    ap.add_argument("--cpu-baseline-seconds", type=float, default=15.0)
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--reference-seconds", type=float, default=150.0,
                    help="--impl reference: oracle seconds over all warm-up and timed steps")
    return ap.parse_args(argv)


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
# What bounds each kernel of the step (everything not listed moves data: HBM).
#   alu            fp32 FMA pipe of the whole GPU (the recurrent matvecs)
#   tensor_bf16    tcgen05 kind::f16 with bf16 operands
#   tensor_tf32x3  tcgen05 kind::tf32, three MMAs per split-precision product
KERNEL_BOUND = {"lstm_fwd": "alu", "lstm_bwd": "alu", "gemm_tc": "tensor_bf16",
                "gemm_tf32x3": "tensor_tf32x3", "gemm_tf32x3_tn": "tensor_tf32x3"}
TF32_PER_BF16 = 1.1 / 2.25   # nominal dense tf32 : bf16 tensor rate


def roofline_for(stat: dict, peaks: dict, peak_src: str, clocks: dict, n_sm: int = 152):
    """Achieved algorithmic rate of one kernel (its totals over the timer
    epochs: launches, total_ms, flops, bytes, serial_steps) against the peak
    of what bounds it; None when the kernel carries no work."""
    name, ms = stat["name"], stat["total_ms"]
    if ms <= 0 or stat["launches"] <= 0:
        return None
    bound = KERNEL_BOUND.get(name, "hbm")
    sec = ms / 1e3
    out = {"kernel": name, "launches": stat["launches"], "avg_launch_ms": ms / stat["launches"]}
    if bound == "hbm":
        if stat["bytes"] <= 0:
            return None
        peak = peaks["hbm_gbs"]
        out.update(bound="hbm", achieved=stat["bytes"] / sec / 1e9, peak=peak, unit="GB/s",
                   peak_source=f"hbm_gbs of {peak_src}",
                   algorithmic_bytes_per_launch=stat["bytes"] / stat["launches"])
    else:
        if stat["flops"] <= 0:
            return None
        if bound == "alu":
            sm_mhz = clocks.get("sm_mhz") or peaks.get("sm_max_mhz", 2070.0)
            peak = n_sm * 128 * 2 * sm_mhz * 1e6 / 1e12
            src = f"{n_sm} SMs x 128 fp32 FMA/clk x 2 x {sm_mhz:.0f} MHz (sampled median)"
            b = "alu"
        elif bound == "tensor_bf16":
            peak = peaks.get("bf16_tflops_sustained") or peaks["bf16_tflops"]
            src = f"bf16_tflops_sustained of {peak_src} (kernel timed inside a long step)"
            b = "tensor"
        else:
            base = peaks.get("bf16_tflops_sustained") or peaks["bf16_tflops"]
            peak = base * TF32_PER_BF16 / 3.0
            src = (f"bf16_tflops_sustained of {peak_src} x {TF32_PER_BF16:.3f} (nominal tf32:bf16) / 3 "
                   "(three tf32 MMAs per split-precision product)")
            b = "tensor"
        out.update(bound=b, achieved=stat["flops"] / sec / 1e12, peak=peak, unit="TFLOP/s",
                   peak_source=src, algorithmic_flops_per_launch=stat["flops"] / stat["launches"])
    out["frac"] = out["achieved"] / out["peak"]
    if stat.get("serial_steps", 0) > 0:
        out["us_per_step"] = ms * 1e3 / stat["serial_steps"]
    return out


def recorded_traffic(kernel: str, workload: str, buckets: int):
    """DRAM bytes per launch of `kernel` from the ncu record committed under
    profiles/ for this workload, or None when there is none or the kernel's
    source has changed since it was taken (sha256 of the source file)."""
    import hashlib
    path = os.path.join(ROOT, "profiles", f"traffic_{workload}.json")
    try:
        rec = json.load(open(path))
        if int(rec.get("buckets", -1)) != buckets:
            return None, None
        if "kernels" in rec:  # several kernels of one source file
            entry = rec["kernels"].get(kernel)
            if entry is None:
                return None, None
        elif rec.get("kernel") == kernel:
            entry = rec
        else:
            return None, None
        src = open(os.path.join(ROOT, rec["source"]), "rb").read()
        if hashlib.sha256(src).hexdigest() != rec.get("source_sha256"):
            return None, None
        return float(entry["dram_bytes_per_launch"]), os.path.relpath(path, ROOT)
    except (OSError, ValueError, KeyError):
        return None, None


def budget_count(ms_per_epoch: float, budget_ms: float, lo: int, hi: int) -> int:
    """How many epochs of `ms_per_epoch` fit in `budget_ms`, within [lo, hi]."""
    n = int(math.ceil(budget_ms / max(ms_per_epoch, 1e-3)))
    return max(lo, min(hi, n))


# ---------------------------------------------------------------------------
def run_native(args, world, rank, local):
    import torch

    from paper_1708_05604_gb300 import binding, build, synth

    build.build()
    binding.lib()
    dev = torch.device("cuda", local)
    torch.cuda.set_device(dev)
    n_sm = torch.cuda.get_device_properties(dev).multi_processor_count
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

    prev = torch.empty_like(params) if world > 1 else None

    def epoch(e, Q, dataset=dd, loss_buf=loss):
        plan = binding.plan_buckets(ds.lengths, Q, w.batch, seed=args.seed, epoch=e)
        order, off = plan["order"], plan["batch_off"]
        if prev is not None:
            prev.copy_(params)
        for k in range(plan["n_batches"]):
            ids = order[off[k]:off[k + 1]]
            lv = loss_buf[off[k]:off[k + 1]]
            ctx.step(dataset, ids, params, grads, lv, stream)
            if opt is None:
                binding.sgd_update(params, grads, LR, stream)
            else:
                opt.step(grads, stream)
        if prev is not None:
            # the replicas' models are combined once per epoch (Section III.B
            # step 5, eq. 3): NCCL all-reduce of the parameters, then
            # bkt_average_models
            import torch.distributed as dist
            dist.all_reduce(params, op=dist.ReduceOp.SUM)
            binding.average_models(params, prev, world, 1e-6, stream)
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
        kstats = ctx.kernel_stats() if with_timer else []
        if with_timer:
            ctx.set_timing(False)
        ctx.sync_status()
        return ms, plans, kstats

    clocks = Clocks(local if not os.environ.get("CUDA_VISIBLE_DEVICES") else 0)
    ms, plans, _ = timed(args.buckets, args.steps, args.warmup, clocks=clocks)
    ms_step = sum(ms) / len(ms)
    ms_max = max_over_ranks(world, ms_step)
    value = world * unpadded / (ms_max / 1e3)
    pe = [p["unpadded_timesteps"] / p["padded_timesteps"] for p in plans]
    clk = clocks.summary()
    infeasible = ctx.infeasible_count()

    # per-kernel durations and work come from separate epochs: the per-launch
    # event records they need would otherwise sit inside the timed epochs
    timer_steps = budget_count(ms_step, 3000.0, 1, max(1, args.steps // 2))
    _, _, kstats = timed(args.buckets, timer_steps, 0, e0=args.warmup, with_timer=True)

    # epoch time vs bucket count (short runs)
    by_q = {str(args.buckets): {"ms_per_epoch": ms_step, "padded_efficiency": float(np.mean(pe)),
                                "dp_cost": plans[0]["dp_cost"], "n_batches": plans[0]["n_batches"],
                                "serial_steps": serial_steps(plans[0], ds), "epochs": len(ms)}}
    q_steps = budget_count(ms_step, 2000.0, 1, max(1, args.steps // 3))
    for qs in [q for q in args.compare_buckets.split(",") if q.strip()]:
        q = int(qs)
        if q == args.buckets:
            continue
        m2, p2, _ = timed(q, q_steps, 0, e0=1000)
        by_q[str(q)] = {"ms_per_epoch": sum(m2) / len(m2),
                        "padded_efficiency": float(np.mean([p["unpadded_timesteps"] / p["padded_timesteps"]
                                                            for p in p2])),
                        "dp_cost": p2[0]["dp_cost"], "n_batches": p2[0]["n_batches"],
                        "serial_steps": serial_steps(p2[0], ds), "epochs": len(m2)}
    by_q = dict(sorted(by_q.items(), key=lambda kv: int(kv[0])))

    # kernel launches in the timed region, per-kernel rooflines, the dominant one
    per_epoch = sum(k["launches"] for k in kstats) / timer_steps + plans[0]["n_batches"]
    launches = round(per_epoch * args.steps)
    peaks, peak_src = measured_peaks()
    total_k = sum(k["total_ms"] for k in kstats) or 1.0
    rooflines = []
    for k in sorted(kstats, key=lambda k: -k["total_ms"]):
        r = roofline_for(k, peaks, peak_src, clk, n_sm)
        if r:
            r["share_of_kernel_time"] = k["total_ms"] / total_k
            rooflines.append(r)
    roof = dict(rooflines[0]) if rooflines else None
    if roof:
        tb, tsrc = recorded_traffic(roof["kernel"], w.name, args.buckets)
        roof["traffic"] = tb
        roof["traffic_source"] = tsrc
    kernel_table = [{"kernel": k["name"], "launches": k["launches"], "total_ms": round(k["total_ms"], 3),
                     "share": round(k["total_ms"] / total_k, 4)}
                    for k in sorted(kstats, key=lambda k: -k["total_ms"])]

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
        e2e_warm = min(args.warmup, 1)
        e2e_steps = budget_count(ms_step, 15000.0, 2, max(2, args.steps))
        e2e_ms = []
        for i in range(e2e_warm + e2e_steps):
            flush.zero_()
            torch.cuda.synchronize(dev)
            t0 = time.perf_counter()
            x_dev.copy_(x_host, non_blocking=True)
            lab_dev.copy_(lab_host, non_blocking=True)
            epoch(5000 + i, args.buckets, dataset=dd2)
            loss_host.copy_(loss, non_blocking=True)
            torch.cuda.synchronize(dev)
            if i >= e2e_warm:
                e2e_ms.append((time.perf_counter() - t0) * 1e3)
        e_ms = max_over_ranks(world, sum(e2e_ms) / len(e2e_ms))
        e2e = {"value": world * unpadded / (e_ms / 1e3), "unit": "timesteps/s",
               "ms_per_step": e_ms, "steps": len(e2e_ms),
               "h2d_bytes_per_step": int(x_host.numel() * 4 + lab_host.numel() * 4),
               "d2h_bytes_per_step": int(loss_host.numel() * 4)}

    cpu = None
    if rank == 0 and not args.no_cpu_baseline:
        cpu = cpu_baseline(args, w, ds, params0, plans[0], args.cpu_baseline_seconds)

    line = {
        "metric": METRIC,
        "optimizer": args.optimizer,
        "value": value, "unit": "timesteps/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms_max, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32" if not w.gemm_bf16 else "bf16+f32",
        "data": "synthetic (seeded; stands in for the paper's handwriting set)",
        "config": {"workload": w.name, "layers": w.n_layers, "bidirectional": w.bidirectional,
                   "hidden": w.hidden, "n_seqs": w.n_seqs, "batch": w.batch,
                   "buckets": args.buckets, "unpadded_timesteps_per_epoch": unpadded,
                   "step": "one epoch: plan + every batch's fwd/bwd/CTC + SGD, rebucketed and reshuffled",
                   "l2": "flushed between timed steps (256 MiB write, outside the events)",
                   "parallelism": "replicas, eq.-3 averaging per epoch" if world > 1 else "1 GPU"},
        "padded_efficiency": float(np.mean(pe)),
        "infeasible_sequences_per_epoch": infeasible / max(1, args.steps),
        "epoch_time_vs_buckets": by_q,
        "clocks": clk,
        "gpu_launches": int(launches),
        "roofline": roof,
        "rooflines": rooflines,
        "kernels": kernel_table,
        "e2e": e2e,
        "cpu_baseline": cpu,
    }
    if rank == 0:
        print(json.dumps(line), flush=True)
    ctx.close()


def serial_steps(plan, ds) -> int:
    """Sum over the plan's batches of the longest length: the recurrence's
    serial time steps per layer and direction in one epoch."""
    off, order = plan["batch_off"], plan["order"]
    return int(sum(int(ds.lengths[order[off[k]:off[k + 1]]].max()) for k in range(plan["n_batches"])))


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
    per_step = max(0.05, args.reference_seconds / max(1, args.steps + args.warmup))
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
            "metric": METRIC,
            "value": value, "unit": "timesteps/s", "n_gpus": world, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": tot_s / args.steps * 1e3,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "gpu_launches": 0,
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
