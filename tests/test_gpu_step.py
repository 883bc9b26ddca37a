"""GPU parity: the CUDA training step (through the C ABI) against the fp64
oracle, element by element per parameter block, on seeded synthetic inputs.
Sizes let the oracle finish in seconds while spanning several tiles, clusters
and ragged tails; the last tests take whole batches of the workloads' own
plans at full size, launched as the benchmark launches them, and compare
every gradient with the oracle (run one sequence per process)."""
import math

import numpy as np
import pytest

import oracle
from paper_1708_05604_gb300 import binding, synth

from gpu_util import BF16_TOL, FP32_TOL, compare, gpu_step, oracle_step, oracle_step_parallel

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built(cuda_device):
    from paper_1708_05604_gb300 import build
    build.build()
    binding.lib()


def tol_for(cfg):
    return BF16_TOL if cfg.get("gemm_bf16") else FP32_TOL


def make_case(wname, n, max_len, seed=0):
    w = synth.WORKLOADS[wname]
    ds = synth.make_workload(w, seed=seed, n_seqs=n, max_len=max_len)
    cfg = w.model_cfg()
    rng = np.random.default_rng(seed + 100)
    params = synth.draw_params(rng, binding.param_count(cfg))
    return cfg, ds, params


# (workload, sequences, length cap): oracle-sized versions of every workload
SMALL = [
    ("lstm1_uni_h32", 16, None),
    ("lstm1_bi_h128", 9, 260),
    ("lstm3_bi_h256_bf16", 3, 70),
    ("lstm2_uni_h512", 3, 90),
    ("lstm3_bi_h256_bf16_bimodal", 3, 60),
]


@pytest.mark.parametrize("wname,n,max_len", SMALL)
def test_step_parity_small(wname, n, max_len):
    cfg, ds, params = make_case(wname, n, max_len)
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, tol_for(cfg))


def tiny_cfg(layers, bi, H, C=7):
    return {"n_layers": layers, "bidirectional": bi, "in_dim": 4, "hidden": H, "n_classes": C,
            "blank": 0}


@pytest.mark.parametrize("layers,bi,H", [(1, True, 5), (2, True, 6), (2, False, 12), (3, True, 8)])
def test_step_parity_odd_shapes(layers, bi, H):
    """Hidden sizes that are not multiples of 4 or of the cluster size."""
    cfg = tiny_cfg(layers, bi, H)
    rng = np.random.default_rng(layers * 7 + H)
    ds = synth.make_dataset([11, 1, 7, 30, 7, 2, 19], 3, rng, n_classes=cfg["n_classes"])
    params = rng.uniform(-0.4, 0.4, size=binding.param_count(cfg)).astype(np.float32)
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, FP32_TOL)


def _ctx_for(cfg, ds, max_batch):
    """A ctx sized for `max_batch` rows: its recurrent geometry is planned for
    that many rows, so a small batch runs the wide-batch kernel variant."""
    return binding.Ctx(cfg, max(int(ds.lengths.sum()), 64 * max_batch), max_batch,
                       max(1, int(ds.label_lengths.max())))


@pytest.mark.parametrize("wname,lengths,max_batch", [
    # 8 rows per 4-CTA cluster, rows ending at different steps, a partial second group
    ("lstm3_bi_h256_bf16", [26, 24, 21, 21, 17, 12, 9, 7, 5, 3, 2], 128),
    # 8 rows per 16-CTA cluster
    ("lstm2_uni_h512", [22, 20, 19, 14, 11, 8, 6, 4, 2, 1], 32),
    # two rows per single-CTA block (rows x directions > SMs)
    ("lstm1_bi_h128", [45, 44, 30, 30, 22, 13, 8, 3, 1], 100),
    ("lstm1_uni_h32", [40, 33, 20, 12, 6, 2, 1], 200),
])
def test_step_parity_wide_batch_kernels(wname, lengths, max_batch):
    """Element-wise parity of the kernel variants that full-size batches use,
    on oracle-sized batches (fp32 contractions, so the 1e-4 bound applies)."""
    w = synth.WORKLOADS[wname]
    rng = np.random.default_rng(4)
    ds = synth.make_dataset(lengths, 4, rng)
    cfg = dict(w.model_cfg(), gemm_bf16=False)
    params = synth.draw_params(rng, binding.param_count(cfg))
    ctx = _ctx_for(cfg, ds, max_batch)
    lg, gg = gpu_step(cfg, ds, params, ctx=ctx)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, FP32_TOL)


@pytest.mark.parametrize("H", [32, 256])
def test_step_parity_longer_than_shared_time_index(H):
    """A sequence longer than the 8,192 time offsets the recurrent kernels
    stage in shared memory (they then read them from global memory), with a
    long label (CTC with four extended-label positions per thread)."""
    cfg = {"n_layers": 1, "bidirectional": H == 32, "in_dim": 4, "hidden": H, "n_classes": 81,
           "blank": 0}
    rng = np.random.default_rng(8)
    ds = synth.make_dataset([8300, 37, 5], 10, rng)
    params = synth.draw_params(rng, binding.param_count(cfg))
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, FP32_TOL)


def test_edge_cases_one_step():
    """Length-1 sequence, empty label, repeated labels, no alignment, equal lengths."""
    cfg = synth.WORKLOADS["lstm1_bi_h128"].model_cfg()
    rng = np.random.default_rng(3)
    ds = synth.make_dataset([1, 40, 40, 40, 25, 9, 6], 3, rng)
    lab = ds.labels.copy()
    U = ds.label_lengths.copy()
    # seq 1: no labels at all
    U[1] = 0
    # seq 2: every label the same (needs blanks between repeats)
    # seq 5: 3 labels that all repeat -> needs 5 steps; length 9 fits
    # seq 6: length 6 with 4 identical labels -> needs 7 steps: no alignment
    U[6] = 4
    labels = []
    for i in range(ds.n):
        if i == 2:
            labels.append(np.full(U[i], 17, np.int32))
        elif i == 5:
            labels.append(np.array([4, 4, 4], np.int32)[:U[i]])
        elif i == 6:
            labels.append(np.full(4, 9, np.int32))
        else:
            labels.append(rng.integers(1, 81, size=U[i]).astype(np.int32))
    labels = np.concatenate(labels)
    off = np.zeros(ds.n + 1, np.int64)
    np.cumsum(U, out=off[1:])
    ds = synth.Dataset(ds.lengths, ds.x, ds.x_off, U.astype(np.int32), labels, off)
    params = synth.draw_params(rng, binding.param_count(cfg))
    ctx = binding.Ctx(cfg, int(ds.lengths.sum()), ds.n, int(ds.label_lengths.max()))
    lg, gg = gpu_step(cfg, ds, params, ctx=ctx)
    lo, go = oracle_step(cfg, ds, params)
    assert math.isinf(lo[6]) and math.isinf(lg[6]) and lg[6] > 0
    compare(cfg, lg, gg, lo, go, FP32_TOL)
    # the sequence without an alignment is counted in the ctx, once
    assert ctx.infeasible_count() == 1
    assert ctx.infeasible_count() == 0
    gpu_step(cfg, ds, params, ctx=ctx)
    gpu_step(cfg, ds, params, ctx=ctx)
    assert ctx.infeasible_count() == 2


def test_single_sequence_and_permutation_invariance():
    """A sequence's loss does not depend on its batch-mates or batch order
    (the packed layout adds no padding to the arithmetic)."""
    cfg, ds, params = make_case("lstm1_bi_h128", 12, 200, seed=5)
    lg, gg = gpu_step(cfg, ds, params)
    perm = np.array([7, 3, 11, 0, 5, 9, 1, 2, 10, 4, 8, 6])
    lp, gp = gpu_step(cfg, ds, params, seq_ids=perm)
    np.testing.assert_allclose(lp, lg[perm], rtol=2e-6)
    for i in (0, 4, 11):
        l1, g1 = gpu_step(cfg, ds, params, seq_ids=[i])
        assert abs(l1[0] - lg[i]) <= 2e-6 * abs(lg[i])
    # the batch gradient is the sum of two halves' gradients
    la, ga = gpu_step(cfg, ds, params, seq_ids=np.arange(6))
    lb, gb = gpu_step(cfg, ds, params, seq_ids=np.arange(6, 12))
    assert np.linalg.norm(ga + gb - gg) <= 1e-5 * np.linalg.norm(gg)


def test_step_is_deterministic():
    cfg, ds, params = make_case("lstm1_bi_h128", 10, 150, seed=2)
    l1, g1 = gpu_step(cfg, ds, params)
    l2, g2 = gpu_step(cfg, ds, params)
    assert np.array_equal(l1, l2) and np.array_equal(g1, g2)


def test_sgd_update():
    """p - lr * g with one fp32 rounding: within one ulp of the operands'
    magnitude of the exact value (lr as the fp32 the kernel receives)."""
    import torch
    rng = np.random.default_rng(0)

    def check(p, g, lr, got):
        lr32 = np.float64(np.float32(lr))
        exact = p.astype(np.float64) - lr32 * g.astype(np.float64)
        scale = np.abs(p.astype(np.float64)) + np.abs(lr32 * g.astype(np.float64))
        assert np.all(np.abs(got.astype(np.float64) - exact) <= 2.0 ** -23 * scale + 1e-30)

    for n in (1, 5, 7409, 100003):
        p = rng.standard_normal(n).astype(np.float32)
        g = rng.standard_normal(n).astype(np.float32)
        tp, tg = torch.from_numpy(p).cuda(), torch.from_numpy(g).cuda()
        binding.sgd_update(tp, tg, 1e-3)
        torch.cuda.synchronize()
        check(p, g, 1e-3, tp.cpu().numpy())
    # unaligned views take the scalar path
    tp = torch.from_numpy(p).cuda()
    tg = torch.from_numpy(g).cuda()
    binding.sgd_update(tp[1:], tg[1:], 0.5)
    torch.cuda.synchronize()
    check(p[1:], g[1:], 0.5, tp[1:].cpu().numpy())


def test_adadelta_update_vs_oracle():
    """ADADELTA (ref. [21]) against the oracle, one update at a time from the
    same fp32 state.  Error budget of the kernel's fp32 arithmetic, in units
    u = 2^-24 of relative error: E[g^2] is an fma of a rounded product (2u);
    dx takes two sums, two IEEE square roots, one IEEE division and one
    product on top (<= 5u); E[dx^2] squares it (10u) and adds two roundings
    (12u); the parameter moves by lr dx (5u of lr |dx|) plus one rounding of
    the result.  Bounds used: 4u, 16u and 8u (|p| + lr |dx|)."""
    import torch
    rng = np.random.default_rng(3)
    rho, eps, lr = 0.95, 1e-6, 1.0
    u = 2.0 ** -24
    for n, offset in ((1, 0), (7409, 0), (100003, 0), (5000, 1)):
        p = torch.from_numpy(rng.standard_normal(n + offset).astype(np.float32)).cuda()[offset:]
        a = torch.zeros(n + offset, device="cuda")[offset:]
        b = torch.zeros(n + offset, device="cuda")[offset:]
        for step in range(5):
            g = torch.from_numpy((rng.standard_normal(n) * 10.0 ** rng.uniform(-3, 1)).astype(np.float32)).cuda()
            p0, a0, b0, g0 = (t.cpu().numpy().astype(np.float64) for t in (p, a, b, g))
            binding.adadelta_update(p, g, a, b, rho, eps, lr)
            torch.cuda.synchronize()
            xe, ae, be = oracle.adadelta(p0, g0, a0, b0, np.float32(rho), np.float32(eps), lr)
            gx, ga, gb = (t.cpu().numpy().astype(np.float64) for t in (p, a, b))
            dx = np.abs(xe - p0) / lr
            assert np.all(np.abs(gx - xe) <= 8 * u * (np.abs(xe) + lr * dx) + 1e-37), (n, step)
            assert np.all(np.abs(ga - ae) <= 4 * u * np.abs(ae) + 1e-37), (n, step)
            assert np.all(np.abs(gb - be) <= 16 * u * np.abs(be) + 1e-37), (n, step)
    # argument checks
    t = torch.zeros(4, device="cuda")
    for bad in ((1.0, 1e-6, 1.0), (0.9, 0.0, 1.0), (0.9, 1e-6, -1.0)):
        with pytest.raises(binding.BktError):
            binding.adadelta_update(t, t, t, t, *bad)


def test_argument_errors():
    import torch
    cfg, ds, params = make_case("lstm1_uni_h32", 4, 50)
    ctx = binding.Ctx(cfg, max_tokens=100, max_batch=2, max_label_len=4)
    dd = binding.DeviceDataset(ds)
    p = torch.from_numpy(params).cuda()
    g = torch.zeros_like(p)
    loss = torch.zeros(4, device="cuda")
    with pytest.raises(binding.BktError) as e:
        ctx.step(dd, [0, 1, 2], p, g, loss)       # more sequences than max_batch
    assert e.value.rc == binding.BKT_EINVAL
    small = binding.Ctx(cfg, max_tokens=10, max_batch=2, max_label_len=40)
    with pytest.raises(binding.BktError):
        small.step(dd, [0, 1], p, g, loss)        # more tokens than the ctx holds
    short = binding.Ctx(cfg, max_tokens=1000, max_batch=4, max_label_len=0)
    with pytest.raises(binding.BktError):
        short.step(dd, [0, 1], p, g, loss)        # labels longer than max_label_len
    # a label equal to the blank is caught on the device
    bad = synth.Dataset(ds.lengths, ds.x, ds.x_off, ds.label_lengths, ds.labels.copy(), ds.lab_off)
    bad.labels[0] = 0
    ctx2 = binding.Ctx(cfg, max_tokens=int(ds.lengths.sum()), max_batch=4,
                       max_label_len=int(ds.label_lengths.max()))
    ctx2.step(binding.DeviceDataset(bad), [0, 1, 2, 3], p, g, loss)
    with pytest.raises(binding.BktError) as e:
        ctx2.sync_status()
    assert e.value.rc == binding.BKT_EDEVICE
    ctx2.sync_status()  # cleared


# ---------------------------------------------------------------------------
# Full-size batches, launched as the benchmark launches them.

def full_batch(wname, Q, which="longest", seed=0):
    w = synth.WORKLOADS[wname]
    ds = synth.make_workload(w, seed=seed)
    plan = binding.plan_buckets(ds.lengths, Q, w.batch, seed=seed, epoch=0)
    batches = [plan["order"][plan["batch_off"][k]:plan["batch_off"][k + 1]]
               for k in range(plan["n_batches"])]
    if which == "longest":
        ids = max(batches, key=lambda b: int(ds.lengths[b].max()))
    else:
        ids = batches[0]
    return w, ds, ids


@pytest.mark.parametrize("wname,Q,which", [
    ("lstm1_uni_h32", 2, "longest"),
    # the longest batch of the 4-bucket plan: 64 sequences, ~58 k tokens
    ("lstm1_bi_h128", 4, "longest"),
    ("lstm1_bi_h128", 1, "first"),
    # the shortest batches of the 16- and 32-bucket plans: 128 sequences,
    # split-K weight gradients over several accumulators
    ("lstm3_bi_h256_bf16", 16, "first"),
    ("lstm3_bi_h256_bf16_bimodal", 32, "first"),
])
def test_full_size_batch_vs_oracle(wname, Q, which):
    """A whole batch of the benchmark's plan, launched as the benchmark
    launches it (ctx sized for the workload), against the oracle element by
    element in every parameter block; the bf16 workloads again with fp32
    contractions at the fp32 bound."""
    w, ds, ids = full_batch(wname, Q, which)
    cfg = w.model_cfg()
    params = synth.draw_params(np.random.default_rng(1), binding.param_count(cfg))
    dd = binding.DeviceDataset(ds)
    lo, go = oracle_step_parallel(cfg, ds, params, ids)
    cfgs = [cfg] + ([dict(cfg, gemm_bf16=False)] if cfg["gemm_bf16"] else [])
    for c in cfgs:
        ctx = binding.Ctx(c, int(np.sort(ds.lengths)[-w.batch:].sum()), w.batch, int(ds.label_lengths.max()))
        lg, gg = gpu_step(c, ds, params, seq_ids=ids, dd=dd, ctx=ctx)
        assert np.all(np.isfinite(gg))
        compare(c, lg, gg, lo, go, tol_for(c))
        ctx.close()


def test_full_length_h512_wide_batch_vs_oracle():
    """Three full-length sequences of the H = 512 workload (two layers, fp32)
    through a ctx sized for its batch of 32: the 16-CTA cluster kernels run
    in their full-batch configuration, over ~3,000-4,000 steps."""
    w = synth.WORKLOADS["lstm2_uni_h512"]
    ds = synth.make_workload(w, seed=0)
    order = np.argsort(-ds.lengths, kind="stable")
    ids = np.array([order[0], order[len(order) // 2], order[-1]])
    cfg = w.model_cfg()
    params = synth.draw_params(np.random.default_rng(1), binding.param_count(cfg))
    dd = binding.DeviceDataset(ds)
    ctx = binding.Ctx(cfg, int(np.sort(ds.lengths)[-w.batch:].sum()), w.batch, int(ds.label_lengths.max()))
    lg, gg = gpu_step(cfg, ds, params, seq_ids=ids, dd=dd, ctx=ctx)
    lo, go = oracle_step_parallel(cfg, ds, params, ids)
    compare(cfg, lg, gg, lo, go, FP32_TOL)
    # the batch gradient is the sum of the sequences' gradients
    _, ga = gpu_step(cfg, ds, params, seq_ids=ids[:1], dd=dd, ctx=ctx)
    _, gb = gpu_step(cfg, ds, params, seq_ids=ids[1:], dd=dd, ctx=ctx)
    assert np.linalg.norm(ga + gb - gg) <= 1e-4 * np.linalg.norm(gg)


@pytest.mark.parametrize("layers,bi,H", [(2, True, 128), (2, False, 512), (3, True, 64)])
def test_bf16_path_with_the_other_recurrent_kernels(layers, bi, H):
    """The bf16 contractions when the recurrent kernels do not write the bf16
    copies themselves (single-CTA kernels at H <= 128, register-tiled
    clusters at H = 512): the step casts them instead.  Parity at the bf16
    bound."""
    cfg = {"n_layers": layers, "bidirectional": bi, "in_dim": 4, "hidden": H, "n_classes": 81, "blank": 0,
           "gemm_bf16": True}
    rng = np.random.default_rng(H + layers)
    ds = synth.make_dataset([61, 47, 33, 30, 12, 5, 1], 8, rng)
    params = synth.draw_params(rng, binding.param_count(cfg))
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, BF16_TOL)


@pytest.mark.parametrize("b", [100, 120, 232])
def test_tensor_core_recurrence_cluster_layouts(b):
    """The H = 256 tensor-core recurrence spreads a batch over one-team
    (16-row) and two-team (32-row) clusters, no more of them than can be
    resident at once (15 on a GB300): 100 rows run on one-team clusters
    only, 120 on six one-team clusters and one two-team cluster per
    direction (its second team partly filled), 232 on two-team clusters only
    (one team empty; more clusters than fit at once).  Rows end at every
    step; one bidirectional layer with bf16 contractions, at the bf16
    bound."""
    cfg = {"n_layers": 1, "bidirectional": True, "in_dim": 4, "hidden": 256, "n_classes": 81, "blank": 0,
           "gemm_bf16": True}
    rng = np.random.default_rng(b)
    ds = synth.make_dataset(rng.integers(1, 15, size=b), 4, rng)
    params = synth.draw_params(rng, binding.param_count(cfg))
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step_parallel(cfg, ds, params, np.arange(ds.n))
    compare(cfg, lg, gg, lo, go, BF16_TOL)


@pytest.mark.parametrize("H,bi,b", [(512, False, 24), (512, False, 32), (512, False, 60), (256, True, 100)])
def test_register_tiled_cluster_layouts(H, bi, b):
    """The fp32 cluster kernels (H = 256 and 512) spread a batch over 4-row
    and 8-row clusters, no more of them than can be resident at once (7
    sixteen-CTA clusters at H = 512): 24 rows run on 4-row clusters only,
    32 on six 4-row clusters and one 8-row cluster, 60 on 8-row clusters
    only (more than fit at once); at H = 256, 100 rows per direction mix
    both.  Rows end at every step; fp32 contractions, at the fp32 bound."""
    cfg = {"n_layers": 1, "bidirectional": bi, "in_dim": 4, "hidden": H, "n_classes": 81, "blank": 0}
    rng = np.random.default_rng(H + b)
    ds = synth.make_dataset(rng.integers(1, 13, size=b), 4, rng)
    params = synth.draw_params(rng, binding.param_count(cfg))
    lg, gg = gpu_step(cfg, ds, params)
    lo, go = oracle_step_parallel(cfg, ds, params, np.arange(ds.n))
    compare(cfg, lg, gg, lo, go, FP32_TOL)


def test_bf16_workload_runs_on_tensor_cores():
    """The bf16 workloads route their contractions through the tcgen05 GEMM
    (and stay within the bf16 tolerance while differing from fp32 rounding)."""
    import torch
    cfg, ds, params = make_case("lstm3_bi_h256_bf16", 4, 80, seed=3)
    ctx = binding.Ctx(cfg, int(ds.lengths.sum()), ds.n, int(ds.label_lengths.max()))
    ctx.set_timing(True)
    lg, gg = gpu_step(cfg, ds, params, ctx=ctx)
    names = {n: c for n, c, _ in ctx.kernel_times()}
    assert names.get("gemm_tc", 0) >= 2 * 2 + 2 * 3 * 2, names   # projections, dX, weight grads
    lo, go = oracle_step(cfg, ds, params)
    worst = compare(cfg, lg, gg, lo, go, BF16_TOL)
    assert worst > 1e-6   # bf16 operands really are in play
    fcfg = dict(cfg, gemm_bf16=False)
    lf, gf = gpu_step(fcfg, ds, params)
    compare(fcfg, lf, gf, lo, go, FP32_TOL)


def test_average_models_vs_oracle():
    """Eq. 3 (Section III.B step 5) on the GPU: from the element-wise sum of K
    models, v / K - beta prev in fp32 (one IEEE division, one fused
    multiply-add: within 2 ulp of the exact value's magnitude terms)."""
    import torch
    rng = np.random.default_rng(9)
    for n, K, beta in ((1, 1, 1e-6), (7409, 2, 1e-6), (100003, 6, 0.25), (5003, 3, 0.0)):
        models = rng.standard_normal((K, n)).astype(np.float32)
        summed = models.astype(np.float64).sum(axis=0).astype(np.float32)   # what the all-reduce delivers
        prev = rng.standard_normal(n).astype(np.float32)
        v = torch.from_numpy(summed).cuda()
        binding.average_models(v, torch.from_numpy(prev).cuda(), K, beta)
        torch.cuda.synchronize()
        exact = oracle.average_models([summed.astype(np.float64) / K], prev.astype(np.float64), float(np.float32(beta)))
        scale = np.abs(summed.astype(np.float64) / K) + abs(beta) * np.abs(prev.astype(np.float64))
        assert np.all(np.abs(v.cpu().numpy().astype(np.float64) - exact) <= 2 * 2.0 ** -24 * scale + 1e-38)
    with pytest.raises(binding.BktError):
        binding.average_models(torch.zeros(4, device="cuda"), torch.zeros(4, device="cuda"), 0)


def test_data_parallel_epoch_on_one_gpu_with_nccl():
    """The replica loop's GPU data plane with one NCCL rank: the all-reduce is
    the identity and eq. 3 leaves (start + delta) - beta * start."""
    import torch
    import torch.distributed as dist

    from paper_1708_05604_gb300 import train
    import socket
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        port = s.getsockname()[1]
    dist.init_process_group("nccl", init_method=f"tcp://127.0.0.1:{port}", rank=0, world_size=1)
    try:
        start = torch.randn(10007, device="cuda")
        delta = torch.randn(10007, device="cuda")
        out = train.data_parallel_epoch(start, np.arange(5), lambda ids: start + delta,
                                        lambda t: dist.all_reduce(t, op=dist.ReduceOp.SUM),
                                        lambda v, prev, k: binding.average_models(v, prev, k, 1e-6), 1)
        torch.cuda.synchronize()
        ref = (start.double() + delta.double()) - 1e-6 * start.double()
        assert torch.allclose(out.double(), ref, rtol=1e-6, atol=1e-6)
    finally:
        dist.destroy_process_group()
