"""Failure detection on the GPU without a GPU fault: every spin-wait of the
library's kernels is bounded.  These tests make a wait run out on purpose
through the ctx's failure-detection hooks (a tiny poll cap, and data that a
host-set flag withholds, so the waited-for bytes never arrive), then check
that the step returns, that bkt_ctx_sync_status reports BKT_ETIMEOUT, and
that the next step with the hooks off matches the oracle."""
import numpy as np
import pytest

from paper_1708_05604_gb300 import binding, synth

from gpu_util import BF16_TOL, FP32_TOL, compare, gpu_step, oracle_step

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def built(cuda_device):
    from paper_1708_05604_gb300 import build
    build.build()
    binding.lib()


def small_case(cfg, lengths, seed):
    rng = np.random.default_rng(seed)
    ds = synth.make_dataset(lengths, 4, rng)
    params = synth.draw_params(rng, binding.param_count(cfg))
    ctx = binding.Ctx(cfg, int(ds.lengths.sum()), ds.n, int(ds.label_lengths.max()))
    return ds, params, ctx


def expect_timeout_then_recover(cfg, ds, params, ctx, withhold, tol):
    ctx.set_wait_faults(poll_cap=1000, withhold=withhold)
    import torch
    p = torch.from_numpy(params).cuda()
    g = torch.zeros_like(p)
    loss = torch.zeros(ds.n, device="cuda")
    ctx.step(binding.DeviceDataset(ds), np.arange(ds.n), p, g, loss)
    with pytest.raises(binding.BktError) as e:
        ctx.sync_status()
    assert e.value.rc == binding.BKT_ETIMEOUT, str(e.value)
    ctx.sync_status()   # the flags were cleared
    ctx.set_wait_faults(0, 0)
    lg, gg = gpu_step(cfg, ds, params, ctx=ctx)
    lo, go = oracle_step(cfg, ds, params)
    compare(cfg, lg, gg, lo, go, tol)


@pytest.mark.parametrize("H,bi,bf16", [(256, True, False), (512, False, False), (256, True, True)])
def test_cluster_exchange_wait_runs_out(H, bi, bf16):
    """CTA 0 of every recurrent cluster withholds its h / partial sums: its
    peers' bounded mbarrier waits expire, the kernels leave their loops and
    report bit 4; the forward kernel and BPTT both take that path (the
    register-tiled fp32 kernels at H = 256 and 512, the tensor-core kernels
    of the bf16 configuration at H = 256)."""
    cfg = {"n_layers": 1, "bidirectional": bi, "in_dim": 4, "hidden": H, "n_classes": 81, "blank": 0,
           "gemm_bf16": bf16}
    ds, params, ctx = small_case(cfg, [14, 11, 9, 5, 2], seed=H)
    expect_timeout_then_recover(cfg, ds, params, ctx, binding.BKT_WITHHOLD_EXCHANGE, BF16_TOL if bf16 else FP32_TOL)
    ctx.close()


@pytest.mark.parametrize("bf16", [True, False])
def test_tensor_core_pipeline_wait_runs_out(bf16):
    """The producers of every tensor-core GEMM withhold their first k slab:
    the MMA issuer's bounded wait expires, the producer drains the loads it
    did issue, and the kernel reports bit 2 (bf16 and 3xTF32 kernels, TMA-fed
    and token-major)."""
    cfg = {"n_layers": 2, "bidirectional": True, "in_dim": 4, "hidden": 64, "n_classes": 81, "blank": 0,
           "gemm_bf16": bf16}
    ds, params, ctx = small_case(cfg, [40, 33, 21, 8], seed=7)
    expect_timeout_then_recover(cfg, ds, params, ctx, binding.BKT_WITHHOLD_TMA, BF16_TOL if bf16 else FP32_TOL)
    ctx.close()


def test_wait_fault_arguments():
    cfg = {"n_layers": 1, "bidirectional": False, "in_dim": 4, "hidden": 32, "n_classes": 81, "blank": 0}
    ctx = binding.Ctx(cfg, 100, 2, 4)
    with pytest.raises(binding.BktError) as e:
        ctx.set_wait_faults(-1, 0)
    assert e.value.rc == binding.BKT_EINVAL
    with pytest.raises(binding.BktError):
        ctx.set_wait_faults(0, 8)
    ctx.set_wait_faults(1, 0)   # raised to the minimum cap
    ctx.set_wait_faults(0, 0)
    ctx.close()
