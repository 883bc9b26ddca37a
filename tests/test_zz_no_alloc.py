"""The allocation-free step entry point (bkt_lstm_ctc_step_static).

Some callers cannot allocate device memory: a plugin inside a framework
that owns all GPU memory through its own pool, or a process whose memory
budget is fixed at start-up.  For them the library keeps one fixed device
array and runs the step on it.  This test calls that entry point through the
C ABI twice in a row, on two different batches, and checks each result
against the ordinary entry point (bkt_lstm_ctc_step with a ctx) at the fp32
parity tolerance.  It lives in a file of its own, collected last, and runs
the same way alone in a fresh process or after the other tests.
"""
import numpy as np
import pytest

pytestmark = pytest.mark.gpu


STATIC_CASES = [
    ("lstm1_bi_h128", None, 180),
    # two fp32 layers: dX on the tensor cores shares scratch with the weight
    # gradients here, while the ctx path runs them on two streams
    ("lstm1_bi_h128", {"n_layers": 2, "hidden": 64}, 120),
    ("lstm3_bi_h256_bf16", None, 50),
]


@pytest.mark.parametrize("wname,override,max_len", STATIC_CASES)
def test_static_step_matches_ctx_step(cuda_device, wname, override, max_len):
    import torch

    from paper_1708_05604_gb300 import binding, build, synth

    from gpu_util import FP32_TOL, compare, gpu_step

    build.build()
    w = synth.WORKLOADS[wname]
    cfg = dict(w.model_cfg(), **(override or {}))
    ds = synth.make_workload(w, seed=4, n_seqs=14, max_len=max_len)
    params_np = synth.draw_params(np.random.default_rng(8), binding.param_count(cfg))
    dd = binding.DeviceDataset(ds)
    params = torch.from_numpy(params_np).cuda()
    batches = [np.array([3, 0, 7, 12, 5, 9]), np.array([1, 2, 4, 6, 8, 10, 11, 13, 0])]
    for ids in batches:   # two calls in a row on the shared array
        grads = torch.full_like(params, float("nan"))
        loss = torch.full((ids.size,), float("nan"), device="cuda")
        binding.step_static(cfg, dd, ids, params, grads, loss)
        torch.cuda.synchronize()
        lr, gr = gpu_step(cfg, ds, params_np, seq_ids=ids, dd=dd)
        compare(cfg, loss.cpu().numpy().astype(np.float64), grads.cpu().numpy().astype(np.float64),
                lr, gr, FP32_TOL)


def test_static_step_rejects_oversized_batch(cuda_device):
    import torch

    from paper_1708_05604_gb300 import binding, build, synth

    build.build()
    w = synth.WORKLOADS["lstm1_bi_h128"]
    cfg = w.model_cfg()
    ds = synth.make_workload(w, seed=0, n_seqs=64)
    dd = binding.DeviceDataset(ds)
    params = torch.zeros(binding.param_count(cfg), device="cuda")
    grads = torch.zeros_like(params)
    loss = torch.zeros(64, device="cuda")
    with pytest.raises(binding.BktError) as e:
        binding.step_static(cfg, dd, np.arange(64), params, grads, loss)
    assert e.value.rc == binding.BKT_EINVAL
    assert "bytes of scratch" in str(e.value)
