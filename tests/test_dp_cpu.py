"""The data-parallel loop of Section III.B (steps 3-5) on CPU ranks: data
portions reshuffled every epoch, each replica trains its portion from the
same parameters, then the replicas' parameters are summed by a collective
(gloo here, NCCL on GPUs) and combined by eq. 3.  The replica's training and
eq. 3 are injected (the oracle's, on the CPU), so the test covers the loop's
host logic and its one exchange with world_size 2."""
import os
import socket

import numpy as np
import pytest

import oracle
from paper_1708_05604_gb300 import binding, synth, train

CFG = {"n_layers": 1, "bidirectional": True, "in_dim": 4, "hidden": 4, "n_classes": 7, "blank": 0}
BETA = 1e-3


def tiny_dataset():
    rng = np.random.default_rng(5)
    L = rng.integers(6, 20, size=12).astype(np.int32)
    return synth.make_dataset(L, 4, rng, n_classes=CFG["n_classes"])


def oracle_train_portion(ds, params_start, portion, epoch, lr=0.05):
    """One SGD epoch of the oracle over the portion, bucketed by the
    library's planner (2 buckets, batches of 3)."""
    p = np.array(params_start, dtype=np.float64)
    batches, _ = train.epoch_batches(ds.lengths, portion, 2, 3, seed=0, epoch=epoch)
    for ids in batches:
        sub = ds.subset(ids)
        _, g = oracle.lstm_ctc_step(CFG, sub.lengths, sub.x.astype(np.float64), sub.label_lengths, sub.labels, p)
        p = oracle.sgd(p, g, lr)
    return p


def _rank(rank, world, port, epochs, out_dir):
    import torch
    import torch.distributed as dist
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    ds = tiny_dataset()
    P = oracle.param_count(1, True, 4, 4, 7)
    params = torch.from_numpy(synth.draw_params(np.random.default_rng(3), P).astype(np.float64))
    train_ids = np.arange(ds.n)
    for e in range(epochs):
        portion = train.data_portions(train_ids, world, seed=11, epoch=e)[rank]

        def train_portion(ids):
            return torch.from_numpy(oracle_train_portion(ds, params.numpy(), ids, e))

        def average(v, prev, k):
            # eq. 3 from the summed parameters: the mean is sum / k
            v.copy_(torch.from_numpy(oracle.average_models([v.numpy() / k], prev.numpy(), BETA)))

        params = train.data_parallel_epoch(params, portion, train_portion,
                                           lambda t: dist.all_reduce(t, op=dist.ReduceOp.SUM), average, world)
    np.save(os.path.join(out_dir, f"rank{rank}.npy"), params.numpy())
    dist.destroy_process_group()


def free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def test_data_portions():
    ids = np.arange(100, 203)
    a = train.data_portions(ids, 4, seed=3, epoch=0)
    b = train.data_portions(ids, 4, seed=3, epoch=1)
    assert len(a) == 4 and sorted(np.concatenate(a).tolist()) == ids.tolist()
    assert max(p.size for p in a) - min(p.size for p in a) <= 1
    assert any(not np.array_equal(x, y) for x, y in zip(a, b))  # reshuffled between epochs
    for x, y in zip(a, train.data_portions(ids, 4, seed=3, epoch=0)):
        assert np.array_equal(x, y)  # reproducible


def test_two_replicas_average_by_eq3(tmp_path):
    import torch.multiprocessing as mp
    binding.lib()   # the planner the replicas use is the library's (host code)
    epochs, world = 2, 2
    ctx = mp.get_context("spawn")
    port = free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, epochs, str(tmp_path))) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=300)
        assert p.exitcode == 0
    got = [np.load(tmp_path / f"rank{r}.npy") for r in range(world)]
    assert np.array_equal(got[0], got[1])   # every replica ends with the same model
    # the same loop written out in one process
    ds = tiny_dataset()
    P = oracle.param_count(1, True, 4, 4, 7)
    v = synth.draw_params(np.random.default_rng(3), P).astype(np.float64)
    for e in range(epochs):
        portions = train.data_portions(np.arange(ds.n), world, seed=11, epoch=e)
        models = [oracle_train_portion(ds, v, portions[r], e) for r in range(world)]
        v = oracle.average_models(models, v, BETA)
    np.testing.assert_allclose(got[0], v, rtol=1e-12, atol=1e-14)
    # and the models really moved and really were averaged
    assert not np.allclose(v, synth.draw_params(np.random.default_rng(3), P))
