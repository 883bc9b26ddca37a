"""Training checkpoints and the per-epoch JSON-lines log (host side, no GPU):
round trip, refusal of damaged or foreign checkpoints, the resume point, and
that the epochs after a resume draw the mini-batches an uninterrupted run
draws (Section III.B step 3: the plan is rebuilt every epoch from the seed)."""
import json

import numpy as np
import pytest

from paper_1708_05604_gb300 import checkpoint, synth, train


def _arrays(seed=0, n=1000):
    r = np.random.default_rng(seed)
    return {"params": r.standard_normal(n).astype(np.float32),
            "eg2": r.random(n).astype(np.float32), "edx2": r.random(n).astype(np.float32)}


def test_round_trip(tmp_path):
    p = str(tmp_path / "ck")
    a = _arrays()
    meta = {"workload": "lstm1_uni_h32", "epoch_next": 3, "epochs": [{"epoch": 0, "train_loss": 1.5}]}
    checkpoint.save(p, a, meta)
    m, b = checkpoint.load(p)
    assert m == meta
    assert list(b) == ["params", "eg2", "edx2"]
    for k in a:
        assert b[k].dtype == np.float32 and np.array_equal(b[k], a[k])
    # a second save replaces the first
    a2 = _arrays(1)
    checkpoint.save(p, a2, {**meta, "epoch_next": 4})
    m, b = checkpoint.load(p)
    assert m["epoch_next"] == 4 and np.array_equal(b["params"], a2["params"])
    assert not list(tmp_path.glob("*.tmp.*"))


def test_damaged_or_foreign_records_are_refused(tmp_path):
    p = str(tmp_path / "ck")
    checkpoint.save(p, _arrays(), {"epoch_next": 1})
    blob = bytearray(open(p + ".bin", "rb").read())
    blob[100] ^= 1
    open(p + ".bin", "wb").write(bytes(blob))
    with pytest.raises(ValueError, match="SHA-256"):
        checkpoint.load(p)
    open(p + ".bin", "wb").write(bytes(blob[:-4]))
    with pytest.raises(ValueError, match="bytes"):
        checkpoint.load(p)
    rec = json.load(open(p + ".json"))
    rec["format"] = "something-else"
    json.dump(rec, open(p + ".json", "w"))
    with pytest.raises(ValueError, match="not a"):
        checkpoint.load(p)
    with pytest.raises(FileNotFoundError):
        checkpoint.load(str(tmp_path / "missing"))


def test_resume_point_and_run_identity(tmp_path):
    ident = train.run_identity("lstm1_uni_h32", 2, "adadelta", "ascending", 0, 0.05, None, None, None, 1234)
    # the identity survives the JSON record unchanged, so a resumed run matches it
    p = str(tmp_path / "ck")
    recs = [{"epoch": 0, "train_loss": 9.0}, {"epoch": 1, "train_loss": 8.0}]
    checkpoint.save(p, _arrays(), {**ident, "epoch_next": 2, "epochs": recs, "wall_s": 1.25,
                                   "val_loss_initial": 10.0})
    meta, _ = checkpoint.load(p)
    start, done, wall, v0 = train.resume_point(meta, ident, 5)
    assert (start, done, wall, v0) == (2, recs, 1.25, 10.0)
    # another bucket count, seed or update rule is another run
    for k, v in [("n_buckets", 4), ("seed", 1), ("optimizer", "sgd"), ("batch_order", "shuffle_batches")]:
        with pytest.raises(ValueError, match=k):
            train.resume_point(meta, {**ident, k: v}, 5)
    # a checkpoint past the requested epoch count
    with pytest.raises(ValueError, match="after epoch"):
        train.resume_point(meta, ident, 1)
    assert train.resume_point(meta, ident, 2)[0] == 2   # nothing left to run


def test_resumed_epochs_draw_the_same_batches():
    w = synth.WORKLOADS["lstm1_bi_h128"]
    ds = synth.make_workload(w, seed=0)
    tr, _ = train.split_validation(ds.n, 0.05, 17)
    for order in ["ascending", "shuffle_batches"]:
        straight = [train.epoch_batches(ds.lengths, tr, 4, w.batch, 0, e, order)[0] for e in range(4)]
        resumed = [train.epoch_batches(ds.lengths, tr, 4, w.batch, 0, e, order)[0] for e in (2, 3)]
        for a, b in zip(straight[2:], resumed):
            assert len(a) == len(b) and all(np.array_equal(x, y) for x, y in zip(a, b))
        # and the epochs differ from one another (the plan is reshuffled every epoch)
        assert any(not np.array_equal(x, y) for x, y in zip(straight[2], straight[3]))


def test_jsonl_log(tmp_path):
    f = tmp_path / "log.jsonl"
    log = checkpoint.JsonlLog(str(f), workload="w", n_buckets=4)
    log({"epoch": 0, "train_loss": 1.0})
    log({"epoch": 1, "train_loss": 0.5, "kernel_ms": {"lstm_fwd": 1.25}})
    lines = [json.loads(x) for x in open(f)]
    assert lines == [{"workload": "w", "n_buckets": 4, "epoch": 0, "train_loss": 1.0},
                     {"workload": "w", "n_buckets": 4, "epoch": 1, "train_loss": 0.5,
                      "kernel_ms": {"lstm_fwd": 1.25}}]


def test_resume_takes_one_bucket_count():
    with pytest.raises(SystemExit):
        train.main(["--buckets", "1,2", "--resume", "/nonexistent/ck"])


class _FakeEvent:
    def __init__(self, enable_timing=False):
        pass

    def record(self, stream=None):
        pass

    def elapsed_time(self, other):
        return 2.0


def _fake_gpu(monkeypatch):
    """The training driver's library and CUDA calls replaced by deterministic
    CPU stand-ins: the step's gradient depends on the parameters and the
    batch, the update on the optimizer state, so a resume that dropped or
    misplaced any of them would change the result."""
    import torch

    from paper_1708_05604_gb300 import binding, build

    class Ctx:
        def __init__(self, *a):
            pass

        def step(self, dd, ids, params, grads, loss, stream=None):
            s = float(np.sum(ids % 13)) / 13.0
            grads.copy_(0.01 * params + s * torch.cos(torch.arange(params.numel(), dtype=params.dtype)))
            loss.fill_(s + float(params[:7].sum()))

        def sync_status(self):
            pass

        def set_timing(self, on):
            pass

        def kernel_stats(self):
            return [{"name": "lstm_fwd", "total_ms": 1.5}]

    class Adadelta:
        def __init__(self, params, rho=0.95, eps=1e-6, lr=1.0):
            self.params = params
            self.eg2, self.edx2 = torch.zeros_like(params), torch.zeros_like(params)

        def step(self, grads, stream=None):
            self.eg2.mul_(0.9).add_(0.1 * grads * grads)
            dx = grads / torch.sqrt(self.eg2 + 1e-3) * torch.sqrt(self.edx2 + 1e-3)
            self.edx2.mul_(0.9).add_(0.1 * dx * dx)
            self.params.sub_(dx)

    monkeypatch.setattr(build, "build", lambda *a, **k: None)
    monkeypatch.setattr(binding, "Ctx", Ctx)
    monkeypatch.setattr(binding, "Adadelta", Adadelta)
    monkeypatch.setattr(binding, "DeviceDataset", lambda ds, device=None: None)
    monkeypatch.setattr(torch.cuda, "synchronize", lambda *a, **k: None)
    monkeypatch.setattr(torch.cuda, "current_stream", lambda *a, **k: None)
    monkeypatch.setattr(torch.cuda, "Event", _FakeEvent)


def test_training_resumed_from_a_checkpoint_matches_an_uninterrupted_run(tmp_path, monkeypatch):
    _fake_gpu(monkeypatch)
    kw = dict(workload="lstm1_uni_h32", n_buckets=2, optimizer="adadelta", seed=3, device="cpu")
    straight = train.train(epochs=3, **kw)
    p = str(tmp_path / "ck")
    logged = []
    first = train.train(epochs=2, checkpoint_path=p, log=logged.append, **kw)
    meta, arrays = checkpoint.load(p)
    assert meta["epoch_next"] == 2 and set(arrays) == {"params", "eg2", "edx2"}
    assert np.array_equal(arrays["params"], first["params"])
    resumed = train.train(epochs=3, resume=p, checkpoint_path=p, log=logged.append, kernel_times=True, **kw)
    assert resumed["resumed_at_epoch"] == 2
    assert np.array_equal(resumed["params"], straight["params"])
    keys = ["epoch", "train_loss", "val_loss", "n_batches", "timesteps", "padded_efficiency"]
    assert [[r[k] for k in keys] for r in resumed["epochs"]] == [[r[k] for k in keys] for r in straight["epochs"]]
    assert resumed["val_loss_initial"] == straight["val_loss_initial"]
    assert [r["epoch"] for r in logged] == [0, 1, 2] and logged[-1]["kernel_ms"] == {"lstm_fwd": 1.5}
    assert logged[0]["timesteps_per_s"] == pytest.approx(logged[0]["timesteps"] / 2e-3)
    # the checkpoint now records the third epoch too
    assert checkpoint.load(p)[0]["epoch_next"] == 3
    # a different run refuses it
    with pytest.raises(ValueError, match="n_buckets"):
        train.train(epochs=4, resume=p, **{**kw, "n_buckets": 3})
