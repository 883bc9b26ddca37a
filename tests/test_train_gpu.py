"""GPU parity of the multi-epoch training driver: two epochs of bucketed
training with ADADELTA (Section III.B steps 3-4) through the library against
the same loop written with the oracle (plan, step, ADADELTA)."""
import numpy as np
import pytest

import oracle
from paper_1708_05604_gb300 import binding, synth, train

pytestmark = pytest.mark.gpu


def oracle_training(workload, Q, epochs, seed, batch_order, n_seqs=None, max_len=None):
    w = synth.WORKLOADS[workload]
    cfg = w.model_cfg()
    ds = synth.make_workload(w, seed=seed, n_seqs=n_seqs, max_len=max_len)
    tr, va = train.split_validation(ds.n, 0.05, seed + 17)
    P = oracle.param_count(cfg["n_layers"], cfg["bidirectional"], cfg["in_dim"], cfg["hidden"],
                           cfg["n_classes"])
    p = synth.draw_params(np.random.default_rng(seed + 1), P).astype(np.float64)
    eg2, edx2 = np.zeros(P), np.zeros(P)
    rho, eps = float(np.float32(0.95)), float(np.float32(1e-6))
    losses = []
    for e in range(epochs):
        plan = oracle.plan(ds.lengths[tr], Q, w.batch, seed=seed, epoch=e, batch_order=batch_order)
        tot, cnt = 0.0, 0
        for k in range(plan["n_batches"]):
            ids = tr[plan["order"][plan["batch_off"][k]:plan["batch_off"][k + 1]]]
            sub = ds.subset(ids)
            loss, g = oracle.lstm_ctc_step(cfg, sub.lengths, sub.x.astype(np.float64),
                                           sub.label_lengths, sub.labels, p)
            p, eg2, edx2 = oracle.adadelta(p, g, eg2, edx2, rho, eps, 1.0)
            tot += float(loss.sum())
            cnt += ids.size
        losses.append(tot / cnt)
    return p, losses


@pytest.mark.parametrize("order", ["ascending", "shuffle_batches"])
def test_two_epochs_adadelta_match_the_oracle(cuda_device, order):
    wl, Q, seed = "lstm1_uni_h32", 2, 0
    rec = train.train(wl, Q, 2, optimizer="adadelta", batch_order=order, seed=seed)
    p_o, losses_o = oracle_training(wl, Q, 2, seed, order)
    p0 = synth.draw_params(np.random.default_rng(seed + 1), p_o.size).astype(np.float64)
    p_g = rec["params"].astype(np.float64)
    # the accumulated update agrees to 1e-3 relative (about ten ADADELTA steps,
    # each a smooth map of fp32 gradients that match to 1e-4)
    d_o, d_g = p_o - p0, p_g - p0
    assert np.linalg.norm(d_g - d_o) / np.linalg.norm(d_o) < 1e-3
    for e, r in enumerate(rec["epochs"]):
        assert abs(r["train_loss"] - losses_o[e]) <= 1e-4 * abs(losses_o[e])
        assert np.isfinite(r["val_loss"])
    # training lowers the held-out loss on this data
    assert rec["epochs"][-1]["val_loss"] < rec["val_loss_initial"]
