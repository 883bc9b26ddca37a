"""Pins for the oracle's training step: torch's CPU LSTM + Linear +
log-softmax + ctc_loss with autograd (an independent implementation of the
same definitions, gate order i, f, g, o, bias_hh = 0), fp64 central finite
differences, per-sequence additivity and the no-alignment rule."""
import math

import numpy as np
import pytest
import torch

import oracle
from paper_1708_05604_gb300 import synth


def torch_step(cfg, ds, params):
    """Loss and gradient from torch modules, one sequence at a time."""
    L, H, C = cfg["n_layers"], cfg["hidden"], cfg["n_classes"]
    bi = cfg["bidirectional"]
    dirs = 2 if bi else 1
    lstm = torch.nn.LSTM(cfg["in_dim"], H, num_layers=L, bidirectional=bi,
                         dtype=torch.float64)
    out = torch.nn.Linear(dirs * H, C, dtype=torch.float64)
    p = torch.tensor(np.asarray(params, np.float64))
    off = 0
    names = []
    with torch.no_grad():
        for layer in range(L):
            D = cfg["in_dim"] if layer == 0 else dirs * H
            for d in range(dirs):
                sfx = f"_l{layer}" + ("_reverse" if d else "")
                for nm, shape in (("weight_ih", (4 * H, D)), ("weight_hh", (4 * H, H)),
                                  ("bias_ih", (4 * H,))):
                    n = int(np.prod(shape))
                    getattr(lstm, nm + sfx).copy_(p[off:off + n].reshape(shape))
                    names.append((getattr(lstm, nm + sfx), off, n))
                    off += n
                getattr(lstm, "bias_hh" + sfx).zero_()
                getattr(lstm, "bias_hh" + sfx).requires_grad_(False)
        n = C * dirs * H
        out.weight.copy_(p[off:off + n].reshape(C, dirs * H))
        names.append((out.weight, off, n))
        off += n
        out.bias.copy_(p[off:off + C])
        names.append((out.bias, off, C))
        off += C
    assert off == p.numel()
    total = 0.0
    losses = []
    for i in range(ds.n):
        x = torch.tensor(ds.seq_x(i), dtype=torch.float64)[:, None, :]
        y, _ = lstm(x)
        lp = torch.log_softmax(out(y[:, 0, :]), dim=1)
        lab = torch.tensor(ds.seq_labels(i), dtype=torch.long)[None, :]
        li = torch.nn.functional.ctc_loss(
            lp[:, None, :], lab, torch.tensor([int(ds.lengths[i])]),
            torch.tensor([int(ds.label_lengths[i])]), blank=cfg["blank"],
            reduction="sum", zero_infinity=True)
        losses.append(float(li.detach()))
        total = total + li
    total.backward()
    g = np.zeros(p.numel())
    for prm, o, n in names:
        g[o:o + n] = prm.grad.detach().numpy().reshape(-1)
    return np.array(losses), g


def small_cfg(layers, bi, H, C=7):
    return {"n_layers": layers, "bidirectional": bi, "in_dim": 4, "hidden": H,
            "n_classes": C, "blank": 0}


@pytest.mark.parametrize("layers,bi,H,C", [(1, False, 5, 7), (1, True, 4, 7), (2, True, 3, 7),
                                           (3, False, 4, 7), (2, False, 6, 7),
                                           # the benchmarked architecture (3 bidirectional
                                           # layers, 81 classes) at a tiny H
                                           (3, True, 4, 81)])
def test_step_matches_torch(layers, bi, H, C):
    cfg = small_cfg(layers, bi, H, C)
    rng = np.random.default_rng(layers * 10 + H + bi)
    ds = synth.make_dataset([9, 4, 13, 7, 1], 3, rng, n_classes=cfg["n_classes"])
    P = oracle.param_count(layers, bi, 4, H, cfg["n_classes"])
    params = rng.uniform(-0.5, 0.5, size=P)
    loss, g = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths,
                                   ds.labels, params)
    tl, tg = torch_step(cfg, ds, params)
    np.testing.assert_allclose(loss, tl, rtol=1e-11)
    np.testing.assert_allclose(g, tg, rtol=1e-9, atol=1e-12)


def test_step_repeat_labels_and_no_alignment():
    cfg = small_cfg(1, True, 4)
    rng = np.random.default_rng(5)
    ds = synth.make_dataset([6, 6, 3], 2, rng, n_classes=cfg["n_classes"])
    # sequence 1: labels with a repeat that still fits; sequence 2: cannot fit
    ds.labels[ds.lab_off[1]:ds.lab_off[2]] = [3, 3, 4]
    ds.labels[ds.lab_off[2]:ds.lab_off[3]] = [2]
    ds2 = synth.make_dataset([3], 1, rng, n_classes=cfg["n_classes"])
    ds2.labels[:] = [5]
    P = oracle.param_count(1, True, 4, 4, cfg["n_classes"])
    params = rng.uniform(-0.5, 0.5, size=P)
    loss, g = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths,
                                   ds.labels, params)
    tl, tg = torch_step(cfg, ds, params)
    np.testing.assert_allclose(loss[:2], tl[:2], rtol=1e-11)
    np.testing.assert_allclose(g, tg, rtol=1e-9, atol=1e-12)
    # a 3-step sequence whose 3 labels are 2, 2, 2 has no alignment
    bad = synth.make_dataset([3], 1, rng, n_classes=cfg["n_classes"])
    bad = synth.Dataset(bad.lengths, bad.x, bad.x_off, np.array([3], np.int32),
                        np.array([2, 2, 2], np.int32), np.array([0, 3], np.int64))
    lb, gb = oracle.lstm_ctc_step(cfg, bad.lengths, bad.x, bad.label_lengths,
                                  bad.labels, params)
    assert math.isinf(lb[0]) and lb[0] > 0 and np.all(gb == 0)


def test_step_finite_differences():
    cfg = small_cfg(2, True, 3, C=5)
    rng = np.random.default_rng(9)
    ds = synth.make_dataset([5, 7], 3, rng, n_classes=cfg["n_classes"])
    P = oracle.param_count(2, True, 4, 3, 5)
    params = rng.uniform(-0.6, 0.6, size=P)
    _, g = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths, ds.labels, params)
    h = 1e-6
    for j in rng.choice(P, size=60, replace=False):
        pp, pm = params.copy(), params.copy()
        pp[j] += h
        pm[j] -= h
        lp = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths, ds.labels, pp)[0].sum()
        lm = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths, ds.labels, pm)[0].sum()
        assert (lp - lm) / (2 * h) == pytest.approx(g[j], abs=2e-7, rel=1e-5)


def test_step_is_a_sum_over_sequences_and_order_free():
    """Padding invariance, oracle side: each sequence's loss and gradient
    depend on that sequence alone, whatever its batch-mates and order."""
    cfg = small_cfg(1, True, 6, C=11)
    rng = np.random.default_rng(2)
    ds = synth.make_dataset([12, 3, 30, 8, 17, 5], 4, rng, n_classes=11)
    P = oracle.param_count(1, True, 4, 6, 11)
    params = rng.uniform(-0.3, 0.3, size=P)
    loss, g = oracle.lstm_ctc_step(cfg, ds.lengths, ds.x, ds.label_lengths, ds.labels, params)
    perm = np.array([4, 0, 5, 2, 1, 3])
    sub = ds.subset(perm)
    loss_p, g_p = oracle.lstm_ctc_step(cfg, sub.lengths, sub.x, sub.label_lengths,
                                       sub.labels, params)
    np.testing.assert_allclose(loss_p, loss[perm], rtol=0, atol=0)
    np.testing.assert_allclose(g_p, g, rtol=1e-12, atol=1e-14)
    acc = np.zeros(P)
    for i in range(ds.n):
        one = ds.subset([i])
        li, gi = oracle.lstm_ctc_step(cfg, one.lengths, one.x, one.label_lengths,
                                      one.labels, params)
        assert li[0] == loss[i]
        acc += gi
    np.testing.assert_allclose(acc, g, rtol=1e-12, atol=1e-14)


def test_sgd():
    p = np.array([1.0, -2.0, 3.0])
    g = np.array([0.5, 0.25, -1.0])
    np.testing.assert_array_equal(oracle.sgd(p, g, 0.1), p - 0.1 * g)


def test_param_count_layout():
    assert oracle.param_count(1, False, 4, 32, 81) == 7409
    assert oracle.param_count(3, True, 4, 256, 81) == 3725905
    assert oracle.param_count(2, False, 4, 512, 81) == 3199569
