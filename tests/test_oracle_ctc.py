"""Pins for the oracle's CTC (the paper's ref. [15], Graves et al. 2006):
brute-force sums over every path, closed forms, torch's CPU ctc_loss, and
finite differences."""
import itertools
import math

import numpy as np
import pytest
import torch

import oracle


def log_softmax(z):
    z = z - z.max(axis=1, keepdims=True)
    return z - np.log(np.exp(z).sum(axis=1, keepdims=True))


def collapse(path, blank=0):
    out, prev = [], None
    for k in path:
        if k != prev and k != blank:
            out.append(k)
        prev = k
    return out


def brute(logits, labels, blank=0):
    """p and d(-ln p)/d logits by enumerating all K^T paths."""
    T, K = logits.shape
    y = np.exp(log_softmax(logits))
    p = 0.0
    post = np.zeros((T, K))
    for path in itertools.product(range(K), repeat=T):
        if collapse(path, blank) == list(labels):
            pr = float(np.prod([y[t, k] for t, k in enumerate(path)]))
            p += pr
            for t, k in enumerate(path):
                post[t, k] += pr
    grad = y - post / p if p > 0 else np.zeros_like(y)
    return p, grad


CASES = [
    (4, 3, [1]), (5, 3, [1, 2]), (5, 3, [1, 1]), (6, 3, [2, 1, 2]),
    (6, 3, [1, 1, 2]), (3, 2, [1, 1]), (6, 3, []), (2, 3, [1, 2]),
    (5, 3, [2, 2, 2]),
]


@pytest.mark.parametrize("T,K,labels", CASES)
def test_ctc_matches_brute_force(T, K, labels):
    rng = np.random.default_rng(T * 31 + K + len(labels))
    logits = rng.normal(size=(T, K)) * 1.5
    p, g = brute(logits, labels)
    loss, go = oracle.ctc(log_softmax(logits), labels)
    if p == 0:
        assert math.isinf(loss) and np.all(go == 0)
    else:
        assert loss == pytest.approx(-math.log(p), rel=1e-12, abs=1e-12)
        np.testing.assert_allclose(go, g, rtol=1e-10, atol=1e-12)


def test_ctc_blank_only_closed_form():
    rng = np.random.default_rng(3)
    lp = log_softmax(rng.normal(size=(9, 5)))
    loss, g = oracle.ctc(lp, [])
    assert loss == pytest.approx(-lp[:, 0].sum(), rel=1e-13)
    expect = np.exp(lp)
    expect[:, 0] -= 1.0
    np.testing.assert_allclose(g, expect, atol=1e-13)


@pytest.mark.parametrize("T,K", [(1, 4), (3, 2), (7, 5), (12, 81)])
def test_ctc_uniform_single_label_closed_form(T, K):
    """Uniform outputs, label 'a': the alignments are blank* a+ blank*, so
    there are T(T+1)/2 of them and p = T(T+1)/2 / K^T."""
    lp = np.full((T, K), -math.log(K))
    loss, _ = oracle.ctc(lp, [1])
    assert loss == pytest.approx(T * math.log(K) - math.log(T * (T + 1) / 2), rel=1e-12)


def test_ctc_infeasible():
    lp = log_softmax(np.zeros((3, 4)))
    loss, g = oracle.ctc(lp, [1, 1, 2])   # needs 4 steps (a blank between the 1s)
    assert math.isinf(loss) and loss > 0 and np.all(g == 0)
    loss, _ = oracle.ctc(lp, [1, 2, 3])   # needs exactly 3
    assert math.isfinite(loss)


@pytest.mark.parametrize("seed", range(6))
def test_ctc_matches_torch(seed):
    rng = np.random.default_rng(seed)
    T = int(rng.integers(5, 60))
    C = 81
    U = int(rng.integers(0, T // 3 + 1))
    labels = rng.integers(1, C, size=U)
    if U >= 2 and seed % 2 == 0:
        labels[1] = labels[0]  # a repeat
    logits = torch.tensor(rng.normal(size=(T, C)) * 2.0, dtype=torch.float64,
                          requires_grad=True)
    lp = torch.log_softmax(logits, dim=1)
    tl = torch.nn.functional.ctc_loss(
        lp[:, None, :], torch.tensor(labels[None, :], dtype=torch.long),
        torch.tensor([T]), torch.tensor([U]), blank=0, reduction="sum")
    tl.backward()
    loss, g = oracle.ctc(lp.detach().numpy(), labels)
    assert loss == pytest.approx(float(tl.detach()), rel=1e-10)
    np.testing.assert_allclose(g, logits.grad.numpy(), rtol=1e-8, atol=1e-11)


def test_ctc_finite_differences():
    rng = np.random.default_rng(11)
    T, C = 8, 6
    labels = [2, 3, 3, 5]
    z = rng.normal(size=(T, C))
    _, g = oracle.ctc(log_softmax(z), labels)
    h = 1e-6
    for t in range(T):
        for k in range(C):
            zp, zm = z.copy(), z.copy()
            zp[t, k] += h
            zm[t, k] -= h
            fd = (oracle.ctc(log_softmax(zp), labels, grad=False)[0]
                  - oracle.ctc(log_softmax(zm), labels, grad=False)[0]) / (2 * h)
            assert fd == pytest.approx(g[t, k], abs=1e-7)
