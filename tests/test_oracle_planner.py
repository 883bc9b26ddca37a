"""Pins for the oracle's planner (Section III.A): brute force over every
boundary tuple, a hand-worked instance, invariants of the objective, and the
plan's structural properties."""
import itertools
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def brute_force(lengths, Q):
    """Every tuple b_1 < ... < b_{Q-1} < lmax, cost per eq. 2 (each sequence
    charged its bucket's upper bound).  Among minimisers, the tuple largest
    when read from b_{Q-1} down to b_1 (the DP's tie rule)."""
    L = np.asarray(lengths)
    lmax = int(L.max())
    best = None
    for cut in itertools.combinations(range(1, lmax), Q - 1):
        bounds = list(cut) + [lmax]
        cost, lo = 0, 0
        for b in bounds:
            cost += b * int(np.sum((L > lo) & (L <= b)))
            lo = b
        key = (cost, tuple(-v for v in reversed(bounds[:-1])))
        if best is None or key < best[0]:
            best = (key, bounds)
    return best[1], best[0][0]


def test_hand_worked_example():
    rows = open(os.path.join(GOLDEN, "dp_worked_example.txt")).read().splitlines()
    rows = [r for r in rows if r and not r.startswith("#")]
    lengths = [int(v) for v in rows[0].split(":")[1].split()]
    f = oracle.histogram(lengths)
    assert f.tolist() == [0, 2, 1, 0, 0, 3, 1, 0, 0, 0, 1]
    for r in rows[1:]:
        parts = r.split()
        Q = int(parts[0][2:])
        if parts[1] == "infeasible":
            with pytest.raises(oracle.OracleError):
                oracle.dynamic_bucketing(f, Q)
            continue
        cost = int(parts[1].split("=")[1])
        bounds = [int(v) for v in parts[2].split("=")[1].split(",")]
        b, c = oracle.dynamic_bucketing(f, Q)
        assert c == cost, (Q, c, cost)
        assert b.tolist() == bounds, (Q, b, bounds)


@pytest.mark.parametrize("seed", range(40))
def test_dp_matches_brute_force(seed):
    rng = np.random.default_rng(1000 + seed)
    lmax = int(rng.integers(2, 13))
    n = int(rng.integers(1, 25))
    L = rng.integers(1, lmax + 1, size=n)
    L[0] = lmax  # make lmax the true maximum
    for Q in range(1, min(4, int(L.max())) + 1):
        b, c = oracle.dynamic_bucketing(oracle.histogram(L), Q)
        bb, cc = brute_force(L, Q)
        assert c == cc and b.tolist() == bb, (L.tolist(), Q, b, c, bb, cc)


@pytest.mark.parametrize("seed", range(10))
def test_dp_invariants(seed):
    rng = np.random.default_rng(seed)
    L = rng.integers(20, 300, size=200).astype(np.int32)
    f = oracle.histogram(L)
    lmax = int(L.max())
    _, c1 = oracle.dynamic_bucketing(f, 1)
    assert c1 == L.size * lmax
    prev = c1
    for Q in (2, 3, 4, 6, 8, 16):
        b, c = oracle.dynamic_bucketing(f, Q)
        assert c <= prev
        assert b[-1] == lmax and np.all(np.diff(b) > 0) and b[0] >= 1
        # the cost equals eq. 2 evaluated at the returned bounds
        lo, cost = 0, 0
        for ub in b:
            cost += int(ub) * int(np.sum((L > lo) & (L <= ub)))
            lo = ub
        assert cost == c
        prev = c
    distinct = np.unique(L).size
    _, cd = oracle.dynamic_bucketing(f, distinct)
    assert cd == int(L.sum())
    # permutation invariance of the whole plan's bounds
    perm = rng.permutation(L.size)
    assert oracle.dynamic_bucketing(oracle.histogram(L[perm]), 5)[0].tolist() == \
        oracle.dynamic_bucketing(f, 5)[0].tolist()


def test_dp_infeasible_and_bad_input():
    with pytest.raises(oracle.OracleError):
        oracle.dynamic_bucketing(oracle.histogram([1, 2, 3]), 4)
    with pytest.raises(oracle.OracleError):
        oracle.histogram([1, 0, 3])


def test_splitmix64_published_stream():
    vals = [int(v, 16) for v in open(os.path.join(GOLDEN, "splitmix64_seed0.txt"))
            .read().split() if v.startswith("0x")]
    assert oracle.splitmix64_stream(0, 4) == vals


def _check_plan(p, L, Q, B):
    n = L.size
    order = p["order"]
    assert sorted(order.tolist()) == list(range(n))
    bounds = p["bounds"]
    lo_of = np.concatenate([[0], bounds[:-1]])
    boff, bb = p["batch_off"], p["batch_bucket"]
    assert boff[0] == 0 and boff[-1] == n
    assert np.all(np.diff(bb) >= 0), "buckets must be emitted shortest first"
    padded = 0
    for k in range(p["n_batches"]):
        ids = order[boff[k]:boff[k + 1]]
        q = bb[k]
        assert 1 <= ids.size <= B
        assert np.all((L[ids] > lo_of[q]) & (L[ids] <= bounds[q]))
        if k + 1 < p["n_batches"] and bb[k + 1] == q:
            assert ids.size == B, "only a bucket's last batch may be partial"
        padded += ids.size * int(L[ids].max())
    assert padded == p["padded_timesteps"]
    # every bucket's members are exactly the sequences within its bounds
    for q in range(Q):
        members = np.concatenate([order[boff[k]:boff[k + 1]]
                                  for k in range(p["n_batches"]) if bb[k] == q]
                                 + [np.zeros(0, np.int32)])
        expect = np.nonzero((L > lo_of[q]) & (L <= bounds[q]))[0]
        assert sorted(members.tolist()) == expect.tolist()


@pytest.mark.parametrize("Q,B", [(1, 16), (2, 16), (4, 7), (8, 64), (3, 1)])
def test_plan_structure(Q, B):
    rng = np.random.default_rng(7)
    L = rng.integers(20, 201, size=300).astype(np.int32)
    p = oracle.plan(L, Q, B, seed=0, epoch=0)
    _check_plan(p, L, Q, B)
    # reproducible, and the epoch reshuffles
    p2 = oracle.plan(L, Q, B, seed=0, epoch=0)
    assert np.array_equal(p["order"], p2["order"])
    p3 = oracle.plan(L, Q, B, seed=0, epoch=1)
    assert np.array_equal(p["bounds"], p3["bounds"])
    assert not np.array_equal(p["order"], p3["order"])
    _check_plan(p3, L, Q, B)


def test_plan_shuffle_is_uniform_enough():
    """Fisher-Yates on a single bucket: every element visits every slot."""
    L = np.full(6, 5, dtype=np.int32)
    counts = np.zeros((6, 6))
    for e in range(3000):
        o = oracle.plan(L, 1, 6, seed=123, epoch=e)["order"]
        counts[np.arange(6), o] += 1
    assert counts.min() > 3000 / 6 * 0.8 and counts.max() < 3000 / 6 * 1.2


def test_plan_empty_bucket_and_q_equals_lmax():
    L = np.array([1, 1, 2, 5, 5, 5, 6, 10], dtype=np.int32)
    p = oracle.plan(L, 6, 2, seed=3, epoch=0)
    assert p["bounds"].tolist() == [1, 2, 5, 6, 9, 10]
    assert 4 not in p["batch_bucket"].tolist()   # bucket (6, 9] is empty
    _check_plan(p, L, 6, 2)
    p = oracle.plan(L, 10, 3, seed=3, epoch=0)
    _check_plan(p, L, 10, 3)
    with pytest.raises(oracle.OracleError):
        oracle.plan(L, 11, 3, seed=3, epoch=0)
