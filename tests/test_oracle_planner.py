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


# ---------------------------------------------------------------------------
# Batch-order variants (bucket-ordering strategies, Section V future work).

def _batches(p):
    o, off = p["order"], p["batch_off"]
    return [tuple(o[off[k]:off[k + 1]].tolist()) for k in range(p["n_batches"])]


ORDERS = ["descending", "shuffle_buckets", "shuffle_batches"]


@pytest.mark.parametrize("mode", ORDERS)
@pytest.mark.parametrize("Q,B", [(1, 16), (4, 7), (8, 64), (3, 1)])
def test_ordered_plan_permutes_whole_batches(mode, Q, B):
    """Every order emits exactly the ascending plan's batches (same members,
    same internal order), with the same bounds, dp cost and padding."""
    rng = np.random.default_rng(11)
    L = rng.integers(20, 201, size=300).astype(np.int32)
    a = oracle.plan(L, Q, B, seed=5, epoch=2)
    p = oracle.plan(L, Q, B, seed=5, epoch=2, batch_order=mode)
    assert np.array_equal(a["bounds"], p["bounds"])
    assert a["dp_cost"] == p["dp_cost"] and a["padded_timesteps"] == p["padded_timesteps"]
    assert a["n_batches"] == p["n_batches"]
    ba, bp = _batches(a), _batches(p)
    assert sorted(ba) == sorted(bp)
    bucket_of = {b: q for b, q in zip(ba, a["batch_bucket"].tolist())}
    assert [bucket_of[b] for b in bp] == p["batch_bucket"].tolist()
    if mode != "shuffle_batches":
        # buckets stay together, each bucket's batches in cut order
        seq = p["batch_bucket"].tolist()
        runs = [q for i, q in enumerate(seq) if i == 0 or seq[i - 1] != q]
        assert len(runs) == len(set(runs))
        for q in set(seq):
            assert [b for b in bp if bucket_of[b] == q] == [b for b in ba if bucket_of[b] == q]
        if mode == "descending":
            assert runs == sorted(runs, reverse=True)


def test_ordered_plan_ascending_is_the_plain_plan():
    L = np.random.default_rng(3).integers(1, 60, size=200).astype(np.int32)
    for e in range(3):
        a = oracle.plan(L, 5, 9, seed=1, epoch=e)
        b = oracle.plan(L, 5, 9, seed=1, epoch=e, batch_order="ascending")
        assert _batches(a) == _batches(b)


def test_shuffle_batches_is_fisher_yates_on_the_continued_stream():
    """Definition check: after the in-bucket shuffles (sum over buckets of
    m_q - 1 draws), the same SplitMix64 stream permutes the list of batches
    with Fisher-Yates, k = n_batches-1 .. 1, j = next() mod (k+1)."""
    L = np.random.default_rng(4).integers(1, 50, size=150).astype(np.int32)
    Q, B, seed, epoch = 4, 6, 9, 1
    a = oracle.plan(L, Q, B, seed=seed, epoch=epoch)
    p = oracle.plan(L, Q, B, seed=seed, epoch=epoch, batch_order="shuffle_batches")
    sizes = np.bincount(a["batch_bucket"], weights=np.diff(a["batch_off"]), minlength=Q)
    used = int(sum(max(int(m) - 1, 0) for m in sizes))
    nb = a["n_batches"]
    state0 = (seed + (epoch + 1) * 0x9E3779B97F4A7C15) % (1 << 64)
    draws = oracle.splitmix64_stream(state0, used + nb)[used:]
    seq = list(range(nb))
    for i, k in enumerate(range(nb - 1, 0, -1)):
        j = draws[i] % (k + 1)
        seq[k], seq[j] = seq[j], seq[k]
    ba = _batches(a)
    assert _batches(p) == [ba[s] for s in seq]


@pytest.mark.parametrize("mode", ["shuffle_buckets", "shuffle_batches"])
def test_order_shuffles_are_uniform_enough(mode):
    """Over many epochs each bucket (batch) takes every position about equally
    often, and the order changes with the epoch."""
    L = np.repeat(np.arange(1, 5, dtype=np.int32), 3)   # 4 buckets of 3 equal lengths
    Q, B = 4, 3                                          # one batch per bucket
    counts = np.zeros((4, 4))
    for e in range(2000):
        p = oracle.plan(L, Q, B, seed=77, epoch=e, batch_order=mode)
        for pos, q in enumerate(p["batch_bucket"].tolist()):
            counts[q, pos] += 1
    assert counts.min() > 2000 / 4 * 0.8 and counts.max() < 2000 / 4 * 1.2


def test_ordered_plan_rejects_unknown_order():
    with pytest.raises(KeyError):
        oracle.plan(np.array([1, 2, 3], np.int32), 2, 2, seed=0, batch_order="zigzag")
