"""Host-side checks of libbkt that need no GPU: the library loads and exports
every entry point include/bkt.h declares, the planner matches the oracle
bit for bit, and the parameter layout and argument checks hold."""
import ctypes
import os
import re

import numpy as np
import pytest

import oracle
from paper_1708_05604_gb300 import binding, synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_1708_05604_gb300 import build
    build.build()
    return binding.lib()


def header_functions():
    names = set()
    for fn in os.listdir(os.path.join(ROOT, "include")):
        if fn.endswith(".h"):
            txt = open(os.path.join(ROOT, "include", fn)).read()
            txt = re.sub(r"/\*.*?\*/", "", txt, flags=re.S)
            names |= set(re.findall(r"\b(bkt_\w+)\s*\(", txt))
    return sorted(names)


def test_exports_every_declared_symbol(lib):
    names = header_functions()
    assert len(names) >= 12
    for n in names:
        assert hasattr(lib, n), f"{n} declared in include/ but not exported"
    assert set(binding.EXPORTS) == set(names)


PLAN_CASES = [(w, Q) for w in synth.WORKLOAD_ORDER for Q in synth.WORKLOADS[w].bucket_counts]


@pytest.mark.parametrize("wname,Q", PLAN_CASES)
@pytest.mark.parametrize("seed", [0, 1, 2])
def test_planner_bit_exact_vs_oracle(lib, wname, Q, seed):
    w = synth.WORKLOADS[wname]
    rng = np.random.default_rng(seed)
    L = synth.draw_lengths(rng, w.n_seqs, w.length_dist)
    for epoch in (0, 3):
        a = binding.plan_buckets(L, Q, w.batch, seed=seed, epoch=epoch)
        b = oracle.plan(L, Q, w.batch, seed=seed, epoch=epoch)
        for k in ("bounds", "order", "batch_off", "batch_bucket"):
            assert np.array_equal(a[k], b[k]), (k, wname, Q, seed, epoch)
        assert a["dp_cost"] == b["dp_cost"]
        assert a["n_batches"] == b["n_batches"]
        assert a["padded_timesteps"] == b["padded_timesteps"]
        assert a["unpadded_timesteps"] == int(L.sum())


@pytest.mark.parametrize("mode", ["descending", "shuffle_buckets", "shuffle_batches"])
@pytest.mark.parametrize("wname,Q", PLAN_CASES[::2])
def test_ordered_planner_bit_exact_vs_oracle(lib, wname, Q, mode):
    w = synth.WORKLOADS[wname]
    L = synth.draw_lengths(np.random.default_rng(5), w.n_seqs, w.length_dist)
    for epoch in (0, 4):
        a = binding.plan_buckets(L, Q, w.batch, seed=5, epoch=epoch, batch_order=mode)
        b = oracle.plan(L, Q, w.batch, seed=5, epoch=epoch, batch_order=mode)
        for k in ("bounds", "order", "batch_off", "batch_bucket"):
            assert np.array_equal(a[k], b[k]), (k, wname, Q, mode, epoch)
        assert a["padded_timesteps"] == b["padded_timesteps"]


def test_ordered_planner_rejects_unknown_order(lib):
    L = np.array([1, 2, 3], np.int32)
    h = ctypes.c_void_p()
    rc = lib.bkt_plan_buckets_ordered(L.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)), 3, 2, 2,
                                      ctypes.c_uint64(0), ctypes.c_uint64(0), 7, ctypes.byref(h))
    assert rc == binding.BKT_EINVAL and not h.value


@pytest.mark.parametrize("seed", range(30))
def test_planner_small_random_vs_oracle(lib, seed):
    rng = np.random.default_rng(500 + seed)
    lmax = int(rng.integers(1, 40))
    n = int(rng.integers(1, 60))
    L = rng.integers(1, lmax + 1, size=n).astype(np.int32)
    for Q in range(1, min(int(L.max()), 8) + 1):
        B = int(rng.integers(1, 9))
        a = binding.plan_buckets(L, Q, B, seed=seed, epoch=seed % 3)
        b = oracle.plan(L, Q, B, seed=seed, epoch=seed % 3)
        for k in ("bounds", "order", "batch_off", "batch_bucket"):
            assert np.array_equal(a[k], b[k]), (k, L.tolist(), Q, B)
        assert a["dp_cost"] == b["dp_cost"]


def test_planner_rejects_bad_input(lib):
    with pytest.raises(binding.BktError) as e:
        binding.plan_buckets([3, 0, 2], 1, 2, 0)
    assert e.value.rc == binding.BKT_EINVAL
    with pytest.raises(binding.BktError):
        binding.plan_buckets([3, 1, 2], 4, 2, 0)   # Q > max length
    with pytest.raises(binding.BktError):
        binding.plan_buckets([3, 1, 2], 1, 0, 0)   # batch 0
    assert "buckets" in lib.bkt_last_error().decode()


def test_param_count_matches_oracle_layout(lib):
    for w in synth.WORKLOADS.values():
        cfg = w.model_cfg()
        assert binding.param_count(cfg) == oracle.param_count(
            cfg["n_layers"], cfg["bidirectional"], cfg["in_dim"], cfg["hidden"], cfg["n_classes"])
    bad = dict(synth.WORKLOADS["lstm1_uni_h32"].model_cfg(), blank=81)
    assert binding.param_count(bad) == 0


@pytest.mark.parametrize("seed", range(12))
def test_planner_tie_heavy_histograms_vs_oracle(lib, seed):
    """Histograms built to create equal-cost bound tuples (flat counts,
    repeated blocks, lengths in arithmetic steps), every Q up to the longest
    length: the library's bounds, cost and plan equal the oracle's."""
    rng = np.random.default_rng(900 + seed)
    kind = seed % 3
    if kind == 0:      # every length once: many tuples of equal cost
        L = np.arange(1, int(rng.integers(2, 60)) + 1, dtype=np.int32)
    elif kind == 1:    # a repeated block of counts
        block = rng.integers(1, 4, size=int(rng.integers(2, 6)))
        counts = np.tile(block, int(rng.integers(2, 12)))
        L = np.repeat(np.arange(1, counts.size + 1), counts).astype(np.int32)
    else:              # lengths on a coarse grid with equal counts
        step = int(rng.integers(2, 7))
        vals = np.arange(step, step * int(rng.integers(3, 25)) + 1, step)
        L = np.repeat(vals, int(rng.integers(1, 4))).astype(np.int32)
    rng.shuffle(L)
    lmax = int(L.max())
    for Q in sorted(set([1, 2, 3, lmax // 2, lmax - 1, lmax]) - {0}):
        if Q < 1 or Q > lmax:
            continue
        a = binding.plan_buckets(L, Q, 4, seed=seed, epoch=1)
        b = oracle.plan(L, Q, 4, seed=seed, epoch=1)
        assert np.array_equal(a["bounds"], b["bounds"]), (Q, a["bounds"], b["bounds"])
        assert a["dp_cost"] == b["dp_cost"]
        for k in ("order", "batch_off", "batch_bucket"):
            assert np.array_equal(a[k], b[k])
