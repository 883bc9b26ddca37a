"""Host logic of the multi-epoch training driver (no GPU): the validation
split, the per-epoch batches against the oracle's plan of the training
subset (bit for bit, every batch order), and the validation batches."""
import numpy as np
import pytest

import oracle
from paper_1708_05604_gb300 import synth, train


@pytest.fixture(scope="module", autouse=True)
def built():
    from paper_1708_05604_gb300 import build
    build.build()


def test_split_validation():
    tr, va = train.split_validation(1024, 0.05, 3)
    assert va.size == 51 and tr.size == 973
    assert np.array_equal(np.sort(np.concatenate([tr, va])), np.arange(1024))
    tr2, va2 = train.split_validation(1024, 0.05, 3)
    assert np.array_equal(va, va2) and np.array_equal(tr, tr2)
    assert not np.array_equal(va, train.split_validation(1024, 0.05, 4)[1])
    tr, va = train.split_validation(10, 0.0, 0)
    assert va.size == 0 and tr.size == 10
    tr, va = train.split_validation(5, 0.01, 0)
    assert va.size == 1


@pytest.mark.parametrize("order", ["ascending", "descending", "shuffle_buckets", "shuffle_batches"])
@pytest.mark.parametrize("wname", ["lstm1_uni_h32", "lstm1_bi_h128"])
def test_epoch_batches_follow_the_oracle_plan(wname, order):
    w = synth.WORKLOADS[wname]
    L = synth.draw_lengths(np.random.default_rng(2), w.n_seqs, w.length_dist)
    tr, _ = train.split_validation(L.size, 0.05, 9)
    Q = w.bucket_counts[-1]
    seen = []
    for e in range(3):
        batches, _ = train.epoch_batches(L, tr, Q, w.batch, 4, e, order)
        p = oracle.plan(L[tr], Q, w.batch, seed=4, epoch=e, batch_order=order)
        expect = [tr[p["order"][p["batch_off"][k]:p["batch_off"][k + 1]]]
                  for k in range(p["n_batches"])]
        assert len(batches) == len(expect)
        for a, b in zip(batches, expect):
            assert np.array_equal(a, b)
        assert np.array_equal(np.sort(np.concatenate(batches)), tr)
        seen.append(np.concatenate(batches))
    assert not np.array_equal(seen[0], seen[1])   # every epoch reshuffles


def test_validation_batches():
    L = np.array([5, 9, 1, 7, 7, 3, 2], np.int32)
    vb = train.validation_batches(L, np.array([0, 1, 3, 4, 6]), 2)
    assert [b.tolist() for b in vb] == [[1, 3], [4, 0], [6]]
