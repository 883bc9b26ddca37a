"""Seeded synthetic workloads (inputs only; none of the method's arithmetic).

The paper trains on proprietary online-handwriting data (Section IV.A, Samsung
S-Note stylus recordings) that is not available; these generators stand in
for it.  Each token is a pen sample [dx, dy, pen_up, dt]; each sequence has a
label string whose length is proportional to its number of samples.

Draw order for one workload, from ``numpy.random.default_rng(seed)``:
  1. sequence lengths (lognormal: floor(exp(N(ln median, sigma)) + 0.5),
     then clipped; uniform: integers, bounds inclusive; bimodal: a fair coin
     per sequence picks the median, then the lognormal draw);
  2. features, all tokens of all sequences in index order:
     dx, dy ~ N(0, 1) as a [n_tok x 2] block, then pen_up ~ Bernoulli(0.05),
     then dt ~ U(0, 1);
  3. labels: U_i = L_i // label_div symbols per sequence, uniform in
     1..n_classes-1 (0 is the CTC blank);
  4. parameters (``draw_params``): every entry ~ U(-0.1, 0.1), float32.

Both the CUDA path and the oracle consume these arrays byte for byte.  This
module is shared by the tests, the benchmark and the smoke check; it imports
neither the product library nor the oracle.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

IN_DIM = 4
N_CLASSES = 81
BLANK = 0


@dataclass(frozen=True)
class Workload:
    """A model shape plus the length/label distribution it trains on."""
    name: str
    n_layers: int
    bidirectional: bool
    hidden: int
    n_seqs: int
    length_dist: tuple          # ("uniform", lo, hi) | ("lognormal", median, sigma, lo, hi)
                                # | ("bimodal", m1, m2, sigma, lo, hi)
    label_div: int
    batch: int
    bucket_counts: tuple
    gemm_bf16: bool
    in_dim: int = IN_DIM
    n_classes: int = N_CLASSES
    blank: int = BLANK
    extra: dict = field(default_factory=dict)

    @property
    def dirs(self) -> int:
        return 2 if self.bidirectional else 1

    def model_cfg(self) -> dict:
        return {"n_layers": self.n_layers, "bidirectional": self.bidirectional,
                "in_dim": self.in_dim, "hidden": self.hidden,
                "n_classes": self.n_classes, "blank": self.blank,
                "gemm_bf16": self.gemm_bf16}


# The five workloads.  Names say what each one is.
WORKLOADS = {
    "lstm1_uni_h32": Workload(
        "lstm1_uni_h32", 1, False, 32, 64, ("uniform", 20, 200), 10, 16, (2,), False),
    "lstm1_bi_h128": Workload(
        "lstm1_bi_h128", 1, True, 128, 1024, ("lognormal", 300.0, 0.6, 30, 1500), 12, 64,
        (1, 4), False),
    "lstm3_bi_h256_bf16": Workload(
        "lstm3_bi_h256_bf16", 3, True, 256, 8192, ("lognormal", 400.0, 0.7, 30, 2000), 12,
        128, (1, 2, 4, 8, 16), True),
    "lstm2_uni_h512": Workload(
        "lstm2_uni_h512", 2, False, 512, 2048, ("uniform", 1500, 4000), 20, 32, (4,), False),
    "lstm3_bi_h256_bf16_bimodal": Workload(
        "lstm3_bi_h256_bf16_bimodal", 3, True, 256, 32768,
        ("bimodal", 150.0, 900.0, 0.5, 20, 3000), 12, 128, (1, 2, 4, 8, 16, 32), True),
}
WORKLOAD_ORDER = list(WORKLOADS)


def _lognormal_lengths(rng, n, median, sigma, lo, hi):
    z = rng.standard_normal(n)
    L = np.floor(np.exp(np.log(median) + sigma * z) + 0.5)
    return np.clip(L, lo, hi).astype(np.int32)


def draw_lengths(rng: np.random.Generator, n: int, dist: tuple) -> np.ndarray:
    kind = dist[0]
    if kind == "uniform":
        _, lo, hi = dist
        return rng.integers(lo, hi, size=n, endpoint=True).astype(np.int32)
    if kind == "lognormal":
        _, median, sigma, lo, hi = dist
        return _lognormal_lengths(rng, n, median, sigma, lo, hi)
    if kind == "bimodal":
        _, m1, m2, sigma, lo, hi = dist
        first = rng.random(n) < 0.5
        z = rng.standard_normal(n)
        med = np.where(first, m1, m2)
        L = np.floor(np.exp(np.log(med) + sigma * z) + 0.5)
        return np.clip(L, lo, hi).astype(np.int32)
    raise ValueError(f"unknown length distribution {kind!r}")


@dataclass
class Dataset:
    """Sequences stored one after another in original index order."""
    lengths: np.ndarray        # int32 [n]
    x: np.ndarray              # float32 [n_tok x in_dim]
    x_off: np.ndarray          # int64 [n+1], row offset of each sequence in x
    label_lengths: np.ndarray  # int32 [n]
    labels: np.ndarray         # int32 [sum U]
    lab_off: np.ndarray        # int64 [n+1]

    @property
    def n(self) -> int:
        return int(self.lengths.size)

    @property
    def n_tok(self) -> int:
        return int(self.x_off[-1])

    def seq_x(self, i: int) -> np.ndarray:
        return self.x[self.x_off[i]:self.x_off[i + 1]]

    def seq_labels(self, i: int) -> np.ndarray:
        return self.labels[self.lab_off[i]:self.lab_off[i + 1]]

    def subset(self, idx) -> "Dataset":
        """The listed sequences, in the listed order, re-packed."""
        idx = np.asarray(idx, dtype=np.int64)
        L = self.lengths[idx]
        U = self.label_lengths[idx]
        x = np.concatenate([self.seq_x(i) for i in idx]) if idx.size else \
            np.zeros((0, self.x.shape[1]), np.float32)
        lab = np.concatenate([self.seq_labels(i) for i in idx]) if idx.size else \
            np.zeros(0, np.int32)
        return Dataset(L.astype(np.int32), np.ascontiguousarray(x, np.float32),
                       _offsets(L), U.astype(np.int32),
                       np.ascontiguousarray(lab, np.int32), _offsets(U))


def _offsets(counts) -> np.ndarray:
    off = np.zeros(len(counts) + 1, dtype=np.int64)
    np.cumsum(np.asarray(counts, dtype=np.int64), out=off[1:])
    return off


def make_dataset(lengths, label_div: int, rng: np.random.Generator,
                 in_dim: int = IN_DIM, n_classes: int = N_CLASSES) -> Dataset:
    """Features and labels for given lengths (draw steps 2 and 3)."""
    L = np.asarray(lengths, dtype=np.int32)
    n_tok = int(L.sum())
    x = np.zeros((n_tok, in_dim), dtype=np.float32)
    x[:, 0:2] = rng.standard_normal((n_tok, 2))
    x[:, 2] = (rng.random(n_tok) < 0.05)
    x[:, 3] = rng.random(n_tok)
    U = (L // label_div).astype(np.int32)
    labels = rng.integers(1, n_classes, size=int(U.sum()), endpoint=False).astype(np.int32)
    return Dataset(L, x, _offsets(L), U, labels, _offsets(U))


def make_workload(w: Workload | str, seed: int = 0, n_seqs: int | None = None,
                  max_len: int | None = None) -> Dataset:
    """Draw steps 1-3 for a workload.  `n_seqs` and `max_len` shrink it
    (fewer sequences; lengths clipped to max_len) for oracle-sized cases."""
    if isinstance(w, str):
        w = WORKLOADS[w]
    rng = np.random.default_rng(seed)
    n = w.n_seqs if n_seqs is None else n_seqs
    L = draw_lengths(rng, n, w.length_dist)
    if max_len is not None:
        L = np.minimum(L, max_len).astype(np.int32)
    return make_dataset(L, w.label_div, rng, w.in_dim, w.n_classes)


def draw_params(rng: np.random.Generator, n_params: int) -> np.ndarray:
    """Draw step 4: every parameter ~ U(-0.1, 0.1), float32."""
    return rng.uniform(-0.1, 0.1, size=n_params).astype(np.float32)
