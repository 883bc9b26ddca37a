"""Training checkpoints: the flat parameter buffer and the optimizer state as
one fp32 blob, with a JSON record beside it.

Section III.B stores each model after a stage of training and starts the
next stage from the stored models.  Here a checkpoint is taken after an
epoch: `<path>.bin` holds the named fp32 arrays back to back (parameters,
then ADADELTA's running averages when that rule is used) and `<path>.json`
their layout, a SHA-256 of the blob and the run's metadata (workload, bucket
count, seed, batch order, the next epoch, the per-epoch records so far).
An epoch's mini-batches are a pure function of (lengths, Q, batch, seed,
epoch, batch order), so a run resumed from a checkpoint replays the
following epochs' batches bit for bit.

Both files are written to a temporary name and moved into place, the blob
first, so a crash leaves either the previous checkpoint or the new one; a
record whose blob does not match its hash is refused.
"""
from __future__ import annotations

import hashlib
import json
import os

import numpy as np

FORMAT = "bkt-checkpoint-1"


def _replace(path: str, data: bytes) -> None:
    tmp = f"{path}.tmp.{os.getpid()}"
    with open(tmp, "wb") as f:
        f.write(data)
        f.flush()
        os.fsync(f.fileno())
    os.replace(tmp, path)


def save(path: str, arrays: dict, meta: dict) -> None:
    """Writes `path`.bin (the arrays, fp32, in the given order) and
    `path`.json (layout, hash, meta).  `meta` must be JSON-serialisable."""
    layout, parts, off = [], [], 0
    for name, a in arrays.items():
        v = np.ascontiguousarray(np.asarray(a, dtype=np.float32).ravel())
        layout.append({"name": str(name), "offset": off, "count": int(v.size)})
        parts.append(v.tobytes())
        off += int(v.size)
    blob = b"".join(parts)
    rec = {"format": FORMAT, "arrays": layout, "floats": off,
           "sha256": hashlib.sha256(blob).hexdigest(), "meta": meta}
    _replace(path + ".bin", blob)
    _replace(path + ".json", (json.dumps(rec, indent=1) + "\n").encode())


def load(path: str):
    """(meta, {name: fp32 array}) of a checkpoint; ValueError when the record
    is not a checkpoint of this format or the blob does not match it."""
    with open(path + ".json") as f:
        rec = json.load(f)
    if rec.get("format") != FORMAT:
        raise ValueError(f"{path}.json: not a {FORMAT} record")
    with open(path + ".bin", "rb") as f:
        blob = f.read()
    if len(blob) != 4 * int(rec["floats"]):
        raise ValueError(f"{path}.bin: {len(blob)} bytes, the record says {4 * int(rec['floats'])}")
    if hashlib.sha256(blob).hexdigest() != rec["sha256"]:
        raise ValueError(f"{path}.bin: contents do not match the record's SHA-256")
    flat = np.frombuffer(blob, dtype=np.float32)
    arrays = {}
    for e in rec["arrays"]:
        o, n = int(e["offset"]), int(e["count"])
        if o < 0 or o + n > flat.size:
            raise ValueError(f"{path}.json: array {e['name']!r} lies outside the blob")
        arrays[e["name"]] = flat[o:o + n].copy()
    return rec["meta"], arrays


def check_compatible(meta: dict, expect: dict) -> None:
    """Raises ValueError naming every key of `expect` whose value differs in
    the checkpoint's meta (a resumed run must continue the same run)."""
    bad = [k for k, v in expect.items() if meta.get(k) != v]
    if bad:
        raise ValueError("checkpoint belongs to another run: " +
                         ", ".join(f"{k} = {meta.get(k)!r} (this run {expect[k]!r})" for k in bad))


class JsonlLog:
    """Appends one JSON object per call to a file, flushed at once, so a
    run's per-epoch metrics can be followed while it runs and survive it."""

    def __init__(self, path: str, **fixed):
        self.path, self.fixed = path, fixed

    def __call__(self, rec: dict) -> None:
        with open(self.path, "a") as f:
            f.write(json.dumps({**self.fixed, **rec}) + "\n")
            f.flush()
