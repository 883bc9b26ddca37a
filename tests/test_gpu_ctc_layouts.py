"""GPU parity of every lane layout of the CTC tables kernel (a8).

The launcher picks K extended-label positions per lane from the batch's
longest label; BKT_CTC_K forces K, read once per process, so each layout runs
in its own child process.  The batch mixes an empty label, one-symbol labels,
repeated symbols, an infeasible row and labels long enough that every K below
16 spans several warps (cross-warp neighbour exchange)."""
import json
import os
import subprocess
import sys

import pytest

pytestmark = pytest.mark.gpu

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))

CHILD = r"""
import json, sys
import numpy as np
sys.path.insert(0, "tests")
from gpu_util import FP32_TOL, compare, gpu_step, oracle_step
from paper_1708_05604_gb300 import binding, build, synth
build.build()
cfg = {"n_layers": 1, "bidirectional": True, "in_dim": 4, "hidden": 16, "n_classes": 9,
       "blank": 0}
rng = np.random.default_rng(31)
L = np.array([1, 2, 7, 40, 130, 301, 520, 4], np.int32)
U = np.array([0, 1, 2, 13, 43, 100, 173, 3], np.int32)
base = synth.make_dataset(L, 3, rng, n_classes=cfg["n_classes"])
labels = rng.integers(1, cfg["n_classes"], size=int(U.sum())).astype(np.int32)
off = np.concatenate([[0], np.cumsum(U)]).astype(np.int64)
labels[off[2]:off[2] + 2] = 4                   # a repeated pair
labels[off[3]:off[3] + 5] = 6                   # a run of repeats
labels[off[7]:off[7] + 3] = 2                   # U + repeats = 5 > L = 4: no alignment
ds = synth.Dataset(L, base.x, base.x_off, U, labels, off)
params = synth.draw_params(rng, binding.param_count(cfg))
lg, gg = gpu_step(cfg, ds, params)
lo, go = oracle_step(cfg, ds, params)
compare(cfg, lg, gg, lo, go, FP32_TOL)
print(json.dumps({"S_max": int(2 * ds.label_lengths.max() + 1),
                  "infeasible": int((~np.isfinite(lo)).sum())}))
"""


@pytest.mark.parametrize("K", [1, 2, 4, 8, 16])
def test_ctc_lane_layout_parity(cuda_device, K):
    env = dict(os.environ, BKT_CTC_K=str(K))
    r = subprocess.run([sys.executable, "-c", CHILD], cwd=ROOT, env=env, capture_output=True,
                       text=True, timeout=600)
    assert r.returncode == 0, r.stdout[-2000:] + r.stderr[-4000:]
    info = json.loads(r.stdout.strip().splitlines()[-1])
    assert info["S_max"] == 347 and info["infeasible"] == 1
