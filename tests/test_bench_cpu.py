"""Host-side logic of bench.py that needs no GPU: the roofline arithmetic
per bound, the epoch budget rule, the committed DRAM-traffic record
(reported only while the kernel source it was taken from is unchanged), the
peak table and the defaults (the full-epoch bimodal sweep)."""
import hashlib
import importlib.util
import json
import os
import shutil

import numpy as np
import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def stat(name, launches, ms, flops=0.0, nbytes=0.0, steps=0):
    return {"name": name, "launches": launches, "total_ms": ms, "flops": flops, "bytes": nbytes,
            "serial_steps": steps}


def test_roofline_alu_arithmetic(bench):
    r = bench.roofline_for(stat("lstm_fwd", 10, 20.0, flops=4.0e10, steps=4000),
                           {"sm_max_mhz": 2000.0}, "measured", {"sm_mhz": 1000.0}, n_sm=152)
    # 4e10 flop in 20 ms = 2 TFLOP/s; 20 ms over 4000 serial steps = 5 us per step
    assert r["bound"] == "alu" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(2.0)
    assert r["peak"] == pytest.approx(152 * 128 * 2 * 1000e6 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert r["us_per_step"] == pytest.approx(5.0)
    assert r["algorithmic_flops_per_launch"] == pytest.approx(4.0e9)
    # no work, no roofline
    assert bench.roofline_for(stat("lstm_fwd", 1, 1.0), {}, "measured", {}) is None


def test_roofline_hbm_arithmetic(bench):
    r = bench.roofline_for(stat("ctc_grad", 4, 4.0, nbytes=2.4e7), {"hbm_gbs": 6000.0}, "measured", {})
    # 2.4e7 B in 4 ms = 6 GB/s
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(6.0)
    assert r["frac"] == pytest.approx(6.0 / 6000.0)
    assert "us_per_step" not in r


def test_roofline_tensor_peaks(bench):
    peaks = {"bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
    r = bench.roofline_for(stat("gemm_tc", 2, 1.0, flops=1.7e15 * 1e-3 * 0.5), peaks, "measured", {})
    assert r["bound"] == "tensor" and r["peak"] == pytest.approx(1700.0)
    assert r["frac"] == pytest.approx(0.5)
    r3 = bench.roofline_for(stat("gemm_tf32x3", 2, 1.0, flops=1e9), peaks, "measured", {})
    assert r3["peak"] == pytest.approx(1700.0 * (1.1 / 2.25) / 3.0)


def test_budget_count(bench):
    assert bench.budget_count(5700.0, 3000.0, 1, 10) == 1
    assert bench.budget_count(20.0, 3000.0, 1, 10) == 10
    assert bench.budget_count(5700.0, 15000.0, 2, 20) == 3
    assert bench.budget_count(0.0, 1.0, 2, 5) == 5


def test_defaults_are_the_full_epoch_sweep(bench):
    a = bench.parse([])
    assert a.workload == "lstm3_bi_h256_bf16_bimodal" and a.buckets == 8
    qs = sorted({a.buckets} | {int(q) for q in a.compare_buckets.split(",")})
    assert qs == [1, 2, 4, 8, 16, 32]
    assert bench.METRIC.startswith("unpadded timesteps/sec")


def test_serial_steps(bench):
    class DS:
        lengths = np.array([5, 9, 2, 7], np.int32)
    plan = {"n_batches": 2, "batch_off": np.array([0, 2, 4]), "order": np.array([2, 0, 1, 3])}
    assert bench.serial_steps(plan, DS) == 5 + 9


def test_recorded_traffic_matches_committed_source(bench):
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic_lstm1_bi_h128.json")))
    src = open(os.path.join(ROOT, rec["source"]), "rb").read()
    same = hashlib.sha256(src).hexdigest() == rec["source_sha256"]
    assert set(rec["kernels"]) == {"lstm_fwd", "lstm_bwd"}
    for k, entry in rec["kernels"].items():
        tb, where = bench.recorded_traffic(k, rec["workload"], rec["buckets"])
        if same:
            assert tb == entry["dram_bytes_per_launch"] and where.endswith("traffic_lstm1_bi_h128.json")
            assert entry["dram_bytes_per_launch"] == pytest.approx(
                entry["dram_read_bytes_per_launch"] + entry["dram_write_bytes_per_launch"], abs=1)
        else:   # the kernels changed since the counters were taken: nothing is reported
            assert tb is None and where is None
        # other workloads or bucket counts have no record
        assert bench.recorded_traffic(k, rec["workload"], rec["buckets"] + 1) == (None, None)
        assert bench.recorded_traffic(k, "lstm2_uni_h512", rec["buckets"]) == (None, None)
    assert bench.recorded_traffic("ctc_tables", rec["workload"], rec["buckets"]) == (None, None)


def test_recorded_traffic_ignored_after_a_source_change(bench, tmp_path, monkeypatch):
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic_lstm1_bi_h128.json")))
    (tmp_path / "profiles").mkdir()
    dst = tmp_path / rec["source"]
    dst.parent.mkdir(parents=True)
    src = open(os.path.join(ROOT, rec["source"]), "rb").read()
    dst.write_bytes(src)
    # make the copy's record match its source, then change the source
    rec["source_sha256"] = hashlib.sha256(src).hexdigest()
    json.dump(rec, open(tmp_path / "profiles" / "traffic_lstm1_bi_h128.json", "w"))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    for k, entry in rec["kernels"].items():
        assert bench.recorded_traffic(k, rec["workload"], rec["buckets"])[0] == entry["dram_bytes_per_launch"]
    dst.write_bytes(src + b"\n// changed\n")
    for k in rec["kernels"]:
        assert bench.recorded_traffic(k, rec["workload"], rec["buckets"]) == (None, None)


def test_measured_peaks_source(bench, tmp_path, monkeypatch):
    peaks, src = bench.measured_peaks()
    if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")):
        assert src == "measured" and peaks.get("hbm_gbs")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    peaks, src = bench.measured_peaks()
    assert src == "fallback" and peaks["hbm_gbs"] == 6800.0


def test_recorded_traffic_per_kernel_record(bench):
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic_lstm3_bi_h256_bf16_bimodal.json")))
    src = open(os.path.join(ROOT, rec["source"]), "rb").read()
    same = hashlib.sha256(src).hexdigest() == rec["source_sha256"]
    for k, entry in rec["kernels"].items():
        tb, where = bench.recorded_traffic(k, rec["workload"], rec["buckets"])
        if same:
            assert tb == entry["dram_bytes_per_launch"] and where.endswith(".json")
            # scaled from the profiled batch by tokens
            prof = entry["dram_read_bytes_profiled"] + entry["dram_write_bytes_profiled"]
            assert tb == pytest.approx(prof * rec["mean_tokens_per_launch"] / rec["scaled_from"]["tokens"])
        else:
            assert tb is None
    assert bench.recorded_traffic("gemm_tc", rec["workload"], rec["buckets"]) == (None, None)


def test_reference_arm_prints_one_contract_line():
    """`bench.py --impl reference` (the oracle on bounded samples, host cores
    only) prints one JSON line with the keys the launch contract names."""
    import subprocess
    import sys
    r = subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), "--impl", "reference",
                        "--workload", "lstm1_uni_h32", "--buckets", "2", "--steps", "2", "--warmup", "1",
                        "--reference-seconds", "1.5"],
                       capture_output=True, text=True, timeout=300, cwd=ROOT)
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [x for x in r.stdout.splitlines() if x.startswith("{")]
    assert len(lines) == 1
    d = json.loads(lines[0])
    for k in ("impl", "metric", "value", "unit", "n_gpus", "steps", "warmup", "ms_per_step",
              "higher_is_better", "scaling", "vs_baseline", "dtype", "config", "cpu_baseline", "e2e"):
        assert k in d, k
    assert d["impl"] == "reference" and d["value"] > 0 and d["unit"] == "timesteps/s"
    assert d["config"]["workload"] == "lstm1_uni_h32"
    assert d["cpu_baseline"]["kind"] == "oracle" and d["cpu_baseline"]["cores"] == 1
    assert d["cpu_baseline"]["value"] == d["value"] == d["e2e"]["value"]
    assert d["e2e"]["h2d_bytes_per_step"] == 0 and d["e2e"]["d2h_bytes_per_step"] == 0
