"""Host-side logic of bench.py that needs no GPU: the roofline arithmetic,
the committed DRAM-traffic record (reported only while the kernel source it
was taken from is unchanged) and the peak table."""
import hashlib
import importlib.util
import json
import os
import shutil

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def bench():
    spec = importlib.util.spec_from_file_location("bench_under_test", os.path.join(ROOT, "bench.py"))
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    return mod


def test_roofline_alu_arithmetic(bench):
    work = {"lstm_fwd": ("alu", 4.0e9)}
    r = bench.roofline_for("lstm_fwd", 10, 20.0, work, {"sm_max_mhz": 2000.0}, "measured",
                           {"sm_mhz": 1000.0})
    # 10 launches in 20 ms: 2 ms each; 4 GFLOP / 2 ms = 2 TFLOP/s
    assert r["bound"] == "alu" and r["unit"] == "TFLOP/s"
    assert r["achieved"] == pytest.approx(2.0)
    assert r["peak"] == pytest.approx(152 * 128 * 2 * 1000e6 / 1e12)
    assert r["frac"] == pytest.approx(r["achieved"] / r["peak"])
    assert bench.roofline_for("other", 1, 1.0, work, {}, "measured", {}) is None


def test_roofline_hbm_arithmetic(bench):
    work = {"ctc_grad": ("hbm", 6.0e6)}
    r = bench.roofline_for("ctc_grad", 4, 4.0, work, {"hbm_gbs": 6000.0}, "measured", {})
    # 1 ms per launch: 6e6 B / 1e-3 s = 6e9 B/s = 6 GB/s
    assert r["bound"] == "hbm" and r["unit"] == "GB/s"
    assert r["achieved"] == pytest.approx(6.0)
    assert r["frac"] == pytest.approx(6.0 / 6000.0)


def test_recorded_traffic_matches_committed_source(bench):
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic_lstm1_bi_h128.json")))
    src = open(os.path.join(ROOT, rec["source"]), "rb").read()
    tb, where = bench.recorded_traffic(rec["kernel"], rec["workload"], rec["buckets"])
    if hashlib.sha256(src).hexdigest() == rec["source_sha256"]:
        assert tb == rec["dram_bytes_per_launch"] and where.endswith("traffic_lstm1_bi_h128.json")
    else:   # the kernel changed since the counters were taken: nothing is reported
        assert tb is None and where is None
    # other workloads or bucket counts have no record
    assert bench.recorded_traffic(rec["kernel"], rec["workload"], rec["buckets"] + 1) == (None, None)
    assert bench.recorded_traffic(rec["kernel"], "lstm2_uni_h512", rec["buckets"]) == (None, None)


def test_recorded_traffic_ignored_after_a_source_change(bench, tmp_path, monkeypatch):
    rec = json.load(open(os.path.join(ROOT, "profiles", "traffic_lstm1_bi_h128.json")))
    (tmp_path / "profiles").mkdir()
    shutil.copy(os.path.join(ROOT, "profiles", "traffic_lstm1_bi_h128.json"), tmp_path / "profiles")
    dst = tmp_path / rec["source"]
    dst.parent.mkdir(parents=True)
    src = open(os.path.join(ROOT, rec["source"]), "rb").read()
    dst.write_bytes(src)
    # make the copy's record match its source, then change the source
    rec["source_sha256"] = hashlib.sha256(src).hexdigest()
    json.dump(rec, open(tmp_path / "profiles" / "traffic_lstm1_bi_h128.json", "w"))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.recorded_traffic(rec["kernel"], rec["workload"], rec["buckets"])[0] == \
        rec["dram_bytes_per_launch"]
    dst.write_bytes(src + b"\n// changed\n")
    assert bench.recorded_traffic(rec["kernel"], rec["workload"], rec["buckets"]) == (None, None)


def test_measured_peaks_source(bench, tmp_path, monkeypatch):
    peaks, src = bench.measured_peaks()
    if os.path.exists(os.path.join(ROOT, "MEASURED_PEAKS.json")):
        assert src == "measured" and peaks.get("hbm_gbs")
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    peaks, src = bench.measured_peaks()
    assert src == "fallback" and peaks["hbm_gbs"] == 6800.0
