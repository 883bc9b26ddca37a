"""The committed profile summaries: short text only, each with the command
that produced it, every ncu command leaving the GPU clocks alone, and each
DRAM-traffic record pointing at a source file of the library."""
import glob
import json
import os
import re

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
PROF = os.path.join(ROOT, "profiles")


def test_profiles_are_short_text():
    files = glob.glob(os.path.join(PROF, "*"))
    assert files
    for f in files:
        assert os.path.splitext(f)[1] in (".md", ".txt", ".json"), f
        assert os.path.getsize(f) < 64 * 1024, f


def test_every_summary_gives_its_command():
    for f in glob.glob(os.path.join(PROF, "*.md")):
        text = open(f).read()
        assert "```" in text and re.search(r"\b(ncu|python)\b", text), f


def test_ncu_commands_leave_the_clocks_alone():
    for f in glob.glob(os.path.join(PROF, "*.md")) + glob.glob(os.path.join(PROF, "*.json")):
        text = open(f).read().replace("\\\n", " ")
        for m in re.finditer(r"(?m)(?:^|[`\"\s])ncu (--[^\n`\"]*)", text):
            cmd = m.group(1)
            if cmd.startswith("-i"):   # reading a report back needs no GPU
                continue
            assert "--clock-control none" in cmd, (os.path.basename(f), cmd[:120])


def test_traffic_records_name_library_sources():
    for f in glob.glob(os.path.join(PROF, "traffic_*.json")):
        rec = json.load(open(f))
        assert os.path.exists(os.path.join(ROOT, rec["source"])), f
        assert rec["source"].startswith("paper_1708_05604_gb300/csrc/"), f
        kernels = rec.get("kernels") or {rec["kernel"]: rec}
        for k, e in kernels.items():
            assert e["dram_bytes_per_launch"] > 0, (f, k)
