"""Host logic of bench.py on the CPU: the DRAM-traffic record and its source
hashes, and the parsing of the clock samples taken during the timed region."""
import hashlib
import json
import os
import sys

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402


def test_measured_traffic_follows_the_source_hashes(tmp_path, monkeypatch):
    src = tmp_path / "k.cu"
    src.write_text("kernel v1\n")
    (tmp_path / "profiles").mkdir()
    rec = {"k<256>": {"dram_read": 1000, "dram_write": 24, "capture": "profiles/k.md",
                      "sources": {"k.cu": hashlib.sha256(b"kernel v1\n").hexdigest()}}}
    (tmp_path / "profiles" / "traffic.json").write_text(json.dumps(rec))
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    assert bench.measured_traffic("k<256>") == 1024
    assert bench.measured_traffic("other") is None
    src.write_text("kernel v2\n")                 # changed since the capture
    assert bench.measured_traffic("k<256>") is None
    src.unlink()
    assert bench.measured_traffic("k<256>") is None


def test_committed_traffic_records_are_well_formed():
    recs = json.load(open(os.path.join(ROOT, "profiles", "traffic.json")))
    kernels = [k for k in recs if not k.startswith("_")]
    assert {"decode_split_kernel<256>", "prefill_kernel<256>"} <= set(kernels)
    for k in kernels:
        r = recs[k]
        assert isinstance(r["dram_read"], int) and isinstance(r["dram_write"], int)
        assert r["dram_read"] > 0 and r["dram_write"] >= 0
        assert os.path.exists(os.path.join(ROOT, r["capture"])), r["capture"]
        for name, sha in r["sources"].items():
            assert os.path.exists(os.path.join(ROOT, name)), name
            assert len(sha) == 64


def _summary(tmp_path, lines):
    s = bench.ClockSampler(0)
    s.path = str(tmp_path / "clocks.csv")
    with open(s.path, "w") as f:
        f.write("\n".join(lines) + "\n")
    s.proc = object()          # a sampler that ran
    return s.summary()


NA = "Not Active"


def test_clock_summary_keeps_loaded_samples_and_active_reasons(tmp_path):
    rows = [
        f"0, 1980, 2070, 95.0, 0x0, {NA}, {NA}, {NA}, {NA}",        # idle: dropped
        f"0, 2070, 2070, 812.5, 0x0, {NA}, {NA}, {NA}, {NA}",
        f"0, 2040, 2070, 1390.0, 0x4, {NA}, {NA}, {NA}, Active",    # power cap
        f"0, 2070, 2070, 900.0, 0x0, {NA}, {NA}, {NA}, {NA}",
        "garbage line",
    ]
    got = _summary(tmp_path, rows)
    assert got["samples"] == 3
    assert got["sm_mhz"] == 2070.0 and got["sm_max_mhz"] == 2070.0
    assert got["power_w_max"] == 1390.0
    assert got["reasons"] == ["sw_power_cap"]


def test_clock_summary_reports_thermal_slowdown(tmp_path):
    rows = [f"0, 1500, 2070, 700.0, 0x20, Active, {NA}, Active, {NA}"] * 3
    got = _summary(tmp_path, rows)
    assert got["sm_mhz"] == 1500.0
    assert got["reasons"] == ["hw_slowdown", "sw_thermal_slowdown"]


def test_clock_summary_without_samples(tmp_path):
    assert _summary(tmp_path, [])["reasons"] == ["no samples"]
    s = bench.ClockSampler(0)
    assert s.summary()["reasons"] == ["nvidia-smi unavailable"]
