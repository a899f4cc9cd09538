"""Host logic of bench.py that needs no GPU: the hash-gated DRAM traffic
read from the committed ncu summary, and the clock record of the timed
region (median SM clock, throttle reasons inside the window)."""
from __future__ import annotations

import os
import sys
import time

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def test_traffic_only_for_the_current_kernel_source(tmp_path, monkeypatch):
    note = tmp_path / "note.md"
    monkeypatch.setattr(bench, "TRAFFIC_NOTE", str(note))
    assert bench.recorded_traffic() is None  # no summary
    h = bench.kernel_source_hash()
    note.write_text(f"text\n    kernel_source_sha256_16: {h}\n    dram_bytes_per_launch: 17045248\n")
    assert bench.recorded_traffic() == 17045248
    other = "0" * 16 if h != "0" * 16 else "1" * 16
    note.write_text(f"    kernel_source_sha256_16: {other}\n    dram_bytes_per_launch: 17045248\n")
    assert bench.recorded_traffic() is None  # counters of another kernel source
    note.write_text(f"    kernel_source_sha256_16: {h}\n")
    assert bench.recorded_traffic() is None  # no figure


def test_committed_summary_names_a_figure():
    text = open(os.path.join(ROOT, "profiles", "block_attn_8b_b1_L4096_bl16.md")).read()
    assert "kernel_source_sha256_16:" in text and "dram_bytes_per_launch:" in text


def _sampler_with(tmp_path, rows):
    path = tmp_path / "clocks.csv"
    path.write_text("".join(",".join(r) + "\n" for r in rows))
    s = object.__new__(bench.ClockSampler)
    s.proc, s.path = None, str(path)
    return s


def _row(t, sm, reasons=("Not Active",) * 4):
    stamp = time.strftime("%Y/%m/%d %H:%M:%S", time.localtime(int(t))) + ".%03d" % int((t % 1) * 1000)
    return [stamp, "0", str(sm), "2070", "900.0", "0x0"] + list(reasons)


def test_clock_summary_uses_samples_inside_the_timed_region(tmp_path):
    t0 = float(int(time.time())) + 0.5
    rows = [_row(t0 - 2.0, 1000, ("Active", "Not Active", "Not Active", "Not Active")),  # before: ignored
            _row(t0 + 0.1, 2070), _row(t0 + 0.2, 2055),
            _row(t0 + 0.3, 2070, ("Not Active", "Not Active", "Not Active", "Active")),
            _row(t0 + 5.0, 900)]  # after: ignored
    out = _sampler_with(tmp_path, rows).summary(t0, t0 + 0.4)
    assert out["samples"] == 3 and out["sm_mhz"] == 2070.0 and out["sm_max_mhz"] == 2070.0
    assert out["reasons"] == ["sw_power_cap"]
    assert not os.path.exists(tmp_path / "clocks.csv")


def test_clock_summary_short_region_falls_back_to_all_samples(tmp_path):
    t0 = float(int(time.time())) + 0.5
    rows = [_row(t0 - 3.0, 2000), _row(t0 + 3.0, 2070, ("Not Active", "Active", "Not Active", "Not Active"))]
    out = _sampler_with(tmp_path, rows).summary(t0, t0 + 0.01)
    assert out["samples"] == 2 and "all samples" in out["note"]
    assert out["reasons"] == ["hw_thermal_slowdown"]


def test_clock_summary_without_nvidia_smi():
    s = object.__new__(bench.ClockSampler)
    s.proc, s.path = None, None
    assert s.summary(0.0, 1.0)["note"] == "nvidia-smi unavailable"
