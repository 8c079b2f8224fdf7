"""bench.py's host-side helpers, without a GPU.

The clock sampler is run against a stand-in `nvidia-smi` (a script on PATH
that prints CSV rows the way the real one does), so that the reasons a
measurement would be rejected for (hardware or thermal slowdown) are seen
and reported; the other helpers are checked on plain inputs.
"""
import os
import stat
import sys
import time

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)
import bench  # noqa: E402

FAKE = """#!/bin/sh
# prints three samples, then idles until terminated
echo "2026/12/02 09:00:00.100, 0, 2070, 2070, 900.00, 0x0000000000000004, Not Active, Not Active, Not Active, Active"
echo "2026/12/02 09:00:00.150, 0, 1980, 2070, 1390.00, 0x0000000000000008, Active, Not Active, Not Active, Not Active"
echo "2026/12/02 09:00:00.200, 0, 2070, 2070, 910.00, 0x0000000000000000, Not Active, Not Active, Not Active, Not Active"
exec sleep 30
"""


def at(stamp):
    return bench.ClockSampler._when(stamp)


@pytest.fixture
def fake_smi(tmp_path, monkeypatch):
    exe = tmp_path / "nvidia-smi"
    exe.write_text(FAKE)
    exe.chmod(exe.stat().st_mode | stat.S_IXUSR)
    monkeypatch.setenv("PATH", f"{tmp_path}{os.pathsep}{os.environ['PATH']}")
    return exe


def test_clock_sampler_reports_slowdowns(fake_smi):
    with bench.ClockSampler(0) as clk:
        deadline = time.time() + 10
        while len(clk.rows) < 3 and time.time() < deadline:
            time.sleep(0.05)
    s = clk.summary()
    assert s["samples"] == 3 and s["window"].startswith("bench run")
    assert s["sm_mhz"] == 2070.0 and s["sm_max_mhz"] == 2070.0
    assert s["reasons"] == ["hw_slowdown", "sw_power_cap"]


def test_clock_sampler_windows(fake_smi):
    """Rows belong to the timed region by nvidia-smi's timestamps: a region
    holding all three reports them alone; one holding fewer than three falls
    back to every row, and says how many the region held."""
    with bench.ClockSampler(0) as clk:
        clk.wait_first()
        deadline = time.time() + 10
        while len(clk.rows) < 3 and time.time() < deadline:
            time.sleep(0.05)
    clk.mark(at("2026/12/02 09:00:00.050"), at("2026/12/02 09:00:00.250"))
    s = clk.summary()
    assert s["window"] == "timed region" and s["samples"] == 3
    clk.mark(at("2026/12/02 09:00:00.120"), at("2026/12/02 09:00:00.160"))
    s = clk.summary()
    assert s["samples"] == 3 and "1 sample(s)" in s["window"]
    assert s["reasons"] == ["hw_slowdown", "sw_power_cap"]
    assert bench.ClockSampler._when("not a time") is None


def test_clock_sampler_without_nvidia_smi(tmp_path, monkeypatch):
    monkeypatch.setenv("PATH", str(tmp_path))          # nothing to run
    with bench.ClockSampler(0) as clk:
        pass
    assert clk.summary() == {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}


def test_visible_gpu_index(monkeypatch):
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "3,5")
    assert bench.visible_gpu_index(0) == 3 and bench.visible_gpu_index(1) == 5
    monkeypatch.setenv("CUDA_VISIBLE_DEVICES", "")
    assert bench.visible_gpu_index(2) == 2


def test_profiled_traffic_needs_the_current_kernel(tmp_path, monkeypatch):
    """The profile's traffic is reported only while the code it was taken on
    is unchanged; a comment edit does not count as a change."""
    monkeypatch.setattr(bench, "ROOT", str(tmp_path))
    (tmp_path / "profiles").mkdir()
    (tmp_path / "include").mkdir()
    src = tmp_path / "paper_2512_22492_gb300" / "csrc"
    src.mkdir(parents=True)
    for name in bench.KERNEL_SOURCES:
        (tmp_path / name).write_text("int x; // a\n")
    (src / "rr_device.cu").write_text("int kernel_v1(void) { return 1; }  // first\n")
    good = bench.kernel_code_hash()
    page = tmp_path / "profiles" / "rr_pack_demo.md"
    page.write_text(f"kernel_code_sha256_16: {good}\ndram_bytes_per_launch_full: 123\n")
    assert bench.profiled_traffic("demo") == 123
    (src / "rr_device.cu").write_text("/* new words */ int kernel_v1(void)\n{\n  return 1;  // said\n}\n")
    assert bench.profiled_traffic("demo") == 123        # comments and layout only
    (src / "rr_device.cu").write_text("int kernel_v1(void) { return 2; }\n")
    assert bench.profiled_traffic("demo") is None       # the code changed since the capture
    (src / "rr_device.cu").write_text("int kernel_v1(void) { return 1; }\n")
    (src / "rr_plan.cpp").write_text("int x = 1;\n")      # so did the planner's
    assert bench.profiled_traffic("demo") is None
    assert bench.profiled_traffic("other") is None


def test_aggregate_and_host_memory():
    assert bench.aggregate_gbs(4, 1_000_000_000, 10.0) == pytest.approx(400.0)
    assert bench.host_memory_bytes() > 1 << 30
