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
    is unchanged (a comment edit does not count as a change), scaled from the
    small captured case to a full launch by the ratio of algorithmic bytes."""
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
    page.write_text(f"kernel_code_sha256_16: {good}\ndram_bytes_per_launch_small: 990\n"
                    f"algorithmic_bytes_small: 1000\n")
    assert bench.profiled_traffic("demo", 1000) == 990
    assert bench.profiled_traffic("demo", 50_000) == 49_500    # scaled to the full launch
    (src / "rr_device.cu").write_text("/* new words */ int kernel_v1(void)\n{\n  return 1;  // said\n}\n")
    assert bench.profiled_traffic("demo", 1000) == 990        # comments and layout only
    (src / "rr_device.cu").write_text("int kernel_v1(void) { return 2; }\n")
    assert bench.profiled_traffic("demo", 1000) is None       # the code changed since the capture
    (src / "rr_device.cu").write_text("int kernel_v1(void) { return 1; }\n")
    (src / "rr_plan.cpp").write_text("int x = 1;\n")          # so did the planner's
    assert bench.profiled_traffic("demo", 1000) is None
    assert bench.profiled_traffic("other", 1000) is None
    (src / "rr_plan.cpp").write_text("int x; // a\n")
    assert bench.profiled_traffic("demo", 1000) == 990
    page.write_text(f"kernel_code_sha256_16: {good}\ndram_bytes_per_launch_full: 123\n")
    assert bench.profiled_traffic("demo", 1000) is None       # full-size figures are not read


def test_aggregate_and_host_memory():
    assert bench.aggregate_gbs(4, 1_000_000_000, 10.0) == pytest.approx(400.0)
    assert bench.host_memory_bytes() > 1 << 30


def test_ready_runs():
    assert bench.ready_runs([True, True, False, True]) == [(0, 2), (3, 4)]
    assert bench.ready_runs([False, False]) == []
    assert bench.ready_runs([]) == []
    assert bench.ready_runs([True] * 3) == [(0, 3)]


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-fsdp2", "tiny-units"])
def test_bucket_source_needs_cover_every_read(name):
    """The pipelined e2e packs a bucket once the first need[b] bytes of the
    source block have landed.  The oracle, given only those bytes (the rest
    zero), must produce that bucket exactly as from the whole source."""
    import numpy as np
    import oracle
    import paper_2512_22492_gb300 as rr
    from synth import device as D
    from tests import _util as U
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = rr.rr_plan_create(m, s, d, desc["bucket_bytes"], rr.PlanOptions(host_only=1))
    need = bench.bucket_source_needs(plan)
    shards = L.host_shards(desc["seed"], desc["specials"])
    starts = D.source_offsets(plan)
    block = np.zeros(starts[-1], np.uint8)
    for i, sh in enumerate(shards):
        block[starts[i]:starts[i] + len(sh)] = sh
    assert need.max() <= starts[-1] and need.min() >= 0
    full, full_cs = L.pack(oracle.Source(shards=shards))
    for b in range(plan.n_buckets):
        cut = block.copy()
        cut[need[b]:] = 0
        part = [cut[starts[i]:starts[i] + len(sh)] for i, sh in enumerate(shards)]
        got, cs = L.pack(oracle.Source(shards=part), first=b, count=1)
        np.testing.assert_array_equal(got[0], full[b], err_msg=f"bucket {b}")


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-tied", "tiny-moe-kvrep", "tiny-units",
                                  "qwen3-0.6b", "qwen3-8b", "qwen3-8b-tp4", "qwen3-30b-a3b",
                                  "qwen3-8b-fsdp2-tp8", "qwen3-30b-a3b-fsdp2-ep8"])
def test_both_arms_print_one_config(name):
    """The reference arm's config, from the oracle's layout, equals the native
    arm's, from the plan's byte counts (a host-only plan: no GPU)."""
    import oracle
    import paper_2512_22492_gb300 as rr
    from tests import _util as U
    w = U.workload(name)
    m, s, d = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep)
    plan = rr.rr_plan_create(m, s, d, w.bucket_bytes, rr.PlanOptions(host_only=True))
    st = plan.stats()
    native = bench.workload_config(w, w.bucket_bytes, plan.n_buckets, st["pack_bytes_read"],
                                   st["unpack_bytes_written"], 2)
    assert native["step_bytes"] == (st["pack_bytes_read"] + st["pack_bytes_written"] +
                                    st["verify_bytes_read"] + st["unpack_bytes_written"])
    assert bench.oracle_config(oracle.workload_layout(w), w, w.bucket_bytes, 2) == native


@pytest.mark.parametrize("name,want", [("qwen3-8b", 1), ("qwen3-30b-a3b-fsdp2-tp8", 1),
                                       ("qwen3-32b-fsdp2-tp8", 2)])
def test_receiver_launch_count(name, want):
    """The verifying unpack's launches per full call: one while every
    destination tensor fits one launch's pointer table (3480 tensors for
    30B-A3B at TP=8), two bucket ranges for Qwen3-32B at TP=8 (4120)."""
    import paper_2512_22492_gb300 as rr
    from tests import _util as U
    w = U.workload(name)
    m, s, d = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep)
    plan = rr.rr_plan_create(m, s, d, w.bucket_bytes, rr.PlanOptions(host_only=True))
    assert bench.receiver_launches(plan) == want
