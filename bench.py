"""Benchmark: one full trainer -> rollout weight sync per step on GB300.

A step is the whole hot path once (RobustRL Section 5.2.1 steps 1-2 and the
Section 5.2.2 check): rr_pack (reshard + bf16 cast + bucket pack + checksum)
and the receiver's rr_unpack_verify_async (buckets -> rollout tensors, with
every bucket's checksum recomputed and compared in the same pass).  Default
workload: Qwen3-8B-shaped fp32 weights in 8 flat FSDP-style shards -> TP=1
bf16 rollout layout with fused QKV / gate_up, 128 MiB buckets, seeded
synthetic values ~N(0, 0.02).

Metric: GB/s of algorithmic bytes (every byte read once, every byte written
once: pack = source bytes + bucket bytes; the receiver = bucket bytes read +
tensor bytes written), plus ms per full model sync (pack + the receiver).
The separate rr_unpack and rr_verify are timed after the step loop as a
breakdown.  Inputs (33 GB of source) are far larger than L2, so no flush is
needed between steps.

End to end (`e2e`): the same step with the trainer's shards in host memory,
by three routes, all timed and the fastest reported -- the copy engines
bringing the source over in pieces while the buckets whose sources have
landed are packed, the pack reading the pinned shards itself over
NVLink-C2C, or the same from ordinary pageable memory where the GPU reads it.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl native|reference]

Under torchrun each rank runs an independent replica on its own GPU (the
path does not shard: replicas only); the value is the bytes of all replicas
over the slowest rank's time.
"""
from __future__ import annotations

import argparse
import atexit
import hashlib
import json
import os
import re
import statistics
import subprocess
import sys
import threading
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "weight-sync reshard+pack GB/s and ms per full model sync; % of HBM roofline"
UNIT = "GB/s"
FALLBACK_HBM_GBS = 6800.0


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["native", "reference"], default="native")
    ap.add_argument("--workload", default="qwen3-8b")
    ap.add_argument("--bucket-mib", type=int, default=0, help="override the bucket size")
    ap.add_argument("--dst-dtype", choices=["bf16", "f16"], default="bf16",
                    help="the rollout's 16-bit element type")
    ap.add_argument("--layers", type=int, default=0,
                    help="keep only the first N decoder layers (a small case of the same "
                         "kernels, for profiler captures); the workload name says so")
    ap.add_argument("--vocab", type=int, default=0,
                    help="with --layers: a smaller vocabulary as well")
    ap.add_argument("--chunk-kib", type=int, default=0, help="plan option: KiB per work item")
    ap.add_argument("--grid", type=int, default=0, help="plan option: persistent grid size")
    ap.add_argument("--sync-verify", action="store_true",
                    help="the receiver uses the synchronous rr_unpack_verify (a host round "
                         "trip per step) instead of rr_unpack_verify_async")
    ap.add_argument("--check-items", action="store_true",
                    help="plan option: kernels check every work item's bounds")
    ap.add_argument("--engine", choices=["auto", "registers"], default="auto",
                    help="plan option: the bulk-copy engine for device buffers (auto) or the "
                         "register path for every call")
    ap.add_argument("--snapshot", action="store_true",
                    help="also time rr_pack straight into pinned host buckets")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--e2e-pieces", type=int, default=16,
                    help="pieces the e2e source copy is cut into (the pack follows each)")
    ap.add_argument("--e2e-route", choices=["auto", "copy", "direct", "pageable"],
                    default="auto",
                    help="e2e source route: copy engines, the pack reading pinned host "
                         "memory directly, the same from pageable host memory, or all "
                         "timed and the fastest reported (auto)")
    ap.add_argument("--e2e-direct-pieces", type=int, default=16,
                    help="bucket ranges of the direct e2e route (the receiver follows each)")
    ap.add_argument("--no-next-rows", action="store_true",
                    help="skip the resume (bucket-range) and relay re-pack timings")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-buckets", type=int, default=2,
                    help="buckets in the oracle's CPU sample")
    return ap.parse_args()


# ---------------------------------------------------------------------------
# Distributed plumbing (replicas only)
# ---------------------------------------------------------------------------

def dist_setup(args):
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if torch.cuda.is_available():
            torch.cuda.set_device(local)
        dist.init_process_group(backend)
    return world, rank, local


L2_BYTES = 129 << 20   # GB300 L2


def host_memory_bytes() -> int:
    try:
        return os.sysconf("SC_PAGE_SIZE") * os.sysconf("SC_PHYS_PAGES")
    except (ValueError, OSError, AttributeError):
        return 1 << 62


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def aggregate_gbs(world: int, bytes_per_replica: int, slowest_ms: float) -> float:
    """Whole-job GB/s: every replica moved bytes_per_replica; the job took as
    long as its slowest rank."""
    return world * bytes_per_replica / (slowest_ms * 1e-3) / 1e9


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch
    import torch.distributed as dist
    dev = "cuda" if torch.cuda.is_available() else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


# ---------------------------------------------------------------------------
# Clocks during the timed region
# ---------------------------------------------------------------------------

class ClockSampler:
    """nvidia-smi sampling the GPU's clocks every 50 ms.

    It is started before the warm-up steps (nvidia-smi takes a few hundred ms
    to print its first row) and stopped after the last measurement.  Each row
    carries nvidia-smi's own timestamp, so rows are assigned to the timed
    region by when they were taken, not by when they arrived.  The summary is
    over the timed region's rows when there are at least three; a shorter
    region (a small workload's few ms) reports the rows of the whole window of
    GPU work instead, and says so."""
    FIELDS = ("timestamp,index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    MIN_ROWS = 3

    def __init__(self, gpu_index: int):
        self.gpu = gpu_index
        self.rows = []          # (seconds since the epoch, fields after the timestamp)
        self.proc = None
        self.window = None      # (start, end) of the timed region, seconds since the epoch

    def __enter__(self):
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "50", "-i", str(self.gpu)],
                stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            self.thread = threading.Thread(target=self._read, daemon=True)
            self.thread.start()
            atexit.register(self.__exit__, None, None, None)   # never outlive the bench
        except OSError:
            self.proc = None
        return self

    @staticmethod
    def _when(stamp: str):
        try:   # "2026/12/02 09:48:40.123", the host's local time
            day, frac = (stamp.split(".") + ["0"])[:2]
            return time.mktime(time.strptime(day, "%Y/%m/%d %H:%M:%S")) + float("0." + frac)
        except (ValueError, OverflowError):
            return None

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 10:
                self.rows.append((self._when(parts[0]), parts[1:]))

    def wait_first(self, timeout: float = 3.0):
        """Returns once nvidia-smi has printed a row (or after `timeout`)."""
        deadline = time.time() + timeout
        while self.proc and not self.rows and time.time() < deadline:
            time.sleep(0.02)

    def mark(self, start: float, end: float):
        self.window = (start, end)

    def __exit__(self, *exc):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except subprocess.TimeoutExpired:
                self.proc.kill()
            self.thread.join(timeout=2)

    def summary(self):
        rows, where = [r for _, r in self.rows], "bench run (no timed-region marks)"
        if self.window:
            a, b = self.window
            timed = [r for w, r in self.rows if w is not None and a <= w <= b]
            if len(timed) >= self.MIN_ROWS:
                rows, where = timed, "timed region"
            else:
                where = (f"warm-up to last measurement ({len(timed)} sample(s) in the "
                         f"{1e3 * (b - a):.0f} ms timed region)")
        if not rows:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["unsampled"]}
        sm = [float(r[1]) for r in rows if r[1].replace(".", "").isdigit()]
        mx = [float(r[2]) for r in rows if r[2].replace(".", "").isdigit()]
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        reasons = sorted({n for r in rows for n, v in zip(names, r[5:9])
                          if v.lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": max(mx) if mx else None,
                "reasons": reasons, "samples": len(rows), "window": where}


def visible_gpu_index(local_rank: int) -> int:
    vis = os.environ.get("CUDA_VISIBLE_DEVICES")
    if vis:
        ids = [v for v in vis.split(",") if v.strip()]
        if local_rank < len(ids) and ids[local_rank].strip().isdigit():
            return int(ids[local_rank])
    return local_rank


# ---------------------------------------------------------------------------
# Peaks and profile summaries
# ---------------------------------------------------------------------------

def same_run_copy_gbs(stream, nbytes: int = 4 << 30, reps: int = 5) -> float:
    """A plain device-to-device torch copy_ of nbytes (read + write counted), timed
    with CUDA events in this run: the copy ceiling of this GPU right now."""
    import torch
    a = torch.empty(nbytes, dtype=torch.uint8, device="cuda")
    b = torch.empty_like(a)
    a.fill_(1)
    with torch.cuda.stream(stream):
        for _ in range(3):
            b.copy_(a)
        e0 = torch.cuda.Event(enable_timing=True)
        e1 = torch.cuda.Event(enable_timing=True)
        e0.record(stream)
        for _ in range(reps):
            b.copy_(a)
        e1.record(stream)
    torch.cuda.synchronize()
    ms = e0.elapsed_time(e1) / reps
    del a, b
    return 2 * nbytes / (ms * 1e-3) / 1e9


def hbm_peak():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    try:
        with open(path) as f:
            return float(json.load(f)["hbm_gbs"]), "measured"
    except (OSError, KeyError, ValueError):
        return FALLBACK_HBM_GBS, "fallback"


KERNEL_SOURCES = ("include/rr.h", "paper_2512_22492_gb300/csrc/rr_device.cu",
                  "paper_2512_22492_gb300/csrc/rr_internal.h",
                  "paper_2512_22492_gb300/csrc/rr_plan.cpp")


def code_only(text: str) -> str:
    """C/C++/CUDA source with comments removed and white space collapsed, so
    that an edit of comments alone keeps a profile's figures current."""
    text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
    text = re.sub(r"//[^\n]*", " ", text)
    return " ".join(text.split())


def kernel_code_hash() -> str:
    """sha256 (first 16 hex digits) of the code of the kernels, of the planner
    that writes their work tables and of the item layouts they share: what a
    profile's DRAM figures depend on."""
    h = hashlib.sha256()
    for name in KERNEL_SOURCES:
        text = open(os.path.join(ROOT, name)).read()
        h.update(name.encode() + b"\0" + code_only(text).encode() + b"\0")
    return h.hexdigest()[:16]


def profiled_traffic(workload: str, algorithmic_bytes: int):
    """DRAM bytes per pack launch of `workload`, from the committed ncu summary
    if it was taken on the current code, else None.

    The counters are captured on a small case of the same kernel (the workload
    cut to its first decoder layers and a small vocabulary: a few GB on the
    device, above L2) and scaled to one full launch by the ratio of the two
    launches' algorithmic bytes; the summary records both figures.  Traffic
    grows with the bytes moved (every byte is read or written once), so the
    ratio carries over."""
    path = os.path.join(ROOT, "profiles", f"rr_pack_{workload}.md")
    try:
        text = open(path).read()
    except OSError:
        return None
    m_hash = re.search(r"kernel_code_sha256_16:\s*([0-9a-f]+)", text)
    m_dram = re.search(r"dram_bytes_per_launch_small:\s*([0-9]+)", text)
    m_alg = re.search(r"algorithmic_bytes_small:\s*([0-9]+)", text)
    if not (m_hash and m_dram and m_alg) or m_hash.group(1) != kernel_code_hash():
        return None
    return round(int(m_dram.group(1)) * algorithmic_bytes / int(m_alg.group(1)))


# ---------------------------------------------------------------------------
# CPU oracle (baseline leg and the reference arm)
# ---------------------------------------------------------------------------

def oracle_sample_setup(w, bucket_bytes):
    """Oracle layout and host shards whose leading bytes (enough for the first
    buckets' sources) hold the seeded values; the rest are lazily zeroed."""
    import numpy as np
    import oracle
    import synth
    L = oracle.workload_layout(w, bucket_bytes=bucket_bytes)
    need = 8 * bucket_bytes          # covers a few buckets' fp32 sources
    flat = np.zeros(L.shard_bytes * L.n_shards, np.uint8)
    for p, (_, _, es) in enumerate(L.params):
        off = int(L.param_offset[p])
        if off >= need:
            break
        n = min(L.param_numel(p), (need - off) // es)
        flat[off:off + n * es] = synth.values_host(n, es, w.seed, off // es, w.specials).view(
            np.uint8)
    shards = [flat[s * L.shard_bytes:(s + 1) * L.shard_bytes] for s in range(L.n_shards)]
    return L, oracle.Source(shards=shards), shards


def oracle_time(L, src, first, count):
    t0 = time.perf_counter()
    moved = L.sync_sample(src, first, count)
    return moved, time.perf_counter() - t0


def cpu_model() -> str:
    """The host CPU's model name (Linux), or the architecture."""
    import platform
    try:
        with open("/proc/cpuinfo") as f:
            for line in f:
                key = line.split(":")[0].strip().lower()
                if key in ("model name", "cpu model", "hardware"):
                    return line.split(":", 1)[1].strip()
        out = subprocess.run(["lscpu"], capture_output=True, text=True, timeout=10).stdout
        for line in out.splitlines():
            if line.lower().startswith("model name"):
                return line.split(":", 1)[1].strip()
    except (OSError, subprocess.SubprocessError):
        pass
    return platform.machine()


def cpu_baseline(w, bucket_bytes, n_buckets_sample):
    L, src, _keep = oracle_sample_setup(w, bucket_bytes)
    moved, dt = oracle_time(L, src, 0, n_buckets_sample)
    return {"value": round(moved / dt / 1e9, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
            "sample": f"buckets 0..{n_buckets_sample - 1} of {L.n_buckets} "
                      f"({n_buckets_sample} x {bucket_bytes >> 20} MiB): pack, unpack of their "
                      f"elements, verify; single-threaded C oracle; {moved / 1e9:.3f} GB in "
                      f"{dt:.2f} s; 1 of {os.cpu_count()} host cores ({cpu_model()})"}


def workload_config(w, bucket_bytes: int, n_buckets: int, pack_read: int, dst_bytes: int,
                    world: int) -> dict:
    """The JSON line's `config`: the workload alone, the same on both arms.
    Its byte counts are the step's algorithmic bytes: pack reads `pack_read`
    source bytes and writes every bucket byte; the receiver reads every bucket
    byte and writes `dst_bytes` of tensors."""
    buckets = n_buckets * bucket_bytes
    step_bytes = pack_read + 2 * buckets + dst_bytes
    resident = pack_read + buckets + dst_bytes
    return {"workload": w.name, "src_dtype": w.src_dtype,
            "dst_dtype": getattr(w, "dst_dtype", "bf16"), "n_shards": w.n_shards,
            "sharding": w.sharding, "expert_parallel": w.ep, "tp": w.tp,
            "bucket_bytes": bucket_bytes, "n_buckets": n_buckets, "step_bytes": step_bytes,
            "l2": ("inputs > L2 (no flush needed)" if resident >= 4 * L2_BYTES else
                   "L2 flushed between steps (512 MiB write outside the step's events)"),
            "parallelism": f"replicas{world}"}


def oracle_config(L, w, bucket_bytes: int, world: int) -> dict:
    """workload_config from the oracle's own layout: every destination element
    reads one source element of its parameter's width and writes 2 bytes."""
    pack_read = sum(nr * nc * L.params[p][2]
                    for _, _, blocks in L.tensors for p, _, nr, _, nc in blocks)
    dst_bytes = 2 * int(sum(L.tensor_numel[:len(L.tensors)]))
    return workload_config(w, bucket_bytes, int(L.n_buckets), int(pack_read), dst_bytes, world)


def path_dtype(w) -> str:
    """What the path computes: an fp32 source is rounded to bf16 (nearest,
    ties to even, in integer arithmetic); a bf16 source is copied bit for bit.
    For a float16 rollout either source is rounded to IEEE binary16."""
    if getattr(w, "dst_dtype", "bf16") == "f16":
        return "f32->f16 (RNE)" if w.src_dtype == "f32" else "bf16->f16 (RNE)"
    return "f32->bf16 (RNE)" if w.src_dtype == "f32" else "bf16 (bit copy)"


def run_reference(args, w, bucket_bytes, world, rank):
    if rank != 0:
        return
    L, src, _keep = oracle_sample_setup(w, bucket_bytes)
    count = 1
    for _ in range(args.warmup):
        oracle_time(L, src, 0, count)
    moved_total, t_total = 0, 0.0
    for _ in range(args.steps):
        moved, dt = oracle_time(L, src, 0, count)
        moved_total += moved
        t_total += dt
    value = moved_total / t_total / 1e9
    line = {
        "impl": "reference", "metric": METRIC, "value": round(value, 4), "unit": UNIT,
        "n_gpus": args.gpus, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": round(t_total / args.steps * 1e3, 3), "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": path_dtype(w), "data": "synthetic",
        "config": oracle_config(L, w, bucket_bytes, args.gpus),
        "path": {"step": f"oracle sync of bucket 0 of {L.n_buckets} per step (a bounded "
                         f"sample of the workload)"},
        "cpu_baseline": {"value": round(value, 4), "unit": UNIT, "cores": 1, "kind": "oracle",
                         "sample": f"bucket 0 of {L.n_buckets} ({bucket_bytes >> 20} MiB): "
                                   "pack, unpack of its elements, verify per step"},
        "e2e": {"value": round(value, 4), "unit": UNIT, "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------------------
# GPU arm
# ---------------------------------------------------------------------------

def _event_ms(fn, stream, reps=3):
    """Mean CUDA-event time of fn() over reps launches after one warm-up."""
    import torch
    fn()
    torch.cuda.synchronize()
    ms = []
    for _ in range(reps):
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        fn()
        b.record(stream)
        torch.cuda.synchronize()
        ms.append(a.elapsed_time(b))
    return statistics.mean(ms)


def next_rows(rr, H, w, plan, buf, t_src, t_bkt, t_dst, stream, peak):
    """Timings of the paths beyond the step: a resumed pull (the middle third of
    the buckets packed and checked-unpacked again, Section 5.2.2; with TP > 1,
    also one rank's buckets packed again), a relay
    re-pack (a rollout holding the TP=1 image serves a TP=4 one straight from
    the buckets it pulled, Section 5.2.1), and the pack for a float16 rollout.
    Algorithmic bytes as for the step."""
    import numpy as np
    import torch
    out = {}
    items, _ = plan.export_pack()

    def pack_range(b0, n):
        # Algorithmic bytes of a range pack: its items' source reads and its
        # whole buckets written.
        sel = (items["bucket"] >= b0) & (items["bucket"] < b0 + n) & (items["kind"] <= 3)
        es = np.where(items["kind"][sel] <= 1, 4, 2)
        read = int((items["row_len"][sel].astype(np.int64) * items["n_rows"][sel] * es).sum())
        wrote = n * plan.bucket_bytes
        ms = _event_ms(lambda: rr.rr_pack_range(plan, b0, n, t_src, t_bkt, buf.checksums,
                                                stream), stream)
        gbs = (read + wrote) / (ms * 1e-3) / 1e9
        return {"buckets": [b0, b0 + n], "ms": round(ms, 3), "bytes": read + wrote,
                "GB/s": round(gbs, 1), "frac_of_peak": round(gbs / peak, 4)}, wrote

    n = plan.n_buckets // 3
    b0 = n
    if n:
        out["resume_pack_range"], wrote = pack_range(b0, n)
        uitems, _ = plan.export_unpack()
        usel = ((uitems["bucket"] >= b0) & (uitems["bucket"] < b0 + n)
                & ((uitems["kind"] == 6) | (uitems["kind"] == 7)))
        uwrote = int(uitems["nbytes"][usel].astype(np.int64).sum())

        def uv():
            n_bad, _ = rr.rr_unpack_verify(plan, t_bkt, buf.checksums, t_dst, stream=stream,
                                           first_bucket=b0, n_buckets=n)
            if n_bad:
                raise RuntimeError("resumed range failed its checksums")
        ms = _event_ms(uv, stream)
        gbs = (wrote + uwrote) / (ms * 1e-3) / 1e9
        out["resume_unpack_verify_range"] = {"buckets": [b0, b0 + n], "ms": round(ms, 3),
                                             "bytes": wrote + uwrote, "GB/s": round(gbs, 1),
                                             "frac_of_peak": round(gbs / peak, 4)}
    if plan.tp > 1:
        # A rollout rank that reconnects pulls its own buckets only (Section
        # 5.2.2): rank tp/2's whole range.
        r = plan.tp // 2
        fb = list(plan.first_bucket_of_rank) + [plan.n_buckets]
        if fb[r + 1] > fb[r]:
            row, _ = pack_range(fb[r], fb[r + 1] - fb[r])
            out["resume_one_rank_pack_range"] = {"rank": r, **row}
    if w.tp == 1 and plan.bucket_bytes % 16 == 0:
        from paper_2512_22492_gb300 import layouts
        m2, s2, d2 = layouts.qwen3_relay(w.shape, 1, 4, from_plan=plan)
        relay = rr.rr_plan_create(m2, s2, d2, plan.bucket_bytes)
        rst = relay.stats()
        store = torch.empty((relay.n_buckets, plan.bucket_bytes), dtype=torch.uint8,
                            device="cuda")
        cs = torch.zeros(relay.n_buckets, dtype=torch.int64, device="cuda")
        r_src = rr.Pointers(relay, "src_shards", buf.buckets)
        ms = _event_ms(lambda: rr.rr_pack(relay, r_src, store, cs, stream), stream)
        nbytes = rst["pack_bytes_read"] + rst["pack_bytes_written"]
        gbs = nbytes / (ms * 1e-3) / 1e9
        out["relay_repack_tp1_to_tp4"] = {"source": "the TP=1 buckets as pulled",
                                          "n_buckets": relay.n_buckets, "ms": round(ms, 3),
                                          "bytes": nbytes, "GB/s": round(gbs, 1),
                                          "frac_of_peak": round(gbs / peak, 4)}
        del store, cs, r_src, relay
    if getattr(w, "dst_dtype", "bf16") == "bf16":
        # The same sync for a float16 rollout (Section 7.4 counts the transferred
        # model as FP16): the same tables and bytes, the float16 cast.  Its pack
        # overwrites the step's buckets, which nothing reads after this.
        m2, s2, d2 = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep,
                                   dst_dtype="f16")
        p16 = rr.rr_plan_create(m2, s2, d2, plan.bucket_bytes)
        cs16 = torch.zeros_like(buf.checksums)
        t16_src = rr.Pointers(p16, "src_shards", buf.shards)
        t16_bkt = rr.Pointers(p16, "buckets", buf.buckets)
        ms = _event_ms(lambda: rr.rr_pack(p16, t16_src, t16_bkt, cs16, stream), stream)
        n_bad, _ = rr.rr_verify(p16, t16_bkt, cs16, stream)
        if n_bad:
            raise RuntimeError("float16 pack: its buckets do not match its checksums")
        st16 = p16.stats()
        nbytes = st16["pack_bytes_read"] + st16["pack_bytes_written"]
        gbs = nbytes / (ms * 1e-3) / 1e9
        out["float16_rollout_pack"] = {"dtype": "f32->f16 (RNE)" if w.src_dtype == "f32"
                                       else "bf16->f16 (RNE)", "ms": round(ms, 3),
                                       "bytes": nbytes, "GB/s": round(gbs, 1),
                                       "frac_of_peak": round(gbs / peak, 4)}
        del p16, cs16, t16_src, t16_bkt
    return out


class BenchStep:
    """The timed step with its buffers: one plan for workload `w`, the source
    filled by the seeded device generator, pointer tables checked once (as a
    caller syncing every training step would hold them), and per step rr_pack
    followed by the receiver's verifying unpack on one stream.

    The receiver's check is stream-ordered by default: each step's {n_bad,
    first_bad} lands in its own row of `results`, read after the timing by
    check_results().  `sync_verify` uses the blocking rr_unpack_verify instead.
    `poison` (a byte) pre-fills buckets and tensors so that unwritten bytes
    show; None leaves them uninitialised."""

    def __init__(self, w, bucket_bytes, opts=None, sync_verify=False, n_rows=64, stream=None,
                 poison=None):
        import torch
        import paper_2512_22492_gb300 as rr
        from synth import device as D
        self.rr, self.w, self.sync_verify = rr, w, sync_verify
        self.stream = stream if stream is not None else torch.cuda.current_stream()
        m, s, d = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep,
                                dst_dtype=w.dst_dtype)
        self.manifest = m
        self.plan = plan = rr.rr_plan_create(m, s, d, bucket_bytes, opts)
        self.buf = buf = D.alloc(plan, poison=poison)
        D.fill_with_generator(buf, m, w.seed, w.specials)
        torch.cuda.synchronize()
        self.t_src = rr.Pointers(plan, "src_shards", buf.shards)
        self.t_bkt = rr.Pointers(plan, "buckets", buf.buckets)
        self.t_dst = rr.Pointers(plan, "dst", buf.dst)
        st = self.stats = plan.stats()
        self.pack_bytes = st["pack_bytes_read"] + st["pack_bytes_written"]
        self.unpack_bytes = st["unpack_bytes_read"] + st["unpack_bytes_written"]
        self.verify_bytes = st["verify_bytes_read"]
        # The receiver's fused pass reads every bucket byte once and writes every tensor byte.
        self.uv_bytes = st["verify_bytes_read"] + st["unpack_bytes_written"]
        self.step_bytes = self.pack_bytes + self.uv_bytes
        self.scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")
        self.n_rows = n_rows
        self.results = torch.full((n_rows, 2), -7, dtype=torch.int64, device="cuda")
        self.used = 0

    def step(self, ev=None):
        """Enqueues one sync; `ev` (three CUDA events) brackets pack and receiver.
        Returns the step's result row (None with sync_verify)."""
        rr, plan, stream = self.rr, self.plan, self.stream
        if ev:
            ev[0].record(stream)
        rr.rr_pack(plan, self.t_src, self.t_bkt, self.buf.checksums, stream)
        if ev:
            ev[1].record(stream)
        row = None
        if self.sync_verify:
            n_bad, _ = rr.rr_unpack_verify(plan, self.t_bkt, self.buf.checksums, self.t_dst,
                                           stream=stream)
            if n_bad:
                raise RuntimeError(f"verify found {n_bad} bad buckets")
        else:
            row = self.results[self.used % self.n_rows]
            self.used += 1
            rr.rr_unpack_verify_async(plan, self.t_bkt, self.buf.checksums, self.t_dst,
                                      self.scratch, row, stream=stream)
        if ev:
            ev[2].record(stream)
        return row

    def check_results(self):
        """Raises unless every step so far verified clean and no kernel of the
        plan gave up a bounded wait (which leaves its output incomplete without
        touching the result rows; the plan's error word says so)."""
        import torch
        torch.cuda.synchronize()
        got = self.results[:min(self.used, self.n_rows)].cpu()
        if self.used and not bool(((got[:, 0] == 0) & (got[:, 1] == -1)).all()):
            raise RuntimeError(f"verify found bad buckets: {got.tolist()}")
        self.rr.rr_plan_check(self.plan, self.stream)


# Pointers one launch carries in its kernel parameters (include/rr.h: a launch
# addresses at most 3968 buckets or destination tensors).
LAUNCH_POINTERS = 3968


def receiver_launches(plan) -> int:
    """Kernel launches of one verifying unpack over every bucket (equally spaced
    buckets): one, unless the buckets' destination tensors exceed one launch's
    pointer table; the call then runs over consecutive bucket ranges whose
    tensor windows fit, one launch each (the rule of include/rr.h), counted
    here from the exported unpack table."""
    import numpy as np
    items, _ = plan.export_unpack()
    copy = items[(items["kind"] == 6) | (items["kind"] == 7)]
    lo = np.full(plan.n_buckets, np.iinfo(np.int64).max, np.int64)
    hi = np.full(plan.n_buckets, -1, np.int64)
    np.minimum.at(lo, copy["bucket"].astype(np.int64), copy["tensor"].astype(np.int64))
    np.maximum.at(hi, copy["bucket"].astype(np.int64), copy["tensor"].astype(np.int64))
    n, b = 0, 0
    while b < plan.n_buckets:
        wlo, whi, e = np.iinfo(np.int64).max, -1, b
        while e < plan.n_buckets:
            nlo, nhi = min(wlo, lo[e]), max(whi, hi[e])
            if (nhi - nlo + 1 if nhi >= nlo else 0) > LAUNCH_POINTERS:
                break
            wlo, whi, e = nlo, nhi, e + 1
        n += 1
        b = max(e, b + 1)
    return n


def bucket_source_needs(plan) -> "np.ndarray":
    """Per bucket: how many leading bytes of the source block (every source
    buffer one after another at 16-byte starts, as synth.device lays them out)
    must have landed before the bucket can be packed -- the end of its farthest
    source row; 0 for a bucket of zero fill only.  From the exported pack table."""
    import numpy as np
    from synth import device as D
    items, _ = plan.export_pack()
    it = items[items["kind"] <= 3]             # the kinds that read the source
    starts = np.asarray(D.source_offsets(plan)[:-1], np.int64)
    src = it["src"].astype(np.uint64)
    shard = (src >> np.uint64(48)).astype(np.int64)
    off = (src & np.uint64((1 << 48) - 1)).astype(np.int64)
    es = np.where(it["kind"] <= 1, 4, 2).astype(np.int64)
    rows = np.maximum(it["n_rows"].astype(np.int64), 1)
    end = starts[shard] + off + ((rows - 1) * it["src_stride"].astype(np.int64)
                                 + it["row_len"].astype(np.int64)) * es
    need = np.zeros(plan.n_buckets, np.int64)
    np.maximum.at(need, it["bucket"].astype(np.int64), end)
    return need


def ready_runs(ready) -> list:
    """Maximal runs [b0, b1) of consecutive True entries."""
    runs, b, n = [], 0, len(ready)
    while b < n:
        if ready[b]:
            e = b
            while e < n and ready[e]:
                e += 1
            runs.append((b, e))
            b = e
        else:
            b += 1
    return runs


class PipelinedE2E:
    """The step end to end through the public API, with the trainer's shards in
    pinned host memory: each step copies the source block host -> device in
    `pieces` pieces on a copy stream, and on the step's stream -- as soon as a
    piece has landed (an event) -- packs every run of buckets whose sources
    have all arrived (rr_pack_range) and hands the run to the receiver
    (rr_unpack_verify_async on that range, its {n_bad, first_bad} in its own
    result row).  The step ends with the checksums and the result rows read
    back to pinned host memory.  The next step's copy waits only for this
    step's last pack, so it overlaps this step's last receiver pass.  Every
    bucket is packed and checked exactly once per step."""

    def __init__(self, bs, host_src, pieces: int = 16, ring_steps: int = 64):
        import numpy as np
        import torch
        self.bs = bs
        plan, buf = bs.plan, bs.buf
        total = buf.flat.numel()
        self.host_src = host_src
        need = bucket_source_needs(plan)
        self.cuts = sorted({min(total, (total * (k + 1) // pieces + 15) // 16 * 16)
                            for k in range(pieces)})
        done = np.zeros(plan.n_buckets, bool)
        self.schedule = []
        for c in self.cuts:
            runs = ready_runs((~done) & (need <= c))
            for b0, b1 in runs:
                done[b0:b1] = True
            self.schedule.append(runs)
        assert done.all() and self.cuts[-1] == total
        self.n_ranges = sum(len(r) for r in self.schedule)
        self.ring = ring_steps
        self.results = torch.full((ring_steps * self.n_ranges, 2), -7, dtype=torch.int64,
                                  device="cuda")
        self.host_cs = torch.empty(buf.checksums.numel(), dtype=torch.int64, pin_memory=True)
        self.host_res = torch.empty((self.n_ranges, 2), dtype=torch.int64, pin_memory=True)
        self.copy_stream = torch.cuda.Stream()
        self.packed = torch.cuda.Event()       # after the last pack enqueued so far
        self.packed.record(bs.stream)
        self.used = 0
        self.h2d_bytes = total
        self.d2h_bytes = self.host_cs.numel() * 8 + self.host_res.numel() * 8

    def step(self):
        import torch
        bs, rr = self.bs, self.bs.rr
        plan, s, cs = bs.plan, bs.stream, self.copy_stream
        cs.wait_event(self.packed)      # the previous step has read the source it overwrites
        landed, prev = [], 0
        with torch.cuda.stream(cs):
            for c in self.cuts:
                bs.buf.flat[prev:c].copy_(self.host_src[prev:c], non_blocking=True)
                e = torch.cuda.Event()
                e.record(cs)
                landed.append(e)
                prev = c
        base = (self.used % self.ring) * self.n_ranges
        self.used += 1
        j = 0
        for e, runs in zip(landed, self.schedule):
            s.wait_event(e)
            for b0, b1 in runs:
                rr.rr_pack_range(plan, b0, b1 - b0, bs.t_src, bs.t_bkt, bs.buf.checksums, s)
                self.packed.record(s)
                rr.rr_unpack_verify_async(plan, bs.t_bkt, bs.buf.checksums, bs.t_dst, bs.scratch,
                                          self.results[base + j], stream=s, first_bucket=b0,
                                          n_buckets=b1 - b0)
                j += 1
        with torch.cuda.stream(s):
            self.host_cs.copy_(bs.buf.checksums, non_blocking=True)
            self.host_res.copy_(self.results[base:base + self.n_ranges], non_blocking=True)

    def check(self):
        import torch
        torch.cuda.synchronize()
        got = self.results[:min(self.used, self.ring) * self.n_ranges].cpu()
        if self.used and not bool(((got[:, 0] == 0) & (got[:, 1] == -1)).all()):
            raise RuntimeError(f"e2e: verify found bad buckets: {got.tolist()}")
        if not bool(((self.host_res[:, 0] == 0) & (self.host_res[:, 1] == -1)).all()):
            raise RuntimeError("e2e: the last step's result rows read back are not clean")
        self.bs.rr.rr_plan_check(self.bs.plan, self.bs.stream)

    def h2d_ceiling_ms(self, reps: int = 2) -> float:
        """One copy of the whole source block host -> device, timed alone on the
        copy stream (best of `reps`): what the link allows this step."""
        import torch
        ms = []
        for _ in range(reps):
            a = torch.cuda.Event(enable_timing=True)
            b = torch.cuda.Event(enable_timing=True)
            with torch.cuda.stream(self.copy_stream):
                a.record(self.copy_stream)
                self.bs.buf.flat.copy_(self.host_src, non_blocking=True)
                b.record(self.copy_stream)
            torch.cuda.synchronize()
            ms.append(a.elapsed_time(b))
        return min(ms)


class DirectE2E:
    """The step end to end with the trainer's shards left in pinned host memory
    and read by the pack itself: given host source pointers, rr_pack runs the
    register path, whose loads cross NVLink-C2C, so no copy engine is involved
    and the source never lands in HBM.  The buckets are cut into `pieces`
    ranges packed one after another (rr_pack_range) on the step's stream; a
    receiver stream of higher priority runs the verifying unpack of each range
    (rr_unpack_verify_async, its own result row) as soon as that range is
    packed, so the receiver overlaps the next range's pack.  The step ends with
    the checksums and the result rows read back to pinned host memory, and the
    step's stream waits for the receiver, so events on it bracket everything."""

    def __init__(self, bs, host_src, pieces: int = 16, ring_steps: int = 64):
        import torch
        from synth import device as D
        self.bs = bs
        plan = bs.plan
        starts = D.source_offsets(plan)
        self.host_src = host_src
        views = [host_src[starts[i]:starts[i] + nb]
                 for i, nb in enumerate(plan.source_buffer_bytes)]
        self.t_host = bs.rr.Pointers(plan, "src_shards", views)
        nb = plan.n_buckets
        pieces = max(1, min(pieces, nb))
        self.ranges = [(nb * k // pieces, nb * (k + 1) // pieces) for k in range(pieces)]
        self.ranges = [r for r in self.ranges if r[1] > r[0]]
        self.n_ranges = len(self.ranges)
        self.ring = ring_steps
        self.results = torch.full((ring_steps * self.n_ranges, 2), -7, dtype=torch.int64,
                                  device="cuda")
        self.scratch = torch.zeros(nb + 4, dtype=torch.int64, device="cuda")
        self.host_cs = torch.empty(bs.buf.checksums.numel(), dtype=torch.int64, pin_memory=True)
        self.host_res = torch.empty((self.n_ranges, 2), dtype=torch.int64, pin_memory=True)
        _least, greatest = torch.cuda.Stream.priority_range()   # lower number: higher priority
        self.recv = torch.cuda.Stream(priority=greatest)
        self.received = torch.cuda.Event()     # after the last step's receiver and read-back
        self.received.record(self.recv)
        self.used = 0
        # Nothing is copied: the pack's own loads read the source over the link.
        self.h2d_bytes = int(bs.stats["pack_bytes_read"])
        self.d2h_bytes = self.host_cs.numel() * 8 + self.host_res.numel() * 8

    def step(self):
        import torch
        bs, rr = self.bs, self.bs.rr
        plan, s, r = bs.plan, bs.stream, self.recv
        cs = bs.buf.checksums
        s.wait_event(self.received)     # the last step's receiver has read what this overwrites
        base = (self.used % self.ring) * self.n_ranges
        self.used += 1
        for j, (b0, b1) in enumerate(self.ranges):
            rr.rr_pack_range(plan, b0, b1 - b0, self.t_host, bs.t_bkt, cs, s)
            e = torch.cuda.Event()
            e.record(s)
            r.wait_event(e)
            rr.rr_unpack_verify_async(plan, bs.t_bkt, cs, bs.t_dst, self.scratch,
                                      self.results[base + j], stream=r, first_bucket=b0,
                                      n_buckets=b1 - b0)
        with torch.cuda.stream(r):
            self.host_cs.copy_(cs, non_blocking=True)
            self.host_res.copy_(self.results[base:base + self.n_ranges], non_blocking=True)
        self.received.record(r)
        s.wait_event(self.received)

    def check(self):
        import torch
        torch.cuda.synchronize()
        got = self.results[:min(self.used, self.ring) * self.n_ranges].cpu()
        if self.used and not bool(((got[:, 0] == 0) & (got[:, 1] == -1)).all()):
            raise RuntimeError(f"e2e (direct): verify found bad buckets: {got.tolist()}")
        if not bool(((self.host_res[:, 0] == 0) & (self.host_res[:, 1] == -1)).all()):
            raise RuntimeError("e2e (direct): the last step's result rows read back are not clean")
        self.bs.rr.rr_plan_check(self.bs.plan, self.bs.stream)


def time_e2e(route, steps, world, stream):
    """Mean ms per step of `route` over `steps` steps after two warm-up steps,
    the slowest rank's, with the result rows checked afterwards."""
    import torch
    for _ in range(2):
        route.step()
    torch.cuda.synchronize()
    barrier(world)
    a = torch.cuda.Event(enable_timing=True)
    b = torch.cuda.Event(enable_timing=True)
    a.record(stream)
    if isinstance(route, PipelinedE2E):
        route.packed.record(stream)     # the first copy starts inside the timed region
    for _ in range(steps):
        route.step()
    b.record(stream)
    torch.cuda.synchronize()
    ms = max_over_ranks(a.elapsed_time(b), world) / steps
    route.check()
    return ms


def run_native(args, w, bucket_bytes, world, rank, local):
    import torch
    import paper_2512_22492_gb300 as rr
    from synth import device as H

    torch.cuda.set_device(local)
    stream = torch.cuda.current_stream()
    opts = None
    if args.chunk_kib or args.grid or args.engine != "auto" or args.check_items:
        opts = rr.PlanOptions(chunk_bytes=args.chunk_kib * 1024, grid_blocks=args.grid,
                              engine=args.engine, check_items=args.check_items)
    bs = BenchStep(w, bucket_bytes, opts, sync_verify=args.sync_verify,
                   n_rows=2 * (max(3, args.warmup) + args.steps) + 8, stream=stream)
    plan, buf, st = bs.plan, bs.buf, bs.stats
    t_src, t_bkt, t_dst = bs.t_src, bs.t_bkt, bs.t_dst
    pack_bytes, unpack_bytes, verify_bytes = bs.pack_bytes, bs.unpack_bytes, bs.verify_bytes
    uv_bytes, step_bytes = bs.uv_bytes, bs.step_bytes
    step, check_results = bs.step, bs.check_results

    # Clocks: sampled from before the warm-up to the last measurement.
    clk = ClockSampler(visible_gpu_index(local)).__enter__()
    clk.wait_first()
    for _ in range(max(3, args.warmup)):
        step()
    torch.cuda.synchronize()

    # Inputs smaller than a few L2 sizes would be served from L2 on the next
    # step: flush it between steps (a 512 MiB write outside the step's events)
    # and take the step time from those events.
    config = workload_config(w, bucket_bytes, plan.n_buckets, st["pack_bytes_read"],
                             st["unpack_bytes_written"], world)
    assert config["step_bytes"] == step_bytes
    flush = None
    if config["l2"].startswith("L2 flushed"):
        flush = torch.empty(512 << 20, dtype=torch.uint8, device="cuda")
    evs = [[torch.cuda.Event(enable_timing=True) for _ in range(3)] for _ in range(args.steps)]
    barrier(world)
    torch.cuda.synchronize()
    t0 = torch.cuda.Event(enable_timing=True)
    t1 = torch.cuda.Event(enable_timing=True)
    wall0 = time.time()
    t0.record(stream)
    for k in range(args.steps):
        if flush is not None:
            flush.fill_(k & 0xFF)
        step(evs[k])
    t1.record(stream)
    torch.cuda.synchronize()
    clk.mark(wall0, time.time())
    barrier(world)
    pack_all = [e[0].elapsed_time(e[1]) for e in evs]
    uv_all = [e[1].elapsed_time(e[2]) for e in evs]
    pack_ms = statistics.mean(pack_all)
    uv_ms = statistics.mean(uv_all)
    if flush is None:
        total_ms = max_over_ranks(t0.elapsed_time(t1), world)
    else:
        total_ms = max_over_ranks(sum(e[0].elapsed_time(e[2]) for e in evs), world)
        del flush
    ms_per_step = total_ms / args.steps
    value = aggregate_gbs(world, step_bytes, ms_per_step)
    check_results()

    # Breakdown only (not part of the step): the receiver's two separate calls.
    # rr_unpack is asynchronous, so its launches are timed back to back; rr_verify
    # returns its count to the host, so each call is timed on its own.
    for _ in range(2):
        rr.rr_unpack(plan, t_bkt, t_dst, stream)
        rr.rr_verify(plan, t_bkt, buf.checksums, stream)
    reps = 3
    u = [torch.cuda.Event(enable_timing=True) for _ in range(reps + 1)]
    u[0].record(stream)
    for k in range(reps):
        rr.rr_unpack(plan, t_bkt, t_dst, stream)
        u[k + 1].record(stream)
    v = [[torch.cuda.Event(enable_timing=True) for _ in range(2)] for _ in range(reps)]
    for e in v:
        e[0].record(stream)
        rr.rr_verify(plan, t_bkt, buf.checksums, stream)
        e[1].record(stream)
    torch.cuda.synchronize()
    unpack_ms = statistics.mean(u[k].elapsed_time(u[k + 1]) for k in range(reps))
    verify_ms = statistics.mean(e[0].elapsed_time(e[1]) for e in v)

    # Checkpoint snapshot: rr_pack writing the buckets into pinned host memory.
    snapshot = None
    if args.snapshot:
        row = (plan.bucket_bytes + 15) // 16 * 16
        hstore = torch.empty((plan.n_buckets, row), dtype=torch.uint8, pin_memory=True)
        hview = hstore[:, :plan.bucket_bytes]
        hcs = torch.zeros_like(buf.checksums)
        rr.rr_pack(plan, t_src, hview, hcs, stream)
        torch.cuda.synchronize()
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        reps = 3
        a.record(stream)
        for _ in range(reps):
            rr.rr_pack(plan, t_src, hview, hcs, stream)
        b.record(stream)
        torch.cuda.synchronize()
        s_ms = a.elapsed_time(b) / reps
        # Versus packing on the device and copying the buckets out.
        c = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        c.record(stream)
        for _ in range(reps):
            rr.rr_pack(plan, t_src, t_bkt, buf.checksums, stream)
            hstore.copy_(buf.bucket_store, non_blocking=True)
        e.record(stream)
        torch.cuda.synchronize()
        c_ms = c.elapsed_time(e) / reps
        # Restore: the verifying unpack straight from the host snapshot (the
        # register path reads the pinned buckets over the link), against a
        # plain copy of the same bucket bytes host -> device in this run.
        n_bad, _ = rr.rr_unpack_verify(plan, hview, hcs, t_dst, stream=stream)
        if n_bad:
            raise RuntimeError(f"snapshot restore: {n_bad} bad buckets")
        r_ms = _event_ms(lambda: rr.rr_unpack_verify(plan, hview, hcs, t_dst, stream=stream),
                         stream)
        h2d_ms = _event_ms(lambda: buf.bucket_store.copy_(hstore, non_blocking=True), stream,
                           reps=2)
        restore_bytes = st["verify_bytes_read"] + st["unpack_bytes_written"]
        snapshot = {"pack_to_host_ms": round(s_ms, 2),
                    "host_GB/s": round(st["pack_bytes_written"] / (s_ms * 1e-3) / 1e9, 1),
                    "pack_then_copy_ms": round(c_ms, 2),
                    "identical": bool(torch.equal(hcs, buf.checksums)),
                    "restore_ms": round(r_ms, 2),
                    "restore_GB/s": round(restore_bytes / (r_ms * 1e-3) / 1e9, 1),
                    "restore_link_GB/s": round(st["verify_bytes_read"] / (r_ms * 1e-3) / 1e9, 1),
                    "h2d_ceiling": {"ms": round(h2d_ms, 2),
                                    "GB/s": round(buf.bucket_store.numel() / (h2d_ms * 1e-3) / 1e9, 1),
                                    "restore_frac": round(h2d_ms / r_ms, 4),
                                    "method": "copy of the pinned snapshot's bucket block host -> "
                                              "device, mean of 2 after one warm-up"}}
        del hstore, hview
        # The same into ordinary (pageable) host memory, where the GPU reaches it
        # through the CPU's page tables (Grace); elsewhere the call is refused.
        pstore = torch.empty((plan.n_buckets, row), dtype=torch.uint8)
        pstore.fill_(0)
        pview = pstore[:, :plan.bucket_bytes]
        pcs = torch.zeros_like(buf.checksums)
        try:
            p_ms = _event_ms(lambda: rr.rr_pack(plan, t_src, pview, pcs, stream), stream)
            n_bad, _ = rr.rr_unpack_verify(plan, pview, pcs, t_dst, stream=stream)
            if n_bad:
                raise RuntimeError(f"pageable snapshot restore: {n_bad} bad buckets")
            pr_ms = _event_ms(lambda: rr.rr_unpack_verify(plan, pview, pcs, t_dst,
                                                          stream=stream), stream)
            snapshot["pageable"] = {
                "pack_to_host_ms": round(p_ms, 2),
                "host_GB/s": round(st["pack_bytes_written"] / (p_ms * 1e-3) / 1e9, 1),
                "identical": bool(torch.equal(pcs, buf.checksums)),
                "restore_ms": round(pr_ms, 2),
                "restore_link_GB/s": round(st["verify_bytes_read"] / (pr_ms * 1e-3) / 1e9, 1),
                "how": "snapshot into and restore from unpinned host memory (mean of 3 "
                       "after one warm-up)"}
        except rr.RRError as exc:
            snapshot["pageable"] = {"refused": str(exc).splitlines()[0]}
        del pstore, pview
        # The device buckets were overwritten by the ceiling copy: pack them again.
        rr.rr_pack(plan, t_src, t_bkt, buf.checksums, stream)
        torch.cuda.synchronize()

    # End to end through the public API with host buffers: every step copies the
    # trainer's shards from pinned host memory, syncs, and reads back the checksums.
    e2e = None
    local_ranks = int(os.environ.get("LOCAL_WORLD_SIZE", str(world)))
    pinned_need = local_ranks * buf.flat.numel()
    if not args.no_e2e and pinned_need > host_memory_bytes() // 2:
        # Every local rank would pin its whole source on the host: refuse
        # rather than exhaust the node's memory.
        e2e = {"skipped": f"{local_ranks} ranks x {buf.flat.numel() / 1e9:.1f} GB of pinned "
                          f"host memory exceed half of this host's "
                          f"{host_memory_bytes() / 1e9:.0f} GB"}
    elif not args.no_e2e and args.sync_verify:
        # The blocking receiver waits on the host every step: copy, then sync.
        host_src = torch.empty(buf.flat.numel(), dtype=torch.uint8, pin_memory=True)
        host_src.copy_(buf.flat)
        host_cs = torch.empty(buf.checksums.numel(), dtype=torch.int64, pin_memory=True)
        h2d, d2h = host_src.numel(), host_cs.numel() * 8

        def e2e_step():
            buf.flat.copy_(host_src, non_blocking=True)
            step()
            host_cs.copy_(buf.checksums, non_blocking=True)

        for _ in range(2):
            e2e_step()
        torch.cuda.synchronize()
        barrier(world)
        a = torch.cuda.Event(enable_timing=True)
        b = torch.cuda.Event(enable_timing=True)
        a.record(stream)
        for _ in range(args.steps):
            e2e_step()
        b.record(stream)
        torch.cuda.synchronize()
        e2e_ms = max_over_ranks(a.elapsed_time(b), world) / args.steps
        check_results()
        e2e = {"value": round(aggregate_gbs(world, step_bytes, e2e_ms), 2), "unit": UNIT,
               "h2d_bytes_per_step": h2d, "d2h_bytes_per_step": d2h,
               "ms_per_step": round(e2e_ms, 3), "pipelined": False}
        del host_src
    elif not args.no_e2e:
        # Routes for the source, all through the public API and all timed:
        # copy engines (the source copied into HBM in pieces, each piece packed
        # as it lands), direct (the pack reads the pinned shards itself) and
        # direct from pageable memory (below).  Which is fastest depends on the
        # machine: where the copy engines run below the link, the SMs' own
        # loads still reach it.  The line reports the fastest and carries all.
        host_src = torch.empty(buf.flat.numel(), dtype=torch.uint8, pin_memory=True)
        host_src.copy_(buf.flat)
        routes = {}
        if args.e2e_route in ("auto", "copy"):
            pe = PipelinedE2E(bs, host_src, pieces=args.e2e_pieces)
            ms = time_e2e(pe, args.steps, world, stream)
            h2d_ms = pe.h2d_ceiling_ms()
            routes["copy_engine"] = {
                "ms_per_step": round(ms, 3), "h2d_bytes_per_step": pe.h2d_bytes,
                "d2h_bytes_per_step": pe.d2h_bytes, "pieces": len(pe.cuts),
                "bucket_ranges_per_step": pe.n_ranges,
                "h2d_ceiling": {"ms": round(h2d_ms, 3),
                                "GB/s": round(pe.h2d_bytes / (h2d_ms * 1e-3) / 1e9, 1),
                                "e2e_frac": round(h2d_ms / ms, 4),
                                "method": "one copy of the whole pinned source block host -> "
                                          "device, alone on the copy stream, best of 2"}}
            del pe
        if args.e2e_route in ("auto", "direct"):
            de = DirectE2E(bs, host_src, pieces=args.e2e_direct_pieces)
            ms = time_e2e(de, args.steps, world, stream)
            routes["direct"] = {
                "ms_per_step": round(ms, 3), "h2d_bytes_per_step": de.h2d_bytes,
                "d2h_bytes_per_step": de.d2h_bytes, "bucket_ranges_per_step": de.n_ranges,
                "link_GB/s": round(de.h2d_bytes / (ms * 1e-3) / 1e9, 1),
                "how": "rr_pack_range reads the pinned host shards (register path over "
                       "NVLink-C2C); the receiver overlaps on a second stream"}
            del de
        refused = {}
        if args.e2e_route in ("auto", "pageable") and 2 * pinned_need <= host_memory_bytes() // 2:
            # The direct route from ordinary (pageable) host memory: a GPU that
            # reads it through the CPU's page tables (Grace) needs no pinning;
            # elsewhere the library refuses it before launching anything.
            pageable = torch.empty(buf.flat.numel(), dtype=torch.uint8)
            pageable.copy_(buf.flat)
            try:
                de = DirectE2E(bs, pageable, pieces=args.e2e_direct_pieces)
                ms = time_e2e(de, args.steps, world, stream)
                routes["direct_pageable"] = {
                    "ms_per_step": round(ms, 3), "h2d_bytes_per_step": de.h2d_bytes,
                    "d2h_bytes_per_step": de.d2h_bytes, "bucket_ranges_per_step": de.n_ranges,
                    "link_GB/s": round(de.h2d_bytes / (ms * 1e-3) / 1e9, 1),
                    "how": "as direct, from pageable (unpinned) host memory"}
                del de
            except rr.RRError as exc:
                refused["direct_pageable"] = str(exc).splitlines()[0]
            del pageable
        best = min(routes, key=lambda k: routes[k]["ms_per_step"])
        e2e_ms = routes[best]["ms_per_step"]
        e2e = {"value": round(aggregate_gbs(world, step_bytes, e2e_ms), 2), "unit": UNIT,
               "h2d_bytes_per_step": routes[best]["h2d_bytes_per_step"],
               "d2h_bytes_per_step": routes[best]["d2h_bytes_per_step"],
               "ms_per_step": e2e_ms, "route": best, "pipelined": True,
               "routes": routes}
        if refused:
            e2e["refused_routes"] = refused
        if "copy_engine" in routes:
            ceil_ms = routes["copy_engine"]["h2d_ceiling"]["ms"]
            e2e["h2d_ceiling_frac"] = round(ceil_ms / e2e_ms, 4)
        del host_src

    peak, peak_kind = hbm_peak()
    more = None if args.no_next_rows else next_rows(rr, H, w, plan, buf, t_src, t_bkt, t_dst,
                                                    stream, peak)
    copy_gbs = same_run_copy_gbs(stream)
    pack_gbs = pack_bytes / (pack_ms * 1e-3) / 1e9
    traffic = (profiled_traffic(w.name, pack_bytes)
               if bucket_bytes == w.bucket_bytes and args.engine == "auto" else None)
    clk.__exit__(None, None, None)
    clocks = clk.summary()
    line = {
        "metric": METRIC, "value": round(value, 2), "unit": UNIT, "n_gpus": world,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": round(ms_per_step, 3),
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": path_dtype(w),
        "data": "synthetic",
        "config": config,
        "path": {"step": "rr_pack + rr_unpack_verify" + ("" if args.sync_verify else "_async") +
                         " (unpack and checksum check fused)",
                 "engine": args.engine, "check_items": args.check_items},
        "ms_per_full_model_sync": round(pack_ms + uv_ms, 3),
        "ops": {
            "pack": {"ms": round(pack_ms, 3), "ms_median": round(statistics.median(pack_all), 3),
                     "ms_best": round(min(pack_all), 3), "bytes": pack_bytes,
                     "GB/s": round(pack_gbs, 1), "frac_of_peak": round(pack_gbs / peak, 4)},
            "unpack_verify": {"ms": round(uv_ms, 3), "ms_median": round(statistics.median(uv_all), 3),
                              "ms_best": round(min(uv_all), 3), "bytes": uv_bytes,
                              "GB/s": round(uv_bytes / (uv_ms * 1e-3) / 1e9, 1),
                              "frac_of_peak": round(uv_bytes / (uv_ms * 1e-3) / 1e9 / peak, 4)},
            "unpack": {"ms": round(unpack_ms, 3), "bytes": unpack_bytes,
                       "GB/s": round(unpack_bytes / (unpack_ms * 1e-3) / 1e9, 1),
                       "frac_of_peak": round(unpack_bytes / (unpack_ms * 1e-3) / 1e9 / peak, 4)},
            "verify": {"ms": round(verify_ms, 3), "bytes": verify_bytes,
                       "GB/s": round(verify_bytes / (verify_ms * 1e-3) / 1e9, 1),
                       "frac_of_peak": round(verify_bytes / (verify_ms * 1e-3) / 1e9 / peak, 4)},
        },
        "roofline": {"bound": "hbm",
                     "kernel": "rr_bulk_kernel (pack)" if args.engine == "auto" else "rr_pack_kernel",
                     "achieved": round(pack_gbs, 1),
                     "peak": peak, "peak_kind": peak_kind, "unit": "GB/s",
                     "frac": round(pack_gbs / peak, 4), "traffic": traffic,
                     "algorithmic_bytes": pack_bytes,
                     "copy_same_run": {"GB/s": round(copy_gbs, 1),
                                       "pack_frac": round(pack_gbs / copy_gbs, 4),
                                       "method": "torch copy_ of 4 GiB on the device, "
                                                 "read + write bytes"}},
        "clocks": clocks,
        # Per step: the pack kernel and the verifying unpack, which writes its
        # own result (bench launches hold a pooled slot each): one kernel, or
        # one per bucket range where the tensors exceed one launch's table.
        "gpu_launches": (1 + receiver_launches(plan)) * args.steps,
        "e2e": e2e,
    }
    if snapshot:
        line["snapshot"] = snapshot
    if more:
        line["next_rows"] = more
    del buf
    torch.cuda.empty_cache()
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        line["cpu_baseline"] = cpu_baseline(w, bucket_bytes, args.cpu_buckets)
    if rank == 0:
        print(json.dumps(line), flush=True)


def main():
    args = parse()
    import synth
    w = (synth.WORKLOADS.get(args.workload) or synth.TEST_WORKLOADS.get(args.workload)
         or synth.EXTRA_WORKLOADS[args.workload])
    if args.layers:
        import dataclasses
        vocab = args.vocab or w.shape.vocab
        w = w.with_(name=f"{w.name}-first{args.layers}layers-vocab{vocab}",
                    shape=dataclasses.replace(w.shape, layers=args.layers, vocab=vocab))
    if args.dst_dtype != "bf16":
        w = w.with_(name=f"{w.name}-{args.dst_dtype}", dst_dtype=args.dst_dtype)
    bucket_bytes = args.bucket_mib * (1 << 20) if args.bucket_mib else w.bucket_bytes
    world, rank, local = dist_setup(args)
    if args.impl == "reference":
        run_reference(args, w, bucket_bytes, world, rank)
    else:
        run_native(args, w, bucket_bytes, world, rank, local)
    if world > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


if __name__ == "__main__":
    main()
