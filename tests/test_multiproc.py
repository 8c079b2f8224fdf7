"""The benchmark's multi-rank path on CPU (gloo, world size 2).

The weight-sync path does not shard across GPUs: under torchrun each rank
runs an independent replica, ranks meet at a barrier around the timed region,
the slowest rank's time counts, and the value is the bytes of all replicas
over that time.  These tests run that plumbing as two gloo processes, and the
reference arm under torchrun, where rank 0 alone prints one line.
"""
import json
import multiprocessing as mp
import os
import socket
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, q):
    os.environ.update(RANK=str(rank), WORLD_SIZE=str(world), LOCAL_RANK=str(rank),
                      MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port),
                      CUDA_VISIBLE_DEVICES="")
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    w, r, _ = bench.dist_setup(None)
    bench.barrier(w)
    slowest = bench.max_over_ranks(10.0 + 5.0 * r, w)   # rank 1 is slower
    q.put((r, w, slowest, bench.aggregate_gbs(w, 2_000_000_000, slowest)))
    bench.barrier(w)
    dist.destroy_process_group()


def test_replicas_take_the_slowest_rank():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    out = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for r, w, slowest, gbs in out:
        assert w == 2 and slowest == 15.0
        # two replicas x 2 GB in 15 ms
        assert abs(gbs - 2 * 2.0 / 0.015) < 1e-6


def test_reference_arm_under_torchrun_prints_once():
    port = free_port()
    env = dict(os.environ, CUDA_VISIBLE_DEVICES="")
    cmd = [sys.executable, "-m", "torch.distributed.run", "--nnodes=1", "--nproc-per-node", "2",
           "--master-addr", "127.0.0.1", "--master-port", str(port),
           os.path.join(ROOT, "bench.py"), "--gpus", "2", "--impl", "reference",
           "--steps", "1", "--warmup", "0", "--bucket-mib", "4"]
    res = subprocess.run(cmd, cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert res.returncode == 0, res.stderr[-2000:]
    lines = [l for l in res.stdout.splitlines() if l.startswith("{")]
    assert len(lines) == 1
    line = json.loads(lines[0])
    assert line["impl"] == "reference" and line["unit"] == "GB/s" and line["value"] > 0
    assert line["e2e"]["h2d_bytes_per_step"] == 0 and line["cpu_baseline"]["kind"] == "oracle"
