"""The largest sync that fits one GPU: the paper's Qwen3-32B (Section 7.1), fp32
in 8 FSDP2 row shards to a TP=8 bf16 rollout, 128 MiB buckets -- 131 GB of
source, 496 buckets (67 GB) and 4,120 rollout tensors (66 GB): 245 GiB of the
GPU's 277 GiB.  It runs the benchmark's own step (bench.BenchStep: rr_pack
over the whole-sync table with its fan-out groups, then the stream-ordered
verifying unpack, which here runs as two launches over bucket ranges: 4,120
tensor pointers exceed one launch's table) and checks, against the oracle and
at any size:

* every result row is {0, -1} and no kernel gave up a bounded wait;
* every checksum equals torch's word sum of its bucket;
* the first and last bucket of every rank, and a few others, equal the
  oracle's byte for byte, checksums too;
* every tensor equals its own bytes in the buckets (tensors and buckets start
  poisoned), and sampled tensors equal the oracle's direct reshard.

The test skips where the GPU has less free memory than the sync needs.
"""
import gc
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu

NAME = "qwen3-32b-fsdp2-tp8"
SAMPLED = [("embed_tokens", 2), ("layers.0.qkv_proj", 3), ("layers.31.o_proj", 0),
           ("layers.63.down_proj", 7), ("layers.40.gate_up_proj", 5),
           ("layers.63.post_attention_layernorm", 6), ("norm", 1), ("lm_head", 4)]


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    gc.collect()
    torch.cuda.empty_cache()
    yield
    gc.collect()
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def test_qwen3_32b_fsdp2_tp8_full_size():
    import bench
    import paper_2512_22492_gb300 as rr
    w = synth.EXTRA_WORKLOADS[NAME]
    m, s, d = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding)
    probe = rr.rr_plan_create(m, s, d, w.bucket_bytes, rr.PlanOptions(host_only=True))
    st = probe.stats()
    need = (sum(probe.source_buffer_bytes) + probe.n_buckets * probe.bucket_bytes +
            st["unpack_bytes_written"])
    free, _total = torch.cuda.mem_get_info()
    if free < need + (6 << 30):
        pytest.skip(f"needs {need / 2**30:.0f} GiB of device memory, {free / 2**30:.0f} GiB free")
    del probe

    bs = bench.BenchStep(w, w.bucket_bytes, poison=0xAB)
    plan, buf = bs.plan, bs.buf
    for _ in range(2):
        bs.step()
    bs.check_results()                        # every row {0, -1}; rr_plan_check clean
    assert bs.results[:2].cpu().tolist() == [[0, -1]] * 2

    B = plan.bucket_bytes
    assert buf.bucket_store.shape[1] == B
    got_cs = buf.checksums.cpu().numpy().view(np.uint64)[:plan.n_buckets]
    words = buf.bucket_store.view(torch.int64)
    torch_cs = np.array([int(words[b].sum().item()) & ((1 << 64) - 1)
                         for b in range(plan.n_buckets)], np.uint64)
    np.testing.assert_array_equal(got_cs, torch_cs)

    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    assert L.n_buckets == plan.n_buckets
    fr = plan.first_bucket_of_rank
    rng = np.random.default_rng(32)
    pick = sorted({*[fr[r] for r in range(plan.tp)], *[fr[r + 1] - 1 for r in range(plan.tp)],
                   *rng.integers(0, plan.n_buckets, 4).tolist()})
    got = {b: buf.bucket_store[b].cpu().numpy() for b in pick}
    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        wants = dict(zip(pick, ex.map(lambda b: L.pack(gen, first=b, count=1), pick)))
    for b in pick:
        want, want_cs = wants[b]
        np.testing.assert_array_equal(got[b], want[0], err_msg=f"bucket {b}")
        assert got_cs[b] == want_cs[0], b

    store = buf.bucket_store.view(-1)
    for t in range(plan.n_tensors):
        start = plan.first_bucket_of_rank[plan.tensor_ranks[t]] * B + plan.tensor_stream_offset[t]
        n = plan.tensor_numel[t]
        assert torch.equal(buf.dst[t][:n], store[start:start + 2 * n].view(torch.int16)), \
            (plan.tensor_names[t], plan.tensor_ranks[t])
    for name, rank in SAMPLED:
        t = L.tensor_index(name, rank)
        assert plan.tensor_names[t] == name and plan.tensor_ranks[t] == rank
        got_t = buf.dst[t][:plan.tensor_numel[t]].cpu().numpy().view(np.uint16)
        np.testing.assert_array_equal(got_t, L.reshard_tensor(gen, t), err_msg=f"{name} {rank}")
