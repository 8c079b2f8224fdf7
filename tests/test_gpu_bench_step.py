"""The benchmark's own step, at full size, against the oracle.

The headline throughput is measured on Qwen3-8B (fp32, 8 flat shards -> TP=1
bf16, 128 MiB buckets) by ``bench.BenchStep``: rr_pack followed by the
stream-ordered rr_unpack_verify_async, both through checked pointer tables, on
one stream (RobustRL Section 5.2.1: the rollout completes its update from what
it pulled; Section 5.2.2: it must know that what it holds is whole).  This
file runs that very object -- the same plan, buffers, tables, calls, kernels
and launch configuration -- for the bench's three warm-up steps, then checks
what the timed steps produce:

* every step's result row is {0, -1} and no kernel gave up a bounded wait;
* every checksum equals torch's word sum of its bucket, and sampled buckets
  equal the oracle's byte for byte (every bucket of this pack is compared
  with the oracle in test_gpu_parity.py);
* every destination tensor equals its own bytes in the buckets (the tensors
  and buckets start poisoned, so an unwritten byte shows), and sampled
  tensors equal the oracle's direct reshard, element for element.
"""
import numpy as np
import pytest
import torch

import oracle
import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


# Tensors compared with the oracle one by one: the first and last layers, a
# row-parallel weight, a norm vector, and the two vocabulary matrices (the
# first and the last bytes of the stream).
SAMPLED = [("embed_tokens", 0), ("layers.0.qkv_proj", 0), ("layers.17.o_proj", 0),
           ("layers.35.down_proj", 0), ("layers.35.post_attention_layernorm", 0), ("norm", 0),
           ("lm_head", 0)]


def test_bench_step_qwen3_8b_full_size():
    import bench
    w = synth.WORKLOADS["qwen3-8b"]
    bs = bench.BenchStep(w, w.bucket_bytes, poison=0xAB)
    plan, buf = bs.plan, bs.buf
    assert bs.step_bytes == 82_161_973_248
    for _ in range(3):          # the bench's warm-up steps; the timed ones repeat them
        bs.step()
    bs.check_results()          # every row {0, -1}; rr_plan_check clean
    assert bs.used == 3
    assert bs.results[:3].cpu().tolist() == [[0, -1]] * 3

    # Checksums: torch's wrapping word sum of every bucket.
    B = plan.bucket_bytes
    assert buf.bucket_store.shape[1] == B
    got_cs = buf.checksums.cpu().numpy().view(np.uint64)[:plan.n_buckets]
    words = buf.bucket_store.view(torch.int64)
    torch_cs = np.array([int(words[b].sum().item()) & ((1 << 64) - 1)
                         for b in range(plan.n_buckets)], np.uint64)
    np.testing.assert_array_equal(got_cs, torch_cs)

    # Sampled buckets against the oracle: first, last, and a few in between.
    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    assert L.n_buckets == plan.n_buckets
    for b in sorted({0, 1, plan.n_buckets // 2, plan.n_buckets - 2, plan.n_buckets - 1}):
        want, want_cs = L.pack(gen, first=b, count=1)
        np.testing.assert_array_equal(buf.bucket_store[b].cpu().numpy(), want[0],
                                      err_msg=f"bucket {b}")
        assert got_cs[b] == want_cs[0]

    # Every tensor against its own bytes in the buckets (TP=1: one stream).
    store = buf.bucket_store.view(-1)
    for t in range(plan.n_tensors):
        start = plan.first_bucket_of_rank[plan.tensor_ranks[t]] * B + plan.tensor_stream_offset[t]
        n = plan.tensor_numel[t]
        want = store[start:start + 2 * n].view(torch.int16)
        assert torch.equal(buf.dst[t][:n], want), plan.tensor_names[t]

    # Sampled tensors against the oracle's direct reshard of the source.
    for name, rank in SAMPLED:
        t = L.tensor_index(name, rank)
        assert plan.tensor_names[t] == name and plan.tensor_ranks[t] == rank
        got = buf.dst[t][:plan.tensor_numel[t]].cpu().numpy().view(np.uint16)
        np.testing.assert_array_equal(got, L.reshard_tensor(gen, t), err_msg=name)
