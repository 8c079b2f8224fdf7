"""The benchmark's end-to-end routes, run as bench.py runs them, against the oracle.

The trainer's shards sit in pinned host memory.  The copy-engine route
(bench.PipelinedE2E) copies them to the device in pieces and packs each run of
buckets as its sources land; the direct route (bench.DirectE2E) packs straight
from host memory, the pack's loads crossing NVLink-C2C, from pinned memory or,
where the GPU reads it, from ordinary pageable memory.  Each hands every bucket
range to the stream-ordered verifying unpack and read the checksums and result
rows back to the host (RobustRL Section 5.2.1: the rollout completes its update
from what it pulled; Section 5.2.2: it must know that what it holds is whole).

The device copy of the source is poisoned before the first step, so the
buckets can only be right if the route brought the host's bytes across.  After
two steps, on Qwen3-0.6B (fp32, 8 flat shards, 36 buckets of 32 MiB):
* every result row is {0, -1} and no kernel gave up a bounded wait;
* every bucket and checksum equals the oracle's, and so do the checksums read
  back to the host;
* every tensor equals its own bytes in the buckets, and sampled tensors equal
  the oracle's direct reshard.
"""
import os
from concurrent.futures import ThreadPoolExecutor

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


@pytest.fixture(scope="module")
def oracle_image():
    w = synth.WORKLOADS["qwen3-0.6b"]
    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        parts = list(ex.map(lambda b: L.pack(gen, first=b, count=1), range(L.n_buckets)))
    want = np.concatenate([p[0] for p in parts])
    want_cs = np.concatenate([p[1] for p in parts]).astype(np.uint64)
    return L, gen, want, want_cs


SAMPLED = ["embed_tokens", "layers.0.qkv_proj", "layers.13.o_proj", "layers.27.down_proj",
           "layers.27.post_attention_layernorm", "norm"]


@pytest.mark.parametrize("route", ["copy_engine", "direct", "direct_pageable"])
def test_e2e_route(route, oracle_image):
    import bench
    if route == "direct_pageable":
        from tests.test_pointers import _pageable_access
        if not _pageable_access():
            pytest.skip("this GPU does not read pageable host memory")
    L, gen, want, want_cs = oracle_image
    w = synth.WORKLOADS["qwen3-0.6b"]
    bs = bench.BenchStep(w, w.bucket_bytes, poison=0xAB)
    plan, buf = bs.plan, bs.buf
    host = torch.empty(buf.flat.numel(), dtype=torch.uint8,
                       pin_memory=route != "direct_pageable")
    host.copy_(buf.flat)
    buf.flat.fill_(0x5A)                     # only the host copy holds the weights now
    torch.cuda.synchronize()
    e2e = bench.PipelinedE2E(bs, host) if route == "copy_engine" else bench.DirectE2E(bs, host)
    for _ in range(2):
        e2e.step()
    e2e.check()                              # result rows {0, -1}; rr_plan_check clean
    assert e2e.used == 2

    assert L.n_buckets == plan.n_buckets
    np.testing.assert_array_equal(buf.bucket_store[:, :plan.bucket_bytes].cpu().numpy(), want)
    np.testing.assert_array_equal(buf.checksums.cpu().numpy().view(np.uint64)[:plan.n_buckets],
                                  want_cs)
    np.testing.assert_array_equal(e2e.host_cs.numpy().view(np.uint64)[:plan.n_buckets], want_cs)
    assert e2e.host_res.tolist() == [[0, -1]] * e2e.n_ranges

    B = plan.bucket_bytes
    store = buf.bucket_store.view(-1)
    for t in range(plan.n_tensors):           # TP=1: one stream, buckets back to back
        start = plan.first_bucket_of_rank[plan.tensor_ranks[t]] * B + plan.tensor_stream_offset[t]
        n = plan.tensor_numel[t]
        assert torch.equal(buf.dst[t][:n], store[start:start + 2 * n].view(torch.int16)), \
            plan.tensor_names[t]
    for name in SAMPLED:
        t = L.tensor_index(name, 0)
        got = buf.dst[t][:plan.tensor_numel[t]].cpu().numpy().view(np.uint16)
        np.testing.assert_array_equal(got, L.reshard_tensor(gen, t), err_msg=name)


@pytest.mark.parametrize("route", ["copy_engine", "direct", "direct_pageable"])
def test_e2e_route_tp4_special_values(route):
    """The same routes on the tiny TP=4 workload with special values (RNE ties,
    subnormals, infinities, NaNs): four ranks' streams, every bucket, checksum
    and tensor against the oracle."""
    import bench
    if route == "direct_pageable":
        from tests.test_pointers import _pageable_access
        if not _pageable_access():
            pytest.skip("this GPU does not read pageable host memory")
    w = synth.TEST_WORKLOADS["tiny-tp4"]
    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    want, want_cs = L.pack(gen)
    bs = bench.BenchStep(w, w.bucket_bytes, poison=0xAB)
    plan, buf = bs.plan, bs.buf
    host = torch.empty(buf.flat.numel(), dtype=torch.uint8,
                       pin_memory=route != "direct_pageable")
    host.copy_(buf.flat)
    buf.flat.fill_(0x5A)
    torch.cuda.synchronize()
    e2e = (bench.PipelinedE2E(bs, host, pieces=4) if route == "copy_engine"
           else bench.DirectE2E(bs, host, pieces=4))
    for _ in range(2):
        e2e.step()
    e2e.check()
    np.testing.assert_array_equal(buf.bucket_store[:, :plan.bucket_bytes].cpu().numpy(), want)
    np.testing.assert_array_equal(e2e.host_cs.numpy().view(np.uint64)[:plan.n_buckets], want_cs)
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(
            buf.dst[t][:plan.tensor_numel[t]].cpu().numpy().view(np.uint16),
            L.unpack_tensor(want, t), err_msg=f"{plan.tensor_names[t]} rank {plan.tensor_ranks[t]}")
