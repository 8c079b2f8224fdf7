"""rr_pack reading the trainer's shards from host memory (pinned, or pageable
where the GPU reads it).

A trainer that keeps its master weights in host RAM (offloaded optimizer
state) hands the pack host pointers: on GB300 the pack's own loads read them
over NVLink-C2C, with no copy into HBM first (RobustRL Section 5.2.1 steps
1-2: reshard, then place the model into the transfer buffer).  That source
takes the register path, whose fp32 vectors are narrowed to 4 elements so
that each warp load uses whole 32-byte sectors of host memory.  Buckets and
checksums are compared with the oracle byte for byte: small workloads (fp32
with special values, bf16, row-sharded, per-unit), random ragged layouts,
row-parallel slices, bucket ranges, the checked kernels, and Qwen3-0.6B in
full.
"""
import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield
    torch.cuda.synchronize()


def host_source_buffers(plan, shards):
    """Device buckets and tensors, and the source block in pinned host memory."""
    flat = torch.from_numpy(np.concatenate([np.asarray(s, np.uint8) for s in shards]))
    flat = flat.pin_memory()
    buf = H.alloc(plan, flat=flat)
    assert not buf.flat.is_cuda and buf.flat.is_pinned()
    return buf


def oracle_pack(L, shards, parallel=False):
    src = oracle.Source(shards=shards)
    if not parallel:
        return L.pack(src)
    # Bucket by bucket on all host cores (the oracle's C calls release the
    # interpreter lock and share no state).
    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        parts = list(ex.map(lambda b: L.pack(src, first=b, count=1), range(L.n_buckets)))
    return (np.concatenate([p[0] for p in parts]),
            np.concatenate([p[1] for p in parts]).astype(np.uint64))


def pack_from_host(desc, parallel=False, **opts):
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], **opts)
    shards = L.host_shards(desc["seed"], desc["specials"])
    buf = host_source_buffers(plan, shards)
    H.pack(buf)
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    want, want_cs = oracle_pack(L, shards, parallel)
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
    return plan, buf, L, want, want_cs


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-moe-kvrep", "tiny-fsdp2",
                                  "tiny-units", "tiny-moe-bf16-specials", "tiny-kvrep-f32"])
def test_small_workloads_from_host(name):
    plan, buf, L, want, _ = pack_from_host(U.workload_desc(name))
    # The receiver on the device, as after any pack.
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    for t in range(len(L.tensors)):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.unpack_tensor(want, t),
                                      err_msg=f"tensor {t}")


@pytest.mark.parametrize("seed", range(12))
def test_random_layouts_from_host(seed):
    pack_from_host(U.random_layout(seed))


@pytest.mark.parametrize("seed", range(6))
def test_random_row_parallel_layouts_from_host(seed):
    pack_from_host(U.random_tp_layout(seed))


@pytest.mark.parametrize("case", ["tiny-tp4", "random-7", "row-parallel-2"])
def test_checked_kernels_from_host(case):
    if case.startswith("random-"):
        desc = U.random_layout(int(case.split("-")[1]))
    elif case.startswith("row-parallel-"):
        desc = U.random_tp_layout(int(case.split("-")[2]))
    else:
        desc = U.workload_desc(case)
    pack_from_host(desc, check_items=True)


def test_bucket_ranges_from_host():
    """rr_pack_range over three ranges, last first, as a pipelined caller runs it."""
    desc = U.workload_desc("tiny-tp4")
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    shards = L.host_shards(desc["seed"], desc["specials"])
    buf = host_source_buffers(plan, shards)
    n = plan.n_buckets
    cuts = [0, n // 3, 2 * n // 3, n]
    for a, b in reversed(list(zip(cuts[:-1], cuts[1:]))):
        rr.rr_pack_range(plan, a, b - a, buf.shards, buf.buckets, buf.checksums)
    torch.cuda.synchronize()
    want, want_cs = L.pack(oracle.Source(shards=shards))
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)


def test_qwen3_0_6b_from_host():
    """Every bucket and checksum of Qwen3-0.6B (fp32, 8 flat shards) packed
    from pinned host memory, and the receiver's tensors after it."""
    plan, buf, L, want, _ = pack_from_host(U.workload_desc("qwen3-0.6b"), parallel=True)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    for t in sorted({0, 1, plan.n_tensors // 2, plan.n_tensors - 1}):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.unpack_tensor(want, t),
                                      err_msg=plan.tensor_names[t])


@pytest.mark.parametrize("name", ["tiny-tp4", "tiny-moe-kvrep", "qwen3-0.6b"])
def test_pageable_host_source(name):
    """On a GPU that reads pageable host memory (Grace, through address
    translation) the trainer's shards need not be pinned: ordinary host
    memory is read by the same kernel, with the same bytes."""
    from tests.test_pointers import _pageable_access
    if not _pageable_access():
        pytest.skip("this GPU does not read pageable host memory (the call refuses it)")
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    shards = L.host_shards(desc["seed"], desc["specials"])
    flat = torch.from_numpy(np.concatenate([np.asarray(x, np.uint8) for x in shards]))
    assert not flat.is_pinned()
    buf = H.alloc(plan, flat=flat)
    H.pack(buf)
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    want, want_cs = oracle_pack(L, shards, parallel=name == "qwen3-0.6b")
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
