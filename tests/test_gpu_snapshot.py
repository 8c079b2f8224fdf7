"""Per-step checkpoint snapshot to host memory (the paper's per-step checkpoint,
Sections 2.3 and 7.4: its blocking part is the GPU -> host-memory copy).

On GB300 the device reaches pinned host memory over NVLink-C2C, so rr_pack can
write its buckets -- the bf16 rollout image with its checksums -- straight into
host RAM, and a recovering process can unpack and verify from there.  Both
directions run on the register path (host-resident buffers).  The host
buckets and checksums are compared with the oracle's pack, and the restored
tensors with the oracle's unpack of its own buckets, byte for byte; the
device path's output must equal them too.
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


def host_buckets(plan, pinned=True):
    row = (plan.bucket_bytes + 15) // 16 * 16
    store = torch.empty((plan.n_buckets, row), dtype=torch.uint8, pin_memory=pinned)
    store.fill_(0xAB)
    return store, store[:, :plan.bucket_bytes]


def oracle_pack(L, desc):
    """The oracle's buckets and checksums, packed bucket by bucket on all host
    cores (its C calls release the interpreter lock and share no state)."""
    gen = oracle.Source(seed=desc["seed"], specials=desc["specials"])
    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        parts = list(ex.map(lambda b: L.pack(gen, first=b, count=1), range(L.n_buckets)))
    return (np.concatenate([p[0] for p in parts]),
            np.concatenate([p[1] for p in parts]).astype(np.uint64))


@pytest.mark.parametrize("where", ["pinned", "pageable"])
@pytest.mark.parametrize("name", ["tiny-tp4", "tiny-moe-kvrep", "qwen3-0.6b"])
def test_snapshot_to_host_and_restore(name, where):
    """`pageable`: the snapshot goes into ordinary host memory, which a GPU that
    reads and writes pageable memory through the CPU's page tables (Grace)
    reaches without pinning."""
    if where == "pageable":
        from tests.test_pointers import _pageable_access
        if not _pageable_access():
            pytest.skip("this GPU does not reach pageable host memory")
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    assert L.n_buckets == plan.n_buckets
    dev = H.alloc(plan, with_dst=False)
    H.fill_with_generator(dev, m, desc["seed"], desc["specials"])
    store, view = host_buckets(plan, pinned=where == "pinned")
    cs = torch.zeros(plan.n_buckets, dtype=torch.int64, device="cuda")
    rr.rr_pack(plan, dev.shards, view, cs)                     # straight into host memory
    H.pack(dev)                                                # and on the device
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    want, want_cs = oracle_pack(L, desc)
    np.testing.assert_array_equal(view.numpy(), want)
    np.testing.assert_array_equal(cs.cpu().numpy().view(np.uint64), want_cs)
    np.testing.assert_array_equal(H.buckets_host(dev), want)
    # Restore: a fresh process image unpacks and verifies from the host snapshot.
    back = H.alloc(plan)
    assert rr.rr_unpack_verify(plan, view, cs, back.dst) == (0, -1)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(H.tensor_host(back, t), L.unpack_tensor(want, t),
                                      err_msg=f"tensor {t} ({plan.tensor_names[t]})")
    # Sampled tensors also against the oracle's direct reshard of the source.
    gen = oracle.Source(seed=desc["seed"], specials=desc["specials"])
    for t in sorted({0, plan.n_tensors // 2, plan.n_tensors - 1}):
        np.testing.assert_array_equal(H.tensor_host(back, t), L.reshard_tensor(gen, t))
    # A damaged host copy is caught, at the right bucket.
    view[plan.n_buckets // 2, 5] ^= 0x20
    assert rr.rr_verify(plan, view, cs) == (1, plan.n_buckets // 2)
