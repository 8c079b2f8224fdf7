"""Per-step checkpoint snapshot to host memory (the paper's per-step checkpoint,
Sections 2.3 and 7.4: its blocking part is the GPU -> host-memory copy).

On GB300 the device reaches pinned host memory over NVLink-C2C, so rr_pack can
write its buckets -- the bf16 rollout image with its checksums -- straight into
host RAM, and a recovering process can unpack and verify from there.  Bucket
bytes written to the host must equal the device path's exactly.
"""
import numpy as np
import pytest
import torch

import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield


def host_buckets(plan):
    row = (plan.bucket_bytes + 15) // 16 * 16
    store = torch.empty((plan.n_buckets, row), dtype=torch.uint8, pin_memory=True)
    store.fill_(0xAB)
    return store, store[:, :plan.bucket_bytes]


@pytest.mark.parametrize("name", ["tiny-tp4", "tiny-moe-kvrep", "qwen3-0.6b"])
def test_snapshot_to_host_and_restore(name):
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    dev = H.alloc(plan)
    H.fill_with_generator(dev, m, desc["seed"], desc["specials"])
    H.pack(dev)
    H.unpack(dev)
    torch.cuda.synchronize()
    store, view = host_buckets(plan)
    cs = torch.zeros(plan.n_buckets, dtype=torch.int64, device="cuda")
    rr.rr_pack(plan, dev.shards, view, cs)                     # straight into host memory
    torch.cuda.synchronize()
    assert torch.equal(cs, dev.checksums[:plan.n_buckets])
    assert torch.equal(view, dev.buckets.cpu())
    # Restore: a fresh process image unpacks and verifies from the host snapshot.
    back = H.alloc(plan)
    assert rr.rr_unpack_verify(plan, view, cs, back.dst) == (0, -1)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        assert torch.equal(back.dst[t], dev.dst[t])
    # A damaged host copy is caught.
    view[plan.n_buckets // 2, 5] ^= 0x20
    assert rr.rr_verify(plan, view, cs) == (1, plan.n_buckets // 2)
