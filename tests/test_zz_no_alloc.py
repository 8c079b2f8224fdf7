"""The allocation-free verify entry point, rr_verify_noalloc, through the C ABI.

It serves callers that cannot allocate device memory when they check the
buckets they pulled (an inference engine that has reserved nearly all device
memory, or code under a memory pool that refuses cudaMalloc).  Its results
must equal rr_verify's -- the check is exact integer work, so equal means
identical -- on two calls in a row, both on intact buckets and after damage,
and it must not change the device's free memory once set up.  This file is
collected last on purpose.
"""
import numpy as np
import pytest
import torch

import paper_2512_22492_gb300 as rr
from paper_2512_22492_gb300 import rr as rrmod
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield


def packed(name, separate=False):
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan, separate_buckets=separate, with_dst=False)
    H.fill_with_generator(buf, m, desc["seed"], desc["specials"])
    H.pack(buf)
    torch.cuda.synchronize()
    return plan, buf


@pytest.mark.parametrize("name,separate", [("tiny-tp4", False), ("tiny-tp4", True),
                                           ("qwen3-0.6b", False)])
def test_matches_rr_verify_twice_in_a_row(name, separate):
    plan, buf = packed(name, separate)
    want = rr.rr_verify(plan, buf.buckets, buf.checksums)
    assert want == (0, -1)
    for _ in range(2):
        assert rrmod.rr_verify_noalloc(buf.buckets, plan.n_buckets, plan.bucket_bytes,
                                       buf.checksums) == want
    # Damage two buckets: both entry points must name the same count and first index.
    bl = H.bucket_list(buf)
    hit = sorted({plan.n_buckets // 2, plan.n_buckets - 1})
    for b in hit:
        bl[b][17] ^= 0x40
    want = rr.rr_verify(plan, buf.buckets, buf.checksums)
    assert want == (len(hit), hit[0])
    for _ in range(2):
        assert rrmod.rr_verify_noalloc(buf.buckets, plan.n_buckets, plan.bucket_bytes,
                                       buf.checksums) == want
    # Repaired: the previous call's state must not leak into the next one.
    for b in hit:
        bl[b][17] ^= 0x40
    for _ in range(2):
        assert rrmod.rr_verify_noalloc(buf.buckets, plan.n_buckets, plan.bucket_bytes,
                                       buf.checksums) == (0, -1)


def test_allocates_nothing_after_setup():
    plan, buf = packed("tiny-tp4")
    rrmod.rr_verify_noalloc(buf.buckets, plan.n_buckets, plan.bucket_bytes, buf.checksums)
    torch.cuda.synchronize()
    free0, _ = torch.cuda.mem_get_info()
    for _ in range(3):
        assert rrmod.rr_verify_noalloc(buf.buckets, plan.n_buckets, plan.bucket_bytes,
                                       buf.checksums) == (0, -1)
    free1, _ = torch.cuda.mem_get_info()
    assert free1 == free0


def test_rejects_more_buckets_than_the_array_holds():
    store = torch.zeros((16385, 16), dtype=torch.uint8, device="cuda")
    cs = torch.zeros(16385, dtype=torch.int64, device="cuda")
    with pytest.raises(rr.RRError) as e:
        rrmod.rr_verify_noalloc(store, 16385, 16, cs)
    assert e.value.status == rrmod.RR_EINVAL
    # The maximum itself is accepted (all-zero buckets have checksum zero).
    assert rrmod.rr_verify_noalloc(store[:16384], 16384, 16, cs) == (0, -1)
