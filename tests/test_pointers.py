"""Pointer tables checked once (rr.Pointers) in place of per-call lists.

The checks are host logic and run without a GPU on a host-only plan: a table
is refused for the wrong role, the wrong count, buffers too small, or a plan
of a different shape.  The GPU tests check that calls through tables give the
same bytes as calls through lists, and that a table built for one plan is
re-checked (not trusted) when handed to another.
"""
import numpy as np
import pytest
import torch

import paper_2512_22492_gb300 as rr
from tests import _util as U


def host_plan(name="tiny-tp4", **kw):
    desc = U.workload_desc(name, **kw)
    m, s, d = U.to_product(desc)
    return rr.rr_plan_create(m, s, d, desc["bucket_bytes"], rr.PlanOptions(host_only=True))


def fake_dst(plan, short=None):
    out = [torch.empty(n, dtype=torch.bfloat16) for n in plan.tensor_numel]
    if short is not None:
        out[short] = torch.empty(plan.tensor_numel[short] - 1, dtype=torch.bfloat16)
    return out


def test_table_checks_on_build():
    plan = host_plan()
    dst = fake_dst(plan)
    t = rr.Pointers(plan, "dst", dst)
    assert len(t) == plan.n_tensors and t.role == "dst" and t.plan is plan
    with pytest.raises(ValueError):
        rr.Pointers(plan, "dst", dst[:-1])                       # one short
    with pytest.raises(ValueError):
        rr.Pointers(plan, "dst", fake_dst(plan, short=3))        # tensor 3 too small
    with pytest.raises(ValueError):
        rr.Pointers(plan, "weights", dst)                        # no such role
    buckets = torch.empty(plan.n_buckets, plan.bucket_bytes, dtype=torch.uint8)
    tb = rr.Pointers(plan, "buckets", buckets)
    assert list(tb.array)[:2] == [buckets.data_ptr(), buckets.data_ptr() + plan.bucket_bytes]
    with pytest.raises(ValueError):
        rr.Pointers(plan, "buckets", buckets[:, :-16])           # rows too short


def test_table_refused_for_the_wrong_role_or_plan():
    """These are refused in Python before any call reaches the library."""
    plan = host_plan()
    dst = rr.Pointers(plan, "dst", fake_dst(plan))
    buckets = rr.Pointers(plan, "buckets",
                          torch.empty(plan.n_buckets, plan.bucket_bytes, dtype=torch.uint8))
    with pytest.raises(ValueError, match="built for dst"):
        rr.rr_unpack(plan, dst, dst)                             # dst table as buckets
    other = host_plan("tiny-moe-tp2")
    with pytest.raises(ValueError):
        rr.rr_unpack(other, buckets, dst)                        # counts differ


def test_recheck_uses_recorded_sizes():
    """A table handed to a plan other than its own is checked entry by entry
    against the sizes recorded when it was built."""
    plan = host_plan()
    twin = host_plan()                                           # same shape, another object
    dst = rr.Pointers(plan, "dst", fake_dst(plan))
    from paper_2512_22492_gb300 import rr as rrmod
    rrmod._check_list(dst, twin.n_tensors, lambda i: 2 * twin.tensor_numel[i], "dst", plan=twin)
    with pytest.raises(ValueError):
        rrmod._check_list(dst, twin.n_tensors, lambda i: 2 * twin.tensor_numel[i] + 2, "dst",
                          plan=twin)


@pytest.mark.gpu
def test_tables_give_the_same_bytes_as_lists():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from tests import gpu_harness as H
    desc = U.workload_desc("tiny-moe-tp2")
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    a, b = H.alloc(plan), H.alloc(plan)
    for x in (a, b):
        H.fill_with_generator(x, m, desc["seed"], desc["specials"])
    H.pack(a)
    H.unpack(a)
    ts = rr.Pointers(plan, "src_shards", b.shards)
    tb = rr.Pointers(plan, "buckets", b.buckets)
    td = rr.Pointers(plan, "dst", b.dst)
    for _ in range(2):
        rr.rr_pack(plan, ts, tb, b.checksums)
        assert rr.rr_unpack_verify(plan, tb, b.checksums, td) == (0, -1)
    torch.cuda.synchronize()
    assert torch.equal(a.bucket_store, b.bucket_store)
    assert torch.equal(a.checksums, b.checksums)
    for t in range(plan.n_tensors):
        assert torch.equal(a.dst[t], b.dst[t])
    for x in b.dst:
        x.fill_(0)
    rr.rr_unpack(plan, tb, td)
    assert rr.rr_verify(plan, tb, b.checksums) == (0, -1)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        assert torch.equal(a.dst[t], b.dst[t])
    np.testing.assert_array_equal(H.checksums_host(a), H.checksums_host(b))


def test_non_contiguous_buffers_are_refused():
    """A strided view would have the library write past what it shows."""
    plan = host_plan()
    dst = fake_dst(plan)
    wide = torch.empty(2 * plan.tensor_numel[0], dtype=torch.bfloat16)
    dst[0] = wide[::2]
    with pytest.raises(ValueError, match="not contiguous"):
        rr.Pointers(plan, "dst", dst)
    buckets = torch.empty(plan.bucket_bytes, plan.n_buckets, dtype=torch.uint8).t()
    with pytest.raises(ValueError, match="contiguous"):
        rr.rr_verify(plan, buckets, torch.empty(plan.n_buckets, dtype=torch.int64))
    cs = torch.empty(2 * plan.n_buckets, dtype=torch.int64)[::2]
    with pytest.raises(ValueError, match="checksums"):
        rr.rr_verify(plan, torch.empty(plan.n_buckets, plan.bucket_bytes, dtype=torch.uint8), cs)


def _pageable_access() -> int:
    import ctypes
    from paper_2512_22492_gb300 import build as B
    from tests.test_c_abi import cudart_dir
    rt = ctypes.CDLL(cudart_dir(B._cuda_home()) + "/libcudart.so")
    v = ctypes.c_int(0)
    assert rt.cudaDeviceGetAttribute(ctypes.byref(v), 88, 0) == 0   # PageableMemoryAccess
    return v.value


@pytest.mark.gpu
def test_pageable_host_buffers_refused_where_unreadable():
    """Ordinary (pageable) host memory is refused with RR_EINVAL unless this GPU
    reads pageable host memory; nothing is launched on it either way."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    if _pageable_access():
        pytest.skip("this GPU reads pageable host memory: nothing to refuse")
    from tests import gpu_harness as H
    from paper_2512_22492_gb300 import rr as rrmod
    desc = U.workload_desc("tiny-tp4")
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan)
    host_buckets = torch.zeros(plan.n_buckets, plan.bucket_bytes, dtype=torch.uint8)
    with pytest.raises(rr.RRError) as e:
        rr.rr_pack(plan, buf.shards, host_buckets, buf.checksums)
    assert e.value.status == rrmod.RR_EINVAL
    with pytest.raises(rr.RRError) as e:
        rr.rr_verify(plan, buf.buckets, torch.zeros(plan.n_buckets, dtype=torch.int64))
    assert e.value.status == rrmod.RR_EINVAL
