"""The stream-ordered verifying unpack (rr_unpack_verify_async) through the C ABI.

It must give what the synchronous rr_unpack_verify gives -- the same tensors,
the same count and first bad bucket, the same per-bucket flags -- with the
result written into device or pinned host memory on the stream, ranges
included, and two streams with their own scratch running at once.
"""
import numpy as np
import pytest
import torch

import oracle
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


def packed(name="tiny-moe-tp2", **opts):
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], **opts)
    buf = H.alloc(plan)
    H.fill_with_generator(buf, m, desc["seed"], desc["specials"])
    H.pack(buf)
    torch.cuda.synchronize()
    return desc, plan, buf


def scratch_for(plan):
    return torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")


@pytest.mark.parametrize("engine", ["auto", "registers"])
@pytest.mark.parametrize("where", ["device", "pinned"])
def test_async_matches_sync(engine, where):
    desc, plan, buf = packed(engine=engine)
    result = (torch.full((2,), 7, dtype=torch.int64, device="cuda") if where == "device"
              else torch.full((2,), 7, dtype=torch.int64).pin_memory())
    rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan), result)
    torch.cuda.synchronize()
    assert result.cpu().tolist() == [0, -1]
    L = U.to_oracle(desc)
    gen = oracle.Source(seed=desc["seed"], specials=desc["specials"])
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(gen, t))
    # Damage two buckets: the count, the first, and the flags follow.
    bl = H.bucket_list(buf)
    bl[5][33] ^= 0x10
    bl[2][0] ^= 0x01
    bad = torch.zeros(plan.n_buckets, dtype=torch.uint8, device="cuda")
    rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan), result,
                              bad=bad)
    torch.cuda.synchronize()
    assert result.cpu().tolist() == [2, 2]
    assert list(np.flatnonzero(bad.cpu().numpy())) == [2, 5]
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (2, 2)


def test_async_ranges_and_empty():
    _, plan, buf = packed()
    result = torch.zeros(2, dtype=torch.int64, device="cuda")
    bl = H.bucket_list(buf)
    bl[7][100] ^= 0x80
    n = plan.n_buckets
    for first, count, want in ((0, 5, [0, -1]), (5, 4, [1, 7]), (8, n - 8, [0, -1]),
                               (3, 0, [0, -1]), (n, 0, [0, -1])):
        result.fill_(9)
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan),
                                  result, first_bucket=first, n_buckets=count)
        torch.cuda.synchronize()
        assert result.cpu().tolist() == want, (first, count)
    rr.rr_plan_check(plan)


def test_two_streams_with_their_own_scratch():
    _, plan, a = packed()
    b = H.alloc(plan)
    b.bucket_store.copy_(a.bucket_store)
    b.checksums.copy_(a.checksums)
    H.bucket_list(b)[4][8] ^= 0x02
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in range(2)]
    results = [torch.zeros(2, dtype=torch.int64, device="cuda") for _ in range(2)]
    scratch = [scratch_for(plan) for _ in range(2)]
    for _ in range(4):
        for buf, st, res, sc in zip((a, b), streams, results, scratch):
            with torch.cuda.stream(st):
                rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, sc, res,
                                          stream=st)
    torch.cuda.synchronize()
    assert results[0].cpu().tolist() == [0, -1]
    assert results[1].cpu().tolist() == [1, 4]


def test_async_refuses_bad_result_and_scratch():
    _, plan, buf = packed()
    pageable = np.zeros(2, np.int64)
    with pytest.raises(rr.RRError) as e:
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan),
                                  int(pageable.ctypes.data))
    assert e.value.status == rrmod.RR_EINVAL
    host_scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64).pin_memory()
    with pytest.raises(rr.RRError) as e:
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, host_scratch,
                                  torch.zeros(2, dtype=torch.int64, device="cuda"))
    assert e.value.status == rrmod.RR_EINVAL
    with pytest.raises(ValueError):
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst,
                                  torch.zeros(3, dtype=torch.int64, device="cuda"),
                                  torch.zeros(2, dtype=torch.int64, device="cuda"))


@pytest.mark.parametrize("grid", [1, 3, 2048])
def test_claimed_units_on_any_grid(grid):
    """The verifying unpack's blocks claim work units: one block taking every
    unit, a few blocks, and more blocks than units (most with none of their
    own) all give the oracle's tensors and the same verdicts, for the whole
    sync and for bucket ranges."""
    desc, plan, buf = packed("tiny-moe-tp2", grid_blocks=grid)
    first, bucket_unit = plan.work_units("unpack")
    assert len(first) - 1 > 3 and len(first) - 1 < 2048
    bl = H.bucket_list(buf)
    bl[6][40] ^= 0x04
    for t in buf.dst:
        t.fill_(0)
    result = torch.zeros(2, dtype=torch.int64, device="cuda")
    bad = torch.zeros(plan.n_buckets, dtype=torch.uint8, device="cuda")
    rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan), result,
                              bad=bad)
    torch.cuda.synchronize()
    assert result.cpu().tolist() == [1, 6]
    assert list(np.flatnonzero(bad.cpu().numpy())) == [6]
    bl[6][40] ^= 0x04                                   # undo: tensors must match the oracle
    L = U.to_oracle(desc)
    gen = oracle.Source(seed=desc["seed"], specials=desc["specials"])
    for first_b, count in ((0, plan.n_buckets), (2, 5), (plan.n_buckets - 1, 1)):
        for t in buf.dst:
            t.fill_(0)
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch_for(plan),
                                  result, first_bucket=first_b, n_buckets=count)
        torch.cuda.synchronize()
        assert result.cpu().tolist() == [0, -1]
        assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst, first_bucket=first_b,
                                   n_buckets=count) == (0, -1)
    for t in buf.dst:
        t.fill_(0)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(gen, t))
    rr.rr_plan_check(plan)
