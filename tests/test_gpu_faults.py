"""Host-side fault injection and robustness checks on the GPU path.

Section 5.2.2 of the paper has a rollout resume or redo a pull after a relay or
trainer failure; the checksums let it tell which buckets it holds intact.
Every data fault here is made on the host side -- bits flipped, buckets
zeroed, swapped, or never received, buffers that do not match the plan -- and
checked through the C ABI.  The only device-side waits (the bulk engine's
barriers) are bounded; the last test makes one run out on purpose, through a
barrier that nothing completes, and checks that the host sees the status and
the context stays usable.  Also: guard bytes around every output stay
untouched, two streams share one plan, and repeated runs give identical bits.
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


def packed(name="tiny-tp4", **kw):
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan, **kw)
    H.fill_with_generator(buf, m, desc["seed"], desc["specials"])
    H.pack(buf)
    torch.cuda.synchronize()
    return desc, plan, buf


def test_damage_is_found_at_the_right_bucket():
    _, plan, buf = packed()
    bl = H.bucket_list(buf)
    assert H.verify(buf) == (0, -1)
    bl[9][1000] ^= 0x01                       # one flipped bit
    assert H.verify(buf) == (1, 9)
    bl[9][1000] ^= 0x01
    saved = bl[30].clone()
    bl[30].zero_()                            # a bucket that never arrived
    assert H.verify(buf) == (1, 30)
    bl[30].copy_(saved)
    a, b = bl[40].clone(), bl[41].clone()     # two buckets delivered in swapped slots
    bl[40].copy_(b)
    bl[41].copy_(a)
    assert H.verify(buf) == (2, 40)
    bl[40].copy_(a)
    bl[41].copy_(b)
    assert H.verify(buf) == (0, -1)


def test_partial_pull_then_resume():
    """A receiver that pulled only some buckets sees exactly the missing ones;
    once it pulls the rest, its unpacked tensors equal a full pull's."""
    desc, plan, sender = packed()
    receiver = H.alloc(plan)
    receiver.checksums.copy_(sender.checksums)
    src_b, dst_b = H.bucket_list(sender), H.bucket_list(receiver)
    got = [b for b in range(plan.n_buckets) if b % 3 != 1]   # every third bucket lost
    for b in got:
        dst_b[b].copy_(src_b[b])
    n_bad, first = H.verify(receiver)
    assert (n_bad, first) == (plan.n_buckets - len(got), 1)
    for b in range(plan.n_buckets):
        if b % 3 == 1:
            dst_b[b].copy_(src_b[b])
    assert H.verify(receiver) == (0, -1)
    H.unpack(receiver)
    H.unpack(sender)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        assert torch.equal(receiver.dst[t], sender.dst[t])


def test_buffers_that_do_not_match_the_plan_are_refused():
    _, plan, buf = packed()
    _, other_plan, other = packed("tiny-moe-tp2")
    with pytest.raises(ValueError):          # buckets of another plan: wrong count / size
        rr.rr_pack(plan, buf.shards, other.buckets, buf.checksums)
    with pytest.raises(ValueError):
        rr.rr_unpack(plan, buf.buckets, other.dst)
    with pytest.raises(ValueError):
        rr.rr_verify(plan, buf.buckets, buf.checksums[:3])


def test_misaligned_pointers_are_refused():
    _, plan, buf = packed()
    shards = list(buf.shards)
    shards[3] += 2
    with pytest.raises(rr.RRError) as e:
        rr.rr_pack(plan, shards, buf.buckets, buf.checksums)
    assert e.value.status == rrmod.RR_EINVAL
    dst = [t.data_ptr() for t in buf.dst]
    dst[5] += 8
    with pytest.raises(rr.RRError) as e:
        rr.rr_unpack(plan, buf.buckets, dst)
    assert e.value.status == rrmod.RR_EINVAL


def test_guard_bytes_stay_untouched():
    """Buckets and tensors placed inside larger allocations with 4 KiB guard
    zones on both sides; after pack + unpack + verify every guard byte is
    still the fill pattern."""
    desc = U.workload_desc("tiny-moe-tp2")
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    G = 4096
    B = plan.bucket_bytes
    slot = G + (B + 15) // 16 * 16 + G
    arena = torch.full((plan.n_buckets * slot,), 0xCD, dtype=torch.uint8, device="cuda")
    bptr = [arena.data_ptr() + i * slot + G for i in range(plan.n_buckets)]
    tarenas = [torch.full((G + 2 * n + G,), 0xCD, dtype=torch.uint8, device="cuda")
               for n in plan.tensor_numel]
    tptr = [a.data_ptr() + G for a in tarenas]
    buf = H.alloc(plan, with_dst=False)
    shards = L.host_shards(desc["seed"], desc["specials"])
    H.fill_from_host(buf, shards)
    rr.rr_pack(plan, buf.shards, bptr, buf.checksums)
    rr.rr_unpack(plan, bptr, tptr)
    assert rr.rr_verify(plan, bptr, buf.checksums) == (0, -1)
    torch.cuda.synchronize()
    a = arena.view(plan.n_buckets, slot).cpu().numpy()
    assert np.all(a[:, :G] == 0xCD) and np.all(a[:, G + B:] == 0xCD)
    want, _ = L.pack(oracle.Source(shards=shards))
    np.testing.assert_array_equal(a[:, G:G + B], want)
    for t, ta in enumerate(tarenas):
        h = ta.cpu().numpy()
        n = 2 * plan.tensor_numel[t]
        assert np.all(h[:G] == 0xCD) and np.all(h[G + n:] == 0xCD), plan.tensor_names[t]
        np.testing.assert_array_equal(h[G:G + n].view(np.uint16), L.unpack_tensor(want, t))


def test_two_streams_share_one_plan():
    desc = U.workload_desc("tiny-tp4")
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    bufs = [H.alloc(plan) for _ in range(2)]
    for b in bufs:
        H.fill_with_generator(b, m, desc["seed"], desc["specials"])
    torch.cuda.synchronize()
    streams = [torch.cuda.Stream() for _ in range(2)]
    for _ in range(5):
        for b, st in zip(bufs, streams):
            with torch.cuda.stream(st):
                H.pack(b, st)
                H.unpack(b, st)
    torch.cuda.synchronize()
    assert torch.equal(bufs[0].bucket_store, bufs[1].bucket_store)
    assert torch.equal(bufs[0].checksums, bufs[1].checksums)
    for t in range(plan.n_tensors):
        assert torch.equal(bufs[0].dst[t], bufs[1].dst[t])


def test_repeated_runs_are_bit_identical():
    _, plan, buf = packed("tiny-moe-tp2")
    first = buf.bucket_store.clone()
    cs = buf.checksums.clone()
    for _ in range(3):
        buf.bucket_store.fill_(0x77)
        H.pack(buf)
        torch.cuda.synchronize()
        assert torch.equal(buf.bucket_store, first)
        assert torch.equal(buf.checksums, cs)


def test_empty_layout():
    """No tensors: zero buckets; every call is a no-op that succeeds."""
    plan = rr.rr_plan_create([rr.Param("a", (4, 4))], rr.SrcLayout(n_shards=2),
                             rr.DstLayout(tp=2, tensors=[]), 64)
    assert plan.n_buckets == 0
    flat = torch.zeros(2 * plan.shard_bytes, dtype=torch.uint8, device="cuda")
    shards = [flat.data_ptr(), flat.data_ptr() + plan.shard_bytes]
    cs = torch.zeros(1, dtype=torch.int64, device="cuda")
    rr.rr_pack(plan, shards, [], cs)
    rr.rr_unpack(plan, [], [])
    assert rr.rr_verify(plan, [], cs) == (0, -1)


def test_bounded_wait_reports_and_context_survives():
    """A device wait that nothing satisfies gives up after about a second, marks
    the plan, and the host sees RR_ECUDA; afterwards the context still works and
    results are still exact."""
    import time
    desc, plan, buf = packed("tiny-tp4")
    rr.rr_plan_check(plan)                                  # clean
    t0 = time.time()
    rr.rr_plan_selftest_wait(plan)
    with pytest.raises(rr.RRError) as e:
        rr.rr_plan_check(plan)
    assert e.value.status == rrmod.RR_ECUDA
    assert time.time() - t0 < 30
    rr.rr_plan_check(plan)                                  # the mark was cleared
    # The verifying calls report a mark left by an earlier kernel too.
    rr.rr_plan_selftest_wait(plan)
    with pytest.raises(rr.RRError):
        rr.rr_verify(plan, buf.buckets, buf.checksums)
    # And the plan keeps working, bit for bit.
    H.pack(buf)
    assert rr.rr_verify(plan, buf.buckets, buf.checksums) == (0, -1)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    L = U.to_oracle(desc)
    want, _ = L.pack(oracle.Source(seed=desc["seed"], specials=desc["specials"]))
    np.testing.assert_array_equal(H.buckets_host(buf), want)
