"""Work units claimed at run time by the bulk-copy engine's blocks.

rr_pack and rr_unpack take a slot (a claim counter, and for pack its sums)
from a pool of 16 per plan.  A slot is free once the launch that last held
it has completed.  When none is, a launch takes the slot handed out longest
ago if that slot's launch ran on its own stream, and waits on the GPU for it.
A launch finds no slot when every slot is held by another stream's launch
still in flight, or when it is being captured into a CUDA graph.  It then
zeroes its checksums first and splits its items evenly over the grid.  These
tests drive every one of those paths and compare bytes with the oracle:
  - more launches in flight on one stream than slots (the stream held back by
    a bounded sleep kernel, so that none of them can complete before the rest
    are enqueued), and meanwhile a second stream's launches, which find every
    slot held;
  - two streams packing and unpacking their own buffers at once;
  - the whole step captured into a CUDA graph and replayed on new inputs;
  - a resumed pull's range calls (clear, pack, unpack, stream-ordered check)
    captured into a CUDA graph and replayed over spoiled buckets.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu

SLEEP_CYCLES = 100_000_000   # about 50 ms at GB300 clocks: longer than enqueueing the calls


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    yield


def setup(name="tiny-moe-tp2"):
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    L = U.to_oracle(desc)
    shards = L.host_shards(desc["seed"], desc["specials"])
    want, want_cs = L.pack(oracle.Source(shards=shards))
    return desc, m, plan, L, shards, want, want_cs


def tensors_want(L, want, plan):
    return [L.unpack_tensor(want, t) for t in range(plan.n_tensors)]


def check(plan, buf, want, want_cs, want_t):
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(H.tensor_host(buf, t), want_t[t])


def test_more_launches_in_flight_than_claim_slots():
    if not hasattr(torch.cuda, "_sleep"):
        pytest.skip("this PyTorch has no bounded sleep kernel to hold the stream")
    desc, m, plan, L, shards, want, want_cs = setup()
    want_t = tensors_want(L, want, plan)
    first = H.alloc(plan)
    H.fill_from_host(first, shards)
    bufs = [H.alloc(plan, flat=first.flat) for _ in range(24)]
    side = [H.alloc(plan, flat=first.flat) for _ in range(2)]
    other = torch.cuda.Stream()
    torch.cuda.synchronize()
    torch.cuda._sleep(SLEEP_CYCLES)            # nothing below can complete until it ends
    for b in bufs:                             # past 16, each waits for the oldest slot
        rr.rr_pack(plan, b.shards, b.buckets, b.checksums)
    for b in bufs:
        rr.rr_unpack(plan, b.buckets, b.dst)
    for b in side:                             # every slot held by the first stream: none
        rr.rr_pack(plan, b.shards, b.buckets, b.checksums, stream=other)
        rr.rr_unpack(plan, b.buckets, b.dst, stream=other)
    torch.cuda.synchronize()
    for b in bufs + side:
        check(plan, b, want, want_cs, want_t)
    # The pool is whole again: later launches claim as usual.
    for b in bufs[:3]:
        for t in b.dst:
            t.fill_(0)
        rr.rr_pack(plan, b.shards, b.buckets, b.checksums)
        rr.rr_unpack(plan, b.buckets, b.dst)
    torch.cuda.synchronize()
    for b in bufs[:3]:
        check(plan, b, want, want_cs, want_t)
    rr.rr_plan_check(plan)


@pytest.mark.parametrize("name", ["tiny-moe-tp2", "qwen3-0.6b"])
def test_two_streams_at_once(name):
    """Each stream packs, unpacks and verifies its own copy, eight times over,
    on one plan; claim slots are shared between the streams' launches."""
    if name == "qwen3-0.6b":
        w = U.workload_desc(name)
        m, s, d = U.to_product(w)
        plan = H.make_plan(m, s, d, w["bucket_bytes"])
        bufs = [H.alloc(plan, poison=None) for _ in range(2)]
        for b in bufs:
            H.fill_with_generator(b, m, w["seed"], w["specials"])
        H.pack(bufs[0])
        H.unpack(bufs[0])
        torch.cuda.synchronize()
        ref_buckets = bufs[0].bucket_store.clone()
        ref_cs = bufs[0].checksums.clone()
        ref_t = [t.clone() for t in bufs[0].dst]
    else:
        desc, m, plan, L, shards, want, want_cs = setup(name)
        bufs = [H.alloc(plan) for _ in range(2)]
        for b in bufs:
            H.fill_from_host(b, shards)
    streams = [torch.cuda.Stream() for _ in bufs]
    torch.cuda.synchronize()
    for _ in range(8):
        for b, st in zip(bufs, streams):
            with torch.cuda.stream(st):
                rr.rr_pack(plan, b.shards, b.buckets, b.checksums, stream=st)
                rr.rr_unpack(plan, b.buckets, b.dst, stream=st)
    torch.cuda.synchronize()
    for b in bufs:
        if name == "qwen3-0.6b":
            assert torch.equal(b.bucket_store, ref_buckets)
            assert torch.equal(b.checksums, ref_cs)
            for t, r in zip(b.dst, ref_t):
                assert torch.equal(t, r)
        else:
            check(plan, b, want, want_cs, tensors_want(L, want, plan))
        assert rr.rr_verify(plan, b.buckets, b.checksums) == (0, -1)


def test_step_captured_in_a_cuda_graph():
    """rr_pack, the stream-ordered verifying unpack and rr_unpack captured once,
    replayed on a second source: the captured launches keep the even split,
    and the bytes are the oracle's for whichever source the replay read."""
    desc, m, plan, L, shards, want, want_cs = setup()
    buf = H.alloc(plan)
    H.fill_from_host(buf, shards)
    ts = rr.Pointers(plan, "src_shards", buf.shards)
    tb = rr.Pointers(plan, "buckets", buf.buckets)
    td = rr.Pointers(plan, "dst", buf.dst)
    other = H.alloc(plan)
    td2 = rr.Pointers(plan, "dst", other.dst)
    scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")
    result = torch.full((2,), 7, dtype=torch.int64, device="cuda")
    # Warm up on a side stream (first-launch set-up stays out of the capture).
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        rr.rr_pack(plan, ts, tb, buf.checksums)
        rr.rr_unpack_verify_async(plan, tb, buf.checksums, td, scratch, result)
        rr.rr_unpack(plan, tb, td2)
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        rr.rr_pack(plan, ts, tb, buf.checksums)
        rr.rr_unpack_verify_async(plan, tb, buf.checksums, td, scratch, result)
        rr.rr_unpack(plan, tb, td2)
    want_t = tensors_want(L, want, plan)
    for source in range(2):
        if source == 1:   # a second trainer step: new weights in the same buffers
            shards2 = [np.ascontiguousarray(s[::-1]) for s in shards]
            H.fill_from_host(buf, shards2)
            want, want_cs = L.pack(oracle.Source(shards=shards2))
            want_t = tensors_want(L, want, plan)
        for t in buf.dst + other.dst:
            t.fill_(0)
        result.fill_(7)
        g.replay()
        torch.cuda.synchronize()
        check(plan, buf, want, want_cs, want_t)
        for t in range(plan.n_tensors):
            np.testing.assert_array_equal(H.tensor_host(other, t), want_t[t])
        assert result.cpu().tolist() == [0, -1]
    rr.rr_plan_check(plan)


def test_range_calls_captured_in_a_cuda_graph():
    """A resumed pull's stream-ordered calls captured once: clear buckets
    [2, 9), pack them again, unpack them and check them; the replay restores
    exactly the oracle's bytes for those buckets and their tensors' bytes."""
    desc, m, plan, L, shards, want, want_cs = setup()
    buf = H.alloc(plan)
    H.fill_from_host(buf, shards)
    H.pack(buf)
    H.unpack(buf)
    torch.cuda.synchronize()
    first, count = 2, 7
    scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")
    result = torch.full((2,), 7, dtype=torch.int64, device="cuda")
    bad = torch.full((plan.n_buckets,), 9, dtype=torch.uint8, device="cuda")

    def calls():
        rr.rr_clear_range(plan, first, count, buf.buckets)
        rr.rr_pack_range(plan, first, count, buf.shards, buf.buckets, buf.checksums)
        rr.rr_unpack_range(plan, first, count, buf.buckets, buf.dst)
        rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch, result,
                                  bad=bad, first_bucket=first, n_buckets=count)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        calls()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g):
        calls()
    # Spoil the range's buckets, checksums and tensors, then replay.
    for b in range(first, first + count):
        H.bucket_list(buf)[b].fill_(0x33)
    buf.checksums[first:first + count].fill_(5)
    for t in buf.dst:
        t.fill_(0)
    result.fill_(7)
    bad.fill_(9)
    g.replay()
    torch.cuda.synchronize()
    idx = list(range(first, first + count))
    np.testing.assert_array_equal(H.buckets_host(buf, idx), want[first:first + count])
    np.testing.assert_array_equal(H.checksums_host(buf)[first:first + count],
                                  want_cs[first:first + count])
    assert result.cpu().tolist() == [0, -1]
    assert not bad[:count].cpu().numpy().any()
    # The tensors' bytes held by those buckets are the oracle's; the rest stay zero.
    _, unpack_first = plan.bucket_items()
    items, _ = plan.export_unpack()
    sel = items[unpack_first[first]:unpack_first[first + count]]
    copied = sel[(sel["kind"] == U.ITEM_COPY_VEC) | (sel["kind"] == U.ITEM_COPY_SCALAR)]
    assert len(copied) > 0
    want_t = tensors_want(L, want, plan)
    for it in copied:
        t, off, nb = int(it["tensor"]), int(it["dst_off"]) // 2, int(it["nbytes"]) // 2
        np.testing.assert_array_equal(H.tensor_host(buf, t)[off:off + nb], want_t[t][off:off + nb])
    rr.rr_plan_check(plan)
