"""Resumable weight sync on the GPU (Section 5.2.2): bucket-range pack, unpack
and verify, per-bucket verify flags, and the clear path, through the C ABI.

A relay that dies mid-pull: the rollout keeps the buckets it verified and
pulls the rest from another relay.  A trainer that dies mid-pull: the partly
received buckets are cleared and the pull starts over.  Ranges are checked
against the oracle bucket by bucket and element by element, and everything
outside a range must stay untouched.
"""
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


def setup(name, **kw):
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan, **kw)
    shards = L.host_shards(desc["seed"], desc["specials"])
    H.fill_from_host(buf, shards)
    return desc, L, plan, buf, shards


def ranges(n, seed):
    rng = np.random.default_rng(seed)
    out = [(0, 0), (0, n), (n - 1, 1), (0, 1), (n, 0)]
    for _ in range(4):
        a = int(rng.integers(0, n))
        out.append((a, int(rng.integers(0, n - a + 1))))
    return out


@pytest.mark.parametrize("name,separate", [("tiny-tp4", False), ("tiny-moe-tp2", True),
                                           ("tiny", False)])
def test_pack_range_touches_only_its_buckets(name, separate):
    desc, L, plan, buf, shards = setup(name, separate_buckets=separate)
    want, want_cs = L.pack(oracle.Source(shards=shards))
    for b0, n in ranges(plan.n_buckets, 3):
        for b in H.bucket_list(buf):
            b.fill_(0xAB)
        buf.checksums.fill_(0x1234)
        rr.rr_pack_range(plan, b0, n, buf.shards, buf.buckets, buf.checksums)
        torch.cuda.synchronize()
        got = H.buckets_host(buf)
        cs = buf.checksums.cpu().numpy().view(np.uint64)
        for b in range(plan.n_buckets):
            if b0 <= b < b0 + n:
                np.testing.assert_array_equal(got[b], want[b], err_msg=f"bucket {b}")
                assert cs[b] == want_cs[b]
            else:
                assert np.all(got[b] == 0xAB) and cs[b] == 0x1234, f"bucket {b} touched"


@pytest.mark.parametrize("name", ["tiny-tp4", "tiny-moe-tp2"])
def test_unpack_range_writes_exactly_its_bytes(name):
    desc, L, plan, buf, shards = setup(name)
    H.pack(buf)
    torch.cuda.synchronize()
    want_b = H.buckets_host(buf)
    B = plan.bucket_bytes
    for b0, n in ranges(plan.n_buckets, 5):
        for t in buf.dst:
            t.fill_(0x5A5A)
        rr.rr_unpack_range(plan, b0, n, buf.buckets, buf.dst)
        torch.cuda.synchronize()
        for t in range(plan.n_tensors):
            got = H.tensor_host(buf, t)
            full = L.unpack_tensor(want_b, t)
            r = plan.tensor_ranks[t]
            pos = plan.first_bucket_of_rank[r] * B + plan.tensor_stream_offset[t] + \
                2 * np.arange(plan.tensor_numel[t], dtype=np.int64)
            inside = (pos >= b0 * B) & (pos < (b0 + n) * B)
            np.testing.assert_array_equal(got[inside], full[inside])
            assert np.all(got[~inside] == 0x5A5A), plan.tensor_names[t]


def test_verify_range_flags():
    desc, L, plan, buf, shards = setup("tiny-tp4")
    H.pack(buf)
    bl = H.bucket_list(buf)
    for b in (3, 4, 17, 40):
        bl[b][b * 7 % plan.bucket_bytes] ^= 0x80
    bad = torch.full((plan.n_buckets,), 7, dtype=torch.uint8, device="cuda")
    assert rr.rr_verify_range(plan, 0, plan.n_buckets, buf.buckets, buf.checksums, bad) == (4, 3)
    flags = bad.cpu().numpy()
    assert set(np.flatnonzero(flags)) == {3, 4, 17, 40} and set(np.unique(flags)) <= {0, 1}
    bad.fill_(7)
    assert rr.rr_verify_range(plan, 10, 20, buf.buckets, buf.checksums, bad) == (1, 17)
    assert list(np.flatnonzero(bad.cpu().numpy()[:20])) == [7] and bad.cpu().numpy()[20] == 7
    assert rr.rr_verify_range(plan, 5, 12, buf.buckets, buf.checksums) == (0, -1)
    with pytest.raises(rr.RRError):
        rr.rr_verify_range(plan, plan.n_buckets - 2, 3, buf.buckets, buf.checksums)


def test_relay_failure_resume():
    """Pull buckets from relay A until it dies, keep what verifies, pull the rest
    from relay B; the result equals one uninterrupted pull."""
    desc, L, plan, trainer, shards = setup("tiny-tp4")
    H.pack(trainer)
    relay_a, relay_b, rollout = (H.alloc(plan) for _ in range(3))
    for r in (relay_a, relay_b):
        r.bucket_store.copy_(trainer.bucket_store)
        r.checksums.copy_(trainer.checksums)
    rollout.checksums.copy_(trainer.checksums)
    n = plan.n_buckets
    k = n // 3
    src, dst = H.bucket_list(relay_a), H.bucket_list(rollout)
    for b in range(k):
        dst[b].copy_(src[b])
    dst[k][:100].copy_(src[k][:100])              # relay A dies halfway through bucket k
    bad = torch.zeros(n, dtype=torch.uint8, device="cuda")
    n_bad, first = rr.rr_verify_range(plan, 0, n, rollout.buckets, rollout.checksums, bad)
    assert first == k and n_bad == n - k
    missing = np.flatnonzero(bad.cpu().numpy())
    rr.rr_unpack_range(plan, 0, k, rollout.buckets, rollout.dst)   # what arrived intact
    src_b = H.bucket_list(relay_b)
    for b in missing:
        dst[b].copy_(src_b[b])
    assert rr.rr_verify_range(plan, k, n - k, rollout.buckets, rollout.checksums) == (0, -1)
    rr.rr_unpack_range(plan, k, n - k, rollout.buckets, rollout.dst)
    H.unpack(trainer)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        assert torch.equal(rollout.dst[t], trainer.dst[t]), plan.tensor_names[t]


def test_trainer_failure_clear_and_repull():
    desc, L, plan, trainer, shards = setup("tiny-moe-tp2")
    rollout = H.alloc(plan)
    H.pack(trainer)
    rollout.checksums.copy_(trainer.checksums)
    src, dst = H.bucket_list(trainer), H.bucket_list(rollout)
    k = plan.n_buckets // 2
    for b in range(k):
        dst[b].copy_(src[b])
    # The trainer dies: the partial pull is cleared.
    rr.rr_clear_range(plan, 0, plan.n_buckets, rollout.buckets)
    torch.cuda.synchronize()
    assert all(int(b.abs().sum()) == 0 for b in dst)
    cs = trainer.checksums.cpu().numpy().view(np.uint64)
    n_zero_cs = int((cs == 0).sum())
    n_bad, _ = rr.rr_verify(plan, rollout.buckets, rollout.checksums)
    assert n_bad == plan.n_buckets - n_zero_cs
    # The trainer is back: it re-packs from its restored state, the rollout pulls again.
    H.pack(trainer)
    for b in range(plan.n_buckets):
        dst[b].copy_(src[b])
    assert rr.rr_verify(plan, rollout.buckets, rollout.checksums) == (0, -1)
    H.unpack(rollout)
    torch.cuda.synchronize()
    want, _ = L.pack(oracle.Source(shards=shards))
    for t in range(plan.n_tensors):
        np.testing.assert_array_equal(H.tensor_host(rollout, t), L.unpack_tensor(want, t))


def test_clear_range_separate_buckets():
    desc, L, plan, buf, shards = setup("tiny-tp4", separate_buckets=True)
    H.pack(buf)
    before = [b.clone() for b in H.bucket_list(buf)]
    rr.rr_clear_range(plan, 5, 9, buf.buckets)
    torch.cuda.synchronize()
    for b, (now, old) in enumerate(zip(H.bucket_list(buf), before)):
        if 5 <= b < 14:
            assert int(now.sum()) == 0, b
        else:
            assert torch.equal(now, old), b


def test_full_size_range_pack_of_one_rank():
    """Qwen3-8B TP=4: pack only rank 2's buckets; they equal the full pack's."""
    w = U.workload("qwen3-8b-tp4")
    desc = U.workload_desc("qwen3-8b-tp4")
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, w.bucket_bytes)
    buf = H.alloc(plan, poison=None, with_dst=False)
    H.fill_with_generator(buf, m, w.seed, w.specials)
    fr = plan.first_bucket_of_rank
    H.pack(buf)
    full = buf.bucket_store[fr[2]:fr[3]].clone()
    full_cs = buf.checksums[fr[2]:fr[3]].clone()
    buf.bucket_store.fill_(0)
    buf.checksums.fill_(0)
    rr.rr_pack_range(plan, fr[2], fr[3] - fr[2], buf.shards, buf.buckets, buf.checksums)
    torch.cuda.synchronize()
    assert torch.equal(buf.bucket_store[fr[2]:fr[3]], full)
    assert torch.equal(buf.checksums[fr[2]:fr[3]], full_cs)
    assert int(buf.bucket_store[:fr[2]].sum()) == 0 and int(buf.bucket_store[fr[3]:].sum()) == 0
    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    want, want_cs = L.pack(gen, first=fr[2] + 3, count=1)
    np.testing.assert_array_equal(H.buckets_host(buf, [fr[2] + 3])[0], want[0])


@pytest.mark.parametrize("name,separate", [("tiny-tp4", False), ("tiny-moe-f32", True),
                                           ("tiny", False)])
def test_unpack_verify_equals_unpack_then_verify(name, separate):
    desc, L, plan, buf, shards = setup(name, separate_buckets=separate)
    H.pack(buf)
    H.unpack(buf)
    torch.cuda.synchronize()
    want = [t.clone() for t in buf.dst]
    for t in buf.dst:
        t.fill_(0x5A5A)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    for t in range(plan.n_tensors):
        assert torch.equal(buf.dst[t], want[t])
    # Damage: a byte inside a tensor, and a byte in an alignment gap or tail
    # (which no tensor holds, so only the checksum can notice it).
    bl = H.bucket_list(buf)
    items, _ = plan.export_unpack()
    gaps = items[items["kind"] >= U.ITEM_READ_VEC]
    g = gaps[len(gaps) // 2]
    bl[int(g["bucket"])][int(g["src_off"])] ^= 0x01
    bl[2][333] ^= 0x10
    hit = sorted({2, int(g["bucket"])})
    bad = torch.zeros(plan.n_buckets, dtype=torch.uint8, device="cuda")
    got = rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst, bad)
    assert got == rr.rr_verify(plan, buf.buckets, buf.checksums) == (len(hit), hit[0])
    assert list(np.flatnonzero(bad.cpu().numpy())) == hit
    # Range form over the second half only.
    h = plan.n_buckets // 2
    got = rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst, first_bucket=h,
                              n_buckets=plan.n_buckets - h)
    assert got == rr.rr_verify_range(plan, h, plan.n_buckets - h, buf.buckets, buf.checksums)


def test_unpack_verify_full_size():
    w = U.workload("qwen3-30b-a3b")
    desc = U.workload_desc("qwen3-30b-a3b")
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, w.bucket_bytes)
    buf = H.alloc(plan, poison=None)
    H.fill_with_generator(buf, m, w.seed, w.specials)
    H.pack(buf)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    B = plan.bucket_bytes
    store = buf.bucket_store.view(-1)
    for t in range(plan.n_tensors):
        start = plan.first_bucket_of_rank[plan.tensor_ranks[t]] * B + plan.tensor_stream_offset[t]
        n = plan.tensor_numel[t]
        assert torch.equal(buf.dst[t][:n], store[start:start + 2 * n].view(torch.int16))
    buf.bucket_store[100, 12345] ^= 1
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (1, 100)
