"""Relay re-pack (Section 5.2.1, step 3): a rollout that holds the new weights
serves another rollout, possibly with another tensor-parallel degree.

The relay's copy is the rollout image in bf16 -- its loaded tensors or the
buckets it pulled.  Re-packing that copy into the target layout must give
exactly what the trainer itself would have packed for the target (the cast
happened once, on the trainer; a bf16 re-pack copies bits).  The expected
buckets come from the oracle packing the original trainer weights straight
into the target layout.
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
from paper_2512_22492_gb300 import layouts
from tests import _util as U

PAIRS = [(4, 4), (4, 2), (2, 4), (4, 1), (1, 4), (2, 1)]


def trainer_image(name, src_tp, src_ep=False):
    """The oracle's trainer source, its TP=src_tp rollout tensors and buckets."""
    return trainer_image_of(U.workload(name), src_tp, src_ep)


def trainer_image_of(w, src_tp, src_ep=False):
    w = w.with_(tp=src_tp, ep=src_ep)
    L = oracle.workload_layout(w)
    src = oracle.Source(shards=L.host_shards(w.seed, w.specials))
    tensors = [L.reshard_tensor(src, t) for t in range(len(L.tensors))]
    buckets, _ = L.pack(src)
    return w, src, tensors, buckets


def expected(w, src, dst_tp, bucket_bytes, dst_ep=False):
    L = oracle.workload_layout(w.with_(tp=dst_tp, ep=dst_ep), bucket_bytes=bucket_bytes)
    return L.pack(src)


# (src_tp, src_ep, dst_tp, dst_ep): tensor-parallel and expert-parallel rollouts
# serving one another.
EP_CASES = [(4, False, 4, True), (4, True, 2, False), (2, True, 4, True), (2, False, 2, True),
            (8, True, 1, False)]


@pytest.mark.parametrize("src_tp,src_ep,dst_tp,dst_ep", EP_CASES)
def test_relay_tables_expert_parallel(src_tp, src_ep, dst_tp, dst_ep):
    w, src, tensors, buckets = trainer_image("tiny-moe-f32", src_tp, src_ep)
    B = 16 * 1024
    want, _ = expected(w, src, dst_tp, B, dst_ep)
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, src_ep=src_ep, dst_ep=dst_ep)
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    got = U.check_and_run_pack(items, [x.view(np.uint8) for x in tensors], plan.n_buckets, B,
                               plan.shard_bytes)
    np.testing.assert_array_equal(got, want)
    m0, s0, d0 = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, src_tp, ep=src_ep)
    src_plan = rr.rr_plan_create(m0, s0, d0, w.bucket_bytes, rr.PlanOptions(host_only=True))
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, from_plan=src_plan, src_ep=src_ep,
                                  dst_ep=dst_ep)
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    got = U.check_and_run_pack(items, [b for b in buckets], plan.n_buckets, B, plan.shard_bytes)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("name", ["tiny", "tiny-moe-f32"])
@pytest.mark.parametrize("src_tp,dst_tp", PAIRS)
def test_relay_tables_from_tensors(name, src_tp, dst_tp):
    w, src, tensors, _ = trainer_image(name, src_tp)
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp)
    B = 16 * 1024
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    shards = [t.view(np.uint8) for t in tensors]
    got = U.check_and_run_pack(items, shards, plan.n_buckets, B, plan.shard_bytes)
    want, _ = expected(w, src, dst_tp, B)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("src_tp,dst_tp", [(4, 2), (2, 4), (1, 2)])
def test_relay_tables_from_buckets(src_tp, dst_tp):
    w, src, _, buckets = trainer_image("tiny-moe-f32", src_tp)
    m0, s0, d0 = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, src_tp)
    src_plan = rr.rr_plan_create(m0, s0, d0, w.bucket_bytes, rr.PlanOptions(host_only=True))
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, from_plan=src_plan)
    B = 8 * 1024
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    got = U.check_and_run_pack(items, [b for b in buckets], plan.n_buckets, B, plan.shard_bytes)
    want, _ = expected(w, src, dst_tp, B)
    np.testing.assert_array_equal(got, want)


@pytest.mark.gpu
@pytest.mark.parametrize("src_tp,dst_tp", [(4, 2), (2, 4), (4, 4), (4, 1)])
def test_relay_on_gpu(src_tp, dst_tp):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w, src, tensors, buckets = trainer_image("tiny-moe-f32", src_tp)
    B = 16 * 1024
    want, want_cs = expected(w, src, dst_tp, B)
    # From the relay's loaded tensors.
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp)
    plan = rr.rr_plan_create(m, s, d, B)
    dev_t = [torch.from_numpy(t.view(np.int16).copy()).cuda() for t in tensors]
    out = torch.full((plan.n_buckets, B), 0xAB, dtype=torch.uint8, device="cuda")
    cs = torch.zeros(plan.n_buckets, dtype=torch.int64, device="cuda")
    rr.rr_pack(plan, dev_t, out, cs)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy(), want)
    np.testing.assert_array_equal(cs.cpu().numpy().view(np.uint64), want_cs)
    # From the buckets it pulled.
    m0, s0, d0 = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, src_tp)
    src_plan = rr.rr_plan_create(m0, s0, d0, w.bucket_bytes, rr.PlanOptions(host_only=True))
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, from_plan=src_plan)
    plan = rr.rr_plan_create(m, s, d, B)
    pulled = torch.from_numpy(buckets.copy()).cuda()
    out.fill_(0xAB)
    rr.rr_pack(plan, pulled, out, cs)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy(), want)
    np.testing.assert_array_equal(cs.cpu().numpy().view(np.uint64), want_cs)


@pytest.mark.gpu
@pytest.mark.parametrize("src_tp,src_ep,dst_tp,dst_ep", EP_CASES[:3])
def test_relay_expert_parallel_on_gpu(src_tp, src_ep, dst_tp, dst_ep):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    w, src, tensors, _ = trainer_image("tiny-moe-f32", src_tp, src_ep)
    B = 16 * 1024
    want, want_cs = expected(w, src, dst_tp, B, dst_ep)
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, src_ep=src_ep, dst_ep=dst_ep)
    plan = rr.rr_plan_create(m, s, d, B)
    dev_t = [torch.from_numpy(t.view(np.int16).copy()).cuda() for t in tensors]
    out = torch.full((plan.n_buckets, B), 0xAB, dtype=torch.uint8, device="cuda")
    cs = torch.zeros(plan.n_buckets, dtype=torch.int64, device="cuda")
    rr.rr_pack(plan, dev_t, out, cs)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(out.cpu().numpy(), want)
    np.testing.assert_array_equal(cs.cpu().numpy().view(np.uint64), want_cs)


@pytest.mark.parametrize("src_tp,dst_tp", [(4, 2), (1, 4)])
def test_relay_of_a_float16_image(src_tp, dst_tp):
    """A float16 rollout relays like a bf16 one: the relay copies the 16-bit
    elements, so re-packing the TP=src_tp float16 image (from its tensors and
    from its buckets) gives the oracle's float16 pack of the TP=dst_tp layout."""
    w0 = U.workload("tiny-moe-f32").with_(dst_dtype="f16")
    w, src, tensors, buckets = trainer_image_of(w0, src_tp)
    B = 16 * 1024
    want, _ = expected(w, src, dst_tp, B)
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp)
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    got = U.check_and_run_pack(items, [t.view(np.uint8) for t in tensors], plan.n_buckets, B,
                               plan.shard_bytes)
    np.testing.assert_array_equal(got, want)
    m0, s0, d0 = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, src_tp, dst_dtype="f16")
    src_plan = rr.rr_plan_create(m0, s0, d0, w.bucket_bytes, rr.PlanOptions(host_only=True))
    m, s, d = layouts.qwen3_relay(w.shape, src_tp, dst_tp, from_plan=src_plan)
    plan = rr.rr_plan_create(m, s, d, B, rr.PlanOptions(host_only=True))
    items, _ = plan.export_pack()
    got = U.check_and_run_pack(items, [b for b in buckets], plan.n_buckets, B, plan.shard_bytes)
    np.testing.assert_array_equal(got, want)
