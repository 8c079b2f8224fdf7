"""GPU parity for a float16 rollout: the same reshard, buckets and checksums with
IEEE binary16 elements (Section 7.4 counts the transferred model as FP16),
against the oracle bit for bit.

* small workloads on both engines: fp32 with special values (ties,
  subnormals, overflow, infinities, NaNs), a bf16 source with special bit
  patterns (widened, then rounded), TP=4, FSDP2 rows, KV replication, per-layer
  units, expert parallel;
* random ragged layouts and random row-parallel layouts (the fan-out groups);
* the pack from pinned host memory; bucket ranges into separately allocated
  buckets;
* full-size Qwen3-8B and Qwen3-30B-A3B: sampled buckets against the oracle,
  every checksum against torch's word sum, sampled tensors against the
  oracle's reshard.
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
    torch.cuda.synchronize()
    torch.cuda.empty_cache()


def f16(desc):
    desc = dict(desc)
    if desc.get("workload") is not None:
        desc["workload"] = desc["workload"].with_(dst_dtype="f16")
    else:
        desc["dst_dtype"] = "f16"
    return desc


def parity(desc, host_source=False, **opts):
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    assert d.dtype == "f16" and L.dst_dtype == "f16"
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], **opts)
    shards = L.host_shards(desc["seed"], desc["specials"])
    if host_source:
        flat = torch.from_numpy(np.concatenate([np.asarray(x, np.uint8) for x in shards]))
        buf = H.alloc(plan, flat=flat.pin_memory())
    else:
        buf = H.alloc(plan)
        H.fill_from_host(buf, shards)
    H.pack(buf)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    rr.rr_plan_check(plan)
    src = oracle.Source(shards=shards)
    want, want_cs = L.pack(src)
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
    for t in range(len(L.tensors)):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(src, t),
                                      err_msg=f"tensor {t}")


@pytest.mark.parametrize("engine", ["auto", "registers"])
@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-moe-bf16-specials", "tiny-fsdp2",
                                  "tiny-moe-kvrep", "tiny-kvrep-f32", "tiny-units",
                                  "tiny-moe-ep4"])
def test_small_workloads_f16(name, engine):
    parity(f16(U.workload_desc(name)), engine=engine)


@pytest.mark.parametrize("seed", range(8))
def test_random_layouts_f16(seed):
    parity(f16(U.random_layout(seed)), engine="registers" if seed % 3 == 0 else "auto")


@pytest.mark.parametrize("seed", range(8))
def test_random_row_parallel_layouts_f16(seed):
    parity(f16(U.random_tp_layout(seed)), engine="registers" if seed % 3 == 0 else "auto")


@pytest.mark.parametrize("name", ["tiny", "tiny-moe-bf16-specials"])
def test_host_source_f16(name):
    parity(f16(U.workload_desc(name)), host_source=True)


def test_item_checks_f16():
    parity(f16(U.workload_desc("tiny-tp4")), check_items=True)
    parity(f16(U.random_tp_layout(2)), check_items=True)


def test_a_bf16_plan_and_an_f16_plan_differ_only_in_the_cast():
    """Same layout, both element types: the same buckets, stream offsets,
    tensor sizes and algorithmic bytes (the element values are checked against
    the oracle by the tests above)."""
    desc = U.workload_desc("tiny-tp4")
    m, s, d = U.to_product(desc)
    m2, s2, d2 = U.to_product(f16(desc))
    a = H.make_plan(m, s, d, desc["bucket_bytes"])
    b = H.make_plan(m2, s2, d2, desc["bucket_bytes"])
    assert (a.n_buckets, a.stream_bytes_per_rank, a.tensor_numel) == \
        (b.n_buckets, b.stream_bytes_per_rank, b.tensor_numel)
    assert a.stats()["pack_bytes_read"] == b.stats()["pack_bytes_read"]


@pytest.mark.parametrize("name,names", [
    ("qwen3-8b", [("embed_tokens", 0), ("layers.17.o_proj", 0), ("norm", 0), ("lm_head", 0)]),
    ("qwen3-30b-a3b", [("layers.0.router", 0), ("layers.47.experts.w2", 0), ("norm", 0)]),
])
def test_full_size_f16_sampled(name, names):
    w = U.workload(name).with_(dst_dtype="f16")
    m, s, d = rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep,
                            dst_dtype="f16")
    plan = H.make_plan(m, s, d, w.bucket_bytes)
    buf = H.alloc(plan, poison=0xAB)
    H.fill_with_generator(buf, m, w.seed, w.specials)
    H.pack(buf)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (0, -1)
    torch.cuda.synchronize()
    np.testing.assert_array_equal(H.checksums_host(buf), H.device_word_sums(buf))
    L = oracle.workload_layout(w)
    assert L.dst_dtype == "f16" and L.n_buckets == plan.n_buckets
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    cs = H.checksums_host(buf)
    rng = np.random.default_rng(16)
    for b in sorted({0, plan.n_buckets - 1, *rng.integers(0, plan.n_buckets, 2).tolist()}):
        want, want_cs = L.pack(gen, first=b, count=1)
        np.testing.assert_array_equal(H.buckets_host(buf, [b])[0], want[0], err_msg=f"bucket {b}")
        assert cs[b] == want_cs[0]
    for nm, rank in names:
        t = L.tensor_index(nm, rank)
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(gen, t),
                                      err_msg=nm)
    buf = None
    torch.cuda.empty_cache()


@pytest.mark.parametrize("engine", ["auto", "registers"])
def test_ranges_and_separate_buckets_f16(engine):
    """rr_pack_range over three ranges (last first) into separately allocated
    buckets (the pointer-table launch shape), float16 destination."""
    desc = f16(U.workload_desc("tiny-tp4"))
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], engine=engine)
    shards = L.host_shards(desc["seed"], desc["specials"])
    buf = H.alloc(plan, separate_buckets=True, with_dst=False)
    H.fill_from_host(buf, shards)
    n = plan.n_buckets
    cuts = [0, n // 3, 2 * n // 3, n]
    for a, b in reversed(list(zip(cuts[:-1], cuts[1:]))):
        rr.rr_pack_range(plan, a, b - a, buf.shards, buf.buckets, buf.checksums)
    torch.cuda.synchronize()
    want, want_cs = L.pack(oracle.Source(shards=shards))
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
