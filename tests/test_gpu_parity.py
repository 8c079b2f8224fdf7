"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle, bit for bit.

Buckets, checksums and unpacked tensors are integer / bit-pattern data, so the
bar is exact equality (RobustRL Section 5.2.1 steps 1-2; Section 5.2.2 for
the checksums).  Small workloads are compared in full.  The full-size
workloads (Qwen3-8B, Qwen3-8B TP=4, Qwen3-30B-A3B) are compared on every
bucket and checksum, the oracle running on all host cores -- at every size of
the TP=4 bucket sweep, and for the further full-size layouts (FSDP2 -> TP=8,
per-layer FSDP1 units, expert parallel) too.  Sampled tensors are compared
with the oracle one by one, plus properties that hold at any size (every
checksum equals a word sum taken by torch; verify finds nothing; every tensor
equals its own bytes in the buckets).
"""
import numpy as np
import pytest
import torch

import oracle
import paper_2512_22492_gb300 as rr
import synth
from paper_2512_22492_gb300 import rr as rrmod
from tests import _util as U
from tests import gpu_harness as H

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    torch.cuda.init()
    yield
    torch.cuda.synchronize()


def full_parity(desc, separate_buckets=False, **opts):
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], **opts)
    # Separately allocated buckets beyond one launch's pointer table run as
    # several launches over bucket ranges.
    buf = H.alloc(plan, separate_buckets=separate_buckets)
    shards = L.host_shards(desc["seed"], desc["specials"])
    H.fill_from_host(buf, shards)
    H.pack(buf)
    H.unpack(buf)
    n_bad, first = H.verify(buf)
    torch.cuda.synchronize()
    want, want_cs = L.pack(oracle.Source(shards=shards))
    got = H.buckets_host(buf)
    np.testing.assert_array_equal(got, want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)
    for t in range(len(L.tensors)):
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(
            oracle.Source(shards=shards), t), err_msg=f"tensor {t}")
    assert (n_bad, first) == (0, -1)
    return buf, L, shards


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-tied", "tiny-moe", "tiny-moe-tp2",
                                  "tiny-moe-f32", "tiny-fsdp2", "tiny-moe-kvrep",
                                  "tiny-kvrep-f32", "tiny-moe-bf16-specials", "tiny-units",
                                  "tiny-moe-ep4", "tiny-moe-units-ep2"])
def test_small_workloads(name):
    full_parity(U.workload_desc(name))


@pytest.mark.parametrize("name", ["tiny-fsdp2", "tiny-moe-kvrep", "tiny-units",
                                  "tiny-moe-units-ep2"])
def test_device_generator_fill_matches_oracle_shards(name):
    """The harness's device fill of a row-sharded or per-layer-unit trainer equals
    the oracle's host shards byte for byte (both indexed by the flat layout)."""
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan, with_dst=False)
    H.fill_with_generator(buf, m, desc["seed"], desc["specials"])
    torch.cuda.synchronize()
    want = np.concatenate(L.host_shards(desc["seed"], desc["specials"]))
    np.testing.assert_array_equal(buf.flat.cpu().numpy(), want)


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4"])
def test_separately_allocated_buckets(name):
    full_parity(U.workload_desc(name), separate_buckets=True)


@pytest.mark.parametrize("chunk", [16, 1040, 4096])
def test_small_chunks_and_buckets(chunk):
    full_parity(U.workload_desc("tiny-tp4", bucket_bytes=8 * 1024), chunk_bytes=chunk)


@pytest.mark.parametrize("seed", range(24))
def test_random_layouts(seed):
    full_parity(U.random_layout(seed), separate_buckets=bool(seed % 2),
                engine="registers" if seed % 3 == 0 else "auto")


@pytest.mark.parametrize("seed", range(16))
def test_random_row_parallel_layouts(seed):
    """Fan-out groups (narrow column slices over several ranks) and their
    fallbacks, through a full rr_pack and, on the bucket-sorted table, through
    rr_pack_range over two ranges; the register engine on every third seed."""
    desc = U.random_tp_layout(seed)
    full_parity(desc, separate_buckets=bool(seed % 2),
                engine="registers" if seed % 3 == 0 else "auto")
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan, with_dst=False)
    shards = L.host_shards(desc["seed"], desc["specials"])
    H.fill_from_host(buf, shards)
    cut = plan.n_buckets // 3
    for a, b in ((cut, plan.n_buckets), (0, cut)):
        rr.rr_pack_range(plan, a, b - a, buf.shards, buf.buckets, buf.checksums)
    torch.cuda.synchronize()
    want, want_cs = L.pack(oracle.Source(shards=shards))
    np.testing.assert_array_equal(H.buckets_host(buf), want)
    np.testing.assert_array_equal(H.checksums_host(buf), want_cs)


@pytest.mark.parametrize("engine", ["auto", "registers"])
@pytest.mark.parametrize("case", ["tiny-tp4", "tiny-moe-units-ep2", "random-7", "random-21",
                                  "row-parallel-2", "row-parallel-9"])
def test_item_checks_pass_on_valid_plans(case, engine):
    """With check_items every kernel checks each work item against the plan's
    buffers; on the plans the planner writes nothing is refused and the bytes
    are the same."""
    if case.startswith("random-"):
        desc = U.random_layout(int(case.split("-")[1]))
    elif case.startswith("row-parallel-"):
        desc = U.random_tp_layout(int(case.split("-")[2]))
    else:
        desc = U.workload_desc(case)
    full_parity(desc, engine=engine, check_items=True)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], engine=engine, check_items=True)
    buf = H.alloc(plan)
    H.fill_from_host(buf, U.to_oracle(desc).host_shards(desc["seed"], desc["specials"]))
    H.pack(buf)
    rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst)
    rr.rr_plan_check(plan)


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-moe-f32", "tiny-fsdp2"])
def test_register_engine(name):
    """The register path (the fallback for host-resident buffers) on device memory."""
    full_parity(U.workload_desc(name), engine="registers")


@pytest.mark.parametrize("chunk", [16, 1040, 65536, 1 << 20])
def test_bulk_engine_piece_splits(chunk):
    """Items longer than a shared-memory stage and multi-row items split into pieces."""
    full_parity(U.workload_desc("tiny-moe-f32", bucket_bytes=256 * 1024), chunk_bytes=chunk)


def many_tensors_desc(n_tensors, bucket_bytes, tp=1):
    """A parameter of n_tensors rows, each row its own destination tensor."""
    return dict(params=[("p", (n_tensors, 16), 2), ("q", (5, 24), 4)],
                tensors=[(f"t{i}", i % tp, [(0, i, 1, 0, 16)]) for i in range(n_tensors)] +
                        [("q", 0, [(1, 0, 5, 0, 24)])],
                tp=tp, sharding="flat", n_shards=3, bucket_bytes=bucket_bytes, align_bytes=16,
                tensor_align=256, seed=31, specials=True)


@pytest.mark.parametrize("engine", ["auto", "registers"])
def test_more_destination_tensors_than_one_launch_addresses(engine):
    """9001 destination tensors: more than one launch's pointer table holds, so
    unpack runs as several launches over bucket ranges whose tensors fit, and
    the verifying forms add one checksum pass.  Full calls, ranges, the async
    form and separately allocated buckets."""
    desc = many_tensors_desc(9000, 64 * 1024)
    full_parity(desc, engine=engine)
    full_parity(desc, separate_buckets=True, engine=engine)
    L = U.to_oracle(desc)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], engine=engine)
    buf = H.alloc(plan)
    shards = L.host_shards(desc["seed"], desc["specials"])
    H.fill_from_host(buf, shards)
    H.pack(buf)
    H.bucket_list(buf)[20][0] ^= 0x04
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst,
                               first_bucket=3, n_buckets=30) == (1, 20)
    res = torch.zeros(2, dtype=torch.int64, device="cuda")
    scratch = torch.zeros(plan.n_buckets + 4, dtype=torch.int64, device="cuda")
    rr.rr_unpack_verify_async(plan, buf.buckets, buf.checksums, buf.dst, scratch, res)
    torch.cuda.synchronize()
    assert res.cpu().tolist() == [1, 20]
    H.bucket_list(buf)[20][0] ^= 0x04
    for x in buf.dst:
        x.fill_(0)
    rr.rr_unpack_range(plan, 0, plan.n_buckets, buf.buckets, buf.dst)
    torch.cuda.synchronize()
    gen = oracle.Source(shards=shards)
    for t_ in (0, 1, 4000, 8999, 9000):
        np.testing.assert_array_equal(H.tensor_host(buf, t_), L.reshard_tensor(gen, t_))


def test_bucket_writing_too_many_tensors_is_refused():
    """One bucket that alone writes more tensors than a launch addresses: pack
    works, unpack is refused with RR_EINVAL before anything is launched."""
    desc = many_tensors_desc(8192, 2 << 20)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"])
    buf = H.alloc(plan)
    H.fill_from_host(buf, U.to_oracle(desc).host_shards(desc["seed"], desc["specials"]))
    H.pack(buf)
    assert H.verify(buf) == (0, -1)
    with pytest.raises(rr.RRError) as e:
        H.unpack(buf)
    assert e.value.status == rrmod.RR_EINVAL


@pytest.mark.parametrize("sharding", ["flat", "rows", "units"])
@pytest.mark.parametrize("engine", ["auto", "registers"])
def test_degenerate_layout(sharding, engine):
    """Zero-size parameters, empty blocks and empty tensors."""
    full_parity(U.degenerate_layout(sharding), engine=engine)


@pytest.mark.parametrize("engine", ["auto", "registers"])
def test_more_separate_buckets_than_one_launch_addresses(engine):
    """4128 separately allocated 1 KiB buckets (with 8 source shards and the
    tensors) exceed one launch's pointer table: pack, unpack and the verifying
    calls run over bucket ranges; damage is still found at the right bucket."""
    desc = U.workload_desc("tiny-tp4", bucket_bytes=1024)
    full_parity(desc, separate_buckets=True, engine=engine)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, desc["bucket_bytes"], engine=engine)
    assert plan.n_buckets > 4000
    buf = H.alloc(plan, separate_buckets=True)
    H.fill_with_generator(buf, m, desc["seed"], desc["specials"])
    H.pack(buf)
    bl = H.bucket_list(buf)
    bl[4100][8] ^= 0x01
    bl[17][0] ^= 0x02
    assert H.verify(buf) == (2, 17)
    assert rr.rr_unpack_verify(plan, buf.buckets, buf.checksums, buf.dst) == (2, 17)
    bad = torch.zeros(plan.n_buckets, dtype=torch.uint8, device="cuda")
    assert rr.rr_verify_range(plan, 100, plan.n_buckets - 100, buf.buckets, buf.checksums,
                              bad=bad) == (1, 4100)
    assert list(np.flatnonzero(bad.cpu().numpy())) == [4100 - 100]


def test_largest_bucket_size():
    """One bucket of the largest size the ABI takes, 2^32 - 16 bytes: the tiny
    model's stream at its start and zeros to its end, so the tail's items sit at
    offsets just under 2^32.  Compared in full with the oracle (4 GiB)."""
    full_parity(U.workload_desc("tiny", bucket_bytes=(1 << 32) - 16))
    torch.cuda.empty_cache()


@pytest.mark.parametrize("grid", [1, 3, 1000])
def test_grid_sizes(grid):
    full_parity(U.workload_desc("tiny-moe-tp2"), grid_blocks=grid)


def test_qwen3_0_6b_full():
    """Qwen3-0.6B, 8 fp32 shards -> TP=1, 32 MiB buckets: every byte compared."""
    full_parity(U.workload_desc("qwen3-0.6b"))


def test_qwen3_0_6b_full_register_engine():
    full_parity(U.workload_desc("qwen3-0.6b"), engine="registers")


def test_device_generator_matches_host():
    n = 5_000_001
    for es, specials in ((4, True), (4, False), (2, False)):
        t = torch.empty(n * es, dtype=torch.uint8, device="cuda")
        synth.fill_dev(t.data_ptr(), n, es, seed=77, first_idx=123456789, specials=specials)
        torch.cuda.synchronize()
        got = t.cpu().numpy().view(np.uint32 if es == 4 else np.uint16)
        np.testing.assert_array_equal(got, synth.values_host(n, es, 77, 123456789, specials))


# ---------------------------------------------------------------------------
# Full-size workloads, sampled
# ---------------------------------------------------------------------------

def sampled_parity(name, bucket_sizes=None, tensors=("norm",), n_random_buckets=3):
    w = U.workload(name)
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    flat = None
    for bb in bucket_sizes or [w.bucket_bytes]:
        plan = H.make_plan(m, s, d, bb)
        buf = H.alloc(plan, poison=None, with_dst=False, flat=flat)
        if flat is None:
            H.fill_with_generator(buf, m, w.seed, w.specials)
            flat = buf.flat
        L = oracle.workload_layout(w, bucket_bytes=bb)
        assert L.n_buckets == plan.n_buckets
        H.pack(buf)
        n_bad, first = H.verify(buf)
        assert (n_bad, first) == (0, -1)
        torch.cuda.synchronize()
        # Property at any size: every checksum equals torch's word sum of its bucket.
        np.testing.assert_array_equal(H.checksums_host(buf), H.device_word_sums(buf))
        rng = np.random.default_rng(bb)
        fr = plan.first_bucket_of_rank
        pick = sorted({0, plan.n_buckets - 1, *[fr[r] for r in range(plan.tp)],
                       *[fr[r + 1] - 1 for r in range(plan.tp)],
                       *rng.integers(0, plan.n_buckets, n_random_buckets).tolist()})
        cs = H.checksums_host(buf)
        for b in pick:
            want, want_cs = L.pack(gen, first=b, count=1)
            np.testing.assert_array_equal(H.buckets_host(buf, [b])[0], want[0],
                                          err_msg=f"bucket {b} (bucket_bytes {bb})")
            assert cs[b] == want_cs[0]
        buf = None


def _unpack_sampled(name, names):
    w = U.workload(name)
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, w.bucket_bytes)
    buf = H.alloc(plan, poison=None)
    H.fill_with_generator(buf, m, w.seed, w.specials)
    H.pack(buf)
    H.unpack(buf)
    assert H.verify(buf) == (0, -1)
    torch.cuda.synchronize()
    L = oracle.workload_layout(w)
    gen = oracle.Source(seed=w.seed, specials=w.specials)
    for nm, rank in names:
        t = L.tensor_index(nm, rank)
        assert plan.tensor_names[t] == nm and plan.tensor_ranks[t] == rank
        np.testing.assert_array_equal(H.tensor_host(buf, t), L.reshard_tensor(gen, t),
                                      err_msg=f"{nm} rank {rank}")
    # Every other tensor, against its own bytes read straight out of the
    # buckets by torch (unpack must be the exact inverse of the stream cut).
    B = plan.bucket_bytes
    assert buf.bucket_store.shape[1] == B
    store = buf.bucket_store.view(-1)
    for t in range(plan.n_tensors):
        r = plan.tensor_ranks[t]
        start = plan.first_bucket_of_rank[r] * B + plan.tensor_stream_offset[t]
        n = 2 * plan.tensor_numel[t]
        want = store[start:start + n].view(torch.int16)
        assert torch.equal(buf.dst[t][:plan.tensor_numel[t]], want), plan.tensor_names[t]


def every_bucket_parity(name, bucket_bytes=None):
    """Every bucket and every checksum of a full-size workload against the oracle,
    in the launch configuration the benchmark times.  The oracle packs the
    buckets one by one in a pool of host threads (its C calls run without the
    interpreter lock, and it keeps no shared state); nothing is sampled."""
    import os
    from concurrent.futures import ThreadPoolExecutor
    w = U.workload(name)
    desc = U.workload_desc(name)
    m, s, d = U.to_product(desc)
    plan = H.make_plan(m, s, d, bucket_bytes or w.bucket_bytes)
    buf = H.alloc(plan, poison=0xAB, with_dst=False)
    H.fill_with_generator(buf, m, w.seed, w.specials)
    H.pack(buf)
    torch.cuda.synchronize()
    got = buf.bucket_store[:, :plan.bucket_bytes].cpu().numpy()
    cs = H.checksums_host(buf)
    buf = None
    torch.cuda.empty_cache()
    L = oracle.workload_layout(w, bucket_bytes=plan.bucket_bytes)
    gen = oracle.Source(seed=w.seed, specials=w.specials)

    def one(b):
        want, want_cs = L.pack(gen, first=b, count=1)
        return b if not (np.array_equal(got[b], want[0]) and cs[b] == want_cs[0]) else -1

    with ThreadPoolExecutor(max_workers=os.cpu_count() or 4) as ex:
        bad = [b for b in ex.map(one, range(plan.n_buckets)) if b >= 0]
    assert bad == [], f"{name}: buckets differing from the oracle: {bad[:10]}"


@pytest.mark.parametrize("name", ["qwen3-8b", "qwen3-8b-tp4", "qwen3-30b-a3b",
                                  "qwen3-8b-fsdp2-tp8", "qwen3-30b-a3b-fsdp2-tp8",
                                  "qwen3-8b-units", "qwen3-30b-a3b-fsdp2-ep8"])
def test_every_bucket_full_size(name):
    every_bucket_parity(name)


@pytest.mark.parametrize("mib", [s >> 20 for s in synth.TP4_BUCKET_SWEEP])
def test_every_bucket_tp4_sweep(mib):
    every_bucket_parity("qwen3-8b-tp4", bucket_bytes=mib << 20)


def test_qwen3_8b_sampled():
    sampled_parity("qwen3-8b", n_random_buckets=4)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-8b", [("layers.0.qkv_proj", 0), ("layers.17.o_proj", 0),
                                 ("layers.35.down_proj", 0), ("layers.35.post_attention_layernorm",
                                                              0), ("norm", 0)])
    torch.cuda.empty_cache()


def test_qwen3_8b_tp4_sampled():
    sampled_parity("qwen3-8b-tp4", n_random_buckets=1)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-8b-tp4", [("layers.3.qkv_proj", 1), ("layers.20.o_proj", 2),
                                     ("layers.35.down_proj", 3), ("layers.7.gate_up_proj", 0),
                                     ("norm", 3)])
    torch.cuda.empty_cache()


def test_qwen3_8b_fsdp2_tp8_sampled():
    """The paper's own trainer sharding (FSDP2) and rollout TP (8)."""
    sampled_parity("qwen3-8b-fsdp2-tp8", n_random_buckets=2)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-8b-fsdp2-tp8", [("layers.9.qkv_proj", 5), ("layers.30.down_proj", 7),
                                           ("norm", 2)])
    torch.cuda.empty_cache()


def test_qwen3_30b_a3b_fsdp2_tp8_sampled():
    """FSDP2 trainer, TP=8 rollout with 4 KV heads: each KV head on two ranks."""
    sampled_parity("qwen3-30b-a3b-fsdp2-tp8", n_random_buckets=1)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-30b-a3b-fsdp2-tp8", [("layers.1.qkv_proj", 3), ("layers.1.qkv_proj", 2),
                                                ("layers.40.experts.w13", 6), ("norm", 7)])
    torch.cuda.empty_cache()


def test_qwen3_8b_units_sampled():
    """FSDP1 wrapping every decoder layer: 37 FlatParameters of 8 shards each."""
    sampled_parity("qwen3-8b-units", n_random_buckets=3)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-8b-units", [("embed_tokens", 0), ("layers.0.qkv_proj", 0),
                                       ("layers.35.down_proj", 0), ("lm_head", 0)])
    torch.cuda.empty_cache()


def test_qwen3_30b_a3b_fsdp2_ep8_sampled():
    """FSDP2 trainer, expert-parallel rollout over 8 ranks: 16 whole experts each."""
    sampled_parity("qwen3-30b-a3b-fsdp2-ep8", n_random_buckets=1)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-30b-a3b-fsdp2-ep8", [("layers.2.experts.w13", 5),
                                                ("layers.47.experts.w2", 7), ("norm", 0)])
    torch.cuda.empty_cache()


def test_qwen3_30b_a3b_sampled():
    sampled_parity("qwen3-30b-a3b", n_random_buckets=2)
    torch.cuda.empty_cache()
    _unpack_sampled("qwen3-30b-a3b", [("layers.0.router", 0), ("layers.47.experts.w2", 0),
                                      ("layers.5.qkv_proj", 0), ("norm", 0)])
    torch.cuda.empty_cache()
