"""Host-side checks of the library's planner (no GPU): the C ABI loads and
exports what include/rr.h declares; host-only plans agree with the oracle on
geometry; their work tables, interpreted item by item, reproduce the oracle's
buckets and tensors; bad descriptions are rejected with the right status."""
import os
import re

import numpy as np
import pytest

import oracle
import paper_2512_22492_gb300 as rr
from paper_2512_22492_gb300 import rr as rrmod
from tests import _util as U

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def declared_functions():
    src = open(os.path.join(ROOT, "include", "rr.h")).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(rr_[a-z_]+)\s*\(", src)))


def test_library_exports_every_declared_symbol():
    import ctypes
    lib = ctypes.CDLL(rrmod.LIBRARY_PATH)
    names = declared_functions()
    assert "rr_pack" in names and "rr_plan_create" in names
    for name in names:
        assert hasattr(lib, name), f"{name} declared in rr.h but not exported"


def host_plan(desc, **opt):
    m, s, d = U.to_product(desc)
    return rr.rr_plan_create(m, s, d, desc["bucket_bytes"], rr.PlanOptions(host_only=True, **opt))


@pytest.mark.parametrize("name", ["tiny", "qwen3-0.6b", "qwen3-8b", "qwen3-8b-tp4",
                                  "qwen3-30b-a3b", "tiny-moe-tp2", "tiny-units",
                                  "tiny-moe-units-ep2", "qwen3-8b-units",
                                  "qwen3-30b-a3b-fsdp2-ep8"])
def test_geometry_matches_oracle(name):
    desc = U.workload_desc(name)
    L = U.to_oracle(desc)
    p = host_plan(desc)
    assert p.n_buckets == L.n_buckets
    assert p.shard_bytes == L.shard_bytes and p.flat_bytes == L.flat_bytes
    if L.sharding == "units":
        assert p.source_buffer_bytes == [int(s) for s in L.unit_shard_bytes
                                         for _ in range(L.n_shards)]
    elif L.sharding != "tensors":
        assert p.source_buffer_bytes == [L.shard_bytes] * L.n_shards
    assert p.param_flat_offset == list(L.param_offset)
    assert p.first_bucket_of_rank == list(L.rank_first_bucket)
    assert p.stream_bytes_per_rank == list(L.rank_stream_bytes)
    assert p.tensor_numel == list(L.tensor_numel)
    assert p.tensor_stream_offset == list(L.tensor_offset)


def run_and_compare(desc, **opt):
    L = U.to_oracle(desc)
    p = host_plan(desc, **opt)
    shards = L.host_shards(desc["seed"], desc["specials"])
    want, want_cs = L.pack(oracle.Source(shards=shards))
    items, first = p.export_pack()
    U.check_partition(first, len(items))
    got = U.check_and_run_pack(items, shards, p.n_buckets, p.bucket_bytes, p.shard_bytes)
    np.testing.assert_array_equal(got, want)
    # The whole-sync table (fan-out groups in place of narrow slices) packs the same bytes.
    fitems, ffirst = p.export_pack_full()
    U.check_partition(ffirst, len(fitems))
    starts = ffirst[:-1][ffirst[:-1] < len(fitems)]
    assert not np.any(fitems["kind"][starts] == U.ITEM_FAN_DST)
    U.check_units(p, len(items), "pack")
    funits, _ = U.check_units(p, len(fitems), "pack_full")
    starts = funits[:-1][funits[:-1] < len(fitems)]
    assert not np.any(fitems["kind"][starts] == U.ITEM_FAN_DST)
    got = U.check_and_run_pack(fitems, shards, p.n_buckets, p.bucket_bytes, p.shard_bytes)
    np.testing.assert_array_equal(got, want)
    uitems, ufirst = p.export_unpack()
    U.check_partition(ufirst, len(uitems))
    U.check_units(p, len(uitems))
    tensors = U.check_and_run_unpack(uitems, want, p.tensor_numel)
    for t, arr in enumerate(tensors):
        np.testing.assert_array_equal(arr, L.unpack_tensor(want, t))
    return p, items


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-tied", "tiny-moe", "tiny-moe-tp2",
                                  "tiny-moe-f32", "tiny-fsdp2", "tiny-units", "tiny-moe-ep4",
                                  "tiny-moe-units-ep2"])
def test_tables_reproduce_oracle_workloads(name):
    run_and_compare(U.workload_desc(name))


@pytest.mark.parametrize("chunk", [16, 48, 4096])
def test_tables_small_chunks(chunk):
    run_and_compare(U.workload_desc("tiny-tp4", bucket_bytes=8 * 1024), chunk_bytes=chunk)


@pytest.mark.parametrize("seed", range(40))
def test_tables_random_layouts(seed):
    run_and_compare(U.random_layout(seed), grid_blocks=7)


@pytest.mark.parametrize("seed", range(48))
def test_tables_random_row_parallel_layouts(seed):
    """Fan-out groups and all their fallbacks, through both tables."""
    run_and_compare(U.random_tp_layout(seed), grid_blocks=5)


def test_random_row_parallel_layouts_exercise_fan_out():
    """The generator above does produce fan-out groups, and plain fallbacks."""
    heads = plain_rows = 0
    for seed in range(48):
        p = host_plan(U.random_tp_layout(seed))
        items, _ = p.export_pack_full()
        heads += int(np.sum((items["kind"] == U.ITEM_FAN_F32) | (items["kind"] == U.ITEM_FAN_BF16)))
        plain_rows += int(p.stats()["n_pack_full_items"] == p.stats()["n_pack_items"])
    assert heads > 100 and plain_rows > 3


@pytest.mark.parametrize("seed", range(6))
def test_tables_medium_layouts(seed):
    """Medium random layouts (many items per bucket, wide and narrow
    row-parallel slices, fused blocks) through both tables."""
    run_and_compare(U.random_medium_layout(seed), grid_blocks=11)


def test_medium_layouts_reach_every_item_kind():
    """The first 40 medium seeds (the GPU parity cases) produce fan-out groups,
    buckets of many items, every TP degree and every sharding."""
    heads = many = 0
    tps, shardings = set(), set()
    for seed in range(40):
        desc = U.random_medium_layout(seed)
        p = host_plan(desc)
        items, _ = p.export_pack_full()
        heads += int(np.sum((items["kind"] == U.ITEM_FAN_F32) | (items["kind"] == U.ITEM_FAN_BF16)))
        many += int(len(items) > 8 * max(1, p.n_buckets))
        tps.add(desc["tp"])
        shardings.add(desc["sharding"])
    assert heads >= 50 and many >= 5
    assert tps == {1, 2, 3, 4, 8} and shardings == {"flat", "rows", "units"}


@pytest.mark.parametrize("sharding", ["flat", "rows", "units"])
def test_degenerate_layout(sharding):
    """Zero-size parameters, empty blocks and empty tensors."""
    p, _ = run_and_compare(U.degenerate_layout(sharding), grid_blocks=3)
    assert p.tensor_numel == [32, 0, 40, 0]


def test_vector_items_dominate_on_aligned_workloads():
    p, items = run_and_compare(U.workload_desc("tiny"))
    data = items[items["kind"] <= U.ITEM_BF16_SCALAR]
    elems = data["row_len"].astype(np.int64) * data["n_rows"]
    vec = elems[data["kind"] == U.ITEM_F32_VEC].sum()
    assert vec == elems.sum(), "an aligned fp32 workload should need no scalar items"


def test_full_size_tables_are_consistent():
    """Qwen3-8B TP=4: metadata-only checks over ~0.5M items."""
    desc = U.workload_desc("qwen3-8b-tp4")
    p = host_plan(desc)
    items, first = p.export_pack()
    U.check_partition(first, len(items))
    n = items["row_len"].astype(np.int64) * items["n_rows"]
    bucket_bytes = np.zeros(p.n_buckets, np.int64)
    np.add.at(bucket_bytes, items["bucket"].astype(np.int64), 2 * n)
    assert np.all(bucket_bytes == p.bucket_bytes)
    assert np.all(items["dst_off"].astype(np.int64) + 2 * n <= p.bucket_bytes)
    assert np.all(2 * n <= 64 * 1024)
    st = p.stats()
    data = items["kind"] <= U.ITEM_BF16_SCALAR
    assert (n[data] * 4).sum() == st["pack_bytes_read"]
    assert np.all(items["kind"][data] == U.ITEM_F32_VEC)


def unit_weights(p, which):
    """Each unit's weight, by the planner's balancing rule (pack: 6 per fp32
    element by vectors, 12 element by element, 4 and 8 for bf16, 2 per zero
    element; unpack: 2 per byte copied by vectors, 4 element by element, 1 per
    byte only read; 1024 more per item, nothing for a fan-out destination)."""
    if which.startswith("unpack"):
        items, _ = p.export_unpack()
        n = items["nbytes"].astype(np.int64)
        per = np.select([items["kind"] == U.ITEM_COPY_VEC, items["kind"] == U.ITEM_COPY_SCALAR],
                        [2, 4], 1)
        w = per * n + 1024
    else:
        items, _ = p.export_pack_full() if which == "pack_full" else p.export_pack()
        n = items["row_len"].astype(np.int64) * items["n_rows"]
        k = items["kind"]
        per = np.select([k == U.ITEM_F32_VEC, k == U.ITEM_F32_SCALAR, k == U.ITEM_BF16_VEC,
                         k == U.ITEM_BF16_SCALAR, k == U.ITEM_FAN_F32, k == U.ITEM_FAN_BF16],
                        [6, 12, 4, 8, 6, 4], 2)
        w = np.where(k == U.ITEM_FAN_DST, 0, per * n + 1024)
    return items, w


def taper(rem, unit, grid, floor=64 * 1024):
    """The claimed-unit size for `rem` weight left before the table's end."""
    return max(min(unit, floor), min(unit, rem // (2 * grid)))


@pytest.mark.parametrize("name,which", [("qwen3-0.6b", "unpack"), ("qwen3-8b", "unpack"),
                                        ("qwen3-30b-a3b-fsdp2-tp8", "unpack"),
                                        ("qwen3-0.6b", "pack"), ("qwen3-8b", "pack")])
def test_bucket_units_on_full_size_tables(name, which):
    """Per-bucket units: a unit's size is about the weight left to the table's
    end over twice the grid, at most 1 MiB (or less where that would leave a
    block of the grid fewer than 32) and at least 64 KiB.  A unit is cut at the
    item reaching its size unless under a quarter of it would be left in the
    bucket, so only a bucket's last unit is lighter; sizes shrink toward the end."""
    p = host_plan(U.workload_desc(name))
    items, w = unit_weights(p, which)
    first, bucket_unit = U.check_units(p, len(items), which)
    grid = p.stats()["unpack_grid_blocks" if which == "unpack" else "grid_blocks"]
    unit = min(1 << 20, max((1 << 20) // 8, int(w.sum()) // (32 * grid)))
    cum = np.concatenate([[0], np.cumsum(w)])
    total = int(cum[-1])
    unit_w = cum[first[1:]] - cum[first[:-1]]
    size = np.array([taper(total - int(cum[f]), unit, grid) for f in first[:-1]])
    assert np.all(np.diff(size) <= 0)
    assert size[0] == unit and size[-1] == min(unit, 64 * 1024)
    assert np.all(unit_w <= size + size // 4 + w.max())
    last = np.zeros(len(unit_w), bool)
    last[bucket_unit[1:][np.diff(bucket_unit) > 0] - 1] = True
    assert np.all(unit_w[~last] >= size[~last])
    assert len(unit_w) >= 16 * grid


@pytest.mark.parametrize("name", ["qwen3-0.6b", "qwen3-8b", "qwen3-30b-a3b-fsdp2-tp8"])
def test_whole_pack_units_on_full_size_tables(name):
    """A pack over every bucket: one own unit per block, together 85% of the
    weight in equal shares (to within one item, or one fan-out group), then
    claimed units of the tapered size (the weight left over twice the grid,
    within [64 KiB, the per-bucket unit size]) plus at most one item."""
    which = "pack_full"
    p = host_plan(U.workload_desc(name))
    items, w = unit_weights(p, which)
    first, _ = U.check_units(p, len(items), which)
    grid = p.stats()["grid_blocks"]
    heaviest = int(w.max())
    if which == "pack_full":   # a fan-out head and its destinations stay together
        heaviest = int(np.add.reduceat(w, np.flatnonzero(w > 0)).max())
    cum = np.concatenate([[0], np.cumsum(w)])
    unit_w = cum[first[1:]] - cum[first[:-1]]
    total = int(cum[-1])
    own = total * 85 // 100
    assert abs(int(cum[first[grid]]) - own) <= heaviest
    assert np.all(np.abs(unit_w[:grid] - own / grid) <= heaviest + 1)
    unit = min(1 << 20, max((1 << 20) // 8, total // (32 * grid)))
    size = np.array([taper(total - int(cum[f]), unit, grid) for f in first[grid:-1]])
    assert np.all(unit_w[grid:] <= size + heaviest)
    assert np.all(unit_w[grid:-1] >= size[:-1])
    assert np.all(np.diff(size) <= 0) and size[-1] == min(unit, 64 * 1024)


def test_fan_out_groups_on_full_size_tables():
    """Qwen3-30B-A3B FSDP2 -> TP=8: every expert down_proj's eight 96-column slices,
    and every attention o_proj's eight 512-column slices, form one group per
    shard run of rows (metadata only)."""
    desc = U.workload_desc("qwen3-30b-a3b-fsdp2-tp8")
    p = host_plan(desc)
    items, first = p.export_pack_full()
    U.check_partition(first, len(items))
    kind = items["kind"]
    heads = np.flatnonzero((kind == U.ITEM_FAN_F32) | (kind == U.ITEM_FAN_BF16))
    assert np.all(items["dst_off"][heads] == 8)
    assert set(np.unique(items["row_len"][heads]).tolist()) == {768, 4096}
    expert = heads[items["row_len"][heads] == 768]
    o_proj = heads[items["row_len"][heads] == 4096]
    # One head per shard run of 256 rows, and a few more where a bucket boundary
    # cuts a run; a row whose slice would straddle a boundary goes out as plain items.
    assert 48 * 128 * 8 <= len(expert) < 48 * 128 * 8 + 64
    assert np.all(items["n_rows"][expert] <= 256)
    fanned_rows = int(items["n_rows"][expert].astype(np.int64).sum())
    assert 48 * 128 * 2048 - 64 <= fanned_rows <= 48 * 128 * 2048
    o_rows = int(items["n_rows"][o_proj].astype(np.int64).sum())
    assert 48 * 2048 - 64 <= o_rows <= 48 * 2048
    dsts = np.flatnonzero(kind == U.ITEM_FAN_DST)
    assert len(dsts) == 8 * len(heads)
    dst_width = items["row_len"][dsts].reshape(-1, 8)
    assert np.all(dst_width == np.where(items["row_len"][heads] == 768, 96, 512)[:, None])
    # Every bucket byte is written exactly once: plain items plus fan-out slices.
    n = items["row_len"].astype(np.int64) * items["n_rows"]
    plain = kind < U.ITEM_FAN_F32
    per_bucket = np.zeros(p.n_buckets, np.int64)
    np.add.at(per_bucket, items["bucket"][plain].astype(np.int64), 2 * n[plain])
    np.add.at(per_bucket, items["bucket"][dsts].astype(np.int64), 2 * n[dsts])
    assert np.all(per_bucket == p.bucket_bytes)
    starts = first[:-1][first[:-1] < len(items)]
    assert not np.any(kind[starts] == U.ITEM_FAN_DST)


def test_rejections():
    params = [rr.Param("a", (4, 6), "f32"), rr.Param("b", (5,), "bf16")]
    src = rr.SrcLayout(n_shards=2)
    good = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 0, [rr.Block(0, 0, 4, 0, 6)])])
    opts = rr.PlanOptions(host_only=True)
    rr.rr_plan_create(params, src, good, 64, opts)

    def status(params=params, src=src, dst=good, bucket=64):
        with pytest.raises(rr.RRError) as e:
            rr.rr_plan_create(params, src, dst, bucket, opts)
        return e.value.status

    bad_rows = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 0, [rr.Block(0, 2, 3, 0, 6)])])
    bad_cols = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 0, [rr.Block(0, 0, 1, 5, 2)])])
    bad_param = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 0, [rr.Block(2, 0, 1, 0, 1)])])
    bad_rank = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 1, [rr.Block(0, 0, 1, 0, 6)])])
    bad_numel = rr.DstLayout(tp=1, tensors=[rr.DstTensor("t", 0, [rr.Block(0, 0, 1, 0, 6)],
                                                         numel=7)])
    assert status(dst=bad_rows) == rrmod.RR_ELAYOUT
    assert status(dst=bad_cols) == rrmod.RR_ELAYOUT
    assert status(dst=bad_param) == rrmod.RR_ELAYOUT
    assert status(dst=bad_rank) == rrmod.RR_ELAYOUT
    assert status(dst=bad_numel) == rrmod.RR_ELAYOUT
    assert status(bucket=12) == rrmod.RR_EINVAL
    assert status(bucket=0) == rrmod.RR_EINVAL
    assert status(src=rr.SrcLayout(n_shards=0)) == rrmod.RR_EINVAL
    overlap = rr.SrcLayout(n_shards=1, param_flat_offset=[0, 64])
    assert status(src=overlap) == rrmod.RR_ELAYOUT
    misaligned = rr.SrcLayout(n_shards=1, param_flat_offset=[2, 200])
    assert status(src=misaligned) == rrmod.RR_ELAYOUT
    assert status(dst=rr.DstLayout(tp=1, tensors=good.tensors, tensor_align_bytes=3)) \
        == rrmod.RR_EINVAL
    # Per-module FSDP1 units.
    rr.rr_plan_create(params, rr.SrcLayout(n_shards=2, sharding="units", units=[1, 0]), good, 64,
                      opts)
    assert status(src=rr.SrcLayout(n_shards=2, sharding="units", units=[0, 2])) \
        == rrmod.RR_EINVAL                                   # unit 1 holds nothing
    assert status(src=rr.SrcLayout(n_shards=2, sharding="units", units=[-1, 0])) \
        == rrmod.RR_EINVAL                                   # unit out of range
    assert status(src=rr.SrcLayout(n_shards=2, sharding="units")) == rrmod.RR_EINVAL
    assert status(src=rr.SrcLayout(n_shards=2, units=[0, 0])) == rrmod.RR_EINVAL   # flat
    assert status(src=rr.SrcLayout(n_shards=2, sharding="units", units=[0, 0],
                                   param_flat_offset=[0, 96])) == rrmod.RR_EINVAL
    assert status(src=rr.SrcLayout(n_shards=40000, sharding="units", units=[0, 1])) \
        == rrmod.RR_EINVAL                                   # 80000 source buffers


def test_host_only_plan_refuses_to_run():
    desc = U.workload_desc("tiny")
    p = host_plan(desc)
    with pytest.raises(rr.RRError) as e:
        rr.rr_pack(p, [16] * p.n_shards, [16] * p.n_buckets, 16, stream=0)
    assert e.value.status == rrmod.RR_EINVAL


@pytest.mark.parametrize("seed", range(12))
def test_bucket_index_and_range_interpretation(seed):
    """Each bucket's items are a contiguous run of both tables; interpreting only
    a bucket range's pack items reproduces the oracle's buckets of that range."""
    desc = U.random_layout(seed)
    L = U.to_oracle(desc)
    p = host_plan(desc)
    items, _ = p.export_pack()
    uitems, _ = p.export_unpack()
    pf, uf = p.bucket_items()
    assert pf[0] == 0 and pf[-1] == len(items) and np.all(np.diff(pf.astype(np.int64)) >= 0)
    assert uf[0] == 0 and uf[-1] == len(uitems) and np.all(np.diff(uf.astype(np.int64)) >= 0)
    for b in range(p.n_buckets):
        assert np.all(items["bucket"][pf[b]:pf[b + 1]] == b)
        assert np.all(uitems["bucket"][uf[b]:uf[b + 1]] == b)
    if p.n_buckets < 2:
        return
    rng = np.random.default_rng(seed)
    b0 = int(rng.integers(0, p.n_buckets - 1))
    b1 = int(rng.integers(b0 + 1, p.n_buckets + 1))
    shards = L.host_shards(desc["seed"], desc["specials"])
    sub = items[pf[b0]:pf[b1]].copy()
    sub["bucket"] -= b0
    got = U.check_and_run_pack(sub, shards, b1 - b0, p.bucket_bytes, p.shard_bytes)
    want, _ = L.pack(oracle.Source(shards=shards), first=b0, count=b1 - b0)
    np.testing.assert_array_equal(got, want)


@pytest.mark.parametrize("case", ["tiny-tp4", "tiny-moe-bf16-specials", "qwen3-8b-fsdp2-tp8",
                                  "random-3", "row-parallel-5"])
def test_float16_rollout_changes_only_the_cast(case):
    """A float16 destination is the same plan as a bf16 one but for the cast the
    kernels apply: every work table, per-block range, work unit and count is
    identical."""
    if case.startswith("random-"):
        desc = U.random_layout(int(case.split("-")[1]))
    elif case.startswith("row-parallel-"):
        desc = U.random_tp_layout(int(case.split("-")[2]))
    else:
        desc = U.workload_desc(case)
    plans = []
    for dtype in ("bf16", "f16"):
        d16 = dict(desc)
        if d16.get("workload") is not None:
            d16["workload"] = d16["workload"].with_(dst_dtype=dtype)
        else:
            d16["dst_dtype"] = dtype
        m, s, d = U.to_product(d16)
        assert d.dtype == dtype
        plans.append(rr.rr_plan_create(m, s, d, desc["bucket_bytes"],
                                       rr.PlanOptions(host_only=True)))
    a, b = plans
    assert a.dst_dtype == "bf16" and b.dst_dtype == "f16"
    assert a.stats() == b.stats()
    for export in ("export_pack", "export_pack_full", "export_unpack"):
        ia, fa = getattr(a, export)()
        ib, fb = getattr(b, export)()
        np.testing.assert_array_equal(ia, ib, err_msg=export)
        np.testing.assert_array_equal(fa, fb, err_msg=export)
    for which in ("pack", "unpack", "pack_full"):
        ua, ub = a.work_units(which), b.work_units(which)
        for x, y in zip(ua, ub):
            np.testing.assert_array_equal(x, y, err_msg=which)
