"""Shared test helpers: layout descriptions handed to both sides, and a numpy
interpreter of the library's exported work tables (host-side planner checks).

A description is plain data (params, tensors, sizes); ``to_oracle`` and
``to_product`` turn the same description into the oracle's and the library's
inputs, so neither side's code reaches the other.
"""
from __future__ import annotations

import numpy as np

import oracle
import synth

ITEM_F32_VEC, ITEM_F32_SCALAR, ITEM_BF16_VEC, ITEM_BF16_SCALAR, ITEM_ZERO_VEC, \
    ITEM_ZERO_SCALAR, ITEM_COPY_VEC, ITEM_COPY_SCALAR, ITEM_READ_VEC, ITEM_READ_SCALAR, \
    ITEM_FAN_F32, ITEM_FAN_BF16, ITEM_FAN_DST = range(13)


def workload(name):
    return (synth.WORKLOADS.get(name) or synth.TEST_WORKLOADS.get(name)
            or synth.EXTRA_WORKLOADS[name])


# ---------------------------------------------------------------------------
# Random adversarial layouts
# ---------------------------------------------------------------------------

def random_layout(seed: int, max_params: int = 7, bucket_choices=(8, 24, 40, 64, 200, 4096, 65536)):
    """Odd shapes, mixed dtypes, mid-row shard cuts, tiny buckets, ragged blocks."""
    rng = np.random.default_rng(seed)
    n_params = int(rng.integers(1, max_params + 1))
    params = []
    for i in range(n_params):
        es = int(rng.choice([2, 4]))
        nd = int(rng.integers(1, 4))
        dims = tuple(int(rng.integers(1, 70)) for _ in range(nd))
        params.append((f"p{i}", dims, es))
    tp = int(rng.integers(1, 4))
    tensors = []
    for t in range(int(rng.integers(1, 9))):
        blocks = []
        for _ in range(int(rng.integers(1, 4))):
            p = int(rng.integers(0, n_params))
            dims = params[p][1]
            rows = dims[0]
            cols = int(np.prod(dims[1:])) if len(dims) > 1 else 1
            r0 = int(rng.integers(0, rows))
            nr = int(rng.integers(0, rows - r0 + 1))
            if rng.random() < 0.4:
                c0, nc = 0, cols
            else:
                c0 = int(rng.integers(0, cols))
                nc = int(rng.integers(0, cols - c0 + 1))
            blocks.append((p, r0, nr, c0, nc))
        tensors.append((f"t{t}", int(rng.integers(0, tp)), blocks))
    desc = dict(params=params, tensors=tensors, tp=tp,
                sharding="rows" if rng.random() < 0.35 else "flat",
                n_shards=int(rng.integers(1, 6)),
                bucket_bytes=int(rng.choice(bucket_choices)),
                align_bytes=int(rng.choice([1, 2, 4, 8, 16, 32])),
                tensor_align=int(rng.choice([2, 4, 16, 256])),
                seed=int(rng.integers(1, 1 << 20)), specials=bool(rng.random() < 0.5))
    # Some flat trainers become per-module FSDP1 units: parameters dealt to
    # units in scattered order, every unit used (a second stream, so the draws
    # above stay what they were).
    extra = np.random.default_rng(seed + 1_000_003)
    if desc["sharding"] == "flat" and extra.random() < 0.4:
        n_units = int(extra.integers(1, n_params + 1))
        units = np.concatenate([np.arange(n_units),
                                extra.integers(0, n_units, n_params - n_units)])
        desc["sharding"] = "units"
        desc["units"] = [int(u) for u in extra.permutation(units)]
    return desc


def random_tp_layout(seed: int):
    """Row-parallel weights cut by columns over several ranks (the planner's
    fan-out groups), with cuts placed to hit every fallback: slice widths that
    are or are not multiples of 8, tensor alignments that keep or break 16-byte
    destinations, small buckets that cut through slices, flat shards that cut
    through rows, partial row ranges, fp32 and bf16, and some whole-row
    (replicated) blocks in between."""
    rng = np.random.default_rng(seed + 7_000_001)
    tp = int(rng.choice([2, 3, 4, 8]))
    n_params = int(rng.integers(2, 6))
    params, per_rank = [], [[] for _ in range(tp)]
    for i in range(n_params):
        es = int(rng.choice([2, 4]))
        w = 8 * int(rng.integers(1, 9)) if rng.random() < 0.8 else int(rng.integers(1, 40))
        extra = 8 * int(rng.integers(1, 3)) if rng.random() < 0.3 else 0
        rows, cols = int(rng.integers(1, 90)), w * tp + extra
        params.append((f"p{i}", (rows, cols), es))
        r0 = int(rng.integers(0, rows)) if rng.random() < 0.3 else 0
        nr = rows - r0 if rng.random() < 0.7 else int(rng.integers(1, rows - r0 + 1))
        c_off = extra if rng.random() < 0.5 else 0
        for r in range(tp):
            per_rank[r].append((f"p{i}.slice", r, [(i, r0, nr, c_off + r * w, w)]))
        if rng.random() < 0.3:
            for r in range(tp):
                per_rank[r].append((f"p{i}.whole", r, [(i, 0, rows, 0, cols)]))
    tensors = []
    for r in range(tp):
        order = rng.permutation(len(per_rank[r]))
        tensors += [per_rank[r][k] for k in order]
    sharding = str(rng.choice(["flat", "flat", "rows", "units"]))
    desc = dict(params=params, tensors=tensors, tp=tp, sharding=sharding,
                n_shards=int(rng.integers(1, 6)),
                bucket_bytes=int(rng.choice([64, 200, 1024, 4096, 8192, 65536])),
                align_bytes=int(rng.choice([16, 16, 4, 32])),
                tensor_align=int(rng.choice([256, 256, 16, 2])),
                seed=int(rng.integers(1, 1 << 20)), specials=bool(rng.random() < 0.5))
    if sharding == "units":
        desc["units"] = [int(u) for u in rng.permutation(np.arange(n_params) % 2)]
    return desc


def random_medium_layout(seed: int, max_elems: int = 6 << 20):
    """Odd shapes at the scale where a bucket holds many work items: parameters
    of up to about 1500 x 3000 elements (at most ``max_elems`` in all), buckets
    of 64 KiB to 4 MiB.  Each parameter reaches the rollout ranks in one of the
    ways a TP rollout cuts a model: rows split over the ranks (column-parallel;
    long contiguous runs), columns split over the ranks (row-parallel; one
    slice per rank in every row, wide or narrow), replicated whole, or fused
    with the next parameter into one tensor (like qkv or gate_up), rows split.
    Row counts that do not divide by TP give the last rank the remainder."""
    rng = np.random.default_rng(seed + 9_000_011)
    tp = int(rng.choice([1, 2, 3, 4, 8]))
    n_params = int(rng.integers(3, 9))
    hows = [str(h) for h in rng.choice(["rows", "cols", "whole", "fused"], size=n_params,
                                       p=[0.3, 0.4, 0.15, 0.15])]
    shapes = []
    for i in range(n_params):
        es = int(rng.choice([2, 4, 4]))
        if hows[i] == "cols" and tp > 1:
            # mostly 8-element multiples over a 16-byte aligned row (fan-out
            # groups), sometimes an odd width or a ragged remainder (fallbacks)
            w = 8 * int(rng.integers(1, 400)) if rng.random() < 0.75 else int(rng.integers(1, 900))
            extra = 8 * int(rng.integers(1, 4)) if rng.random() < 0.3 else 0
            dims = (int(rng.integers(1, 1500)), w * tp + extra)
        elif rng.random() < 0.2:
            dims = (int(rng.integers(1, 5000)),)
        else:
            dims = (int(rng.integers(1, 1500)), int(rng.integers(1, 3000)))
        shapes.append([dims, es])
    total = sum(int(np.prod(d)) for d, _ in shapes)
    if total > max_elems:                     # shrink rows until the layout fits
        f = max_elems / total
        for s in shapes:
            d = s[0]
            s[0] = (max(1, int(d[0] * f)),) + tuple(d[1:])
    params = [(f"p{i}", tuple(d), es) for i, (d, es) in enumerate(shapes)]

    def row_split(rows):
        h = rows // tp
        return [(r * h, (rows - r * h) if r == tp - 1 else h) for r in range(tp)]

    tensors, i = [[] for _ in range(tp)], 0
    while i < n_params:
        dims = params[i][1]
        rows = dims[0]
        cols = int(np.prod(dims[1:])) if len(dims) > 1 else 1
        how = hows[i]
        if how == "cols" and cols >= tp:
            w = cols // tp
            c_off = 8 * int(rng.integers(0, (cols - w * tp) // 8 + 1))
            for r in range(tp):
                tensors[r].append((f"p{i}.cols", r, [(i, 0, rows, c_off + r * w, w)]))
        elif how == "whole" or (how == "cols" and cols < tp):
            for r in range(tp):
                tensors[r].append((f"p{i}.whole", r, [(i, 0, rows, 0, cols)]))
        elif how == "fused" and i + 1 < n_params:
            j = i + 1
            cj = int(np.prod(params[j][1][1:])) if len(params[j][1]) > 1 else 1
            for r, ((a0, an), (b0, bn)) in enumerate(zip(row_split(rows),
                                                          row_split(params[j][1][0]))):
                tensors[r].append((f"p{i}+p{j}", r, [(i, a0, an, 0, cols), (j, b0, bn, 0, cj)]))
            i += 1
        else:
            for r, (r0, nr) in enumerate(row_split(rows)):
                tensors[r].append((f"p{i}.rows", r, [(i, r0, nr, 0, cols)]))
        i += 1
    flat_tensors = []
    for r in range(tp):
        order = rng.permutation(len(tensors[r])) if rng.random() < 0.5 else range(len(tensors[r]))
        flat_tensors += [tensors[r][k] for k in order]
    sharding = str(rng.choice(["flat", "flat", "rows", "units"]))
    desc = dict(params=params, tensors=flat_tensors, tp=tp, sharding=sharding,
                n_shards=int(rng.integers(1, 9)),
                bucket_bytes=int(rng.choice([1 << 16, (1 << 16) + 8, 1 << 18, 1 << 20,
                                             (3 << 20) + 16, 4 << 20])),
                align_bytes=int(rng.choice([16, 16, 16, 4, 32])),
                tensor_align=int(rng.choice([256, 256, 16, 2])),
                seed=int(rng.integers(1, 1 << 20)), specials=bool(rng.random() < 0.5))
    if sharding == "units":
        n_units = int(rng.integers(1, n_params + 1))
        units = np.concatenate([np.arange(n_units), rng.integers(0, n_units, n_params - n_units)])
        desc["units"] = [int(u) for u in rng.permutation(units)]
    return desc


def degenerate_layout(sharding: str = "flat"):
    """Parameters with a zero dimension, empty blocks, and destination tensors
    with no elements at all, among ordinary ones."""
    desc = dict(params=[("a", (0, 8), 4), ("b", (3, 0), 2), ("c", (5, 16), 4), ("d", (0,), 2)],
                tensors=[("t0", 0, [(0, 0, 0, 0, 8), (2, 1, 2, 0, 16)]),
                         ("t1", 1, [(1, 0, 3, 0, 0)]),
                         ("t2", 1, [(2, 0, 5, 3, 8), (3, 0, 0, 0, 1)]), ("t3", 0, [])],
                tp=2, sharding=sharding, n_shards=3, bucket_bytes=64, align_bytes=16,
                tensor_align=256, seed=5, specials=True)
    if sharding == "units":
        desc["units"] = [0, 1, 0, 1]
    return desc


def workload_desc(name, bucket_bytes=None, dst_dtype=None):
    w = workload(name)
    if dst_dtype is not None:
        w = w.with_(dst_dtype=dst_dtype)
    from oracle import qwen3
    params = qwen3.manifest(w.shape, w.src_elem_bytes)
    return dict(params=params, tensors=None, workload=w, tp=w.tp, n_shards=w.n_shards,
                bucket_bytes=bucket_bytes or w.bucket_bytes, align_bytes=16, tensor_align=256,
                seed=w.seed, specials=w.specials)


def to_oracle(desc) -> "oracle.Layout":
    if desc.get("workload") is not None:
        return oracle.workload_layout(desc["workload"], bucket_bytes=desc["bucket_bytes"])
    return oracle.Layout(desc["params"], desc["tensors"], n_shards=desc["n_shards"],
                         tp=desc["tp"], bucket_bytes=desc["bucket_bytes"],
                         align_bytes=desc["align_bytes"], tensor_align=desc["tensor_align"],
                         sharding=desc.get("sharding", "flat"), units=desc.get("units"),
                         dst_dtype=desc.get("dst_dtype", "bf16"))


def to_product(desc):
    import paper_2512_22492_gb300 as rr
    if desc.get("workload") is not None:
        w = desc["workload"]
        return rr.qwen3_sync(w.shape, w.src_dtype, w.n_shards, w.tp, w.sharding, ep=w.ep,
                             dst_dtype=w.dst_dtype)
    manifest = [rr.Param(n, d, "f32" if es == 4 else "bf16") for n, d, es in desc["params"]]
    src = rr.SrcLayout(n_shards=desc["n_shards"], align_bytes=desc["align_bytes"],
                       sharding=desc.get("sharding", "flat"), units=desc.get("units"))
    dst = rr.DstLayout(tp=desc["tp"], tensor_align_bytes=desc["tensor_align"],
                       tensors=[rr.DstTensor(n, r, [rr.Block(*b) for b in blocks])
                                for n, r, blocks in desc["tensors"]],
                       dtype=desc.get("dst_dtype", "bf16"))
    return manifest, src, dst


# ---------------------------------------------------------------------------
# Work-table interpreter (what the kernels are specified to do with each item)
# ---------------------------------------------------------------------------

def check_and_run_pack(items, shards, n_buckets, bucket_bytes, shard_bytes):
    """Applies pack items to host shards; asserts every item's preconditions and
    that every bucket byte is written exactly once.  Returns the buckets."""
    out = np.zeros((n_buckets, bucket_bytes), np.uint8)
    hits = np.zeros((n_buckets, bucket_bytes), np.uint16)
    items = list(items)
    skip = 0
    for j, it in enumerate(items):
        if skip:
            skip -= 1
            continue
        kind, b, off = int(it["kind"]), int(it["bucket"]), int(it["dst_off"])
        assert kind != ITEM_FAN_DST, "fan-out destination without its head"
        if kind in (ITEM_FAN_F32, ITEM_FAN_BF16):
            es = 4 if kind == ITEM_FAN_F32 else 2
            span, R, st = int(it["row_len"]), int(it["n_rows"]), int(it["src_stride"])
            shard, soff = int(it["src"]) >> 48, int(it["src"]) & ((1 << 48) - 1)
            assert soff % 16 == 0 and (span * es) % 16 == 0 and (st * es) % 16 == 0
            assert soff + ((R - 1) * st + span) * es <= min(shard_bytes, len(shards[shard]))
            rows = np.stack([shards[shard][soff + i * st * es:soff + (i * st + span) * es]
                             for i in range(R)])
            skip = off
            covered = np.zeros(span, np.int32)
            for d in items[j + 1:j + 1 + off]:
                assert int(d["kind"]) == ITEM_FAN_DST and int(d["n_rows"]) == R
                c0, w = int(d["src"]), int(d["row_len"])
                db, doff = int(d["bucket"]), int(d["dst_off"])
                assert w % 8 == 0 and doff % 16 == 0 and (c0 * es) % 16 == 0
                assert 0 <= db < n_buckets and doff + 2 * R * w <= bucket_bytes
                covered[c0:c0 + w] += 1
                raw = np.zeros((R, w), np.uint32)
                for k in range(es):
                    raw |= rows[:, c0 * es + k:(c0 + w) * es:es].astype(np.uint32) << (8 * k)
                vals = oracle.rne_bf16(raw) if es == 4 else raw.astype(np.uint16)
                out[db, doff:doff + 2 * R * w] = vals.reshape(-1).astype("<u2").view(np.uint8)
                hits[db, doff:doff + 2 * R * w] += 1
            assert np.all(covered <= 1), "fan-out slices overlap"
            continue
        L, R, st = int(it["row_len"]), int(it["n_rows"]), int(it["src_stride"])
        n = L * R
        assert 0 <= b < n_buckets and off % 2 == 0 and off + 2 * n <= bucket_bytes
        hits[b, off:off + 2 * n] += 1
        if kind in (ITEM_ZERO_VEC, ITEM_ZERO_SCALAR):
            assert R == 1
            if kind == ITEM_ZERO_VEC:
                assert off % 16 == 0 and L % 8 == 0
            out[b, off:off + 2 * n] = 0
            continue
        es = 4 if kind in (ITEM_F32_VEC, ITEM_F32_SCALAR) else 2
        shard, soff = int(it["src"]) >> 48, int(it["src"]) & ((1 << 48) - 1)
        if kind in (ITEM_F32_VEC, ITEM_BF16_VEC):
            assert off % 16 == 0 and L % 8 == 0 and soff % 16 == 0
            assert R == 1 or (st * es) % 16 == 0
        assert soff + ((R - 1) * st + L) * es <= min(shard_bytes, len(shards[shard]))
        idx = soff + (np.arange(R, dtype=np.int64)[:, None] * st * es
                      + np.arange(L, dtype=np.int64)[None, :] * es).ravel()
        raw = np.zeros(idx.size, np.uint32)
        for k in range(es):
            raw |= shards[shard][idx + k].astype(np.uint32) << (8 * k)
        vals = oracle.rne_bf16(raw) if es == 4 else raw.astype(np.uint16)
        out[b, off:off + 2 * n] = vals.astype("<u2").view(np.uint8)
    assert hits.min() == 1 and hits.max() == 1, "bucket bytes not written exactly once"
    return out


def check_and_run_unpack(items, buckets, tensor_numel):
    """Applies unpack items; asserts their preconditions, that every tensor byte
    is written once, and that copy + read items together read every bucket byte
    exactly once (what the verifying unpack relies on)."""
    dst = [np.zeros(2 * n, np.uint8) for n in tensor_numel]
    hits = [np.zeros(2 * n, np.uint16) for n in tensor_numel]
    reads = np.zeros(buckets.shape, np.uint16)
    for it in items:
        kind, b, so = int(it["kind"]), int(it["bucket"]), int(it["src_off"])
        t, do, nb = int(it["tensor"]), int(it["dst_off"]), int(it["nbytes"])
        assert nb % 2 == 0 and so + nb <= buckets.shape[1]
        if kind in (ITEM_COPY_VEC, ITEM_READ_VEC):
            assert so % 16 == 0 and nb % 16 == 0
        reads[b, so:so + nb] += 1
        if kind in (ITEM_READ_VEC, ITEM_READ_SCALAR):
            continue
        assert do + nb <= dst[t].size
        if kind == ITEM_COPY_VEC:
            assert do % 16 == 0
        dst[t][do:do + nb] = buckets[b, so:so + nb]
        hits[t][do:do + nb] += 1
    for h in hits:
        assert h.size == 0 or (h.min() == 1 and h.max() == 1), "dst bytes not written once"
    assert reads.size == 0 or (reads.min() == 1 and reads.max() == 1), \
        "bucket bytes not read exactly once by the unpack table"
    return [d.view("<u2") for d in dst]


def check_partition(first, n_items):
    first = np.asarray(first, np.int64)
    assert first[0] == 0 and first[-1] == n_items
    assert np.all(np.diff(first) >= 0)


def check_units(plan, n_items, which="unpack"):
    """The bulk-copy engine's work units of one table tile its items.  In the
    per-bucket tables ("pack", "unpack") no unit is empty or spans two buckets
    and bucket b's units cover exactly its items, so any bucket range is a
    contiguous run of whole units; the whole-sync pack's ("pack_full") start
    with one own unit per block of the grid."""
    first, bucket_unit = plan.work_units(which)
    first = first.astype(np.int64)
    if which == "pack_full":
        # One own unit per block, then the claimed ones; units may be empty.
        grid = plan.stats()["grid_blocks"]
        assert len(first) >= grid + 2
        assert first[0] == 0 and first[-1] == n_items and np.all(np.diff(first) >= 0)
        return first, None
    if n_items == 0:
        assert len(first) == 1 and first[0] == 0
        return first, bucket_unit
    assert first[0] == 0 and first[-1] == n_items
    assert np.all(np.diff(first) > 0)
    pack_first, unpack_first = plan.bucket_items()
    bucket_first = pack_first if which == "pack" else unpack_first
    bucket_unit = bucket_unit.astype(np.int64)
    assert bucket_unit[0] == 0 and bucket_unit[-1] == len(first) - 1
    assert np.all(np.diff(bucket_unit) >= 0)
    for b in range(plan.n_buckets):
        lo, hi = bucket_first[b], bucket_first[b + 1]
        u0, u1 = bucket_unit[b], bucket_unit[b + 1]
        assert (u1 > u0) == (hi > lo)
        if hi > lo:
            assert first[u0] == lo and first[u1] == hi
    return first, bucket_unit
