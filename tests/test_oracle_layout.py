"""Pins for the oracle's source addressing, reshard, stream/bucket cut, checksum,
unpack and verify (RobustRL Section 5.2.1 steps 1-2 and Section 5.2.2).

The paper prints no worked example for this path, so the oracle is pinned by:
* a hand-worked example (tests/golden/layout_worked_example.json);
* hand-derived Qwen3 manifests and rollout tensor lists
  (tests/golden/qwen3_rollout_worked_example.json): registration order, fused
  orders, TP row and column cuts, KV replication, expert parallel, units;
* a PyTorch restatement of the rollout layout (vLLM-style cat/chunk/stack on
  whole parameter tensors, then byte-level concatenation into streams and
  buckets) on scaled-down workloads of every family;
* invariants: shard-count invariance, coverage counts, unpack(pack) = reshard,
  checksum linearity, numpy's wrapping uint64 sum.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
import synth
from oracle import qwen3

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "layout_worked_example.json")


def _int(x):
    return int(x, 16) if isinstance(x, str) else int(x)


# ---------------------------------------------------------------------------
# Hand-worked example
# ---------------------------------------------------------------------------

def _golden_layout():
    g = json.load(open(GOLDEN))
    params = [(p["name"], tuple(p["dims"]), p["elem_bytes"]) for p in g["params"]]
    tensors = [(t["name"], t["rank"], [tuple(b) for b in t["blocks"]]) for t in g["tensors"]]
    L = oracle.Layout(params, tensors, n_shards=g["n_shards"], tp=g["tp"],
                      bucket_bytes=g["bucket_bytes"], align_bytes=g["align_bytes"],
                      tensor_align=g["tensor_align"])
    # Build the flat source by hand from the expected offsets, then cut it.
    e = g["expect"]
    flat = bytearray(e["shard_bytes"] * g["n_shards"])
    for p, off in zip(g["params"], e["param_offset"]):
        for k, v in enumerate(p["bits"]):
            flat[off + k * p["elem_bytes"]: off + (k + 1) * p["elem_bytes"]] = \
                _int(v).to_bytes(p["elem_bytes"], "little")
    S = e["shard_bytes"]
    shards = [np.frombuffer(bytes(flat[s * S:(s + 1) * S]), np.uint8)
              for s in range(g["n_shards"])]
    return g, L, shards


def test_golden_layout_numbers():
    g, L, _ = _golden_layout()
    e = g["expect"]
    assert list(L.param_offset) == e["param_offset"]
    assert L.flat_bytes == e["flat_bytes"]
    assert L.shard_bytes == e["shard_bytes"]
    assert list(L.tensor_numel) == e["tensor_numel"]
    assert list(L.tensor_offset) == e["tensor_offset"]
    assert list(L.rank_stream_bytes) == e["rank_stream_bytes"]
    assert list(L.rank_first_bucket) == e["rank_first_bucket"]


def test_golden_values():
    g, L, shards = _golden_layout()
    e = g["expect"]
    src = oracle.Source(shards=shards)
    for t, want in enumerate(e["tensors_bf16"]):
        np.testing.assert_array_equal(L.reshard_tensor(src, t),
                                      np.array([_int(x) for x in want], np.uint16))
    buckets, cs = L.pack(src)
    for b, hx in enumerate(e["buckets_hex"]):
        assert buckets[b].tobytes().hex() == hx
    assert [int(c) for c in cs] == [_int(c) for c in e["checksums"]]


# ---------------------------------------------------------------------------
# PyTorch restatement of the rollout layout
# ---------------------------------------------------------------------------

def _param_tensors(params, flat_offsets, seed, specials):
    """Whole parameter tensors (as integer bit patterns) for the generator's values."""
    out = {}
    for (name, dims, es), off in zip(params, flat_offsets):
        n = int(np.prod(dims))
        vals = synth.values_host(n, es, seed, first_idx=off // es, specials=specials)
        t = torch.from_numpy(vals.view(np.int32 if es == 4 else np.int16).copy())
        out[name] = t.view(*dims)
    return out


def _flat_offsets(params, align=16):
    offs, off = [], 0
    for _, dims, es in params:
        a = max(align, es)
        off = (off + a - 1) // a * a
        offs.append(off)
        off += int(np.prod(dims)) * es
    return offs


def _to_bf16_bits(t: torch.Tensor) -> torch.Tensor:
    """fp32 bit patterns -> bf16 bit patterns: PyTorch's conversion for numbers, the
    stated NaN rule for NaNs; a bf16 source passes through."""
    if t.dtype == torch.int16:
        return t
    conv = t.view(torch.float32).to(torch.bfloat16).view(torch.int16)
    u = t.to(torch.int64) & 0xFFFFFFFF
    nan = (u & 0x7FFFFFFF) > 0x7F800000
    nan_bits = ((u >> 16) | 0x40).to(torch.int32).to(torch.int16)
    return torch.where(nan, nan_bits, conv)


def _to_f16_bits(t: torch.Tensor) -> torch.Tensor:
    """fp32 (or bf16, widened exactly) bit patterns -> IEEE binary16 bit
    patterns: PyTorch's conversion for numbers, the stated NaN rule for NaNs."""
    u = t.to(torch.int64) & (0xFFFF if t.dtype == torch.int16 else 0xFFFFFFFF)
    if t.dtype == torch.int16:
        u = u << 16
    f = u.to(torch.int32).view(torch.float32)
    conv = f.to(torch.float16).view(torch.int16)
    nan = (u & 0x7FFFFFFF) > 0x7F800000
    nan_bits = (((u >> 16) & 0x8000) | 0x7E00 | ((u >> 13) & 0x1FF)).to(torch.int32).to(torch.int16)
    return torch.where(nan, nan_bits, conv)


def restate_rollout(shape, P, tp, ep=False, dst_dtype="bf16"):
    """Per rank, the rollout tensors built the way an inference engine's loader
    would; ep: each rank loads its own experts whole; dst_dtype: the rollout's
    16-bit type."""
    H = shape.hidden

    def kv(t, r):
        # Fewer KV heads than ranks: each rank loads one whole head, shared.
        if tp <= shape.n_kv:
            return t.chunk(tp, 0)[r]
        return t.view(shape.n_kv, shape.head_dim, -1)[r * shape.n_kv // tp]

    ranks = []
    for r in range(tp):
        ts = [P["model.embed_tokens.weight"].chunk(tp, 0)[r]]
        for i in range(shape.layers):
            pre = f"model.layers.{i}."
            a = pre + "self_attn."
            ts.append(torch.cat([P[a + "q_proj.weight"].chunk(tp, 0)[r],
                                 kv(P[a + "k_proj.weight"], r),
                                 kv(P[a + "v_proj.weight"], r)], 0))
            ts.append(P[a + "o_proj.weight"].chunk(tp, 1)[r])
            ts.append(P[a + "q_norm.weight"])
            ts.append(P[a + "k_norm.weight"])
            ts.append(P[pre + "input_layernorm.weight"])
            ts.append(P[pre + "post_attention_layernorm.weight"])
            if shape.n_experts and ep:
                ex = pre + "mlp.experts."
                mine = torch.arange(shape.n_experts).chunk(tp)[r].tolist()
                ts.append(P[pre + "mlp.gate.weight"])
                ts.append(torch.stack([torch.cat([P[f"{ex}{e}.gate_proj.weight"],
                                                  P[f"{ex}{e}.up_proj.weight"]], 0)
                                       for e in mine]))
                ts.append(torch.stack([P[f"{ex}{e}.down_proj.weight"] for e in mine]))
            elif shape.n_experts:
                ex = pre + "mlp.experts."
                ts.append(P[pre + "mlp.gate.weight"])
                ts.append(torch.stack([
                    torch.cat([P[f"{ex}{e}.gate_proj.weight"].chunk(tp, 0)[r],
                               P[f"{ex}{e}.up_proj.weight"].chunk(tp, 0)[r]], 0)
                    for e in range(shape.n_experts)]))
                ts.append(torch.stack([P[f"{ex}{e}.down_proj.weight"].chunk(tp, 1)[r]
                                       for e in range(shape.n_experts)]))
            else:
                m = pre + "mlp."
                ts.append(torch.cat([P[m + "gate_proj.weight"].chunk(tp, 0)[r],
                                     P[m + "up_proj.weight"].chunk(tp, 0)[r]], 0))
                ts.append(P[m + "down_proj.weight"].chunk(tp, 1)[r])
        ts.append(P["model.norm.weight"])
        if not shape.tied:
            ts.append(P["lm_head.weight"].chunk(tp, 0)[r])
        assert all(t.shape[-1] in (H, t.shape[-1]) for t in ts)
        cast = _to_f16_bits if dst_dtype == "f16" else _to_bf16_bits
        ranks.append([cast(t.contiguous()) for t in ts])
    return ranks


def restate_buckets(ranks, bucket_bytes, tensor_align=256):
    out = []
    for tensors in ranks:
        stream = bytearray()
        for t in tensors:
            stream += bytes((-len(stream)) % tensor_align)
            stream += t.numpy().tobytes()
        stream += bytes((-len(stream)) % bucket_bytes)
        out += [bytes(stream[i:i + bucket_bytes]) for i in range(0, len(stream), bucket_bytes)]
    return out


def fsdp2_shards(params, P, n, align=16):
    """Trainer shards as FSDP2 holds them: every parameter cut on dim 0 with
    torch.chunk, each chunk padded to the first chunk's rows; per shard the
    chunks follow one another in manifest order at `align`-byte starts."""
    offs, off = [], 0
    for name, dims, es in params:
        c = -(-dims[0] // n)
        off = (off + max(align, es) - 1) // max(align, es) * max(align, es)
        offs.append(off)
        off += c * int(np.prod(dims[1:], dtype=np.int64)) * es
    S = (off + 15) // 16 * 16
    shards = [np.zeros(S, np.uint8) for _ in range(n)]
    for (name, dims, es), o in zip(params, offs):
        for s_, ch in enumerate(torch.chunk(P[name], n, dim=0)):
            b = np.frombuffer(ch.contiguous().numpy().tobytes(), np.uint8)
            shards[s_][o:o + b.size] = b
    return shards


def fsdp1_unit_shards(params, P, n, align=16):
    """Trainer shards as FSDP1 holds them when every decoder layer is wrapped:
    one FlatParameter per layer and one for the root (embedding, final norm,
    lm_head); each is its parameters flattened and concatenated in manifest
    order at `align`-byte starts, zero-padded to a multiple of 16 * n bytes and
    cut into n equal shards.  Returned unit by unit (root first, then layers)."""
    def unit(name):
        return 1 + int(name.split(".")[2]) if name.startswith("model.layers.") else 0
    n_units = 1 + max(unit(name) for name, _, _ in params)
    shards = []
    for u in range(n_units):
        flat = bytearray()
        for name, dims, es in params:
            if unit(name) != u:
                continue
            flat += bytes((-len(flat)) % max(align, es))
            flat += P[name].contiguous().numpy().tobytes()
        flat += bytes((-len(flat)) % (16 * n))
        shards += [np.frombuffer(bytes(c.numpy().tobytes()), np.uint8).copy()
                   for c in torch.frombuffer(bytearray(flat), dtype=torch.uint8).chunk(n)]
    return shards


RESTATE = ["tiny", "tiny-tp4", "tiny-tied", "tiny-moe", "tiny-moe-tp2", "tiny-moe-f32",
           "tiny-fsdp2", "tiny-moe-kvrep", "tiny-kvrep-f32", "tiny-moe-bf16-specials",
           "tiny-units", "tiny-moe-ep4", "tiny-moe-units-ep2"]


def _workload(name):
    return (synth.WORKLOADS.get(name) or synth.TEST_WORKLOADS.get(name)
            or synth.EXTRA_WORKLOADS[name])


@pytest.mark.parametrize("name", RESTATE)
def test_oracle_matches_restatement(name):
    w = _workload(name)
    L = oracle.workload_layout(w)
    P = _param_tensors(L.params, _flat_offsets(L.params), w.seed, w.specials)
    ranks = restate_rollout(w.shape, P, w.tp, ep=w.ep)
    # Per-tensor reshard, straight from trainer shards: materialised by the
    # oracle for a flat trainer, built with torch for FSDP2 and per-layer FSDP1.
    if w.sharding in ("rows", "units"):
        build = fsdp2_shards if w.sharding == "rows" else fsdp1_unit_shards
        shards = build(L.params, P, w.n_shards)
        host = L.host_shards(w.seed, w.specials)
        assert len(shards) == len(host)
        for a, b in zip(shards, host):
            np.testing.assert_array_equal(a, b)
    else:
        shards = L.host_shards(w.seed, w.specials)
    src = oracle.Source(shards=shards)
    flat_t = [t for rank in ranks for t in rank]
    order = [i for r in range(w.tp) for i, (_, rk, _) in enumerate(L.tensors) if rk == r]
    assert len(order) == len(flat_t)
    for t_idx, want in zip(order, flat_t):
        got = L.reshard_tensor(src, t_idx)
        np.testing.assert_array_equal(got, want.reshape(-1).numpy().view(np.uint16),
                                      err_msg=L.tensors[t_idx][0])
    # Buckets and checksums.
    want_b = restate_buckets(ranks, w.bucket_bytes)
    buckets, cs = L.pack(src)
    assert buckets.shape[0] == len(want_b)
    for b, wb in enumerate(want_b):
        assert buckets[b].tobytes() == wb, f"bucket {b}"
        assert int(cs[b]) == int(np.frombuffer(wb, "<u8").sum(dtype=np.uint64))


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-moe-bf16-specials", "tiny-fsdp2",
                                  "tiny-kvrep-f32"])
def test_oracle_matches_restatement_f16(name):
    """The same restatement for a float16 rollout: PyTorch's float16 conversion
    of the loader-built tensors (the stated NaN rule for NaNs), then the same
    stream and buckets."""
    w = _workload(name).with_(dst_dtype="f16")
    L = oracle.workload_layout(w)
    assert L.dst_dtype == "f16"
    P = _param_tensors(L.params, _flat_offsets(L.params), w.seed, w.specials)
    ranks = restate_rollout(w.shape, P, w.tp, ep=w.ep, dst_dtype="f16")
    if w.sharding == "rows":
        shards = fsdp2_shards(L.params, P, w.n_shards)
    else:
        shards = L.host_shards(w.seed, w.specials)
    src = oracle.Source(shards=shards)
    flat_t = [t for rank in ranks for t in rank]
    order = [i for r in range(w.tp) for i, (_, rk, _) in enumerate(L.tensors) if rk == r]
    for t_idx, want in zip(order, flat_t):
        np.testing.assert_array_equal(L.reshard_tensor(src, t_idx),
                                      want.reshape(-1).numpy().view(np.uint16),
                                      err_msg=L.tensors[t_idx][0])
    want_b = restate_buckets(ranks, w.bucket_bytes)
    buckets, cs = L.pack(src)
    for b, wb in enumerate(want_b):
        assert buckets[b].tobytes() == wb, f"bucket {b}"
        assert int(cs[b]) == int(np.frombuffer(wb, "<u8").sum(dtype=np.uint64))


# ---------------------------------------------------------------------------
# Invariants
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("n_shards,sharding", [(1, "flat"), (2, "flat"), (3, "flat"),
                                               (7, "flat"), (8, "flat"), (13, "flat"),
                                               (1, "rows"), (3, "rows"), (8, "rows"),
                                               (13, "rows"), (300, "rows"),
                                               (1, "units"), (3, "units"), (8, "units")])
def test_shard_count_invariance(n_shards, sharding):
    w = synth.TEST_WORKLOADS["tiny-tp4"]
    ref_L = oracle.workload_layout(w.with_(n_shards=1))
    ref, ref_cs = ref_L.pack(oracle.Source(shards=ref_L.host_shards(w.seed, w.specials)))
    L = oracle.workload_layout(w.with_(n_shards=n_shards, sharding=sharding))
    got, cs = L.pack(oracle.Source(shards=L.host_shards(w.seed, w.specials)))
    np.testing.assert_array_equal(got, ref)
    np.testing.assert_array_equal(cs, ref_cs)


def test_generator_mode_matches_buffer_mode():
    w = synth.TEST_WORKLOADS["tiny-moe-f32"]
    L = oracle.workload_layout(w)
    a, ca = L.pack(oracle.Source(shards=L.host_shards(w.seed, w.specials)))
    b, cb = L.pack(oracle.Source(seed=w.seed, specials=w.specials))
    np.testing.assert_array_equal(a, b)
    np.testing.assert_array_equal(ca, cb)


@pytest.mark.parametrize("name", ["qwen3-0.6b", "qwen3-8b", "qwen3-8b-tp4", "qwen3-30b-a3b",
                                  "tiny-moe-tp2", "qwen3-8b-fsdp2-tp8",
                                  "qwen3-30b-a3b-fsdp2-tp8", "qwen3-30b-a3b-fsdp2-ep8"])
def test_coverage_counts(name):
    """Every parameter element is read tp times if replicated, once otherwise, and
    within one rank no parameter element is read twice (metadata only: full sizes)."""
    w = _workload(name)
    params = qwen3.manifest(w.shape, w.src_elem_bytes)
    tensors = qwen3.rollout_tensors(w.shape, params, w.tp, ep=w.ep)
    area = np.zeros(len(params), np.int64)
    per_rank = {}
    for _, r, blocks in tensors:
        for (p, r0, nr, c0, nc) in blocks:
            area[p] += nr * nc
            per_rank.setdefault((r, p), []).append((r0, nr, c0, nc))
    for p, (pname, dims, _) in enumerate(params):
        numel = int(np.prod(dims))
        replicated = len(dims) == 1 or pname.endswith("mlp.gate.weight")
        kv = pname.endswith(("k_proj.weight", "v_proj.weight"))
        times = w.tp if replicated else (max(1, w.tp // w.shape.n_kv) if kv else 1)
        assert area[p] == numel * times, pname
    for (r, p), rects in per_rank.items():
        # Rectangles of one rank on one parameter must not overlap.
        for i in range(len(rects)):
            for j in range(i + 1, len(rects)):
                a, b = rects[i], rects[j]
                rows = a[0] < b[0] + b[1] and b[0] < a[0] + a[1]
                cols = a[2] < b[2] + b[3] and b[2] < a[2] + a[3]
                assert not (rows and cols), (r, params[p][0])


@pytest.mark.parametrize("name", ["tiny", "tiny-tp4", "tiny-moe-tp2"])
def test_unpack_of_pack_is_reshard(name):
    w = _workload(name)
    L = oracle.workload_layout(w)
    src = oracle.Source(shards=L.host_shards(w.seed, w.specials))
    buckets, _ = L.pack(src)
    for t in range(len(L.tensors)):
        np.testing.assert_array_equal(L.unpack_tensor(buckets, t), L.reshard_tensor(src, t))


def test_checksum_against_numpy_and_linearity():
    rng = np.random.default_rng(5)
    for n in (8, 64, 4096, 1 << 20):
        buf = rng.integers(0, 256, size=n, dtype=np.uint8)
        assert oracle.checksum(buf) == int(buf.view("<u8").sum(dtype=np.uint64))
    allff = np.full(1 << 12, 0xFF, np.uint8)
    assert oracle.checksum(allff) == ((1 << 64) - 1) * (len(allff) // 8) % (1 << 64)
    for off in range(0, 64, 2):
        buf = np.zeros(64, np.uint8)
        buf[off:off + 2] = [0x34, 0x12]
        assert oracle.checksum(buf) == 0x1234 << (8 * (off % 8))


def test_verify_flags_damage():
    w = synth.WORKLOADS["tiny"]
    L = oracle.workload_layout(w)
    buckets, cs = L.pack(oracle.Source(seed=w.seed, specials=w.specials))
    assert L.verify(buckets, cs) == (0, -1)
    bad = buckets.copy()
    bad[5, 1234] ^= 0x10
    assert L.verify(bad, cs) == (1, 5)
    bad[11] = 0
    assert L.verify(bad, cs) == (2, 5)
    swapped = buckets.copy()
    swapped[[2, 3]] = swapped[[3, 2]]
    assert L.verify(swapped, cs) == (2, 2)


QWEN3_GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "qwen3_rollout_worked_example.json")


def test_qwen3_layout_worked_example():
    """The oracle's Qwen3 manifest, FSDP1 units and rollout tensors (Section 7.1:
    a verl FSDP trainer, a vLLM TP rollout) against the hand-derived lists.
    Looked up through ``oracle.qwen3`` at call time."""
    g = json.load(open(QWEN3_GOLDEN))
    base = None
    for case in g["cases"]:
        shape = synth.ModelShape("golden", **case["shape"])
        params = oracle.qwen3.manifest(shape, 4)
        tensors = oracle.qwen3.rollout_tensors(shape, params, case["tp"], ep=case["ep"])
        got = [[n, r, [list(b) for b in bl]] for n, r, bl in tensors]
        if "manifest" in case:
            assert [[n, list(d)] for n, d, _ in params] == case["manifest"], case["name"]
            assert oracle.qwen3.layer_units(params) == case["units"], case["name"]
            assert got == case["tensors"], case["name"]
            base = case["tensors"]
        else:                                # expert parallel: only w13 and w2 change
            want = {(n, r): bl for n, r, bl in case["tensors_differing_from_tp"]}
            expect = [[n, r, want.get((n, r), bl)] for n, r, bl in base]
            assert got == expect, case["name"]


def test_layout_rejects_bad_input():
    params = [("a", (4, 4), 4)]
    with pytest.raises(RuntimeError):
        oracle.Layout(params, [("t", 0, [(0, 2, 3, 0, 4)])], 1, 1, 64)   # rows out of range
    with pytest.raises(RuntimeError):
        oracle.Layout(params, [("t", 1, [(0, 0, 1, 0, 4)])], 1, 1, 64)   # rank out of range
    with pytest.raises(RuntimeError):
        oracle.Layout(params, [("t", 0, [(0, 0, 1, 0, 4)])], 1, 1, 12)   # bucket % 8 != 0


ROWS_GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "rows_sharding_worked_example.json")


def test_rows_sharding_golden():
    g = json.load(open(ROWS_GOLDEN))
    params = [(p["name"], tuple(p["dims"]), p["elem_bytes"]) for p in g["params"]]
    tensors = [(t["name"], t["rank"], [tuple(b) for b in t["blocks"]]) for t in g["tensors"]]
    L = oracle.Layout(params, tensors, n_shards=g["n_shards"], tp=g["tp"],
                      bucket_bytes=g["bucket_bytes"], align_bytes=g["align_bytes"],
                      tensor_align=g["tensor_align"], sharding="rows")
    e = g["expect"]
    assert list(L.chunk_rows) == e["chunk_rows"]
    assert list(L.param_offset) == e["param_offset"]
    assert L.shard_bytes == e["shard_bytes"]
    assert list(L.param_gen_base) == e["param_gen_base"]
    shards = [bytearray(e["shard_bytes"]) for _ in range(g["n_shards"])]
    for pl in g["placement"]:
        p = g["params"][pl["param"]]
        es = p["elem_bytes"]
        for k in range(pl["n_elems"]):
            v = _int(p["bits"][pl["first_elem"] + k])
            o = pl["offset"] + k * es
            shards[pl["shard"]][o:o + es] = v.to_bytes(es, "little")
    src = oracle.Source(shards=[np.frombuffer(bytes(s), np.uint8) for s in shards])
    for t, want in enumerate(e["tensors_bf16"]):
        np.testing.assert_array_equal(L.reshard_tensor(src, t),
                                      np.array([_int(x) for x in want], np.uint16))
    buckets, cs = L.pack(src)
    assert [b.tobytes().hex() for b in buckets] == e["buckets_hex"]
    assert [int(c) for c in cs] == [_int(c) for c in e["checksums"]]


def test_shard_size_rule_edge():
    """Hand-derived: one bf16 parameter of 65 elements (130 bytes) over 4 flat
    shards.  The total rounds up to a multiple of 16 * 4 = 64 bytes: 192, so
    S = 48 (not 32: 4 x 32 = 128 bytes would not hold byte 129).  Element 64
    (flat bytes 128-129) is shard 128 // 48 = 2, offset 128 - 96 = 32."""
    L = oracle.Layout([("p", (65,), 2)], [("t", 0, [(0, 64, 1, 0, 1)])], n_shards=4, tp=1,
                      bucket_bytes=16)
    assert L.shard_bytes == 48
    shards = [np.zeros(48, np.uint8) for _ in range(4)]
    shards[2][32:34] = [0x34, 0x12]
    got = L.reshard_tensor(oracle.Source(shards=shards), 0)
    assert list(got) == [0x1234]


def test_unit_sharding_worked_example():
    """Two FSDP1 units over 2 shards, worked by hand.

    Unit 0 holds a (3 bf16) and c (5 bf16); unit 1 holds b (10 f32).
    Unit 0: a at byte 0 (6 B); c at the next 16-byte start, 16 (10 B); the end,
    26, pads to a multiple of 16 * 2 = 32, so S_0 = 16: a is in buffer 0 at 0,
    c in buffer 1 at 0.  Unit 1: b at 0 (40 B) pads to 64, S_1 = 32: b's
    elements 0..7 are buffer 2 bytes 0..31, elements 8 and 9 buffer 3 bytes 0..7."""
    params = [("a", (3,), 2), ("b", (10,), 4), ("c", (5,), 2)]
    tensors = [("c", 0, [(2, 0, 5, 0, 1)]), ("b", 0, [(1, 0, 10, 0, 1)])]
    L = oracle.Layout(params, tensors, n_shards=2, tp=1, bucket_bytes=64, sharding="units",
                      units=[0, 1, 0])
    assert list(L.param_offset) == [0, 0, 16]
    assert list(L.unit_shard_bytes) == [16, 32]
    bufs = [np.zeros(16, np.uint8), np.zeros(16, np.uint8), np.zeros(32, np.uint8),
            np.zeros(32, np.uint8)]
    bufs[1][0:10] = np.array([0x11, 0x3F, 0x22, 0x3F, 0x33, 0x3F, 0x44, 0x3F, 0x55, 0x3F],
                             np.uint8)                      # c = bf16 0x3F11 .. 0x3F55
    b_vals = np.arange(1, 11, dtype=np.float32)             # b = 1.0 .. 10.0, exact in bf16
    bufs[2][:] = b_vals[:8].view(np.uint8)
    bufs[3][0:8] = b_vals[8:].view(np.uint8)
    src = oracle.Source(shards=bufs)
    assert list(L.reshard_tensor(src, 0)) == [0x3F11, 0x3F22, 0x3F33, 0x3F44, 0x3F55]
    want_b = (b_vals.view(np.uint32) >> 16).astype(np.uint16)
    np.testing.assert_array_equal(L.reshard_tensor(src, 1), want_b)


def test_unit_shard_size_rule_edge():
    """A unit whose size over the shard count truncates onto a multiple of 16.

    Unit 0 holds p (25 bf16 = 50 B) over 3 shards: 50 pads to 96 (a multiple of
    16 * 3), so S_0 = 32 and element 24 (byte 48) is buffer 1 at byte 16.  Unit
    1 holds q (4 f32 = 16 B): 16 pads to 48, S_1 = 16, buffers 3..5."""
    params = [("p", (25,), 2), ("q", (4,), 4)]
    tensors = [("p", 0, [(0, 0, 25, 0, 1)]), ("q", 0, [(1, 0, 4, 0, 1)])]
    L = oracle.Layout(params, tensors, n_shards=3, tp=1, bucket_bytes=128, sharding="units",
                      units=[0, 1])
    assert list(L.unit_shard_bytes) == [32, 16]
    bufs = [np.zeros(32, np.uint8) for _ in range(3)] + [np.zeros(16, np.uint8) for _ in range(3)]
    p_vals = np.arange(0x3F00, 0x3F00 + 25, dtype=np.uint16)
    flat0 = np.zeros(96, np.uint8)
    flat0[:50] = p_vals.view(np.uint8)
    for s in range(3):
        bufs[s][:] = flat0[32 * s:32 * (s + 1)]
    assert bufs[1][16] == 0x18 and bufs[1][17] == 0x3F       # element 24 where it belongs
    bufs[3][:] = np.full(4, 0xC0000000, np.uint32).view(np.uint8)   # q = -2.0 each
    src = oracle.Source(shards=bufs)
    np.testing.assert_array_equal(L.reshard_tensor(src, 0), p_vals)
    assert list(L.reshard_tensor(src, 1)) == [0xC000] * 4
