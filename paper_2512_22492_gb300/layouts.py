"""Layout descriptions for Qwen3-family models: trainer manifest -> rollout tensors.

The C library knows nothing about models; a weight sync is described to it
as a parameter manifest plus, per rollout tensor, a list of 2-D blocks of
those parameters.  This module writes those descriptions for Qwen3 dense and
MoE decoders, as the paper's system uses them (RobustRL Section 7.1: FSDP
trainer, vLLM rollout with tensor parallelism; Section 5.2.1 step 1: the
weights are re-laid out in the rollout's sharding).

Trainer manifest: module-registration order of the Hugging Face Qwen3 model.
Rollout tensors, per rank r of TP = t, in this order:
  embed_tokens        rows r of t of the embedding
  per layer:          qkv_proj = [q; k; v] (row slices), o_proj (column slice),
                      q_norm, k_norm, input_layernorm, post_attention_layernorm
                      (replicated), then
                      dense: gate_up_proj = [gate; up] (row slices), down_proj
                             (column slice)
                      MoE:   router (replicated), experts.w13 = stacked
                             [gate_e; up_e] (row slices), experts.w2 = stacked
                             down_e (column slices)
  norm                replicated
  lm_head             rows r of t, unless tied to the embedding
When t exceeds the number of KV heads, k and v are not split but replicated
by head: rank r holds KV head r * n_kv // t.  With expert parallelism
(ep=True) the experts are not sliced but dealt out whole: rank r holds
experts [r * E / t, (r + 1) * E / t), so its w13 and w2 stack E / t full
experts; attention stays tensor-parallel and the router replicated.

Trainer sources: one flat FSDP1 FlatParameter ("flat"), FSDP2 per-parameter
dim-0 shards ("rows"), or FSDP1 wrapping every decoder layer ("units"): unit
0 is the root (embedding, final norm, lm_head), unit 1 + i is layer i.
"""
from __future__ import annotations

from typing import Dict, List, Tuple

from .rr import Block, DstLayout, DstTensor, Param, SrcLayout


def qwen3_manifest(shape, dtype: str = "f32") -> List[Param]:
    """Trainer parameters of a Qwen3 decoder (``shape`` has layers, hidden, n_q,
    n_kv, head_dim, intermediate, vocab, tied, n_experts, moe_intermediate)."""
    h, d = shape.hidden, shape.head_dim
    out = [Param("model.embed_tokens.weight", (shape.vocab, h), dtype)]
    for i in range(shape.layers):
        L = f"model.layers.{i}"
        out += [Param(f"{L}.self_attn.q_proj.weight", (shape.n_q * d, h), dtype),
                Param(f"{L}.self_attn.k_proj.weight", (shape.n_kv * d, h), dtype),
                Param(f"{L}.self_attn.v_proj.weight", (shape.n_kv * d, h), dtype),
                Param(f"{L}.self_attn.o_proj.weight", (h, shape.n_q * d), dtype),
                Param(f"{L}.self_attn.q_norm.weight", (d,), dtype),
                Param(f"{L}.self_attn.k_norm.weight", (d,), dtype)]
        if getattr(shape, "n_experts", 0):
            m = shape.moe_intermediate
            out.append(Param(f"{L}.mlp.gate.weight", (shape.n_experts, h), dtype))
            for e in range(shape.n_experts):
                out += [Param(f"{L}.mlp.experts.{e}.gate_proj.weight", (m, h), dtype),
                        Param(f"{L}.mlp.experts.{e}.up_proj.weight", (m, h), dtype),
                        Param(f"{L}.mlp.experts.{e}.down_proj.weight", (h, m), dtype)]
        else:
            m = shape.intermediate
            out += [Param(f"{L}.mlp.gate_proj.weight", (m, h), dtype),
                    Param(f"{L}.mlp.up_proj.weight", (m, h), dtype),
                    Param(f"{L}.mlp.down_proj.weight", (h, m), dtype)]
        out += [Param(f"{L}.input_layernorm.weight", (h,), dtype),
                Param(f"{L}.post_attention_layernorm.weight", (h,), dtype)]
    out.append(Param("model.norm.weight", (h,), dtype))
    if not shape.tied:
        out.append(Param("lm_head.weight", (shape.vocab, h), dtype))
    return out


class _Slicer:
    """Blocks of named parameters: whole, r-th row range, r-th column range."""

    def __init__(self, manifest: List[Param], tp: int):
        self.idx: Dict[str, int] = {p.name: i for i, p in enumerate(manifest)}
        self.mat: Dict[str, Tuple[int, int]] = {}
        for p in manifest:
            rows = p.shape[0] if len(p.shape) else 1
            cols = 1
            for s in p.shape[1:]:
                cols *= s
            self.mat[p.name] = (rows, cols)
        self.tp = tp

    def whole(self, name: str) -> Block:
        rows, cols = self.mat[name]
        return Block(self.idx[name], 0, rows, 0, cols)

    def rows(self, name: str, r: int) -> Block:
        rows, cols = self.mat[name]
        if rows % self.tp:
            raise ValueError(f"{name}: {rows} rows do not divide over TP={self.tp}")
        n = rows // self.tp
        return Block(self.idx[name], r * n, n, 0, cols)

    def kv_rows(self, name: str, r: int, n_heads: int, head_dim: int) -> Block:
        """k/v rows of rank r: a row slice, or one whole replicated head when the
        ranks outnumber the heads."""
        if self.tp <= n_heads:
            return self.rows(name, r)
        if self.tp % n_heads:
            raise ValueError(f"TP={self.tp} is not a multiple of {n_heads} KV heads")
        _, cols = self.mat[name]
        h = r * n_heads // self.tp
        return Block(self.idx[name], h * head_dim, head_dim, 0, cols)

    def cols(self, name: str, r: int) -> Block:
        rows, cols = self.mat[name]
        if cols % self.tp:
            raise ValueError(f"{name}: {cols} columns do not divide over TP={self.tp}")
        n = cols // self.tp
        return Block(self.idx[name], 0, rows, r * n, n)


def qwen3_layer_units(manifest: List[Param]) -> List[int]:
    """FSDP1 units when every decoder layer is wrapped: the unit of each
    parameter, 1 + i for layer i and 0 for the root's own parameters."""
    units = []
    for p in manifest:
        parts = p.name.split(".")
        units.append(1 + int(parts[2]) if parts[:2] == ["model", "layers"] else 0)
    return units


def qwen3_rollout(shape, manifest: List[Param], tp: int = 1,
                  tensor_align_bytes: int = 256, ep: bool = False) -> DstLayout:
    """Rollout (inference-engine) tensors for TP = tp, rank-major; ep=True
    deals the experts out whole instead of slicing each one."""
    s = _Slicer(manifest, tp)
    if ep and getattr(shape, "n_experts", 0) % tp:
        raise ValueError(f"{shape.n_experts} experts do not divide over {tp} ranks")
    tensors: List[DstTensor] = []
    for r in range(tp):
        def add(name, blocks):
            tensors.append(DstTensor(name, r, blocks))

        add("embed_tokens", [s.rows("model.embed_tokens.weight", r)])
        for i in range(shape.layers):
            L = f"model.layers.{i}"
            a = f"{L}.self_attn"
            add(f"layers.{i}.qkv_proj",
                [s.rows(f"{a}.q_proj.weight", r),
                 s.kv_rows(f"{a}.k_proj.weight", r, shape.n_kv, shape.head_dim),
                 s.kv_rows(f"{a}.v_proj.weight", r, shape.n_kv, shape.head_dim)])
            add(f"layers.{i}.o_proj", [s.cols(f"{a}.o_proj.weight", r)])
            add(f"layers.{i}.q_norm", [s.whole(f"{a}.q_norm.weight")])
            add(f"layers.{i}.k_norm", [s.whole(f"{a}.k_norm.weight")])
            add(f"layers.{i}.input_layernorm", [s.whole(f"{L}.input_layernorm.weight")])
            add(f"layers.{i}.post_attention_layernorm",
                [s.whole(f"{L}.post_attention_layernorm.weight")])
            if getattr(shape, "n_experts", 0):
                E = shape.n_experts
                x = f"{L}.mlp.experts"
                add(f"layers.{i}.router", [s.whole(f"{L}.mlp.gate.weight")])
                if ep:
                    mine = range(r * E // tp, (r + 1) * E // tp)
                    add(f"layers.{i}.experts.w13",
                        [b for e in mine for b in (s.whole(f"{x}.{e}.gate_proj.weight"),
                                                   s.whole(f"{x}.{e}.up_proj.weight"))])
                    add(f"layers.{i}.experts.w2",
                        [s.whole(f"{x}.{e}.down_proj.weight") for e in mine])
                else:
                    add(f"layers.{i}.experts.w13",
                        [b for e in range(E) for b in (s.rows(f"{x}.{e}.gate_proj.weight", r),
                                                       s.rows(f"{x}.{e}.up_proj.weight", r))])
                    add(f"layers.{i}.experts.w2",
                        [s.cols(f"{x}.{e}.down_proj.weight", r) for e in range(E)])
            else:
                add(f"layers.{i}.gate_up_proj", [s.rows(f"{L}.mlp.gate_proj.weight", r),
                                                 s.rows(f"{L}.mlp.up_proj.weight", r)])
                add(f"layers.{i}.down_proj", [s.cols(f"{L}.mlp.down_proj.weight", r)])
        add("norm", [s.whole("model.norm.weight")])
        if not shape.tied:
            add("lm_head", [s.rows("lm_head.weight", r)])
    return DstLayout(tp=tp, tensors=tensors, tensor_align_bytes=tensor_align_bytes)


def qwen3_sync(shape, dtype: str, n_shards: int, tp: int, sharding: str = "flat",
               ep: bool = False, dst_dtype: str = "bf16"):
    """(manifest, source layout, destination layout) for one Qwen3 weight sync.
    sharding: "flat" (one FSDP1 FlatParameter cut evenly), "rows" (FSDP2:
    every parameter cut on dim 0) or "units" (FSDP1 wrapping every decoder
    layer); ep: expert-parallel rollout; dst_dtype: the rollout's 16-bit
    element type, "bf16" or "f16"."""
    manifest = qwen3_manifest(shape, dtype)
    units = qwen3_layer_units(manifest) if sharding == "units" else None
    src = SrcLayout(n_shards=n_shards, align_bytes=16, sharding=sharding, units=units)
    dst = qwen3_rollout(shape, manifest, tp, ep=ep)
    dst.dtype = dst_dtype
    return manifest, src, dst


# ---------------------------------------------------------------------------
# Relay re-pack (Section 5.2.1, step 3): a rollout that already holds the new
# weights serves others.  Its copy is the rollout layout in bf16 -- either the
# buckets it pulled, or the tensors it loaded -- and the rollout it serves may
# use another tensor-parallel degree.
# ---------------------------------------------------------------------------

def rollout_as_source(dst: DstLayout):
    """The tensors of a rollout layout as bf16 source parameters.

    Tensor t becomes parameter t of shape [sum of its blocks' rows, cols] (its
    blocks share one column count).  Also returns, per trainer parameter, the
    pieces that hold it: (source tensor, first row in that tensor, block)."""
    params: List[Param] = []
    pieces: Dict[int, List[Tuple[int, int, Block]]] = {}
    for t, T in enumerate(dst.tensors):
        cols = {b.ncols for b in T.blocks if b.nrows and b.ncols}
        if len(cols) > 1:
            raise ValueError(f"{T.name}: blocks of different widths cannot form a matrix")
        width = cols.pop() if cols else 1
        rows = sum(b.nrows for b in T.blocks if b.nrows and b.ncols)
        params.append(Param(f"rank{T.rank}.{T.name}", (rows, width), "bf16"))
        ro = 0
        for b in T.blocks:
            if not (b.nrows and b.ncols):
                continue
            pieces.setdefault(b.param, []).append((t, ro, b))
            ro += b.nrows
    return params, pieces


def _translate(blk: Block, pieces) -> List[Block]:
    """Blocks over source tensors holding `blk`'s elements in its row-major order."""
    r0, r1 = blk.row0, blk.row0 + blk.nrows
    c0, c1 = blk.col0, blk.col0 + blk.ncols
    if r1 <= r0 or c1 <= c0:
        return []
    seen, cand = set(), []
    for t, ro, b in pieces:
        rect = (b.row0, b.nrows, b.col0, b.ncols)
        if rect in seen:          # a replica (norms, router, shared KV heads): one is enough
            continue
        if b.row0 < r1 and r0 < b.row0 + b.nrows and b.col0 < c1 and c0 < b.col0 + b.ncols:
            seen.add(rect)
            cand.append((t, ro, b))
    cuts = sorted({r0, r1} | {min(max(b.row0, r0), r1) for _, _, b in cand}
                  | {min(max(b.row0 + b.nrows, r0), r1) for _, _, b in cand})
    out: List[Block] = []
    for ra, rb in zip(cuts, cuts[1:]):
        if rb <= ra:
            continue
        band = sorted((x for x in cand if x[2].row0 <= ra and rb <= x[2].row0 + x[2].nrows),
                      key=lambda x: x[2].col0)
        spans, c = [], c0
        for t, ro, b in band:
            a, z = max(c, b.col0), min(c1, b.col0 + b.ncols)
            if a > c:
                raise ValueError("the source does not hold every element of the target")
            if z > a:
                spans.append((t, ro, b, a, z))
                c = z
        if c < c1:
            raise ValueError("the source does not hold every element of the target")
        if len(spans) == 1:
            t, ro, b, a, z = spans[0]
            out.append(Block(t, ro + ra - b.row0, rb - ra, a - b.col0, z - a))
        else:
            for r in range(ra, rb):        # row-parallel pieces side by side: row by row
                for t, ro, b, a, z in spans:
                    out.append(Block(t, ro + r - b.row0, 1, a - b.col0, z - a))
    return out


def relayout(source: DstLayout, target: DstLayout) -> DstLayout:
    """`target` (blocks on trainer parameters) re-expressed on the tensors of
    `source` (the parameters that ``rollout_as_source(source)`` returns)."""
    _, pieces = rollout_as_source(source)
    tensors = [DstTensor(T.name, T.rank,
                         [nb for b in T.blocks for nb in _translate(b, pieces.get(b.param, []))])
               for T in target.tensors]
    return DstLayout(tp=target.tp, tensors=tensors, tensor_align_bytes=target.tensor_align_bytes)


def qwen3_relay(shape, src_tp: int, dst_tp: int, from_plan=None, src_ep: bool = False,
                dst_ep: bool = False):
    """(manifest, source layout, destination layout) for a relay that holds the
    TP=src_tp rollout image and serves a TP=dst_tp rollout (either side may
    deal its experts out whole: src_ep / dst_ep).

    from_plan=None: the relay re-packs from its loaded tensors (one buffer per
    tensor, in the order of the TP=src_tp rollout layout).  from_plan=<the
    plan that packed the image>: it re-packs straight from the buckets it
    pulled (the buckets, in order, are the shards; bucket_bytes must be a
    multiple of 16).

    A relay copies 16-bit elements bit for bit, so the same layout serves a
    bfloat16 and a float16 image alike: its manifest reads the elements as
    bf16 and its destination keeps the default type (no cast)."""
    logical = qwen3_manifest(shape, "bf16")
    src = qwen3_rollout(shape, logical, src_tp, ep=src_ep)
    params, _ = rollout_as_source(src)
    dst = relayout(src, qwen3_rollout(shape, logical, dst_tp, ep=dst_ep))
    if from_plan is None:
        return params, SrcLayout(n_shards=len(params), sharding="tensors"), dst
    B = from_plan.bucket_bytes
    offsets = [from_plan.first_bucket_of_rank[from_plan.tensor_ranks[t]] * B
               + from_plan.tensor_stream_offset[t] for t in range(len(params))]
    return params, SrcLayout(n_shards=from_plan.n_buckets, param_flat_offset=offsets,
                             shard_bytes=B), dst
