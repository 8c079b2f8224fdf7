"""Oracle-side description of a Qwen3 trainer manifest and its rollout layout.

TEST INFRASTRUCTURE ONLY (see ``oracle/__init__.py``).  Written independently
of the CUDA library's own layout helpers; the two meet only through the
workload shapes in ``synth``.

Trainer side (RobustRL Section 7.1: verl + PyTorch FSDP): parameters in
module-registration order of a Qwen3 decoder,
    embed_tokens; per layer: q_proj, k_proj, v_proj, o_proj, q_norm, k_norm,
    then the MLP (dense: gate_proj, up_proj, down_proj; MoE: the router
    ``mlp.gate`` then, for each expert, gate_proj, up_proj, down_proj),
    input_layernorm, post_attention_layernorm; final norm; lm_head unless tied.

Rollout side (Section 7.1: vLLM, tensor parallel): per rank, in this order,
    embed; per layer: qkv, o, q_norm, k_norm, input_ln, post_ln, then
    gate_up, down (dense) or router, w13, w2 (MoE); final norm; lm_head.
with qkv = [q; k; v] and gate_up = w13[e] = [gate; up] stacked along the
output dimension.  Under TP = t, rank r takes the r-th of t equal row ranges
of the column-parallel weights (q, k, v, gate, up, embedding, lm_head, each
expert's gate/up) and the r-th of t equal column ranges of the row-parallel
weights (o_proj, down_proj, each expert's down_proj); norms and the router
are replicated on every rank.  When TP exceeds the number of KV heads, each
KV head is replicated instead: rank r takes the rows of head r * n_kv // t of
k and of v (t / n_kv ranks per head).  Expert-parallel rollout (ep): the
experts are not cut; rank r takes experts r*E/t .. (r+1)*E/t - 1 whole, in
order, into its w13 and w2 (attention as above, router replicated).

Per-layer FSDP1 units: each decoder layer's parameters form one unit (layer
i is unit i + 1); the parameters outside the layers (embedding, final norm,
lm_head) form the root unit 0.

A block is (param index, row0, nrows, col0, ncols) on the parameter's
[rows = d0, cols = d1 * d2 * ...] view.
"""
from __future__ import annotations

from typing import List, Tuple

Param = Tuple[str, Tuple[int, ...], int]          # name, dims, element bytes
Block = Tuple[int, int, int, int, int]            # param, row0, nrows, col0, ncols
Tensor = Tuple[str, int, List[Block]]             # name, rank, blocks


def manifest(shape, elem_bytes: int) -> List[Param]:
    H, hd = shape.hidden, shape.head_dim
    Q, K = shape.n_q * hd, shape.n_kv * hd
    out: List[Param] = [("model.embed_tokens.weight", (shape.vocab, H), elem_bytes)]
    for i in range(shape.layers):
        pre = f"model.layers.{i}."
        out += [
            (pre + "self_attn.q_proj.weight", (Q, H), elem_bytes),
            (pre + "self_attn.k_proj.weight", (K, H), elem_bytes),
            (pre + "self_attn.v_proj.weight", (K, H), elem_bytes),
            (pre + "self_attn.o_proj.weight", (H, Q), elem_bytes),
            (pre + "self_attn.q_norm.weight", (hd,), elem_bytes),
            (pre + "self_attn.k_norm.weight", (hd,), elem_bytes),
        ]
        if shape.n_experts:
            E, Im = shape.n_experts, shape.moe_intermediate
            out.append((pre + "mlp.gate.weight", (E, H), elem_bytes))
            for e in range(E):
                ep = pre + f"mlp.experts.{e}."
                out += [
                    (ep + "gate_proj.weight", (Im, H), elem_bytes),
                    (ep + "up_proj.weight", (Im, H), elem_bytes),
                    (ep + "down_proj.weight", (H, Im), elem_bytes),
                ]
        else:
            I = shape.intermediate
            out += [
                (pre + "mlp.gate_proj.weight", (I, H), elem_bytes),
                (pre + "mlp.up_proj.weight", (I, H), elem_bytes),
                (pre + "mlp.down_proj.weight", (H, I), elem_bytes),
            ]
        out += [
            (pre + "input_layernorm.weight", (H,), elem_bytes),
            (pre + "post_attention_layernorm.weight", (H,), elem_bytes),
        ]
    out.append(("model.norm.weight", (H,), elem_bytes))
    if not shape.tied:
        out.append(("lm_head.weight", (shape.vocab, H), elem_bytes))
    return out


def _view(dims) -> Tuple[int, int]:
    rows = dims[0]
    cols = 1
    for d in dims[1:]:
        cols *= d
    return rows, cols


def layer_units(params: List[Param]) -> List[int]:
    out = []
    for name, _, _ in params:
        if name.startswith("model.layers."):
            layer = int(name[len("model.layers."):].split(".", 1)[0])
            out.append(layer + 1)
        else:
            out.append(0)
    return out


def rollout_tensors(shape, params: List[Param], tp: int, ep: bool = False) -> List[Tensor]:
    index = {name: i for i, (name, _, _) in enumerate(params)}
    view = {name: _view(dims) for name, dims, _ in params}

    def whole(name) -> Block:
        rows, cols = view[name]
        return (index[name], 0, rows, 0, cols)

    def row_slice(name, r) -> Block:
        rows, cols = view[name]
        assert rows % tp == 0, f"{name}: {rows} rows do not split over TP={tp}"
        n = rows // tp
        return (index[name], r * n, n, 0, cols)

    def kv_slice(name, r) -> Block:
        # TP <= n_kv: a row range of whole heads; TP > n_kv: one replicated head.
        if tp <= shape.n_kv:
            return row_slice(name, r)
        assert tp % shape.n_kv == 0, f"TP={tp} is not a multiple of {shape.n_kv} KV heads"
        rows, cols = view[name]
        h = r * shape.n_kv // tp
        return (index[name], h * shape.head_dim, shape.head_dim, 0, cols)

    def col_slice(name, r) -> Block:
        rows, cols = view[name]
        assert cols % tp == 0, f"{name}: {cols} columns do not split over TP={tp}"
        n = cols // tp
        return (index[name], 0, rows, r * n, n)

    tensors: List[Tensor] = []
    for r in range(tp):
        tensors.append(("embed_tokens", r, [row_slice("model.embed_tokens.weight", r)]))
        for i in range(shape.layers):
            pre = f"model.layers.{i}."
            a = pre + "self_attn."
            tensors += [
                (f"layers.{i}.qkv_proj", r, [row_slice(a + "q_proj.weight", r),
                                              kv_slice(a + "k_proj.weight", r),
                                              kv_slice(a + "v_proj.weight", r)]),
                (f"layers.{i}.o_proj", r, [col_slice(a + "o_proj.weight", r)]),
                (f"layers.{i}.q_norm", r, [whole(a + "q_norm.weight")]),
                (f"layers.{i}.k_norm", r, [whole(a + "k_norm.weight")]),
                (f"layers.{i}.input_layernorm", r, [whole(pre + "input_layernorm.weight")]),
                (f"layers.{i}.post_attention_layernorm", r,
                 [whole(pre + "post_attention_layernorm.weight")]),
            ]
            if shape.n_experts:
                E = shape.n_experts
                ex = pre + "mlp.experts."
                w13: List[Block] = []
                w2: List[Block] = []
                if ep:
                    assert E % tp == 0, f"{E} experts do not split over {tp} ranks"
                    per = E // tp
                    for e in range(r * per, (r + 1) * per):
                        w13 += [whole(f"{ex}{e}.gate_proj.weight"),
                                whole(f"{ex}{e}.up_proj.weight")]
                        w2.append(whole(f"{ex}{e}.down_proj.weight"))
                else:
                    for e in range(E):
                        w13 += [row_slice(f"{ex}{e}.gate_proj.weight", r),
                                row_slice(f"{ex}{e}.up_proj.weight", r)]
                        w2.append(col_slice(f"{ex}{e}.down_proj.weight", r))
                tensors += [
                    (f"layers.{i}.router", r, [whole(pre + "mlp.gate.weight")]),
                    (f"layers.{i}.experts.w13", r, w13),
                    (f"layers.{i}.experts.w2", r, w2),
                ]
            else:
                m = pre + "mlp."
                tensors += [
                    (f"layers.{i}.gate_up_proj", r, [row_slice(m + "gate_proj.weight", r),
                                                      row_slice(m + "up_proj.weight", r)]),
                    (f"layers.{i}.down_proj", r, [col_slice(m + "down_proj.weight", r)]),
                ]
        tensors.append(("norm", r, [whole("model.norm.weight")]))
        if not shape.tied:
            tensors.append(("lm_head", r, [row_slice("lm_head.weight", r)]))
    return tensors
