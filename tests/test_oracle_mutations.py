"""The oracle's pins catch plausible mistakes.

Each case below plants one mistake in a copy of oracle/rr_oracle.c -- a
dropped term, a wrong bit, a transposed index, a missed alignment, a wrong
byte order -- builds that copy on its own, and runs a battery of the pins
(hand-worked golden examples, the brute-force cast check, the PyTorch
restatement of the layout, the numpy checksum, round trip and verify) against
it.  The same is done with mistakes planted in a copy of oracle/qwen3.py (the
oracle's Qwen3 manifest and rollout layout), loaded in place of the real
module.  Every planted mistake must make the battery fail, and the real oracle
must pass it.  Nothing here touches a GPU.
"""
import importlib.util
import os
import subprocess

import numpy as np
import pytest

import oracle
from tests import test_oracle_cast as cast_pins
from tests import test_oracle_layout as layout_pins

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "rr_oracle.c")
QWEN3_SRC = os.path.join(ROOT, "oracle", "qwen3.py")

# (name, text in rr_oracle.c, replacement)
MUTATIONS = [
    ("nan loses the quiet bit", "return (uint16_t)((b >> 16) | 0x0040u);",
     "return (uint16_t)(b >> 16);"),
    ("round half up, not to even", "return (uint16_t)((b + 0x7FFFu + ((b >> 16) & 1u)) >> 16);",
     "return (uint16_t)((b + 0x8000u) >> 16);"),
    ("wrong kept bit", "((b >> 16) & 1u)", "((b >> 15) & 1u)"),
    ("infinity taken for a NaN", "if ((b & 0x7FFFFFFFu) > 0x7F800000u)",
     "if ((b & 0x7FFFFFFFu) >= 0x7F800000u)"),
    ("bf16 source rounded again", "return elem_bytes == 4 ? orc_rne_bf16(bits) : (uint16_t)bits;",
     "return orc_rne_bf16(bits << (elem_bytes == 2 ? 16 : 0));"),
    ("block rows and columns transposed",
     "int64_t row = B->row0 + jj / B->ncols;\n            int64_t col = B->col0 + jj % B->ncols;",
     "int64_t row = B->row0 + jj % B->nrows;\n            int64_t col = B->col0 + jj / B->nrows;"),
    ("parameters not aligned", "off = align_up(off, a);", "off = off + 0 * a;"),
    ("tensors not aligned in the stream",
     "int64_t start = align_up(L->rank_stream_bytes[T->rank], L->tensor_align);",
     "int64_t start = L->rank_stream_bytes[T->rank];"),
    ("shard size ignores the shard count",
     "L->shard_bytes = align_up(flat_end, 16 * (int64_t)L->n_shards) / L->n_shards;",
     "L->shard_bytes = align_up(flat_end / L->n_shards, 16);"),
    ("big-endian checksum words", "word |= (uint64_t)bytes[k + i] << (8 * i);",
     "word |= (uint64_t)bytes[k + i] << (8 * (7 - i));"),
    ("buckets numbered from the wrong rank",
     "L->rank_first_bucket[r + 1] = L->rank_first_bucket[r] + nb;",
     "L->rank_first_bucket[r + 1] = nb;"),
    ("unpack ignores the rank's first bucket",
     "const uint8_t* bucket = buckets[first + pos / L->bucket_bytes];",
     "const uint8_t* bucket = buckets[pos / L->bucket_bytes];"),
    ("verify counts the good buckets",
     "if (orc_checksum(buckets[b], L->bucket_bytes) != checksums[b]) {",
     "if (orc_checksum(buckets[b], L->bucket_bytes) == checksums[b]) {"),
    ("FSDP2 chunks rounded down", "int64_t c = (P->rows + L->n_shards - 1) / L->n_shards;",
     "int64_t c = P->rows / L->n_shards + (P->rows < L->n_shards);"),
    ("values indexed by the in-shard offset",
     "L->param_gen_base[p] = start / P->elem_bytes;",
     "L->param_gen_base[p] = (start % 4096) / P->elem_bytes;"),
    ("little-endian source bytes read reversed", "v |= (uint32_t)byte << (8 * i);",
     "v |= (uint32_t)byte << (8 * (es - 1 - i));"),
    ("unit buffers numbered shard-major", "int64_t buf = (int64_t)u * L->n_shards + f / Su;",
     "int64_t buf = (f / Su) * L->n_units + u;"),
    ("unit size not padded for the shard count",
     "L->unit_shard_bytes[u] = align_up(local, 16 * (int64_t)L->n_shards) / L->n_shards;",
     "L->unit_shard_bytes[u] = align_up(local / L->n_shards, 16);"),
    ("unit parameters not aligned",
     "                local = align_up(local, a);\n                L->param_offset[p] = local;",
     "                L->param_offset[p] = local + 0 * a;"),
    ("block column offset dropped", "int64_t col = B->col0 + jj % B->ncols;",
     "int64_t col = jj % B->ncols;"),
    ("rows strided by the block width, not the parameter's",
     "source_bits(L, S, B->param, row * P->cols + col, &bits);",
     "source_bits(L, S, B->param, row * B->ncols + col, &bits);"),
    ("FSDP2 chunk read from the shard's start, not the parameter's",
     "int64_t o = L->param_offset[p] + (e - s * L->chunk_rows[p] * P->cols) * es;",
     "int64_t o = (e - s * L->chunk_rows[p] * P->cols) * es;"),
    ("flat byte read from the shard before", "*out = S->shards[s][f % L->shard_bytes];",
     "*out = S->shards[s > 0 ? s - 1 : 0][f % L->shard_bytes];"),
    ("checksum drops the last word", "for (int64_t k = 0; k + 8 <= n; k += 8) {",
     "for (int64_t k = 0; k + 16 <= n; k += 8) {"),
    ("bucket gaps and tail not zero", "memset(out, 0, (size_t)L->bucket_bytes);",
     "memset(out, 0xFF, (size_t)L->bucket_bytes);"),
    ("unpack reads big-endian elements",
     "out[j - j0] = (uint16_t)(bucket[o] | (bucket[o + 1] << 8));",
     "out[j - j0] = (uint16_t)(bucket[o + 1] | (bucket[o] << 8));"),
    ("verify reports the last bad bucket, not the first", "if (bad == 0) *first_bad = b;",
     "*first_bad = b;"),
    ("f16: NaN loses the quiet bit",
     "return (uint16_t)(sign | 0x7E00u | ((mag >> 13) & 0x01FFu));",
     "return (uint16_t)(sign | 0x7C00u | ((mag >> 13) & 0x01FFu));"),
    ("f16: rounding half up, not to even",
     "if (r > half || (r == half && (q & 1u))) q += 1;", "if (r >= half) q += 1;"),
    ("f16: overflow saturates to the largest finite",
     "h = bits >= 0x7C00 ? 0x7C00u : (uint32_t)bits;",
     "h = bits >= 0x7C00 ? 0x7BFFu : (uint32_t)bits;"),
    ("f16: subnormal spacing off by one", "h = (uint32_t)round_shift(sig, 126 - e);",
     "h = (uint32_t)round_shift(sig, 127 - e);"),
    ("f16: exponent bias off by one", "const int64_t bits = ((int64_t)(E + 14) << 10) + (int64_t)n;",
     "const int64_t bits = ((int64_t)(E + 15) << 10) + (int64_t)n;"),
    ("f16: bf16 source not widened",
     "if (dst_dtype == 1) return orc_rne_f16(elem_bytes == 4 ? bits : bits << 16);",
     "if (dst_dtype == 1) return orc_rne_f16(bits);"),
]


# (name, text in qwen3.py, replacement)
QWEN3_MUTATIONS = [
    ("qkv fused as [q; v; k]",
     'kv_slice(a + "k_proj.weight", r),\n                                              '
     'kv_slice(a + "v_proj.weight", r)]',
     'kv_slice(a + "v_proj.weight", r),\n                                              '
     'kv_slice(a + "k_proj.weight", r)]'),
    ("gate_up fused as [up; gate]",
     'row_slice(m + "gate_proj.weight", r),\n                                                      '
     'row_slice(m + "up_proj.weight", r)]',
     'row_slice(m + "up_proj.weight", r),\n                                                      '
     'row_slice(m + "gate_proj.weight", r)]'),
    ("w13 stacked as [up; gate]",
     'w13 += [row_slice(f"{ex}{e}.gate_proj.weight", r),\n                                '
     'row_slice(f"{ex}{e}.up_proj.weight", r)]',
     'w13 += [row_slice(f"{ex}{e}.up_proj.weight", r),\n                                '
     'row_slice(f"{ex}{e}.gate_proj.weight", r)]'),
    ("o_proj cut by rows", '[col_slice(a + "o_proj.weight", r)]',
     '[row_slice(a + "o_proj.weight", r)]'),
    ("expert down_proj cut by rows", 'w2.append(col_slice(f"{ex}{e}.down_proj.weight", r))',
     'w2.append(row_slice(f"{ex}{e}.down_proj.weight", r))'),
    ("column slices all start at column 0", "return (index[name], 0, rows, r * n, n)",
     "return (index[name], 0, rows, 0, n)"),
    ("row slices in reverse rank order", "return (index[name], r * n, n, 0, cols)",
     "return (index[name], (tp - 1 - r) * n, n, 0, cols)"),
    ("KV heads shared round-robin", "h = r * shape.n_kv // tp", "h = r % shape.n_kv"),
    ("experts dealt round-robin under EP", "for e in range(r * per, (r + 1) * per):",
     "for e in range(r, E, tp):"),
    ("layer i put in unit i, with the root", "out.append(layer + 1)", "out.append(layer)"),
    ("router registered after the experts",
     '            out.append((pre + "mlp.gate.weight", (E, H), elem_bytes))\n'
     '            for e in range(E):\n'
     '                ep = pre + f"mlp.experts.{e}."\n'
     '                out += [\n'
     '                    (ep + "gate_proj.weight", (Im, H), elem_bytes),\n'
     '                    (ep + "up_proj.weight", (Im, H), elem_bytes),\n'
     '                    (ep + "down_proj.weight", (H, Im), elem_bytes),\n'
     '                ]\n',
     '            for e in range(E):\n'
     '                ep = pre + f"mlp.experts.{e}."\n'
     '                out += [\n'
     '                    (ep + "gate_proj.weight", (Im, H), elem_bytes),\n'
     '                    (ep + "up_proj.weight", (Im, H), elem_bytes),\n'
     '                    (ep + "down_proj.weight", (H, Im), elem_bytes),\n'
     '                ]\n'
     '            out.append((pre + "mlp.gate.weight", (E, H), elem_bytes))\n'),
    ("down_proj registered before up_proj",
     '                (pre + "mlp.up_proj.weight", (I, H), elem_bytes),\n'
     '                (pre + "mlp.down_proj.weight", (H, I), elem_bytes),\n',
     '                (pre + "mlp.down_proj.weight", (H, I), elem_bytes),\n'
     '                (pre + "mlp.up_proj.weight", (I, H), elem_bytes),\n'),
    ("o_proj registered as [Q, hidden]", '(pre + "self_attn.o_proj.weight", (H, Q), elem_bytes)',
     '(pre + "self_attn.o_proj.weight", (Q, H), elem_bytes)'),
    ("tied models keep lm_head", "    if not shape.tied:\n        out.append",
     "    if True:\n        out.append"),
]

def battery():
    """A compact run of the pins.  Returns the name of the first that fails, or None."""
    checks = [
        ("golden numbers", layout_pins.test_golden_layout_numbers),
        ("golden values", layout_pins.test_golden_values),
        ("rows golden", layout_pins.test_rows_sharding_golden),
        ("cast named cases", cast_pins.test_named_cases),
        ("cast structured", cast_pins.test_structured_against_brute_force),
        ("cast NaN", cast_pins.test_nan_properties),
        ("f16 named cases", cast_pins.test_f16_named_cases),
        ("f16 ties", cast_pins.test_f16_ties_against_brute_force_and_numpy),
        ("f16 NaN", cast_pins.test_f16_nan_properties),
        ("f16 from bf16", cast_pins.test_f16_from_every_bfloat16_pattern),
        ("checksum", layout_pins.test_checksum_against_numpy_and_linearity),
        ("verify", layout_pins.test_verify_flags_damage),
        ("restatement tiny-tp4", lambda: layout_pins.test_oracle_matches_restatement("tiny-tp4")),
        ("restatement tiny-moe-tp2",
         lambda: layout_pins.test_oracle_matches_restatement("tiny-moe-tp2")),
        ("restatement tiny-fsdp2", lambda: layout_pins.test_oracle_matches_restatement("tiny-fsdp2")),
        ("restatement bf16 specials",
         lambda: layout_pins.test_oracle_matches_restatement("tiny-moe-bf16-specials")),
        ("shard size edge", layout_pins.test_shard_size_rule_edge),
        ("units golden", layout_pins.test_unit_sharding_worked_example),
        ("unit shard size edge", layout_pins.test_unit_shard_size_rule_edge),
        ("restatement tiny-units", lambda: layout_pins.test_oracle_matches_restatement("tiny-units")),
        ("restatement EP", lambda: layout_pins.test_oracle_matches_restatement("tiny-moe-ep4")),
        ("restatement KV replication",
         lambda: layout_pins.test_oracle_matches_restatement("tiny-moe-kvrep")),
        ("qwen3 golden", layout_pins.test_qwen3_layout_worked_example),
        ("round trip", lambda: layout_pins.test_unpack_of_pack_is_reshard("tiny-tp4")),
        ("shard invariance", lambda: layout_pins.test_shard_count_invariance(7, "flat")),
    ]
    for name, fn in checks:
        try:
            fn()
        except Exception:        # an assertion or an oracle error code
            return name
    return None


def _with_library(path):
    saved = oracle._lib
    oracle._lib = oracle.load(path)
    try:
        return battery()
    finally:
        oracle._lib = saved


def _with_qwen3(path):
    spec = importlib.util.spec_from_file_location("oracle_qwen3_mutant", path)
    mod = importlib.util.module_from_spec(spec)
    spec.loader.exec_module(mod)
    saved = oracle.qwen3
    oracle.qwen3 = mod
    try:
        return battery()
    finally:
        oracle.qwen3 = saved


def test_real_oracle_passes_the_battery():
    assert battery() is None


@pytest.mark.parametrize("name,old,new", MUTATIONS, ids=[m[0] for m in MUTATIONS])
def test_planted_mistake_is_caught(name, old, new, tmp_path):
    src = open(SRC).read()
    assert src.count(old) == 1, f"mutation site not found exactly once: {name}"
    mutant = tmp_path / "mutant.c"
    mutant.write_text(src.replace(old, new))
    so = tmp_path / "libmutant.so"
    subprocess.check_call(["gcc", "-O1", "-std=c11", "-fPIC", "-shared", "-o", str(so),
                           str(mutant)])
    failed = _with_library(str(so))
    assert failed is not None, f"no pin catches: {name}"


@pytest.mark.parametrize("name,old,new", QWEN3_MUTATIONS, ids=[m[0] for m in QWEN3_MUTATIONS])
def test_planted_layout_mistake_is_caught(name, old, new, tmp_path):
    src = open(QWEN3_SRC).read()
    assert src.count(old) == 1, f"mutation site not found exactly once: {name}"
    mutant = tmp_path / "qwen3_mutant.py"
    mutant.write_text(src.replace(old, new))
    failed = _with_qwen3(str(mutant))
    assert failed is not None, f"no pin catches: {name}"
