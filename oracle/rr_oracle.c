/*
 * CPU oracle for the trainer -> rollout weight-synchronisation hot path.
 *
 * TEST INFRASTRUCTURE ONLY.  Only the tests, the smoke check and the CPU
 * baseline / reference arm of the benchmark may load this file.  It shares no
 * code with the CUDA library and is written to be read against its definition,
 * not to be fast: single thread, scalar, one element at a time.
 *
 * What it computes (RobustRL, Section 5.2.1, the UCX-based weight update):
 *   (1) reshard: the trainer's parameters, held as flat FSDP-style shards, are
 *       re-laid into the rollout engine's layout (step 1 of that section);
 *   (2) the rollout holds 16-bit weights (Section 7.4 sizes the transferred
 *       model at two bytes per parameter); here the cast is float32 ->
 *       bfloat16, round-to-nearest-even;
 *   (3) the model is copied, one layer after another, into a transfer buffer
 *       (step 2);
 *       here that buffer is a sequence of fixed-size buckets;
 *   (4) each bucket carries a 64-bit word-sum so that a rollout that
 *       reconnects after a failure (Section 5.2.2, "Relay server failure
 *       during pulling", "Trainer failure during pulling") can check what it
 *       pulled;
 *   (5) unpack: buckets back to the rollout's tensors; (6) verify.
 *
 * The paper prints no layout, byte format or checksum; the definitions below
 * are the readings taken here, stated once:
 *
 *  Source, flat sharding (FSDP1-style).  Parameters are concatenated in
 *  manifest order into one flat byte buffer; each starts at a multiple of
 *  max(align_bytes, element size) (or at explicitly given offsets); gap bytes
 *  are zero.  The total is padded up to a multiple of 16 * n_shards (or a
 *  shard size S is given) and cut into n_shards equal shards of S bytes: flat
 *  byte f lives in shard f / S at offset f % S.
 *
 *  Source, row sharding (FSDP2 Shard(0), the torch.chunk rule).  Each
 *  parameter is cut on its first dimension: with c = ceil(rows / n_shards),
 *  shard s holds rows [s*c, min((s+1)*c, rows)) padded to c rows.  In every
 *  shard the parameters' chunks follow one another in manifest order, each
 *  starting at a multiple of max(align_bytes, element size); S is the end of
 *  the last chunk rounded up to 16.  Row r, column k of parameter p is in
 *  shard r / c at offset off_p + ((r - s*c) * cols + k) * element size.
 *
 *  Source, one buffer per parameter.  Parameter p is "shard" p, row-major
 *  from byte 0.
 *
 *  Source, unit sharding (FSDP1 wrapping modules separately, each with its
 *  own FlatParameter).  Every parameter belongs to one unit; a unit is laid
 *  out exactly like the flat source above but on its own: its parameters in
 *  manifest order from offset 0, each aligned, the total padded to a multiple
 *  of 16 * n_shards and cut into n_shards shards of S_u bytes.  The shard
 *  buffers are numbered unit by unit: shard s of unit u is buffer
 *  u * n_shards + s.
 *
 *  A parameter of shape [d0, d1, ...] is viewed as a matrix [rows = d0,
 *  cols = d1 * d2 * ...] (cols = 1 for a vector).  Generated values are
 *  indexed by the element's position in the flat layout whatever the
 *  sharding, so one seed gives the same parameters under every sharding.
 *
 *  Destination.  A destination tensor is a list of blocks (param, row0, nrows,
 *  col0, ncols); its elements are the blocks' elements taken block by block,
 *  each block row by row: element j of a block is the parameter element at
 *  row row0 + j / ncols, column col0 + j % ncols.
 *
 *  Cast.  float32 bits b -> bfloat16: a NaN (|b| > 0x7F800000) keeps its sign
 *  and top payload with the quiet bit forced, (b >> 16) | 0x0040; any other
 *  value rounds to nearest, ties to even: (b + 0x7FFF + ((b >> 16) & 1)) >> 16
 *  (so +-0 and subnormals are kept, overflow carries into +-inf and +-inf map
 *  to themselves).  A bfloat16 source is copied bit for bit.
 *
 *  Cast to float16 instead (the rollout's 16-bit weights as IEEE binary16;
 *  Section 7.4 calls the transferred model FP16).  A float32 value is rounded
 *  to the nearest binary16 value, ties to the even significand: binary16
 *  values are the multiples of 2^(E - 10) in the binade [2^E, 2^(E+1)) for
 *  E = -14 .. 15, and the multiples of 2^-24 below 2^-14 (subnormals, kept);
 *  a value that rounds to 2^16 or more is an infinity.  +-0 and +-inf map to
 *  themselves.  A NaN keeps its sign and its top payload bits with the quiet
 *  bit forced: sign | 0x7E00 | ((b >> 13) & 0x01FF), never an infinity.  A
 *  bfloat16 source is first widened exactly (its bits shifted up by 16) and
 *  then rounded the same way.
 *
 *  Stream and buckets.  Each rollout rank r has a byte stream holding its
 *  destination tensors in the given order, each starting at the next multiple
 *  of tensor_align; elements are little-endian.  The stream is cut every
 *  bucket_bytes; the last bucket and all alignment gaps are zero.  Buckets are
 *  numbered rank-major.
 *
 *  Checksum.  cs[b] = sum over k of the little-endian 64-bit word at bytes
 *  [8k, 8k + 8) of bucket b, modulo 2^64 (bucket_bytes % 8 == 0).
 */
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

typedef struct {
    int64_t rows;
    int64_t cols;
    int32_t elem_bytes; /* 4: float32, 2: bfloat16 */
    int32_t pad_;
} orc_param;

typedef struct {
    int32_t param;
    int32_t pad_;
    int64_t row0, nrows, col0, ncols;
} orc_block;

typedef struct {
    int32_t rank;
    int32_t n_blocks;
    const orc_block* blocks;
} orc_tensor;

typedef struct {
    /* description */
    int32_t n_params;
    int32_t n_shards;
    const orc_param* params;
    int64_t align_bytes;
    int32_t n_tensors;
    int32_t tp;
    const orc_tensor* tensors;
    int64_t tensor_align;
    int64_t bucket_bytes;
    /* derived by orc_layout_compute(), arrays owned by the caller */
    int64_t* param_offset;      /* [n_params] flat byte offset of each parameter   */
    int64_t* tensor_numel;      /* [n_tensors]                                      */
    int64_t* tensor_offset;     /* [n_tensors] byte offset in its rank's stream     */
    int64_t* rank_stream_bytes; /* [tp]                                             */
    int64_t* rank_first_bucket; /* [tp + 1]; rank_first_bucket[tp] = bucket count   */
    int64_t flat_bytes;         /* end of the last parameter (row sharding: of the
                                   last chunk within a shard)                      */
    int64_t shard_bytes;        /* S                                                */
    /* description, continued */
    int32_t sharding;           /* 0: flat, 1: rows, 2: one buffer per parameter     */
    int32_t pad_;
    int64_t shard_bytes_in;     /* flat: explicit S, or 0                           */
    const int64_t* explicit_offset; /* flat: explicit offsets, or NULL              */
    /* derived, continued */
    int64_t* chunk_rows;        /* [n_params] rows: c per parameter                 */
    int64_t* param_gen_base;    /* [n_params] flat element index of element 0       */
    /* description, continued: unit sharding (3) */
    int32_t n_units;
    int32_t pad2_;
    const int32_t* param_unit;  /* [n_params] unit of each parameter                */
    /* derived, continued */
    int64_t* unit_shard_bytes;  /* [n_units] S_u                                    */
    /* description, continued: destination element type */
    int32_t dst_dtype;          /* 0: bfloat16, 1: float16                          */
    int32_t pad3_;
} orc_layout;

/* Where source values come from: real shard buffers, or a generator that maps
 * an element index (flat byte offset / element size) to its bits. */
typedef uint32_t (*orc_value_fn)(const void* ctx, int64_t elem_index, int32_t elem_bytes);

typedef struct {
    const uint8_t* const* shards; /* n_shards host buffers of shard_bytes, or NULL */
    orc_value_fn gen;             /* used when shards == NULL                       */
    const void* gen_ctx;
} orc_source;

enum { ORC_OK = 0, ORC_EINVAL = -1, ORC_ENOMEM = -2, ORC_ESOURCE = -3 };

static int64_t align_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }

/* ---------------------------------------------------------------- layout */

int orc_layout_compute(orc_layout* L) {
    if (L->n_params < 0 || L->n_shards < 1 || L->align_bytes < 1 || L->tp < 1 ||
        L->n_tensors < 0 || L->tensor_align < 2 || L->tensor_align % 2 != 0 ||
        L->bucket_bytes < 8 || L->bucket_bytes % 8 != 0)
        return ORC_EINVAL;

    /* Source, flat layout first: parameters one after another, each aligned
     * (or at the given offsets).  Generated values are indexed by it. */
    int64_t off = 0, flat_end = 0;
    for (int32_t p = 0; p < L->n_params; ++p) {
        const orc_param* P = &L->params[p];
        if (P->rows < 0 || P->cols < 0 || (P->elem_bytes != 2 && P->elem_bytes != 4))
            return ORC_EINVAL;
        int64_t a = L->align_bytes > P->elem_bytes ? L->align_bytes : P->elem_bytes;
        int64_t start;
        if (L->explicit_offset) {
            start = L->explicit_offset[p];
            if (start < 0 || start % P->elem_bytes != 0) return ORC_EINVAL;
        } else {
            off = align_up(off, a);
            start = off;
            off += P->rows * P->cols * P->elem_bytes;
        }
        L->param_offset[p] = start;
        L->param_gen_base[p] = start / P->elem_bytes;
        int64_t end = start + P->rows * P->cols * P->elem_bytes;
        if (end > flat_end) flat_end = end;
    }
    if (L->sharding == 0) {
        L->flat_bytes = flat_end;
        L->shard_bytes = align_up(flat_end, 16 * (int64_t)L->n_shards) / L->n_shards;
        if (L->shard_bytes_in) {
            if (L->shard_bytes_in % 16 != 0 || L->shard_bytes_in * L->n_shards < flat_end)
                return ORC_EINVAL;
            L->shard_bytes = L->shard_bytes_in;
        }
    } else if (L->sharding == 3) {
        /* Units: every unit is a flat layout of its own parameters. */
        if (L->explicit_offset || L->shard_bytes_in || L->n_units < 1 || !L->param_unit)
            return ORC_EINVAL;
        int64_t biggest = 0, longest = 0;
        for (int32_t u = 0; u < L->n_units; ++u) {
            int64_t local = 0, members = 0;
            for (int32_t p = 0; p < L->n_params; ++p) {
                if (L->param_unit[p] != u) continue;
                const orc_param* P = &L->params[p];
                int64_t a = L->align_bytes > P->elem_bytes ? L->align_bytes : P->elem_bytes;
                local = align_up(local, a);
                L->param_offset[p] = local;
                local += P->rows * P->cols * P->elem_bytes;
                ++members;
            }
            if (members == 0) return ORC_EINVAL;
            L->unit_shard_bytes[u] = align_up(local, 16 * (int64_t)L->n_shards) / L->n_shards;
            if (L->unit_shard_bytes[u] > biggest) biggest = L->unit_shard_bytes[u];
            if (local > longest) longest = local;
        }
        for (int32_t p = 0; p < L->n_params; ++p)
            if (L->param_unit[p] < 0 || L->param_unit[p] >= L->n_units) return ORC_EINVAL;
        L->flat_bytes = longest;
        L->shard_bytes = biggest;
    } else if (L->sharding == 2) {
        /* One buffer per parameter. */
        if (L->explicit_offset || L->shard_bytes_in || L->n_shards != L->n_params)
            return ORC_EINVAL;
        int64_t biggest = 0;
        for (int32_t p = 0; p < L->n_params; ++p) {
            const orc_param* P = &L->params[p];
            int64_t bytes = P->rows * P->cols * P->elem_bytes;
            if (bytes > biggest) biggest = bytes;
        }
        L->flat_bytes = biggest;
        L->shard_bytes = biggest;
    } else {
        /* Row sharding: every shard holds each parameter's chunk of c rows. */
        if (L->explicit_offset || L->shard_bytes_in) return ORC_EINVAL;
        int64_t local = 0;
        for (int32_t p = 0; p < L->n_params; ++p) {
            const orc_param* P = &L->params[p];
            int64_t c = (P->rows + L->n_shards - 1) / L->n_shards;
            int64_t a = L->align_bytes > P->elem_bytes ? L->align_bytes : P->elem_bytes;
            local = align_up(local, a);
            L->chunk_rows[p] = c;
            L->param_offset[p] = local;
            local += c * P->cols * P->elem_bytes;
        }
        L->flat_bytes = local;
        L->shard_bytes = align_up(local, 16);
    }

    /* Destination: per-rank streams. */
    for (int32_t r = 0; r < L->tp; ++r) L->rank_stream_bytes[r] = 0;
    for (int32_t t = 0; t < L->n_tensors; ++t) {
        const orc_tensor* T = &L->tensors[t];
        if (T->rank < 0 || T->rank >= L->tp || T->n_blocks < 0) return ORC_EINVAL;
        int64_t numel = 0;
        for (int32_t k = 0; k < T->n_blocks; ++k) {
            const orc_block* B = &T->blocks[k];
            if (B->param < 0 || B->param >= L->n_params) return ORC_EINVAL;
            const orc_param* P = &L->params[B->param];
            if (B->row0 < 0 || B->nrows < 0 || B->row0 + B->nrows > P->rows) return ORC_EINVAL;
            if (B->col0 < 0 || B->ncols < 0 || B->col0 + B->ncols > P->cols) return ORC_EINVAL;
            numel += B->nrows * B->ncols;
        }
        int64_t start = align_up(L->rank_stream_bytes[T->rank], L->tensor_align);
        L->tensor_numel[t] = numel;
        L->tensor_offset[t] = start;
        L->rank_stream_bytes[T->rank] = start + 2 * numel;
    }
    L->rank_first_bucket[0] = 0;
    for (int32_t r = 0; r < L->tp; ++r) {
        int64_t nb = (L->rank_stream_bytes[r] + L->bucket_bytes - 1) / L->bucket_bytes;
        L->rank_first_bucket[r + 1] = L->rank_first_bucket[r] + nb;
    }
    return ORC_OK;
}

/* ------------------------------------------------------------------ cast */

uint16_t orc_rne_bf16(uint32_t b) {
    if ((b & 0x7FFFFFFFu) > 0x7F800000u) return (uint16_t)((b >> 16) | 0x0040u);
    return (uint16_t)((b + 0x7FFFu + ((b >> 16) & 1u)) >> 16);
}

void orc_rne_bf16_array(const uint32_t* in, uint16_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = orc_rne_bf16(in[i]);
}

/* Nearest integer to v / 2^sh, ties to even (sh >= 1). */
static uint64_t round_shift(uint64_t v, int32_t sh) {
    if (sh > 40) return 0; /* v < 2^24: below half of one unit */
    uint64_t q = v >> sh;
    uint64_t r = v - (q << sh);
    uint64_t half = 1ull << (sh - 1);
    if (r > half || (r == half && (q & 1u))) q += 1;
    return q;
}

uint16_t orc_rne_f16(uint32_t b) {
    const uint16_t sign = (uint16_t)((b >> 16) & 0x8000u);
    const uint32_t mag = b & 0x7FFFFFFFu;
    if (mag > 0x7F800000u) return (uint16_t)(sign | 0x7E00u | ((mag >> 13) & 0x01FFu));
    if (mag == 0x7F800000u) return (uint16_t)(sign | 0x7C00u);
    /* |x| = sig * 2^(e - 150), sig the significand with its leading bit */
    int32_t e = (int32_t)(mag >> 23);
    uint64_t sig = mag & 0x7FFFFFu;
    if (e == 0)
        e = 1; /* float32 subnormal */
    else
        sig |= 0x800000u;
    uint32_t h;
    if (mag >= 0x38800000u) {
        /* |x| >= 2^-14: the binade of |x| is 2^E with E = e - 127; binary16
         * spacing there is 2^(E - 10), so n = |x| / 2^(E - 10) = sig / 2^13,
         * an integer in [2^10, 2^11] after rounding.  The value n * 2^(E - 10)
         * is encoded as exponent field E + 15 and mantissa n - 2^10, i.e.
         * ((E + 14) << 10) + n; n = 2^11 carries into the next binade. */
        const int32_t E = e - 127;
        const uint64_t n = round_shift(sig, 13);
        const int64_t bits = ((int64_t)(E + 14) << 10) + (int64_t)n;
        h = bits >= 0x7C00 ? 0x7C00u : (uint32_t)bits;
    } else {
        /* |x| < 2^-14: the multiples of 2^-24; n = |x| / 2^-24 = sig * 2^(e - 126),
         * at most 2^10 (which is 2^-14, the smallest normal, encoded as n). */
        h = (uint32_t)round_shift(sig, 126 - e);
    }
    return (uint16_t)(sign | h);
}

void orc_rne_f16_array(const uint32_t* in, uint16_t* out, int64_t n) {
    for (int64_t i = 0; i < n; ++i) out[i] = orc_rne_f16(in[i]);
}

/* The 16-bit destination element for source bits of elem_bytes. */
static uint16_t cast_to_dst(uint32_t bits, int32_t elem_bytes, int32_t dst_dtype) {
    if (dst_dtype == 1) return orc_rne_f16(elem_bytes == 4 ? bits : bits << 16);
    return elem_bytes == 4 ? orc_rne_bf16(bits) : (uint16_t)bits;
}

/* ---------------------------------------------------------------- source */

static int source_byte(const orc_layout* L, const orc_source* S, int64_t f, uint8_t* out) {
    int64_t s = f / L->shard_bytes;
    if (s >= L->n_shards || S->shards[s] == NULL) return ORC_ESOURCE;
    *out = S->shards[s][f % L->shard_bytes];
    return ORC_OK;
}

/* Bits of element e (row-major) of parameter p (little-endian). */
static int source_bits(const orc_layout* L, const orc_source* S, int32_t p, int64_t e,
                       uint32_t* bits) {
    const orc_param* P = &L->params[p];
    const int32_t es = P->elem_bytes;
    if (S->shards == NULL) {
        *bits = S->gen(S->gen_ctx, L->param_gen_base[p] + e, es);
        return ORC_OK;
    }
    uint32_t v = 0;
    if (L->sharding == 0) {
        int64_t f = L->param_offset[p] + e * es;
        for (int32_t i = 0; i < es; ++i) {
            uint8_t byte;
            int rc = source_byte(L, S, f + i, &byte);
            if (rc) return rc;
            v |= (uint32_t)byte << (8 * i);
        }
    } else if (L->sharding == 2) {
        if (p >= L->n_shards || S->shards[p] == NULL) return ORC_ESOURCE;
        for (int32_t i = 0; i < es; ++i) v |= (uint32_t)S->shards[p][e * es + i] << (8 * i);
    } else if (L->sharding == 3) {
        const int32_t u = L->param_unit[p];
        const int64_t Su = L->unit_shard_bytes[u];
        for (int32_t i = 0; i < es; ++i) {
            int64_t f = L->param_offset[p] + e * es + i;   /* byte within the unit */
            int64_t buf = (int64_t)u * L->n_shards + f / Su;
            if (S->shards[buf] == NULL) return ORC_ESOURCE;
            v |= (uint32_t)S->shards[buf][f % Su] << (8 * i);
        }
    } else {
        int64_t row = e / P->cols;
        int64_t s = row / L->chunk_rows[p];
        int64_t o = L->param_offset[p] + (e - s * L->chunk_rows[p] * P->cols) * es;
        if (s >= L->n_shards || S->shards[s] == NULL) return ORC_ESOURCE;
        for (int32_t i = 0; i < es; ++i) v |= (uint32_t)S->shards[s][o + i] << (8 * i);
    }
    *bits = v;
    return ORC_OK;
}

/* ------------------------------------------------------------- reshard */

/* Elements j0 .. j1-1 of destination tensor t, cast to bfloat16. */
int orc_tensor_elements(const orc_layout* L, const orc_source* S, int32_t t, int64_t j0,
                        int64_t j1, uint16_t* out) {
    const orc_tensor* T = &L->tensors[t];
    int64_t base = 0; /* index in the tensor of the current block's first element */
    for (int32_t k = 0; k < T->n_blocks; ++k) {
        const orc_block* B = &T->blocks[k];
        const orc_param* P = &L->params[B->param];
        int64_t n = B->nrows * B->ncols;
        int64_t lo = j0 > base ? j0 : base;
        int64_t hi = j1 < base + n ? j1 : base + n;
        for (int64_t j = lo; j < hi; ++j) {
            int64_t jj = j - base;
            int64_t row = B->row0 + jj / B->ncols;
            int64_t col = B->col0 + jj % B->ncols;
            uint32_t bits;
            int rc = source_bits(L, S, B->param, row * P->cols + col, &bits);
            if (rc) return rc;
            out[j - j0] = cast_to_dst(bits, P->elem_bytes, L->dst_dtype);
        }
        base += n;
    }
    return ORC_OK;
}

/* The whole of destination tensor t, straight from the source (no buckets). */
int orc_reshard_tensor(const orc_layout* L, const orc_source* S, int32_t t, uint16_t* out) {
    return orc_tensor_elements(L, S, t, 0, L->tensor_numel[t], out);
}

/* ----------------------------------------------------------------- pack */

static int32_t rank_of_bucket(const orc_layout* L, int64_t b) {
    for (int32_t r = 0; r < L->tp; ++r)
        if (b < L->rank_first_bucket[r + 1]) return r;
    return -1;
}

/* Bucket b's bytes (bucket_bytes of them). */
int orc_pack_bucket(const orc_layout* L, const orc_source* S, int64_t b, uint8_t* out) {
    int32_t r = rank_of_bucket(L, b);
    if (b < 0 || r < 0) return ORC_EINVAL;
    int64_t lo = (b - L->rank_first_bucket[r]) * L->bucket_bytes;
    int64_t hi = lo + L->bucket_bytes;
    memset(out, 0, (size_t)L->bucket_bytes);
    for (int32_t t = 0; t < L->n_tensors; ++t) {
        if (L->tensors[t].rank != r) continue;
        int64_t t_lo = L->tensor_offset[t];
        int64_t t_hi = t_lo + 2 * L->tensor_numel[t];
        int64_t a = lo > t_lo ? lo : t_lo;
        int64_t z = hi < t_hi ? hi : t_hi;
        if (a >= z) continue;
        int64_t j0 = (a - t_lo) / 2, j1 = (z - t_lo) / 2;
        uint16_t* tmp = (uint16_t*)malloc((size_t)(j1 - j0) * 2);
        if (!tmp) return ORC_ENOMEM;
        int rc = orc_tensor_elements(L, S, t, j0, j1, tmp);
        if (rc) {
            free(tmp);
            return rc;
        }
        for (int64_t j = j0; j < j1; ++j) {
            int64_t pos = t_lo + 2 * j - lo;
            out[pos] = (uint8_t)(tmp[j - j0] & 0xFF);
            out[pos + 1] = (uint8_t)(tmp[j - j0] >> 8);
        }
        free(tmp);
    }
    return ORC_OK;
}

/* ------------------------------------------------------------- checksum */

uint64_t orc_checksum(const uint8_t* bytes, int64_t n) {
    uint64_t sum = 0;
    for (int64_t k = 0; k + 8 <= n; k += 8) {
        uint64_t word = 0;
        for (int i = 0; i < 8; ++i) word |= (uint64_t)bytes[k + i] << (8 * i);
        sum += word;
    }
    return sum;
}

/* Buckets first .. first+count-1 and their checksums, into out (count * bucket_bytes). */
int orc_pack_range(const orc_layout* L, const orc_source* S, int64_t first, int64_t count,
                   uint8_t* out, uint64_t* checksums) {
    for (int64_t i = 0; i < count; ++i) {
        uint8_t* bucket = out + i * L->bucket_bytes;
        int rc = orc_pack_bucket(L, S, first + i, bucket);
        if (rc) return rc;
        checksums[i] = orc_checksum(bucket, L->bucket_bytes);
    }
    return ORC_OK;
}

/* --------------------------------------------------------------- unpack */

/* Elements j0 .. j1-1 of destination tensor t read back out of the buckets
 * (buckets[b] = bucket b's bytes; buckets not needed may be NULL). */
int orc_unpack_elements(const orc_layout* L, const uint8_t* const* buckets, int32_t t,
                        int64_t j0, int64_t j1, uint16_t* out) {
    const orc_tensor* T = &L->tensors[t];
    int64_t first = L->rank_first_bucket[T->rank];
    for (int64_t j = j0; j < j1; ++j) {
        int64_t pos = L->tensor_offset[t] + 2 * j;
        const uint8_t* bucket = buckets[first + pos / L->bucket_bytes];
        if (bucket == NULL) return ORC_ESOURCE;
        int64_t o = pos % L->bucket_bytes;
        out[j - j0] = (uint16_t)(bucket[o] | (bucket[o + 1] << 8));
    }
    return ORC_OK;
}

/* The whole of destination tensor t read back out of the buckets. */
int orc_unpack_tensor(const orc_layout* L, const uint8_t* const* buckets, int32_t t,
                      uint16_t* out) {
    return orc_unpack_elements(L, buckets, t, 0, L->tensor_numel[t], out);
}

/* --------------------------------------------------------------- verify */

/* Number of buckets whose recomputed checksum differs from checksums[b]; the
 * first such index in *first_bad (-1 if none). */
int64_t orc_verify(const orc_layout* L, const uint8_t* const* buckets, const uint64_t* checksums,
                   int64_t first, int64_t count, int64_t* first_bad) {
    int64_t bad = 0;
    *first_bad = -1;
    for (int64_t b = first; b < first + count; ++b) {
        if (orc_checksum(buckets[b], L->bucket_bytes) != checksums[b]) {
            if (bad == 0) *first_bad = b;
            ++bad;
        }
    }
    return bad;
}
