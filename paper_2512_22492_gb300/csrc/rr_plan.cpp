// Host planner: compiles a manifest, a source shard layout, a destination
// (rollout) layout and a bucket size into the work tables that the pack and
// unpack kernels walk.
//
// RobustRL Section 5.2.1, step 1 (re-lay the trainer's weights out in the
// rollout's sharding) and step 2 (fill a transfer buffer with the model, one
// layer after another): the plan is that reshard expressed as a table of
// strided gathers, each landing in one fixed-size bucket.
//
// A work item never crosses a source shard, a bucket, or `chunk_bytes` of
// destination; items are emitted rank by rank in stream order, so the table
// is sorted by (bucket, offset).  Items whose addresses and lengths allow it
// are 16-byte vector items; the rest (ragged heads and tails, misaligned
// sources, odd row lengths) are scalar items.
//
// A second, whole-sync table serves a full-range pack on the bulk-copy
// engine: the same items, except that narrow column slices of the same
// parameter rows for several ranks (row-parallel weights under tensor
// parallelism) become fan-out groups that read each source row once.
#include <algorithm>
#include <climits>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <map>
#include <new>
#include <tuple>

#include "rr_internal.h"

namespace {

thread_local std::string g_error;

constexpr int64_t kDefaultChunkBytes = 64 * 1024;
// Balancing weights (build-time overridable for tuning sweeps).
#ifndef RR_ITEM_OVERHEAD
#define RR_ITEM_OVERHEAD 1024
#endif
#ifndef RR_ZERO_WEIGHT
#define RR_ZERO_WEIGHT 2
#endif
#ifndef RR_OWN_SHARE_PCT
#define RR_OWN_SHARE_PCT 85
#endif
#ifndef RR_TAPER
#define RR_TAPER 1
#endif
#ifndef RR_TAPER_FLOOR
#define RR_TAPER_FLOOR (64 * 1024)
#endif
#ifndef RR_FAN_HEAD_CHUNKS
#define RR_FAN_HEAD_CHUNKS 32
#endif
#ifndef RR_FAN_END_PCT
#define RR_FAN_END_PCT 80
#endif
constexpr int64_t kItemOverhead = RR_ITEM_OVERHEAD;   // balancing weight of one item, in bytes
constexpr int64_t kZeroWeight = RR_ZERO_WEIGHT;       // weight of one zero-filled element
constexpr int64_t kUnitWeight = 1 << 20;   // largest claimed work unit (weight), and the
constexpr int32_t kUnitsPerBlock = 32;     //   units wanted per block of the grid
constexpr int64_t kMaxShardOffset = (int64_t(1) << 48) - 1;
// Fan-out groups: at most kMaxFanDst column slices over a joint span of at
// most kFanMaxRowBytes of source per row (one pack stage of the bulk-copy
// engine holds a whole row; the kernel refuses a wider head).
constexpr int64_t kMaxFanDst = 16;
constexpr int64_t kFanMaxRowBytes = 48 * 1024;

int64_t align_up(int64_t x, int64_t a) { return (x + a - 1) / a * a; }
bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

// One member of a fan-out group: a column slice of the group's rows that lands
// contiguously in rank `rank`'s stream at byte `pos`.
struct FanSlice {
    int32_t rank;
    int64_t pos, col0, ncols;
};

class Builder {
public:
    explicit Builder(rr_plan* p) : P(p), chunk_elems(p->chunk_bytes / 2), out(&p->pack_items) {}

    // Pack items go to `o` from here on (the bucket-sorted table by default).
    void set_out(std::vector<rr_pack_item>* o) { out = o; }

    // ---- pack ------------------------------------------------------------

    // Where element e of parameter p lives: shard, byte offset in it, and how
    // many bytes from there on stay contiguous in that shard and in p.
    struct Loc {
        int64_t shard, off, room;
    };
    Loc loc(int32_t p, int64_t e) const {
        const int32_t es = P->es[p];
        if (P->sharding == RR_SHARD_FLAT) {
            const int64_t S = P->shard_bytes;
            const int64_t f = P->param_off[p] + e * es;
            return {f / S, f % S, S - f % S};
        }
        if (P->sharding == RR_SHARD_TENSORS)
            return {p, e * es, (P->rows[p] * P->cols[p] - e) * es};
        if (P->sharding == RR_SHARD_UNITS) {
            const int32_t u = P->unit_of[p];
            const int64_t S = P->unit_shard_bytes[u];
            const int64_t f = P->param_off[p] + e * es;
            return {int64_t(u) * P->unit_shards + f / S, f % S, S - f % S};
        }
        const int64_t cols = P->cols[p], c = P->chunk_rows[p];
        const int64_t sh = e / cols / c;
        const int64_t end = std::min((sh + 1) * c, P->rows[p]) * cols;   // p's last element in sh
        return {sh, P->param_off[p] + (e - sh * c * cols) * es, (end - e) * es};
    }

    // Emits the items of one strided run of parameter p: n rows of l elements,
    // row i starting at parameter element first + i * st, landing contiguously
    // in rank `rank`'s stream at byte `pos0`.
    void pack_run(int32_t p, int64_t first, int64_t l, int64_t n, int64_t st, int32_t rank,
                  int64_t pos0) {
        if (l == 0 || n == 0) return;
        const int32_t es = P->es[p];
        const int64_t B = P->bucket_bytes;
        const int64_t fb = P->rank_first_bucket[rank];
        int64_t i = 0, c = 0;
        while (i < n) {
            const int64_t pos = pos0 + 2 * (i * l + c);
            const int64_t bl = pos / B, boff = pos - bl * B;
            const int64_t brem = (B - boff) / 2;                      // elements left in bucket
            const Loc at = loc(p, first + i * st + c);
            const int64_t sh = at.shard, soff = at.off;
            const int64_t srem = at.room / es;                        // elements left in shard
            if (c == 0 && n - i > 1 && l <= chunk_elems) {
                int64_t k = std::min({n - i, chunk_elems / l, brem / l});
                const int64_t room = at.room;
                const int64_t kshard = room >= l * es ? (room - l * es) / (st * es) + 1 : 0;
                k = std::min(k, kshard);
                if (k >= 2) {
                    pack_rows(es, sh, soff, fb + bl, boff, l, k, st);
                    i += k;
                    continue;
                }
            }
            const int64_t len = std::min({l - c, chunk_elems, brem, srem});
            pack_piece(es, sh, soff, fb + bl, boff, len);
            c += len;
            if (c == l) {
                c = 0;
                ++i;
            }
        }
    }

    // Zero fill of stream bytes [a, b) of rank `rank` (alignment gaps, last bucket's tail).
    void zero_range(int32_t rank, int64_t a, int64_t b) {
        const int64_t B = P->bucket_bytes;
        const int64_t fb = P->rank_first_bucket[rank];
        while (a < b) {
            const int64_t bl = a / B, boff = a - bl * B;
            const int64_t len = std::min({(b - a) / 2, (B - boff) / 2, chunk_elems});
            split3(RR_ITEM_ZERO_VEC, RR_ITEM_ZERO_SCALAR, 2, 0, 0, fb + bl, boff, len, true);
            a += 2 * len;
        }
    }

    // ---- unpack ----------------------------------------------------------

    void unpack_tensor(int32_t t) {
        const int64_t B = P->bucket_bytes;
        const int64_t fb = P->rank_first_bucket[P->tensor_rank[t]];
        const int64_t nbytes = 2 * P->tensor_numel[t];
        int64_t x = 0;
        while (x < nbytes) {
            const int64_t pos = P->tensor_off[t] + x;
            const int64_t bl = pos / B, boff = pos - bl * B;
            int64_t len = std::min({nbytes - x, B - boff, P->chunk_bytes});
            copy_piece(fb + bl, boff, t, x, len);
            x += len;
        }
    }

    // Stream bytes [a, b) of rank `rank` that belong to no tensor: read (and
    // checksummed) only by the verifying unpack.
    void read_gap(int32_t rank, int64_t a, int64_t b) {
        const int64_t B = P->bucket_bytes;
        const int64_t fb = P->rank_first_bucket[rank];
        while (a < b) {
            const int64_t bl = a / B;
            int64_t boff = a - bl * B;
            int64_t len = std::min({b - a, B - boff, P->chunk_bytes});
            int64_t h = std::min((16 - boff % 16) % 16, len);
            if (h) {
                emit_copy(RR_ITEM_READ_SCALAR, fb + bl, boff, -1, 0, h);
                boff += h;
                a += h;
                len -= h;
            }
            const int64_t body = len / 16 * 16;
            if (body) {
                emit_copy(RR_ITEM_READ_VEC, fb + bl, boff, -1, 0, body);
                boff += body;
                a += body;
                len -= body;
            }
            if (len) {
                emit_copy(RR_ITEM_READ_SCALAR, fb + bl, boff, -1, 0, len);
                a += len;
            }
        }
    }

    // Rows [row0, row0 + nrows) of parameter p, columns [cmin, cmin + span),
    // are cut into column slices m (sorted, adjacent) for several ranks: one
    // fan-out head per run of rows that stays in one shard and keeps every
    // slice inside one bucket, followed by one destination item per slice.
    // Rows that straddle a shard or put a slice across a bucket boundary go
    // out as plain items.
    void fan_group(int32_t p, int64_t row0, int64_t nrows, int64_t cmin, int64_t span,
                   const std::vector<FanSlice>& m) {
        const int32_t es = P->es[p];
        const int64_t C = P->cols[p], B = P->bucket_bytes;
        // Heads are cut into stage-sized pieces by the kernel; this only bounds
        // the balancing granularity (RR_FAN_HEAD_CHUNKS chunks of source per head).
        const int64_t max_rows =
            std::max<int64_t>(1, RR_FAN_HEAD_CHUNKS * P->chunk_bytes / (span * es));
        int64_t i = 0;
        while (i < nrows) {
            const Loc at = loc(p, (row0 + i) * C + cmin);
            int64_t k = 0;
            if (at.room >= span * es && at.off % 16 == 0) {
                k = std::min({nrows - i, (at.room - span * es) / (C * es) + 1, max_rows});
                for (const FanSlice& s : m) {
                    const int64_t boff = (s.pos + 2 * i * s.ncols) % B;
                    k = std::min(k, (B - boff) / (2 * s.ncols));
                }
            }
            if (k < 1) {
                for (const FanSlice& s : m)
                    pack_run(p, (row0 + i) * C + s.col0, s.ncols, 1, C, s.rank,
                             s.pos + 2 * i * s.ncols);
                ++i;
                continue;
            }
            const int64_t fb0 = P->rank_first_bucket[m[0].rank];
            rr_pack_item h;
            h.src = (uint64_t(at.shard) << 48) | uint64_t(at.off);
            h.dst_off = uint32_t(m.size());
            h.bucket = uint32_t(fb0 + (m[0].pos + 2 * i * m[0].ncols) / B);
            h.row_len = uint32_t(span);
            h.n_rows = uint32_t(k);
            h.src_stride = uint32_t(C);
            h.kind = uint16_t(es == 4 ? RR_ITEM_FAN_F32 : RR_ITEM_FAN_BF16);
            h.reserved = 0;
            out->push_back(h);
            for (const FanSlice& s : m) {
                const int64_t at_pos = s.pos + 2 * i * s.ncols;
                rr_pack_item d;
                d.src = uint64_t(s.col0 - cmin);
                d.dst_off = uint32_t(at_pos % B);
                d.bucket = uint32_t(P->rank_first_bucket[s.rank] + at_pos / B);
                d.row_len = uint32_t(s.ncols);
                d.n_rows = uint32_t(k);
                d.src_stride = 0;
                d.kind = uint16_t(RR_ITEM_FAN_DST);
                d.reserved = 0;
                out->push_back(d);
            }
            i += k;
        }
    }

    int64_t pack_read = 0;

private:
    rr_plan* P;
    int64_t chunk_elems;
    std::vector<rr_pack_item>* out;

    void emit_pack(int kind, int64_t shard, int64_t soff, int64_t bucket, int64_t boff,
                   int64_t row_len, int64_t n_rows, int64_t stride) {
        rr_pack_item it;
        it.src = (uint64_t(shard) << 48) | uint64_t(soff);
        it.dst_off = uint32_t(boff);
        it.bucket = uint32_t(bucket);
        it.row_len = uint32_t(row_len);
        it.n_rows = uint32_t(n_rows);
        it.src_stride = uint32_t(stride);
        it.kind = uint16_t(kind);
        it.reserved = 0;
        out->push_back(it);
        if (kind <= RR_ITEM_BF16_SCALAR && out == &P->pack_items)
            pack_read += row_len * n_rows * (kind <= RR_ITEM_F32_SCALAR ? 4 : 2);
    }

    // One row piece: scalar head up to 16-byte destination alignment, vector
    // body when the source is then 16-byte aligned too, scalar tail.
    void split3(int vec_kind, int sc_kind, int32_t es, int64_t shard, int64_t soff,
                int64_t bucket, int64_t boff, int64_t len, bool src_free) {
        int64_t h = ((16 - boff % 16) % 16) / 2;
        h = std::min(h, len);
        if (h) {
            emit_pack(sc_kind, shard, soff, bucket, boff, h, 1, h);
            soff += h * es;
            boff += 2 * h;
            len -= h;
        }
        const int64_t body = len / 8 * 8;
        if (body && (src_free || soff % 16 == 0)) {
            emit_pack(vec_kind, shard, soff, bucket, boff, body, 1, body);
            soff += body * es;
            boff += 2 * body;
            len -= body;
        }
        if (len) emit_pack(sc_kind, shard, soff, bucket, boff, len, 1, len);
    }

    void pack_piece(int32_t es, int64_t shard, int64_t soff, int64_t bucket, int64_t boff,
                    int64_t len) {
        if (es == 4)
            split3(RR_ITEM_F32_VEC, RR_ITEM_F32_SCALAR, 4, shard, soff, bucket, boff, len, false);
        else
            split3(RR_ITEM_BF16_VEC, RR_ITEM_BF16_SCALAR, 2, shard, soff, bucket, boff, len,
                   false);
    }

    void pack_rows(int32_t es, int64_t shard, int64_t soff, int64_t bucket, int64_t boff,
                   int64_t l, int64_t k, int64_t st) {
        const bool vec = boff % 16 == 0 && l % 8 == 0 && soff % 16 == 0 && (st * es) % 16 == 0;
        const int kind = es == 4 ? (vec ? RR_ITEM_F32_VEC : RR_ITEM_F32_SCALAR)
                                 : (vec ? RR_ITEM_BF16_VEC : RR_ITEM_BF16_SCALAR);
        emit_pack(kind, shard, soff, bucket, boff, l, k, st);
    }

    void emit_copy(int kind, int64_t bucket, int64_t boff, int32_t t, int64_t x, int64_t len) {
        rr_unpack_item it;
        it.dst_off = uint64_t(x);
        it.src_off = uint32_t(boff);
        it.bucket = uint32_t(bucket);
        it.tensor = uint32_t(t);
        it.nbytes = uint32_t(len);
        it.kind = uint32_t(kind);
        it.reserved = 0;
        P->unpack_items.push_back(it);
    }

    void copy_piece(int64_t bucket, int64_t boff, int32_t t, int64_t x, int64_t len) {
        if ((boff - x) % 16 != 0) {   // source and destination phases differ
            emit_copy(RR_ITEM_COPY_SCALAR, bucket, boff, t, x, len);
            return;
        }
        int64_t h = std::min((16 - boff % 16) % 16, len);
        if (h) {
            emit_copy(RR_ITEM_COPY_SCALAR, bucket, boff, t, x, h);
            boff += h;
            x += h;
            len -= h;
        }
        const int64_t body = len / 16 * 16;
        if (body) {
            emit_copy(RR_ITEM_COPY_VEC, bucket, boff, t, x, body);
            boff += body;
            x += body;
            len -= body;
        }
        if (len) emit_copy(RR_ITEM_COPY_SCALAR, bucket, boff, t, x, len);
    }
};

int64_t pack_weight(const rr_pack_item& it) {
    const int64_t n = int64_t(it.row_len) * it.n_rows;
    switch (it.kind) {
        case RR_ITEM_F32_VEC: return 6 * n + kItemOverhead;
        case RR_ITEM_F32_SCALAR: return 12 * n + kItemOverhead;
        case RR_ITEM_BF16_VEC: return 4 * n + kItemOverhead;
        case RR_ITEM_BF16_SCALAR: return 8 * n + kItemOverhead;
        case RR_ITEM_FAN_F32: return 6 * n + kItemOverhead;
        case RR_ITEM_FAN_BF16: return 4 * n + kItemOverhead;
        case RR_ITEM_FAN_DST: return 0;
        default: return kZeroWeight * n + kItemOverhead;
    }
}

int64_t unpack_weight(const rr_unpack_item& it) {
    switch (it.kind) {
        case RR_ITEM_COPY_VEC: return 2 * int64_t(it.nbytes) + kItemOverhead;
        case RR_ITEM_COPY_SCALAR: return 4 * int64_t(it.nbytes) + kItemOverhead;
        default: return int64_t(it.nbytes) + kItemOverhead;
    }
}

// Cuts items [0, n) into `grid` contiguous ranges of roughly equal weight.
template <class Item, class W>
void partition(const std::vector<Item>& items, int32_t grid, std::vector<uint32_t>& first, W w) {
    first.assign(size_t(grid) + 1, uint32_t(items.size()));
    first[0] = 0;
    int64_t total = 0;
    for (const Item& it : items) total += w(it);
    int64_t cum = 0;
    int32_t g = 1;
    for (size_t i = 0; i < items.size() && g < grid; ++i) {
        cum += w(items[i]);
        while (g < grid && cum * grid >= total * g) first[g++] = uint32_t(i + 1);
    }
}

// Claimed units get smaller toward the end of the table (guided
// self-scheduling): a unit that starts with `rem` weight left before the end is
// about rem / (2 * grid), clamped to [floor, unit_weight].  Blocks drain HBM at
// unequal rates and stop within one unit of one another; with the last units
// small, they stop together.
int64_t taper_size(int64_t rem, int64_t unit_weight, int32_t grid) {
    if (!RR_TAPER) return unit_weight;
    const int64_t floor = std::min<int64_t>(unit_weight, RR_TAPER_FLOOR);
    return std::max(floor, std::min(unit_weight, rem / (2 * int64_t(std::max(1, grid)))));
}

// Work units for a kernel whose blocks claim work as they run out of it.  Each
// bucket's items are cut into units (a unit never spans two buckets, so a
// bucket-range call takes a contiguous run of units) of about taper_size of
// the weight left to the table's end: first[u] is the first item of unit u,
// bucket_unit[b] the first unit of bucket b.  Small units claimed one at a
// time let the fast blocks take more of them, and all finish together.  Within
// a bucket a cut falls after the item that reaches the unit's size, unless
// less than a quarter unit would be left in the bucket; no unit is empty.
template <class Item, class W>
void bucket_units(const std::vector<Item>& items, const std::vector<uint32_t>& bucket_first,
                  int64_t unit_weight, int32_t grid, std::vector<uint32_t>& first,
                  std::vector<uint32_t>& bucket_unit, W w) {
    first.clear();
    bucket_unit.assign(bucket_first.size(), 0);
    int64_t rem = 0;   // weight from the current item to the end of the table
    for (const Item& it : items) rem += w(it);
    for (size_t b = 0; b + 1 < bucket_first.size(); ++b) {
        bucket_unit[b] = uint32_t(first.size());
        const uint32_t lo = bucket_first[b], hi = bucket_first[b + 1];
        if (lo == hi) continue;
        int64_t left = 0;   // weight left in this bucket
        for (uint32_t i = lo; i < hi; ++i) left += w(items[i]);
        uint32_t i = lo;
        while (i < hi) {
            first.push_back(i);
            const int64_t size = taper_size(rem, unit_weight, grid);
            int64_t cum = 0;
            while (i < hi) {
                const int64_t wi = w(items[i++]);
                cum += wi;
                rem -= wi;
                left -= wi;
                if (cum >= size && left * 4 >= size) break;
            }
        }
    }
    bucket_unit.back() = uint32_t(first.size());
    first.push_back(bucket_first.empty() ? 0 : bucket_first.back());
}

// Units for a launch over every bucket (the table it runs is fixed): blocks
// first drain kOwnShare of the table's weight in equal contiguous shares (unit
// g < grid is block g's own: no claims, long runs), then claim units of
// taper_size over the rest.  Own units may be empty.  A cut never falls before
// a fan-out destination item (a head and its destinations stay in one unit).
constexpr int64_t kOwnShareNum = RR_OWN_SHARE_PCT, kOwnShareDen = 100;
template <class Item, class W>
void whole_units(const std::vector<Item>& items, int32_t grid, int64_t unit_weight,
                 std::vector<uint32_t>& first, W w) {
    int64_t total = 0;
    for (const Item& it : items) total += w(it);
    const int64_t own = total * kOwnShareNum / kOwnShareDen;
    first.assign(size_t(grid) + 1, uint32_t(items.size()));
    first[0] = 0;
    int64_t cum = 0;
    size_t i = 0;
    // Own shares: the cut before unit g at the first item boundary reaching own * g / grid.
    for (int64_t g = 1; g <= grid; ++g) {
        while (i < items.size() &&
               (cum < own * g / grid || (i < items.size() && items[i].kind == RR_ITEM_FAN_DST)))
            cum += w(items[i++]);
        first[size_t(g)] = uint32_t(i);
    }
    // Claimed units over the rest, smaller toward the end.
    while (i < items.size()) {
        const int64_t size = taper_size(total - cum, unit_weight, grid);
        int64_t u = 0;
        while (i < items.size() && (u < size || items[i].kind == RR_ITEM_FAN_DST)) {
            const int64_t wi = w(items[i++]);
            u += wi;
            cum += wi;
        }
        first.push_back(uint32_t(i));
    }
    if (first.size() == size_t(grid) + 1) first.push_back(uint32_t(items.size()));
}

// Claimed-unit weight for a table: about kUnitsPerBlock units per block of the
// grid, none above kUnitWeight (small enough to even out the finish), none
// below kUnitWeight / 8 (each costs the producer one claim).
template <class Item, class W>
int64_t unit_weight_for(const std::vector<Item>& items, int32_t grid, W w) {
    int64_t total = 0;
    for (const Item& it : items) total += w(it);
    const int64_t per_block = total / (int64_t(kUnitsPerBlock) * std::max(1, grid));
    return std::min(kUnitWeight, std::max(kUnitWeight / 8, per_block));
}

rr_status validate_and_describe(rr_plan* P, const rr_param* manifest, int32_t n_params,
                                const rr_src_layout* src, const rr_dst_layout* dst,
                                size_t bucket_bytes) {
    if (n_params < 0 || (n_params > 0 && !manifest) || !src || !dst)
        return rr_fail(RR_EINVAL, "null manifest / layout pointer or negative n_params");
    if (bucket_bytes < 8 || bucket_bytes % 8 != 0 || bucket_bytes > (size_t(1) << 32) - 16)
        return rr_fail(RR_EINVAL, "bucket_bytes must be a multiple of 8 in [8, 2^32 - 16]");
    if (src->n_shards < 1 || src->n_shards > 65535)
        return rr_fail(RR_EINVAL, "n_shards must be in [1, 65535]");
    if (src->align_bytes < 1) return rr_fail(RR_EINVAL, "align_bytes must be >= 1");
    if (dst->tp < 1) return rr_fail(RR_EINVAL, "tp must be >= 1");
    if (dst->n_tensors < 0 || (dst->n_tensors > 0 && !dst->tensors))
        return rr_fail(RR_EINVAL, "bad destination tensor list");
    if (!is_pow2(dst->tensor_align_bytes) || dst->tensor_align_bytes < 2)
        return rr_fail(RR_EINVAL, "tensor_align_bytes must be a power of two >= 2");
    if (dst->dtype != RR_DST_BF16 && dst->dtype != RR_DST_F16)
        return rr_fail(RR_EINVAL, "unknown destination dtype %d", dst->dtype);

    P->n_params = n_params;
    P->rows.resize(n_params);
    P->cols.resize(n_params);
    P->es.resize(n_params);
    P->param_off.resize(n_params);
    for (int32_t p = 0; p < n_params; ++p) {
        const rr_param& m = manifest[p];
        if (m.ndim < 0 || m.ndim > 4) return rr_fail(RR_EINVAL, "param %d: ndim %d", p, m.ndim);
        if (m.dtype != RR_F32 && m.dtype != RR_BF16)
            return rr_fail(RR_EINVAL, "param %d: bad dtype", p);
        int64_t rows = m.ndim ? m.shape[0] : 1, cols = 1;
        for (int32_t d = 0; d < m.ndim; ++d)
            if (m.shape[d] < 0) return rr_fail(RR_EINVAL, "param %d: negative dim", p);
        for (int32_t d = 1; d < m.ndim; ++d) cols *= m.shape[d];
        if (cols > 0xFFFFFFFFll) return rr_fail(RR_ELAYOUT, "param %d: row too long", p);
        P->rows[p] = rows;
        P->cols[p] = cols;
        P->es[p] = m.dtype == RR_F32 ? 4 : 2;
    }

    // Source offsets.
    int64_t end = 0;
    if (src->sharding != RR_SHARD_FLAT && src->sharding != RR_SHARD_ROWS &&
        src->sharding != RR_SHARD_TENSORS && src->sharding != RR_SHARD_UNITS)
        return rr_fail(RR_EINVAL, "unknown sharding %d", src->sharding);
    if (src->sharding != RR_SHARD_UNITS && (src->n_units || src->param_unit))
        return rr_fail(RR_EINVAL, "units are given only with RR_SHARD_UNITS");
    P->sharding = src->sharding;
    if (src->sharding == RR_SHARD_UNITS) {
        if (src->param_flat_offset || src->shard_bytes)
            return rr_fail(RR_EINVAL, "unit sharding takes no explicit offsets or shard size");
        const int32_t U = src->n_units;
        if (U < 1 || !src->param_unit)
            return rr_fail(RR_EINVAL, "unit sharding needs n_units >= 1 and param_unit");
        if (int64_t(U) * src->n_shards > 65535)
            return rr_fail(RR_EINVAL, "n_units * n_shards must be at most 65535");
        P->unit_shards = src->n_shards;
        P->unit_of.assign(src->param_unit, src->param_unit + n_params);
        std::vector<int64_t> uend(U, 0);
        std::vector<char> used(U, 0);
        for (int32_t p = 0; p < n_params; ++p) {   // manifest order within each unit
            const int32_t u = P->unit_of[p];
            if (u < 0 || u >= U) return rr_fail(RR_EINVAL, "param %d: unit %d out of range", p, u);
            used[u] = 1;
            uend[u] = align_up(uend[u], std::max<int64_t>(src->align_bytes, P->es[p]));
            P->param_off[p] = uend[u];
            uend[u] += P->rows[p] * P->cols[p] * P->es[p];
        }
        P->unit_shard_bytes.resize(U);
        for (int32_t u = 0; u < U; ++u) {
            if (!used[u]) return rr_fail(RR_EINVAL, "unit %d holds no parameter", u);
            P->unit_shard_bytes[u] = align_up(uend[u], 16 * int64_t(src->n_shards)) / src->n_shards;
            end = std::max(end, uend[u]);
            P->shard_bytes = std::max(P->shard_bytes, P->unit_shard_bytes[u]);
        }
        P->flat_bytes = end;
        P->n_shards = U * src->n_shards;
    } else if (src->sharding == RR_SHARD_TENSORS) {
        if (src->param_flat_offset || src->shard_bytes)
            return rr_fail(RR_EINVAL, "per-tensor sources take no explicit offsets or shard size");
        if (src->n_shards != n_params)
            return rr_fail(RR_EINVAL, "per-tensor sources need n_shards (%d) == n_params (%d)",
                           src->n_shards, n_params);
        for (int32_t p = 0; p < n_params; ++p) {
            P->param_off[p] = 0;
            end = std::max(end, P->rows[p] * P->cols[p] * P->es[p]);
        }
        P->flat_bytes = end;
        P->n_shards = src->n_shards;
        P->shard_bytes = end;   // the largest parameter
    } else if (src->sharding == RR_SHARD_ROWS) {
        if (src->param_flat_offset || src->shard_bytes)
            return rr_fail(RR_EINVAL, "row sharding takes no explicit offsets or shard size");
        P->chunk_rows.resize(n_params);
        for (int32_t p = 0; p < n_params; ++p) {
            const int64_t c = (P->rows[p] + src->n_shards - 1) / src->n_shards;
            P->chunk_rows[p] = c;
            end = align_up(end, std::max<int64_t>(src->align_bytes, P->es[p]));
            P->param_off[p] = end;
            end += c * P->cols[p] * P->es[p];
        }
        P->flat_bytes = end;
        P->n_shards = src->n_shards;
        P->shard_bytes = align_up(end, 16);
    } else if (src->param_flat_offset) {
        std::vector<std::pair<int64_t, int64_t>> spans;
        for (int32_t p = 0; p < n_params; ++p) {
            const int64_t o = src->param_flat_offset[p];
            const int64_t sz = P->rows[p] * P->cols[p] * P->es[p];
            if (o < 0 || o % P->es[p] != 0)
                return rr_fail(RR_ELAYOUT, "param %d: flat offset %lld not a multiple of %d", p,
                               (long long)o, P->es[p]);
            P->param_off[p] = o;
            if (sz) spans.emplace_back(o, o + sz);
            end = std::max(end, o + sz);
        }
        std::sort(spans.begin(), spans.end());
        for (size_t i = 1; i < spans.size(); ++i)
            if (spans[i].first < spans[i - 1].second)
                return rr_fail(RR_ELAYOUT, "explicit parameter offsets overlap");
    } else {
        for (int32_t p = 0; p < n_params; ++p) {
            end = align_up(end, std::max<int64_t>(src->align_bytes, P->es[p]));
            P->param_off[p] = end;
            end += P->rows[p] * P->cols[p] * P->es[p];
        }
    }
    if (src->sharding == RR_SHARD_FLAT) {
        P->flat_bytes = end;
        P->n_shards = src->n_shards;
        P->shard_bytes = align_up(end, 16 * int64_t(src->n_shards)) / src->n_shards;
        if (src->shard_bytes) {
            if (src->shard_bytes % 16 != 0 || src->shard_bytes * src->n_shards < end)
                return rr_fail(RR_ELAYOUT,
                               "shard_bytes %lld: not a multiple of 16, or %d shards of it do "
                               "not cover the %lld bytes of parameters",
                               (long long)src->shard_bytes, src->n_shards, (long long)end);
            P->shard_bytes = src->shard_bytes;
        }
    }
    if (P->shard_bytes > kMaxShardOffset) return rr_fail(RR_ELAYOUT, "shards too large");

    // Destination streams.
    P->dst_f16 = dst->dtype == RR_DST_F16 ? 1 : 0;
    P->tp = dst->tp;
    P->n_tensors = dst->n_tensors;
    P->tensor_align = dst->tensor_align_bytes;
    P->bucket_bytes = int64_t(bucket_bytes);
    P->tensor_rank.resize(dst->n_tensors);
    P->tensor_numel.resize(dst->n_tensors);
    P->tensor_off.resize(dst->n_tensors);
    P->rank_stream_bytes.assign(dst->tp, 0);
    for (int32_t t = 0; t < dst->n_tensors; ++t) {
        const rr_dst_tensor& T = dst->tensors[t];
        if (T.rank < 0 || T.rank >= dst->tp)
            return rr_fail(RR_ELAYOUT, "tensor %d: rank %d outside [0, %d)", t, T.rank, dst->tp);
        if (T.n_blocks < 0 || (T.n_blocks > 0 && !T.blocks))
            return rr_fail(RR_EINVAL, "tensor %d: bad block list", t);
        int64_t numel = 0;
        for (int32_t k = 0; k < T.n_blocks; ++k) {
            const rr_block& b = T.blocks[k];
            if (b.param < 0 || b.param >= n_params)
                return rr_fail(RR_ELAYOUT, "tensor %d block %d: param %d out of range", t, k,
                               b.param);
            const int64_t R = P->rows[b.param], C = P->cols[b.param];
            if (b.row0 < 0 || b.nrows < 0 || b.row0 + b.nrows > R || b.col0 < 0 || b.ncols < 0 ||
                b.col0 + b.ncols > C)
                return rr_fail(RR_ELAYOUT,
                               "tensor %d block %d: rows [%lld,+%lld) cols [%lld,+%lld) outside "
                               "param %d's [%lld, %lld]",
                               t, k, (long long)b.row0, (long long)b.nrows, (long long)b.col0,
                               (long long)b.ncols, b.param, (long long)R, (long long)C);
            numel += b.nrows * b.ncols;
        }
        if (T.numel != numel)
            return rr_fail(RR_ELAYOUT, "tensor %d: numel %lld but blocks cover %lld", t,
                           (long long)T.numel, (long long)numel);
        const int64_t start = align_up(P->rank_stream_bytes[T.rank], P->tensor_align);
        P->tensor_rank[t] = T.rank;
        P->tensor_numel[t] = numel;
        P->tensor_off[t] = start;
        P->rank_stream_bytes[T.rank] = start + 2 * numel;
    }
    P->rank_first_bucket.assign(size_t(dst->tp) + 1, 0);
    int64_t nb = 0;
    for (int32_t r = 0; r < dst->tp; ++r) {
        nb += (P->rank_stream_bytes[r] + P->bucket_bytes - 1) / P->bucket_bytes;
        if (nb > 0x7FFFFFFF) return rr_fail(RR_ELAYOUT, "too many buckets");
        P->rank_first_bucket[r + 1] = int32_t(nb);
    }
    P->n_buckets = int32_t(nb);
    return RR_OK;
}

// Fan-out groups: blocks of the same parameter rows whose column slices are
// narrow, 16-byte aligned, and tile one contiguous span.  Returns, per group,
// its slices; marks each member block in `member` ([tensor][block] -> group).
struct FanGroup {
    int32_t param;
    int64_t row0, nrows, cmin, span;
    std::vector<FanSlice> slices;
};

std::vector<FanGroup> find_fan_groups(const rr_plan* P, const rr_dst_layout* dst,
                                      std::vector<std::vector<int32_t>>& member) {
    std::map<std::tuple<int32_t, int64_t, int64_t>, std::vector<std::pair<int32_t, int32_t>>> by;
    member.assign(size_t(P->n_tensors), {});
    for (int32_t t = 0; t < P->n_tensors; ++t) {
        const rr_dst_tensor& T = dst->tensors[t];
        member[t].assign(size_t(T.n_blocks), -1);
        for (int32_t k = 0; k < T.n_blocks; ++k) {
            const rr_block& bl = T.blocks[k];
            if (bl.nrows > 0 && bl.ncols > 0 && bl.ncols < P->cols[bl.param])
                by[{bl.param, bl.row0, bl.nrows}].push_back({t, k});
        }
    }
    std::vector<FanGroup> groups;
    for (auto& kv : by) {
        auto& v = kv.second;
        if (v.size() < 2 || int64_t(v.size()) > kMaxFanDst) continue;
        const int32_t p = std::get<0>(kv.first);
        const int32_t es = P->es[p];
        const int64_t C = P->cols[p];
        std::vector<FanSlice> s;
        for (auto [t, k] : v) {
            const rr_block& bl = dst->tensors[t].blocks[k];
            int64_t pos = P->tensor_off[t];
            for (int32_t j = 0; j < k; ++j)
                pos += 2 * dst->tensors[t].blocks[j].nrows * dst->tensors[t].blocks[j].ncols;
            s.push_back({P->tensor_rank[t], pos, bl.col0, bl.ncols});
        }
        std::vector<size_t> order(s.size());
        for (size_t i = 0; i < order.size(); ++i) order[i] = i;
        std::sort(order.begin(), order.end(),
                  [&](size_t a, size_t b) { return s[a].col0 < s[b].col0; });
        std::vector<FanSlice> m;
        for (size_t i : order) m.push_back(s[i]);
        const int64_t cmin = m[0].col0;
        bool ok = (C * es) % 16 == 0 && P->bucket_bytes % 16 == 0;
        for (size_t i = 0; i < m.size() && ok; ++i) {
            ok = m[i].ncols % 8 == 0 &&
                 ((m[i].col0 - cmin) * es) % 16 == 0 && m[i].pos % 16 == 0 &&
                 (i == 0 || m[i].col0 == m[i - 1].col0 + m[i - 1].ncols);
        }
        const int64_t span = m.back().col0 + m.back().ncols - cmin;
        if (!ok || span * es > kFanMaxRowBytes) continue;
        const int32_t g = int32_t(groups.size());
        for (auto [t, k] : v) member[t][k] = g;
        groups.push_back({p, std::get<1>(kv.first), std::get<2>(kv.first), cmin, span, m});
    }
    return groups;
}

void build_tables(rr_plan* P, const rr_dst_layout* dst) {
    Builder b(P);
    std::vector<std::vector<int32_t>> member;
    const std::vector<FanGroup> groups = find_fan_groups(P, dst, member);
    std::vector<std::pair<size_t, size_t>> fanned;   // regular items of grouped blocks
    for (int32_t r = 0; r < P->tp; ++r) {
        int64_t cursor = 0;   // end of the previous tensor in the stream
        for (int32_t t = 0; t < P->n_tensors; ++t) {
            if (P->tensor_rank[t] != r) continue;
            b.zero_range(r, cursor, P->tensor_off[t]);
            int64_t pos = P->tensor_off[t];
            const rr_dst_tensor& T = dst->tensors[t];
            for (int32_t k = 0; k < T.n_blocks; ++k) {
                const rr_block& bl = T.blocks[k];
                const int64_t C = P->cols[bl.param];
                const size_t before = P->pack_items.size();
                if (bl.ncols == C)   // whole rows: one contiguous run
                    b.pack_run(bl.param, bl.row0 * C, bl.nrows * bl.ncols, 1, bl.nrows * bl.ncols,
                               r, pos);
                else
                    b.pack_run(bl.param, bl.row0 * C + bl.col0, bl.ncols, bl.nrows, C, r, pos);
                if (member[t][k] >= 0) fanned.push_back({before, P->pack_items.size()});
                pos += 2 * bl.nrows * bl.ncols;
            }
            cursor = pos;
        }
        const int64_t nb = P->rank_first_bucket[r + 1] - P->rank_first_bucket[r];
        b.zero_range(r, cursor, nb * P->bucket_bytes);
        cursor = 0;
        for (int32_t t = 0; t < P->n_tensors; ++t) {
            if (P->tensor_rank[t] != r) continue;
            b.read_gap(r, cursor, P->tensor_off[t]);
            b.unpack_tensor(t);
            cursor = P->tensor_off[t] + 2 * P->tensor_numel[t];
        }
        b.read_gap(r, cursor, nb * P->bucket_bytes);
    }
    // Both tables are sorted by bucket: index their per-bucket item ranges.
    auto index = [&](auto& items, std::vector<uint32_t>& first) {
        first.assign(size_t(P->n_buckets) + 1, uint32_t(items.size()));
        size_t i = 0;
        for (int32_t bk = 0; bk < P->n_buckets; ++bk) {
            while (i < items.size() && int64_t(items[i].bucket) < bk) ++i;
            first[bk] = uint32_t(i);
        }
    };
    index(P->pack_items, P->pack_bucket_first);
    index(P->unpack_items, P->unpack_bucket_first);
    // Which destination tensors each bucket's unpack items write (a launch's
    // pointer table holds only the window of tensors its buckets need).
    P->bucket_tensor_lo.assign(size_t(P->n_buckets), INT32_MAX);
    P->bucket_tensor_hi.assign(size_t(P->n_buckets), -1);
    for (const rr_unpack_item& it : P->unpack_items) {
        if (it.kind != RR_ITEM_COPY_VEC && it.kind != RR_ITEM_COPY_SCALAR) continue;
        P->bucket_tensor_lo[it.bucket] = std::min(P->bucket_tensor_lo[it.bucket], int32_t(it.tensor));
        P->bucket_tensor_hi[it.bucket] = std::max(P->bucket_tensor_hi[it.bucket], int32_t(it.tensor));
    }
    partition(P->pack_items, P->grid_blocks, P->pack_block_first, pack_weight);
    partition(P->unpack_items, P->unpack_grid_blocks, P->unpack_block_first, unpack_weight);
    bucket_units(P->unpack_items, P->unpack_bucket_first,
                 unit_weight_for(P->unpack_items, P->unpack_grid_blocks, unpack_weight),
                 P->unpack_grid_blocks, P->unpack_unit_first, P->unpack_bucket_unit,
                 unpack_weight);
    bucket_units(P->pack_items, P->pack_bucket_first,
                 unit_weight_for(P->pack_items, P->grid_blocks, pack_weight), P->grid_blocks,
                 P->pack_unit_first, P->pack_bucket_unit, pack_weight);
    // Summed weights: a bucket-range call splits its items over the grid by them.
    auto prefix = [](const auto& items, std::vector<unsigned long long>& out, auto w) {
        out.assign(items.size() + 1, 0ull);
        for (size_t i = 0; i < items.size(); ++i) out[i + 1] = out[i] + uint64_t(w(items[i]));
    };
    prefix(P->pack_items, P->pack_weight_prefix, pack_weight);
    prefix(P->unpack_items, P->unpack_weight_prefix, unpack_weight);

    // Whole-sync table: the grouped blocks' plain items give way to fan-out groups.
    P->full_items.clear();
    P->full_block_first.clear();
    if (!groups.empty()) {
        std::vector<char> drop(P->pack_items.size(), 0);
        for (auto [lo, hi] : fanned)
            for (size_t i = lo; i < hi; ++i) drop[i] = 1;
        std::vector<rr_pack_item> kept, fan;
        for (size_t i = 0; i < P->pack_items.size(); ++i)
            if (!drop[i]) kept.push_back(P->pack_items[i]);
        b.set_out(&fan);
        for (const FanGroup& g : groups) b.fan_group(g.param, g.row0, g.nrows, g.cmin, g.span, g.slices);
        b.set_out(&P->pack_items);
        // Spread the fan-out heads (with their destinations, and the plain items
        // of rows that fell back) evenly through the first part of the table,
        // so that every block's own share gets its part of them and the heads
        // are done by RR_FAN_END_PCT of the table's weight: a head cannot be
        // split, and the claimed units at the end should all be small.
        std::vector<size_t> unit_start;   // fan items in runs: a head and its destinations
        for (size_t i = 0; i < fan.size(); ++i)
            if (fan[i].kind != RR_ITEM_FAN_DST) unit_start.push_back(i);
        unit_start.push_back(fan.size());
        const size_t U = unit_start.size() - 1;
        int64_t w_kept = 0, w_fan = 0;
        for (const rr_pack_item& it : kept) w_kept += pack_weight(it);
        for (const rr_pack_item& it : fan) w_fan += pack_weight(it);
        // The plain items the heads are spread over: the first `span_kept` of them.
        const int64_t room = (w_kept + w_fan) * RR_FAN_END_PCT / 100 - w_fan;
        const size_t span_kept =
            w_kept <= 0 || room <= 0
                ? 0
                : std::min(kept.size(), size_t(double(kept.size()) * double(room) / double(w_kept)));
        P->full_items.reserve(kept.size() + fan.size());
        size_t k = 0;
        for (size_t u = 0; u < U; ++u) {
            const size_t upto = span_kept * u / U;
            for (; k < upto; ++k) P->full_items.push_back(kept[k]);
            for (size_t i = unit_start[u]; i < unit_start[u + 1]; ++i)
                P->full_items.push_back(fan[i]);
        }
        for (; k < kept.size(); ++k) P->full_items.push_back(kept[k]);
        partition(P->full_items, P->grid_blocks, P->full_block_first, pack_weight);
        // A block never starts on a fan-out destination item.
        auto& f = P->full_block_first;
        for (size_t g = 1; g + 1 < f.size(); ++g) {
            f[g] = std::max(f[g], f[g - 1]);
            while (f[g] < P->full_items.size() && P->full_items[f[g]].kind == RR_ITEM_FAN_DST) ++f[g];
        }
    }

    // Units of a pack over every bucket.
    const std::vector<rr_pack_item>& whole = P->full_items.empty() ? P->pack_items : P->full_items;
    whole_units(whole, P->grid_blocks, unit_weight_for(whole, P->grid_blocks, pack_weight),
                P->pack_whole_unit_first, pack_weight);

    rr_plan_stats& s = P->stats;
    s.n_pack_items = int64_t(P->pack_items.size());
    s.n_unpack_items = int64_t(P->unpack_items.size());
    s.grid_blocks = P->grid_blocks;
    s.unpack_grid_blocks = P->unpack_grid_blocks;
    s.verify_grid_blocks = P->verify_grid_blocks;
    s.n_buckets = P->n_buckets;
    s.n_shards = P->n_shards;
    s.n_tensors = P->n_tensors;
    s.bucket_bytes = P->bucket_bytes;
    s.pack_bytes_read = b.pack_read;
    s.pack_bytes_written = int64_t(P->n_buckets) * P->bucket_bytes;
    int64_t dst_bytes = 0;
    for (int32_t t = 0; t < P->n_tensors; ++t) dst_bytes += 2 * P->tensor_numel[t];
    s.unpack_bytes_read = dst_bytes;
    s.unpack_bytes_written = dst_bytes;
    s.verify_bytes_read = int64_t(P->n_buckets) * P->bucket_bytes;
    s.n_pack_full_items = int64_t(P->full_items.empty() ? P->pack_items.size()
                                                        : P->full_items.size());
}

}  // namespace

rr_status rr_fail(rr_status s, const char* fmt, ...) {
    char buf[512];
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(buf, sizeof buf, fmt, ap);
    va_end(ap);
    g_error = buf;
    return s;
}

void rr_clear_error() { g_error.clear(); }

extern "C" {

rr_status rr_plan_create_ex(const rr_param* manifest, int32_t n_params,
                            const rr_src_layout* src, const rr_dst_layout* dst,
                            size_t bucket_bytes, const rr_plan_options* opts, rr_plan** out) {
    RR_TRACE("rr_plan_create");
    rr_clear_error();
    if (!out) return rr_fail(RR_EINVAL, "out is NULL");
    *out = nullptr;
    rr_plan* P = new (std::nothrow) rr_plan();
    if (!P) return rr_fail(RR_ENOMEM, "host allocation failed");
    rr_status st = RR_OK;
    try {
        st = validate_and_describe(P, manifest, n_params, src, dst, bucket_bytes);
        if (st == RR_OK) {
            P->host_only = opts && opts->host_only;
            P->chunk_bytes = opts && opts->chunk_bytes ? opts->chunk_bytes : kDefaultChunkBytes;
            if (P->chunk_bytes < 16 || P->chunk_bytes % 16 != 0 || P->chunk_bytes > (1 << 30))
                st = rr_fail(RR_EINVAL, "chunk_bytes must be a multiple of 16 in [16, 2^30]");
        }
        if (st == RR_OK) {
            P->check_items = opts && opts->check_items ? 1 : 0;
            P->engine = opts ? opts->engine : RR_ENGINE_AUTO;
            if (P->engine != RR_ENGINE_AUTO && P->engine != RR_ENGINE_REGISTERS)
                st = rr_fail(RR_EINVAL, "unknown engine %d", P->engine);
            rr_grids g{152 * 2, 152 * 2, 152 * 2, 152 * 4, 152 * 4, 152 * 4};
            if (st == RR_OK && !P->host_only) st = rr_device_default_grid(&g);
            const bool bulk = P->engine == RR_ENGINE_AUTO;
            P->grid_blocks = bulk ? g.bulk_pack : g.reg_pack;
            P->unpack_grid_blocks = bulk ? g.bulk_unpack : g.reg_unpack;
            P->reg_pack_grid = g.reg_pack;
            P->reg_unpack_grid = g.reg_unpack;
            P->reg_vunpack_grid = g.reg_vunpack;
            P->verify_grid_blocks = g.verify;
            if (opts && opts->grid_blocks > 0)
                P->grid_blocks = P->unpack_grid_blocks = P->verify_grid_blocks = P->reg_pack_grid =
                    P->reg_unpack_grid = P->reg_vunpack_grid = opts->grid_blocks;
        }
        if (st == RR_OK) {
            build_tables(P, dst);
            if (P->pack_items.size() >= 0xFFFFFFFFull || P->unpack_items.size() >= 0xFFFFFFFFull ||
                P->full_items.size() >= 0xFFFFFFFFull)
                st = rr_fail(RR_ELAYOUT, "too many work items; raise chunk_bytes");
        }
        if (st == RR_OK && !P->host_only) st = rr_device_upload(P);
    } catch (const std::bad_alloc&) {
        st = rr_fail(RR_ENOMEM, "host allocation failed while planning");
    }
    if (st != RR_OK) {
        rr_device_release(P);
        delete P;
        return st;
    }
    *out = P;
    return RR_OK;
}

rr_status rr_plan_create(const rr_param* manifest, int32_t n_params, const rr_src_layout* src,
                         const rr_dst_layout* dst, size_t bucket_bytes, rr_plan** out) {
    return rr_plan_create_ex(manifest, n_params, src, dst, bucket_bytes, nullptr, out);
}

void rr_plan_destroy(rr_plan* plan) {
    if (!plan) return;
    rr_device_release(plan);
    delete plan;
}

rr_status rr_plan_query(const rr_plan* P, int32_t* n_buckets, int64_t* stream_bytes_per_rank,
                        int32_t* first_bucket_of_rank) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (n_buckets) *n_buckets = P->n_buckets;
    if (stream_bytes_per_rank)
        std::copy(P->rank_stream_bytes.begin(), P->rank_stream_bytes.end(), stream_bytes_per_rank);
    if (first_bucket_of_rank)
        std::copy(P->rank_first_bucket.begin(), P->rank_first_bucket.end(), first_bucket_of_rank);
    return RR_OK;
}

rr_status rr_plan_source(const rr_plan* P, int64_t* shard_bytes, int64_t* flat_bytes,
                         int64_t* param_flat_offset) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (shard_bytes) *shard_bytes = P->shard_bytes;
    if (flat_bytes) *flat_bytes = P->flat_bytes;
    if (param_flat_offset) std::copy(P->param_off.begin(), P->param_off.end(), param_flat_offset);
    return RR_OK;
}

rr_status rr_plan_source_buffers(const rr_plan* P, int32_t* n_buffers, int64_t* buffer_bytes) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (n_buffers) *n_buffers = P->n_shards;
    if (!buffer_bytes) return RR_OK;
    for (int32_t i = 0; i < P->n_shards; ++i) {
        if (P->sharding == RR_SHARD_TENSORS)
            buffer_bytes[i] = P->rows[i] * P->cols[i] * P->es[i];
        else if (P->sharding == RR_SHARD_UNITS)
            buffer_bytes[i] = P->unit_shard_bytes[i / P->unit_shards];
        else
            buffer_bytes[i] = P->shard_bytes;
    }
    return RR_OK;
}

rr_status rr_plan_tensors(const rr_plan* P, int64_t* tensor_numel, int64_t* tensor_stream_offset) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (tensor_numel) std::copy(P->tensor_numel.begin(), P->tensor_numel.end(), tensor_numel);
    if (tensor_stream_offset)
        std::copy(P->tensor_off.begin(), P->tensor_off.end(), tensor_stream_offset);
    return RR_OK;
}

rr_status rr_plan_get_stats(const rr_plan* P, rr_plan_stats* stats) {
    if (!P || !stats) return rr_fail(RR_EINVAL, "NULL argument");
    *stats = P->stats;
    return RR_OK;
}

rr_status rr_plan_export_pack(const rr_plan* P, rr_pack_item* items, int64_t cap,
                              uint32_t* block_first) {
    if (!P || (cap > 0 && !items)) return rr_fail(RR_EINVAL, "NULL argument");
    const int64_t n = std::min<int64_t>(cap, int64_t(P->pack_items.size()));
    if (n > 0) std::memcpy(items, P->pack_items.data(), size_t(n) * sizeof(rr_pack_item));
    if (block_first)
        std::copy(P->pack_block_first.begin(), P->pack_block_first.end(), block_first);
    return RR_OK;
}

rr_status rr_plan_export_pack_full(const rr_plan* P, rr_pack_item* items, int64_t cap,
                                   uint32_t* block_first) {
    if (!P || (cap > 0 && !items)) return rr_fail(RR_EINVAL, "NULL argument");
    if (P->full_items.empty()) return rr_plan_export_pack(P, items, cap, block_first);
    const int64_t n = std::min<int64_t>(cap, int64_t(P->full_items.size()));
    if (n > 0) std::memcpy(items, P->full_items.data(), size_t(n) * sizeof(rr_pack_item));
    if (block_first)
        std::copy(P->full_block_first.begin(), P->full_block_first.end(), block_first);
    return RR_OK;
}

rr_status rr_plan_export_unpack(const rr_plan* P, rr_unpack_item* items, int64_t cap,
                                uint32_t* block_first) {
    if (!P || (cap > 0 && !items)) return rr_fail(RR_EINVAL, "NULL argument");
    const int64_t n = std::min<int64_t>(cap, int64_t(P->unpack_items.size()));
    if (n > 0) std::memcpy(items, P->unpack_items.data(), size_t(n) * sizeof(rr_unpack_item));
    if (block_first)
        std::copy(P->unpack_block_first.begin(), P->unpack_block_first.end(), block_first);
    return RR_OK;
}

rr_status rr_plan_bucket_items(const rr_plan* P, uint32_t* pack_first, uint32_t* unpack_first) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (pack_first)
        std::copy(P->pack_bucket_first.begin(), P->pack_bucket_first.end(), pack_first);
    if (unpack_first)
        std::copy(P->unpack_bucket_first.begin(), P->unpack_bucket_first.end(), unpack_first);
    return RR_OK;
}

rr_status rr_plan_work_units(const rr_plan* P, int32_t which, int32_t* n_units,
                             uint32_t* unit_first, uint32_t* bucket_unit) {
    if (!P || !n_units) return rr_fail(RR_EINVAL, "NULL argument");
    const std::vector<uint32_t>* first = nullptr;
    const std::vector<uint32_t>* bu = nullptr;
    switch (which) {
        case RR_UNITS_PACK: first = &P->pack_unit_first; bu = &P->pack_bucket_unit; break;
        case RR_UNITS_PACK_FULL: first = &P->pack_whole_unit_first; break;
        case RR_UNITS_UNPACK: first = &P->unpack_unit_first; bu = &P->unpack_bucket_unit; break;
        default: return rr_fail(RR_EINVAL, "which must be one of the RR_UNITS_ values");
    }
    if (bucket_unit && !bu) return rr_fail(RR_EINVAL, "the whole-sync pack's units have no bucket index");
    *n_units = first->empty() ? 0 : int32_t(first->size()) - 1;
    if (unit_first) std::copy(first->begin(), first->end(), unit_first);
    if (bucket_unit) std::copy(bu->begin(), bu->end(), bucket_unit);
    return RR_OK;
}

const char* rr_status_str(rr_status s) {
    switch (s) {
        case RR_OK: return "RR_OK";
        case RR_EINVAL: return "RR_EINVAL: invalid argument";
        case RR_ENOMEM: return "RR_ENOMEM: out of memory";
        case RR_ECUDA: return "RR_ECUDA: CUDA error";
        case RR_ELAYOUT: return "RR_ELAYOUT: inconsistent layout";
        case RR_EMISMATCH: return "RR_EMISMATCH: checksum mismatch";
    }
    return "unknown rr_status";
}

const char* rr_last_error(void) { return g_error.c_str(); }

}  // extern "C"
