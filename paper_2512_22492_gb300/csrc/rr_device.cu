// Device side of the weight-sync hot path for GB300 (sm_103a): the pack
// (gather + bf16 cast + bucket write + checksum), unpack and verify kernels,
// and the C-ABI entry points that launch them.
//
// RobustRL Section 5.2.1 (steps 1-2: reshard, then place the model layer by
// layer into a transfer buffer) and Section 5.2.2 (a rollout that resumes or
// restarts a pull must know which parts of the buffer it holds intact).
//
// Two engines read the same work tables.  The bulk-copy engine
// (rr_bulk_kernel, the default when every buffer is device memory) has one
// producer warp per block stage source bytes into a shared-memory ring --
// cp.async.bulk for long runs, the warp's 16-byte cp.async for short rows --
// while consumer warps cast or copy from shared memory to the destination.
// The register path (rr_pack_kernel, rr_unpack_kernel, rr_verify_kernel)
// moves 16-byte vectors through registers; it serves host-resident buffers
// and the standalone verify.
//
// Every kernel is persistent: one launch walks the whole work table.  On the
// register path each block takes a contiguous, weight-balanced range of it.
// On the bulk-copy engine blocks take work units: their own first, then the
// next unclaimed one (an atomic counter) until none are left, so that blocks
// draining HBM at unequal rates still finish together.  The work is pure
// data movement bound by HBM bandwidth; the cast is integer arithmetic in
// registers, and the checksum is accumulated per warp and flushed with one
// 64-bit atomic per warp per bucket change.
#include <cuda_runtime.h>

#include <algorithm>
#include <climits>
#include <cstring>
#include <mutex>

#include "rr_internal.h"

namespace {

// Launch shape (overridable at build time for tuning sweeps).
#ifndef RR_THREADS
#define RR_THREADS 256
#endif
#ifndef RR_UNROLL
#define RR_UNROLL 4
#endif
#ifndef RR_PACK_MIN_BLOCKS
#define RR_PACK_MIN_BLOCKS 2
#endif
#ifndef RR_LD_HINT
#define RR_LD_HINT 0
#endif
#ifndef RR_ST_HINT
#define RR_ST_HINT 0
#endif
// The verifying register-path unpack has a shape of its own (measured on GB300:
// with 256-thread blocks it ran Qwen3-0.6B at 0.78 of the copy ceiling, with
// 128-thread blocks and 16 vectors in flight per thread at 0.99; the plain
// unpack and the pack run best at 256).
#ifndef RR_VUNPACK_THREADS
#define RR_VUNPACK_THREADS 128
#endif
#ifndef RR_VUNPACK_VECS
#define RR_VUNPACK_VECS 16
#endif
constexpr int kThreads = RR_THREADS;   // threads per block: pack, plain unpack, verify
constexpr int kUnroll = RR_UNROLL;     // 16-byte vectors in flight per thread
constexpr int kSmallPtrs = 64;      // pointer-table sizes of the two launch shapes
constexpr int kLargePtrs = 3968;    // keeps the kernel parameters under 32 KB
constexpr int64_t kVerifyChunk = 64 * 1024;
constexpr unsigned int kErrWaitTimeout = 1;       // plan error word: a bounded wait ran out
constexpr unsigned int kErrBadItem = 2;           // a work item outside its buffers, refused

// Sizes a kernel checks each work item against when the plan asks for it
// (src_bytes == NULL: no checks).  An item outside them is skipped and marks
// the plan's error word.
struct ItemBounds {
    const int64_t* src_bytes;     // bytes of each source buffer (pack)
    const int64_t* tensor_bytes;  // bytes of each destination tensor (unpack)
    int64_t bucket_bytes;
    int32_t n_src, n_buckets;
    int32_t n_tensors, pad;
    unsigned int* err;
};

// ---------------------------------------------------------------------------
// Launch arguments (passed by value in the kernel parameter space, so that a
// plan can run concurrently on several streams with different buffers).
// ---------------------------------------------------------------------------

template <int NPTR>
struct PackArgs {
    const rr_pack_item* items;
    const uint32_t* block_first;   // balanced per-block ranges, or NULL: split
    uint32_t item_begin;           //   [item_begin, item_end) over the grid by
    uint32_t item_end;             //   the items' weights (weight_prefix)
    const unsigned long long* weight_prefix;
    ItemBounds chk;
    unsigned long long* checksums;
    char* bucket_base;        // equally spaced buckets: base + b * stride
    uint64_t bucket_stride;   // 0: bucket b is ptr[n_shards + b - bucket_lo]
    int32_t n_shards;
    int32_t bucket_lo;        // table mode: the first bucket the table holds
    const void* ptr[NPTR];    // shards, then (table mode) buckets bucket_lo, ...
};

template <int NPTR>
struct UnpackArgs {
    const rr_unpack_item* items;
    const uint32_t* block_first;   // as in PackArgs
    uint32_t item_begin;
    uint32_t item_end;
    const unsigned long long* weight_prefix;
    ItemBounds chk;
    // Verifying unpack only (as in VerifyArgs): per-bucket sums of the range
    // [first_bucket, first_bucket + n_buckets), counters, expected sums, flags.
    unsigned long long* sums;
    unsigned long long* counters;
    const unsigned long long* expected;
    uint8_t* bad;
    int32_t first_bucket;
    int32_t n_buckets;
    const char* bucket_base;
    uint64_t bucket_stride;
    int32_t dst_base;         // index in ptr[] of destination tensor 0
    int32_t bucket_lo;        // table mode: the first bucket the table holds
    // Claimed work units (claim NULL: none, the split above).  unit_first holds
    // the first item of each of n_units units and one past the last; block g
    // walks unit g, then claims the next unclaimed unit (atomicAdd on *claim,
    // zero at launch) until none are left.  claim is counters + 3.
    const uint32_t* unit_first;
    unsigned long long* claim;
    uint32_t n_units;
    uint32_t reset_claims;    // counters are a pooled slot's: its last block leaves them zero
    long long* result;        // verifying: {n_bad, first_bad or -1} written at the end, or NULL
    const void* ptr[NPTR];    // (table mode) buckets bucket_lo, ..., then destination tensors
};

template <int NPTR>
struct VerifyArgs {
    unsigned long long* sums;       // [n_buckets], zeroed
    unsigned long long* counters;   // [4]: blocks done, n_bad, max(ULLONG_MAX - bad index)
    const unsigned long long* expected;   // indexed by global bucket
    uint8_t* bad;                   // optional [n_buckets]: 1 where the sum differs
    int32_t first_bucket;           // the range checked is [first_bucket, +n_buckets)
    int32_t bucket_lo;              // table mode: the first bucket the table holds
    const char* bucket_base;
    uint64_t bucket_stride;
    uint64_t bucket_bytes;
    uint64_t chunk_bytes;
    uint64_t chunks_per_bucket;
    uint64_t total_chunks;
    int32_t n_buckets;
    int32_t pad;
    const void* ptr[NPTR];          // (table mode) buckets
};

// ---------------------------------------------------------------------------
// Small device helpers
// ---------------------------------------------------------------------------

// Streaming 16-byte load of data read exactly once (read-only for the kernel).
__device__ __forceinline__ uint4 ld_stream(const void* p) {
    uint4 r;
#if RR_LD_HINT == 1
    asm volatile("ld.global.nc.L1::no_allocate.L2::256B.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
#elif RR_LD_HINT == 2
    asm volatile("ld.global.cs.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
#else
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(r.x), "=r"(r.y), "=r"(r.z), "=r"(r.w)
                 : "l"(p));
#endif
    return r;
}

// 16-byte store of data written exactly once.
__device__ __forceinline__ void st_stream(void* p, uint4 v) {
#if RR_ST_HINT == 1
    asm volatile("st.global.cs.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
#else
    asm volatile("st.global.v4.u32 [%0], {%1, %2, %3, %4};" ::"l"(p), "r"(v.x), "r"(v.y),
                 "r"(v.z), "r"(v.w)
                 : "memory");
#endif
}

// 8-byte store of data written exactly once.
__device__ __forceinline__ void st_stream8(void* p, uint32_t x, uint32_t y) {
    asm volatile("st.global.v2.u32 [%0], {%1, %2};" ::"l"(p), "r"(x), "r"(y) : "memory");
}

// float32 bits -> value whose upper half is the bfloat16 result: round to
// nearest even by adding 0x7FFF plus the lowest kept bit; a NaN instead
// keeps its upper half with the quiet bit set (no rounding, so it can never
// carry into the exponent and become an infinity).
__device__ __forceinline__ uint32_t round_hi(uint32_t x) {
    const uint32_t r = x + 0x7FFFu + ((x >> 16) & 1u);
    return (x & 0x7FFFFFFFu) > 0x7F800000u ? (x | 0x00400000u) : r;
}

// Two float32 -> two bfloat16 packed little-endian in one word.
__device__ __forceinline__ uint32_t cast2(uint32_t a, uint32_t b) {
    return __byte_perm(round_hi(a), round_hi(b), 0x7632);
}

__device__ __forceinline__ uint16_t cast1(uint32_t a) { return uint16_t(round_hi(a) >> 16); }

// float32 bits -> IEEE binary16 bits.  Numbers take the hardware conversion,
// cvt.rn (round to nearest, ties to even; subnormals kept, overflow to +-inf);
// a NaN is replaced by the quiet NaN that keeps its sign and top payload bits,
// whatever NaN the conversion gives.
__device__ __forceinline__ bool is_nan32(uint32_t x) { return (x & 0x7FFFFFFFu) > 0x7F800000u; }

__device__ __forceinline__ uint32_t nan_f16(uint32_t x) {
    return ((x >> 16) & 0x8000u) | 0x7E00u | ((x >> 13) & 0x01FFu);
}

// Two float32 -> two binary16 packed little-endian in one word (a low), by the
// conversion alone (numbers only).
__device__ __forceinline__ uint32_t cvt_f16x2(uint32_t a, uint32_t b) {
    uint32_t r;
    asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(r) : "f"(__uint_as_float(b)), "f"(__uint_as_float(a)));
    return r;
}

// The same with NaNs replaced by the stated rule.
__device__ __forceinline__ uint32_t cast2_f16(uint32_t a, uint32_t b) {
    uint32_t r = cvt_f16x2(a, b);
    if (is_nan32(a)) r = (r & 0xFFFF0000u) | nan_f16(a);
    if (is_nan32(b)) r = (r & 0x0000FFFFu) | (nan_f16(b) << 16);
    return r;
}

__device__ __forceinline__ uint16_t cast1_f16(uint32_t a) {
    uint16_t h;
    asm("cvt.rn.f16.f32 %0, %1;" : "=h"(h) : "f"(__uint_as_float(a)));
    return is_nan32(a) ? uint16_t(nan_f16(a)) : h;
}

// The destination element type of a pack: bfloat16 (F16 false: a float32
// source is rounded, a bfloat16 one copied) or float16 (a bfloat16 source is
// widened exactly, then rounded like a float32 one).
template <bool F16>
struct DstCast {
    static __device__ __forceinline__ uint32_t f32x2(uint32_t a, uint32_t b) {
        return F16 ? cast2_f16(a, b) : cast2(a, b);
    }
    static __device__ __forceinline__ uint16_t f32(uint32_t a) {
        return F16 ? cast1_f16(a) : cast1(a);
    }
    // Two bfloat16 packed in a word.
    static __device__ __forceinline__ uint32_t bf16x2(uint32_t w) {
        return F16 ? cast2_f16(w << 16, w & 0xFFFF0000u) : w;
    }
    static __device__ __forceinline__ uint16_t bf16(uint16_t h) {
        return F16 ? cast1_f16(uint32_t(h) << 16) : h;
    }
    static __device__ __forceinline__ uint4 bf16x8(uint4 v) {
        if (!F16) return v;
        // One test for the eight elements: a bfloat16 is a NaN when its
        // magnitude exceeds 0x7F80.  Without one, the conversions need no patch.
        const uint32_t m = __vmaxu2(__vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu),
                                    __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu));
        if (__vcmpgtu2(m, 0x7F807F80u) != 0)
            return make_uint4(bf16x2(v.x), bf16x2(v.y), bf16x2(v.z), bf16x2(v.w));
        return make_uint4(cvt_f16x2(v.x << 16, v.x & 0xFFFF0000u),
                          cvt_f16x2(v.y << 16, v.y & 0xFFFF0000u),
                          cvt_f16x2(v.z << 16, v.z & 0xFFFF0000u),
                          cvt_f16x2(v.w << 16, v.w & 0xFFFF0000u));
    }
};

__device__ __forceinline__ unsigned long long words(uint4 v) {
    return ((unsigned long long)v.y << 32 | v.x) + ((unsigned long long)v.w << 32 | v.z);
}

__device__ __forceinline__ unsigned long long warp_sum(unsigned long long v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}

__device__ __forceinline__ void flush(unsigned long long* dst, unsigned long long acc) {
    acc = warp_sum(acc);
    if ((threadIdx.x & 31) == 0 && acc != 0ull) atomicAdd(dst, acc);
}

// The source extent of a data item: the bytes from its first source element to
// the end of its last row.
__device__ __forceinline__ uint64_t src_extent(uint32_t rows, uint32_t row_len, uint32_t stride,
                                               uint32_t es) {
    return rows ? ((uint64_t)(rows - 1) * stride + row_len) * es : 0;
}

// Whether a pack item (or fan-out destination) lies inside the plan's buffers.
__device__ __forceinline__ bool pack_item_in(const ItemBounds& b, const rr_pack_item& d) {
    if (!b.src_bytes) return true;
    const uint64_t n = (uint64_t)d.row_len * d.n_rows;
    bool ok = d.bucket < (uint32_t)b.n_buckets;
    if (d.kind <= RR_ITEM_BF16_SCALAR || d.kind == RR_ITEM_FAN_F32 || d.kind == RR_ITEM_FAN_BF16) {
        const uint32_t es =
            (d.kind <= RR_ITEM_F32_SCALAR || d.kind == RR_ITEM_FAN_F32) ? 4u : 2u;
        const uint32_t sh = (uint32_t)(d.src >> 48);
        const uint64_t off = d.src & 0xFFFFFFFFFFFFull;
        ok = ok && sh < (uint32_t)b.n_src &&
             off + src_extent(d.n_rows, d.row_len, d.src_stride, es) <= (uint64_t)b.src_bytes[sh];
        if (d.kind <= RR_ITEM_BF16_SCALAR) ok = ok && d.dst_off + 2 * n <= (uint64_t)b.bucket_bytes;
    } else if (d.kind == RR_ITEM_ZERO_VEC || d.kind == RR_ITEM_ZERO_SCALAR ||
               d.kind == RR_ITEM_FAN_DST) {
        ok = ok && d.dst_off + 2 * n <= (uint64_t)b.bucket_bytes;
    } else {
        ok = false;
    }
    return ok;
}

// As pack_item_in, called uniformly by a warp or block; its first thread marks
// a refusal in the plan's error word.
__device__ __forceinline__ bool pack_item_ok(const ItemBounds& b, const rr_pack_item& d) {
    const bool ok = pack_item_in(b, d);
    if (!ok && threadIdx.x % 32 == 0) atomicExch(b.err, kErrBadItem);
    return ok;
}

// Whether an unpack item lies inside its bucket and (a copy) its tensor.
__device__ __forceinline__ bool unpack_item_ok(const ItemBounds& b, const rr_unpack_item& d) {
    if (!b.src_bytes) return true;
    bool ok = d.bucket < (uint32_t)b.n_buckets &&
              (uint64_t)d.src_off + d.nbytes <= (uint64_t)b.bucket_bytes;
    if (d.kind == RR_ITEM_COPY_VEC || d.kind == RR_ITEM_COPY_SCALAR)
        ok = ok && d.tensor < (uint32_t)b.n_tensors &&
             d.dst_off + d.nbytes <= (uint64_t)b.tensor_bytes[d.tensor];
    else
        ok = ok && (d.kind == RR_ITEM_READ_VEC || d.kind == RR_ITEM_READ_SCALAR);
    if (!ok && threadIdx.x % 32 == 0) atomicExch(b.err, kErrBadItem);
    return ok;
}

// This block's item range: the plan's balanced split for a full call, an even
// split of [begin, end) for a bucket-range call.
// First item i in [lo, hi] with prefix[i] >= w (prefix is non-decreasing).
__device__ __forceinline__ uint32_t lower_item(const unsigned long long* prefix, uint32_t lo,
                                               uint32_t hi, unsigned long long w) {
    while (lo < hi) {
        const uint32_t mid = lo + (hi - lo) / 2;
        if (prefix[mid] < w)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

__device__ __forceinline__ void block_items(const uint32_t* block_first,
                                            const unsigned long long* prefix, uint32_t begin,
                                            uint32_t end, uint32_t* i0, uint32_t* i1) {
    if (block_first) {
        *i0 = block_first[blockIdx.x];
        *i1 = block_first[blockIdx.x + 1];
    } else if (prefix) {
        // Split points at equal shares of the range's weight; neighbouring blocks
        // compute the same point, so the ranges tile [begin, end).
        const unsigned long long w0 = prefix[begin], w = prefix[end] - w0;
        *i0 = blockIdx.x == 0 ? begin
                              : lower_item(prefix, begin, end, w0 + w * blockIdx.x / gridDim.x);
        *i1 = blockIdx.x + 1 == gridDim.x
                  ? end
                  : lower_item(prefix, begin, end, w0 + w * (blockIdx.x + 1) / gridDim.x);
    } else {
        const uint64_t n = end - begin;
        *i0 = begin + (uint32_t)(n * blockIdx.x / gridDim.x);
        *i1 = begin + (uint32_t)(n * (blockIdx.x + 1) / gridDim.x);
    }
}

template <int NPTR>
__device__ __forceinline__ char* bucket_of(const PackArgs<NPTR>& a, uint32_t b) {
    return a.bucket_stride ? a.bucket_base + (uint64_t)b * a.bucket_stride
                           : (char*)a.ptr[a.n_shards + (b - a.bucket_lo)];
}

// ---------------------------------------------------------------------------
// Pack
// ---------------------------------------------------------------------------

// Vector item: n_rows rows of row_len (multiple of 8) elements, 16-byte
// aligned source rows and destination.  One "vector" is 8 elements: 32 (fp32)
// or 16 (bf16) source bytes, 16 destination bytes.  Thread t handles vectors
// t, t + T, t + 2T, ...; (row, vector-in-row) is advanced incrementally.
template <int ES, bool F16>
__device__ __forceinline__ unsigned long long pack_vec(const char* src, char* dst,
                                                       const rr_pack_item& d) {
    using D = DstCast<F16>;
    // A bf16 vector is one 16-byte load instead of two: twice as many of them
    // keep the same bytes in flight per thread.
    constexpr int U = ES == 4 ? kUnroll : 2 * kUnroll;
    const uint32_t vpr = d.row_len >> 3;
    const uint32_t nvec = vpr * d.n_rows;
    const uint64_t stride = (uint64_t)d.src_stride * ES;
    const uint32_t dq = kThreads / vpr, dr = kThreads - dq * vpr;
    uint32_t v = threadIdx.x;
    uint32_t r = v / vpr, c = v - r * vpr;
    unsigned long long acc = 0;
    while (v < nvec) {
        uint4 x[U][ES / 2];
        uint32_t vv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            vv[u] = v;
            if (v < nvec) {
                const char* p = src + r * stride + (uint64_t)c * (8 * ES);
                x[u][0] = ld_stream(p);
                if (ES == 4) x[u][ES / 2 - 1] = ld_stream(p + 16);
            }
            v += kThreads;
            c += dr;
            r += dq;
            if (c >= vpr) {
                c -= vpr;
                ++r;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (vv[u] < nvec) {
                uint4 o;
                if (ES == 4) {
                    o.x = D::f32x2(x[u][0].x, x[u][0].y);
                    o.y = D::f32x2(x[u][0].z, x[u][0].w);
                    o.z = D::f32x2(x[u][ES / 2 - 1].x, x[u][ES / 2 - 1].y);
                    o.w = D::f32x2(x[u][ES / 2 - 1].z, x[u][ES / 2 - 1].w);
                } else {
                    o = D::bf16x8(x[u][0]);
                }
                st_stream(dst + (uint64_t)vv[u] * 16, o);
                acc += words(o);
            }
        }
    }
    return acc;
}

// fp32 vector item with its source in host memory: vectors of 4 elements, one
// 16-byte load and one 8-byte store each, so that a warp's load instruction
// covers 512 contiguous source bytes.  Over NVLink-C2C a load instruction that
// uses half of every 32-byte sector it touches (the two 16-byte halves of an
// 8-element vector, loaded by two instructions) moves each sector twice: with
// 8-element vectors the pack read pinned host memory at half the link's rate.
// The destination is 16-byte aligned, so each store is one whole checksum word.
template <bool F16>
__device__ __forceinline__ unsigned long long pack_vec_f32_narrow(const char* src, char* dst,
                                                                  const rr_pack_item& d) {
    using D = DstCast<F16>;
    constexpr int U = 2 * kUnroll;
    const uint32_t vpr = d.row_len >> 2;
    const uint32_t nvec = vpr * d.n_rows;
    const uint64_t stride = (uint64_t)d.src_stride * 4;
    const uint32_t dq = kThreads / vpr, dr = kThreads - dq * vpr;
    uint32_t v = threadIdx.x;
    uint32_t r = v / vpr, c = v - r * vpr;
    unsigned long long acc = 0;
    while (v < nvec) {
        uint4 x[U];
        uint32_t vv[U];
#pragma unroll
        for (int u = 0; u < U; ++u) {
            vv[u] = v;
            if (v < nvec) x[u] = ld_stream(src + r * stride + (uint64_t)c * 16);
            v += kThreads;
            c += dr;
            r += dq;
            if (c >= vpr) {
                c -= vpr;
                ++r;
            }
        }
#pragma unroll
        for (int u = 0; u < U; ++u) {
            if (vv[u] < nvec) {
                const uint32_t lo = D::f32x2(x[u].x, x[u].y), hi = D::f32x2(x[u].z, x[u].w);
                st_stream8(dst + (uint64_t)vv[u] * 8, lo, hi);
                acc += (unsigned long long)hi << 32 | lo;
            }
        }
    }
    return acc;
}

// Scalar item: any alignment and row length; one element per thread-step.
// Each element's checksum contribution is its bits shifted to its byte
// position within the 64-bit word it lands in.
template <int ES, bool F16>
__device__ __forceinline__ unsigned long long pack_scalar(const char* src, char* dst,
                                                          const rr_pack_item& d) {
    using D = DstCast<F16>;
    const uint32_t L = d.row_len;
    const uint32_t n = L * d.n_rows;
    const uint64_t stride = (uint64_t)d.src_stride * ES;
    const uint32_t dq = kThreads / L, dr = kThreads - dq * L;
    uint32_t e = threadIdx.x;
    uint32_t r = e / L, c = e - r * L;
    unsigned long long acc = 0;
    for (; e < n; e += kThreads) {
        const char* p = src + r * stride + (uint64_t)c * ES;
        uint16_t h;
        if (ES == 4)
            h = D::f32(*(const uint32_t*)p);
        else
            h = D::bf16(*(const uint16_t*)p);
        *(uint16_t*)(dst + 2ull * e) = h;
        acc += (unsigned long long)h << (8 * ((d.dst_off + 2 * e) & 7));
        c += dr;
        r += dq;
        if (c >= L) {
            c -= L;
            ++r;
        }
    }
    return acc;
}

// HOST_SRC: the source is in host memory (fp32 vectors of 4 elements).
// F16: the rollout's elements are float16 (else bfloat16).
template <int NPTR, bool CHECK, bool HOST_SRC, bool F16>
__global__ void __launch_bounds__(kThreads, RR_PACK_MIN_BLOCKS) rr_pack_kernel(const __grid_constant__ PackArgs<NPTR> a) {
    uint32_t i0, i1;
    block_items(a.block_first, a.weight_prefix, a.item_begin, a.item_end, &i0, &i1);
    unsigned long long acc = 0;
    uint32_t cur = 0xFFFFFFFFu;
    // The next item's load is in flight while the current one is moved.
    rr_pack_item next;
    if (i0 < i1) next = a.items[i0];
    for (uint32_t it = i0; it < i1; ++it) {
        const rr_pack_item d = next;
        if (it + 1 < i1) next = a.items[it + 1];
        if (CHECK && !pack_item_ok(a.chk, d)) continue;
        if (d.bucket != cur) {
            if (cur != 0xFFFFFFFFu) flush(a.checksums + cur, acc);
            cur = d.bucket;
            acc = 0;
        }
        char* dst = bucket_of(a, d.bucket) + d.dst_off;
        const char* src = (const char*)a.ptr[d.src >> 48] + (d.src & 0xFFFFFFFFFFFFull);
        switch (d.kind) {
            case RR_ITEM_F32_VEC:
                acc += HOST_SRC ? pack_vec_f32_narrow<F16>(src, dst, d)
                                : pack_vec<4, F16>(src, dst, d);
                break;
            case RR_ITEM_BF16_VEC: acc += pack_vec<2, F16>(src, dst, d); break;
            case RR_ITEM_F32_SCALAR: acc += pack_scalar<4, F16>(src, dst, d); break;
            case RR_ITEM_BF16_SCALAR: acc += pack_scalar<2, F16>(src, dst, d); break;
            case RR_ITEM_ZERO_VEC:
                for (uint32_t v = threadIdx.x; v < (d.row_len >> 3); v += kThreads)
                    st_stream(dst + 16ull * v, make_uint4(0, 0, 0, 0));
                break;
            default:  // RR_ITEM_ZERO_SCALAR
                for (uint32_t e = threadIdx.x; e < d.row_len; e += kThreads)
                    *(uint16_t*)(dst + 2ull * e) = 0;
                break;
        }
    }
    if (cur != 0xFFFFFFFFu) flush(a.checksums + cur, acc);
}

// ---------------------------------------------------------------------------
// Checksum comparison, run by whichever block finishes last (a ticket counter;
// no block waits for another).  sums[i] belongs to bucket first + i.
// ---------------------------------------------------------------------------

// The last block's result: counters[1] mismatches, the lowest one's index
// from counters[2] (which holds ULLONG_MAX - index), or -1.
__device__ __forceinline__ void write_result(unsigned long long* counters, long long* result) {
    const unsigned long long nb = atomicAdd(&counters[1], 0ull);
    result[0] = (long long)nb;
    result[1] = nb ? (long long)(ULLONG_MAX - atomicAdd(&counters[2], 0ull)) : -1ll;
}

__device__ void compare_in_last_block(unsigned long long* counters,
                                      const unsigned long long* sums,
                                      const unsigned long long* expected, uint8_t* bad,
                                      int32_t first, int32_t n, long long* result = nullptr) {
    __shared__ bool last;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        last = atomicAdd(&counters[0], 1ull) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last) return;
    __threadfence();
    for (int32_t i = threadIdx.x; i < n; i += blockDim.x) {
        const int32_t b = first + i;
        const bool differs = __ldcg(sums + i) != expected[b];
        if (bad) bad[i] = differs ? 1 : 0;
        if (differs) {
            atomicAdd(&counters[1], 1ull);
            atomicMax(&counters[2], ULLONG_MAX - (unsigned long long)b);
        }
    }
    if (result) {
        __syncthreads();
        if (threadIdx.x == 0) write_result(counters, result);
    }
}

// ---------------------------------------------------------------------------
// Unpack
// ---------------------------------------------------------------------------

// Launch shape of rr_unpack_kernel: threads per block and 16-byte vectors in
// flight per thread (plain: twice the pack's depth, one load per vector).
template <bool VERIFY>
struct RegUnpackShape {
    static constexpr int kBlock = VERIFY ? RR_VUNPACK_THREADS : kThreads;
    static constexpr int kVecs = VERIFY ? RR_VUNPACK_VECS : 2 * kUnroll;
};

// Copies each item's bytes from its bucket to its tensor.  With VERIFY it also
// sums every bucket byte it reads (the gap READ items too) into the bucket's
// checksum and compares at the end, so the buckets are read once for both.
template <int NPTR, bool VERIFY, bool CHECK>
__global__ void __launch_bounds__(RegUnpackShape<VERIFY>::kBlock, 4) rr_unpack_kernel(const __grid_constant__ UnpackArgs<NPTR> a) {
    constexpr int T = RegUnpackShape<VERIFY>::kBlock;
    constexpr int U = RegUnpackShape<VERIFY>::kVecs;
    __shared__ uint32_t next_unit[2];   // the claimed unit, double-buffered by parity
    uint32_t i0 = 0, i1 = 0;
    uint32_t walked = 0;              // units this block has walked
    unsigned long long pending = 0;   // thread 0: the claim in flight
    if (!a.claim) {
        block_items(a.block_first, a.weight_prefix, a.item_begin, a.item_end, &i0, &i1);
    } else {
        if (blockIdx.x < a.n_units) {
            i0 = a.unit_first[blockIdx.x];
            i1 = a.unit_first[blockIdx.x + 1];
        }
        if (threadIdx.x == 0) pending = atomicAdd(a.claim, 1ull);   // the unit after this one
    }
    unsigned long long acc = 0;
    uint32_t cur = 0xFFFFFFFFu;
    for (;;) {
        // The next item's load is in flight while the current one is moved.
        rr_unpack_item next;
        if (i0 < i1) next = a.items[i0];
        for (uint32_t it = i0; it < i1; ++it) {
            const rr_unpack_item d = next;
            if (it + 1 < i1) next = a.items[it + 1];
            if (!VERIFY && d.kind >= RR_ITEM_READ_VEC) continue;
            if (CHECK && !unpack_item_ok(a.chk, d)) continue;
            if (VERIFY && d.bucket != cur) {
                if (cur != 0xFFFFFFFFu) flush(a.sums + (cur - a.first_bucket), acc);
                cur = d.bucket;
                acc = 0;
            }
            const char* src = (a.bucket_stride ? a.bucket_base + (uint64_t)d.bucket * a.bucket_stride
                                               : (const char*)a.ptr[d.bucket - a.bucket_lo]) +
                              d.src_off;
            const bool copy = d.kind == RR_ITEM_COPY_VEC || d.kind == RR_ITEM_COPY_SCALAR;
            char* dst = copy ? (char*)a.ptr[a.dst_base + d.tensor] + d.dst_off : nullptr;
            if (d.kind == RR_ITEM_COPY_VEC || d.kind == RR_ITEM_READ_VEC) {
                const uint32_t nvec = d.nbytes >> 4;
                for (uint32_t v = threadIdx.x; v < nvec; v += T * U) {
                    uint4 x[U];
#pragma unroll
                    for (int u = 0; u < U; ++u)
                        if (v + u * T < nvec) x[u] = ld_stream(src + 16ull * (v + u * T));
#pragma unroll
                    for (int u = 0; u < U; ++u) {
                        if (v + u * T < nvec) {
                            if (copy) st_stream(dst + 16ull * (v + u * T), x[u]);
                            if (VERIFY) acc += words(x[u]);
                        }
                    }
                }
            } else {
                for (uint32_t e = threadIdx.x; e < (d.nbytes >> 1); e += T) {
                    const uint16_t h = *(const uint16_t*)(src + 2ull * e);
                    if (copy) *(uint16_t*)(dst + 2ull * e) = h;
                    if (VERIFY) acc += (unsigned long long)h << (8 * ((d.src_off + 2 * e) & 7));
                }
            }
        }
        if (!a.claim) break;
        // The next unit: the claim issued when this one began (its latency hid
        // behind the walk), published by thread 0 in this unit's parity slot
        // (the other slot may still be read by warps leaving the previous
        // barrier), then the following claim goes out at once.  One barrier
        // per unit.
        const uint32_t par = walked++ & 1u;
        if (threadIdx.x == 0)
            next_unit[par] = pending < (unsigned long long)(a.n_units - min(a.n_units, gridDim.x))
                                 ? gridDim.x + (uint32_t)pending
                                 : a.n_units;
        __syncthreads();
        const uint32_t u = next_unit[par];
        if (u >= a.n_units) break;
        if (threadIdx.x == 0) pending = atomicAdd(a.claim, 1ull);
        i0 = a.unit_first[u];
        i1 = a.unit_first[u + 1];
    }
    if (a.claim && a.reset_claims) {
        // A pooled slot's counters go back to zero for its next launch: the
        // block that takes the last ticket (counters[0]) resets them.  Every
        // block gets here only after its last claim has returned.
        __syncthreads();
        if (threadIdx.x == 0) {
            __threadfence();
            if (atomicAdd(&a.counters[0], 1ull) == gridDim.x - 1) {
                __threadfence();
                atomicExch(a.claim, 0ull);
                atomicExch(&a.counters[0], 0ull);
            }
        }
    }
    if (VERIFY) {
        if (cur != 0xFFFFFFFFu) flush(a.sums + (cur - a.first_bucket), acc);
        compare_in_last_block(a.counters, a.sums, a.expected, a.bad, a.first_bucket,
                              a.n_buckets, a.result);
    }
}

// ---------------------------------------------------------------------------
// Verify
// ---------------------------------------------------------------------------

template <int NPTR>
__global__ void __launch_bounds__(kThreads, 4) rr_verify_kernel(const __grid_constant__ VerifyArgs<NPTR> a) {
    const uint64_t c0 = a.total_chunks * blockIdx.x / gridDim.x;
    const uint64_t c1 = a.total_chunks * (blockIdx.x + 1) / gridDim.x;
    unsigned long long acc = 0;
    uint32_t cur = 0xFFFFFFFFu;
    for (uint64_t ch = c0; ch < c1; ++ch) {
        const uint32_t bl = (uint32_t)(ch / a.chunks_per_bucket);   // index within the range
        const uint64_t off = (ch - (uint64_t)bl * a.chunks_per_bucket) * a.chunk_bytes;
        const uint64_t len = min(a.chunk_bytes, a.bucket_bytes - off);
        if (bl != cur) {
            if (cur != 0xFFFFFFFFu) flush(a.sums + cur, acc);
            cur = bl;
            acc = 0;
        }
        const uint32_t b = a.first_bucket + bl;
        const char* p = (a.bucket_stride ? a.bucket_base + (uint64_t)b * a.bucket_stride
                                         : (const char*)a.ptr[b - a.bucket_lo]) + off;
        const uint32_t nvec = (uint32_t)(len >> 4);
        for (uint32_t v = threadIdx.x; v < nvec; v += kThreads * kUnroll) {
            uint4 x[kUnroll];
#pragma unroll
            for (int u = 0; u < kUnroll; ++u)
                if (v + u * kThreads < nvec) x[u] = ld_stream(p + 16ull * (v + u * kThreads));
#pragma unroll
            for (int u = 0; u < kUnroll; ++u)
                if (v + u * kThreads < nvec) acc += words(x[u]);
        }
        if ((len & 15) && threadIdx.x == 0)   // a trailing 8-byte word
            acc += *(const unsigned long long*)(p + (len & ~15ull));
    }
    if (cur != 0xFFFFFFFFu) flush(a.sums + cur, acc);

    compare_in_last_block(a.counters, a.sums, a.expected, a.bad, a.first_bucket, a.n_buckets);
}

// ---------------------------------------------------------------------------
// Bulk-copy engine (cp.async.bulk + mbarrier), the default for buffers in
// device memory.  One producer lane per block turns the block's work items
// into pieces: long contiguous or row-strided 16-byte-aligned runs are loaded
// into a ring of shared-memory stages with cp.async.bulk (rows of a strided
// run land back to back); ragged, misaligned and zero-fill work passes
// through as metadata only.  Consumer warps wait for a stage, cast or copy it
// to the destination with 16-byte stores, accumulate the checksum, and
// release the stage.  Memory latency is hidden by the ring, not by registers.
//
// Every wait is bounded: a wait that runs out sets the plan's error word,
// lets its block's loads land, and returns (the host reports it as RR_ECUDA).
// ---------------------------------------------------------------------------

// Stage ring shape per direction (build-time overridable for tuning sweeps).
#ifndef RR_PACK_STAGE_KB
#define RR_PACK_STAGE_KB 48
#endif
#ifndef RR_PACK_STAGES
#define RR_PACK_STAGES 3
#endif
#ifndef RR_PACK_WARPS
#define RR_PACK_WARPS 8
#endif
#ifndef RR_UNPACK_STAGE_KB
#define RR_UNPACK_STAGE_KB 32
#endif
#ifndef RR_UNPACK_STAGES
#define RR_UNPACK_STAGES 3
#endif
#ifndef RR_UNPACK_WARPS
#define RR_UNPACK_WARPS 4
#endif

template <int MODE>
struct BulkShape {
    static constexpr int kWarps = MODE == 0 ? RR_PACK_WARPS : RR_UNPACK_WARPS;
    static constexpr int kStageBytes = (MODE == 0 ? RR_PACK_STAGE_KB : RR_UNPACK_STAGE_KB) * 1024;
    static constexpr int kStages = MODE == 0 ? RR_PACK_STAGES : RR_UNPACK_STAGES;
    static constexpr int kThreads = 32 * (kWarps + 1);
    static constexpr int kSmem = kStages * kStageBytes;
};
constexpr uint32_t kWaitLimit = 1u << 20;        // tries, each suspending at most kWaitHintNs
constexpr uint32_t kWaitHintNs = 1000;
constexpr uint64_t kWaitDeadlineNs = 1000000000;  // and at most one second of wall clock

enum : uint16_t {
    PC_CAST = 1,      // stage holds fp32 rows -> bf16 destination
    PC_COPY = 2,      // stage holds bf16 -> destination
    PC_READ = 3,      // stage holds bf16 that is only summed (verifying unpack gaps)
    PC_SCALAR = 4,    // element by element from global memory
    PC_ZERO_VEC = 5,  // 16-byte zero stores
    PC_ZERO_SCALAR = 6,
    PC_END = 7,
    PC_FAN = 8        // stage holds whole rows; every fan-out destination takes its slice
};

constexpr uint32_t kMinBulkRowBytes = 1024;
constexpr uint32_t kMaxFanDst = 16; // fan-out destinations per head (the planner's limit)

struct Piece {
    const char* src;      // first source element (global)
    char* dst;            // first destination element (global), NULL for PC_READ
    uint64_t src_stride;  // bytes between source rows
    uint32_t n;           // destination elements (2 bytes each)
    uint32_t rows;        // source rows
    uint32_t row_len;     // elements per source row
    uint32_t sum_bucket;  // bucket the checksum contribution belongs to
    uint32_t sum_off;     // byte offset of element 0 in that bucket
    uint16_t kind;
    uint16_t es;          // source element bytes
};

template <int NPTR>
struct BulkArgs {
    const void* items;           // rr_pack_item (MODE 0) or rr_unpack_item
    uint32_t n_items;            // items in that table (the producer reads ahead, never past)
    const uint32_t* block_first; // as in PackArgs
    uint32_t item_begin;
    uint32_t item_end;
    const unsigned long long* weight_prefix;
    ItemBounds chk;
    char* bucket_base;
    uint64_t bucket_stride;
    int32_t n_shards;            // pack: ptr[0 .. n_shards) are the shards
    int32_t dst_base;            // unpack: index in ptr[] of destination tensor 0
    int32_t bucket_lo;           // table mode: the first bucket the table holds
    int32_t pad_;
    unsigned long long* sums;    // pack: sums by global bucket; verify: range sums
    unsigned long long* counters;// {ticket, n_bad, max(~0 - bad index), claim}
    const unsigned long long* expected;
    uint8_t* bad;
    int32_t first_bucket;        // the call's range [first_bucket, first_bucket + n_buckets)
    int32_t n_buckets;
    unsigned int* err;
    // Claimed work units (NULL: none).  block_first then holds the first item
    // of each of n_units units (and one past the last): unit g < gridDim.x is
    // block g's own, the rest go to whichever block asks next (atomicAdd on
    // *claim = counters[3], zero at launch).
    unsigned long long* claim;
    uint32_t n_units;
    // The launch holds a pooled slot (counters, and sums for pack and the
    // verifying unpack): its last block leaves them zero for the slot's next
    // launch.
    uint32_t reset_claims;
    unsigned long long* sums_out;  // pack through a slot: checksums[b] = sums[b] at the end
    long long* result;             // verifying unpack: {n_bad, first_bad or -1}, or NULL
    const void* ptr[NPTR];
};

static_assert(sizeof(rr_pack_item) == 32 && sizeof(rr_unpack_item) == 32,
              "the producer's item window moves 32-byte items as two 16-byte words");

// A 32-byte work item as two 16-byte words (the window's unit of transfer).
template <class Item>
union ItemWords {
    uint4 w[2];
    Item item;
};

// Lane `src`'s two words, for every lane of the warp.
__device__ __forceinline__ void shfl_words(const uint4& a, const uint4& b, int src, uint4& x,
                                           uint4& y) {
    x.x = __shfl_sync(0xFFFFFFFFu, a.x, src);
    x.y = __shfl_sync(0xFFFFFFFFu, a.y, src);
    x.z = __shfl_sync(0xFFFFFFFFu, a.z, src);
    x.w = __shfl_sync(0xFFFFFFFFu, a.w, src);
    y.x = __shfl_sync(0xFFFFFFFFu, b.x, src);
    y.y = __shfl_sync(0xFFFFFFFFu, b.y, src);
    y.z = __shfl_sync(0xFFFFFFFFu, b.z, src);
    y.w = __shfl_sync(0xFFFFFFFFu, b.w, src);
}

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
    return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t global_ns() {
    uint64_t t;
    asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
    return t;
}

__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity, unsigned int* err) {
    const uint64_t t0 = global_ns();
    for (uint32_t it = 0; it < kWaitLimit; ++it) {
        if ((it & 255) == 255 && global_ns() - t0 > kWaitDeadlineNs) break;
        uint32_t done;
        asm volatile(
            "{ .reg .pred p; mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3; "
            "selp.u32 %0, 1, 0, p; }"
            : "=r"(done)
            : "r"(bar), "r"(parity), "n"(kWaitHintNs)
            : "memory");
        if (done) return true;
    }
    atomicExch(err, kErrWaitTimeout);
    return false;
}

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
    asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// Short aligned rows (16-byte aligned, row bytes a multiple of 16) gathered
// into a stage by the whole producer warp: 16-byte cp.async copies, lane l
// taking vectors l, l + 32, ...; the rows land back to back.  Each lane's
// copies are tracked by the stage's full barrier: the counted form of
// cp.async.mbarrier.arrive raises the barrier's pending count now and arrives
// once the lane's copies have landed, so the phase cannot complete before them
// (the caller's own arrival, after a __syncwarp, is the one the count expects).
__device__ __forceinline__ void gather_async(uint32_t stage, uint32_t full_bar, const char* src,
                                             uint64_t src_stride, uint32_t rows,
                                             uint32_t row_bytes, uint32_t lane) {
    const uint32_t vpr = row_bytes >> 4;
    const uint32_t nv = vpr * rows;
    const uint32_t dq = 32 / vpr, dr = 32 - dq * vpr;
    uint32_t r = lane / vpr, c = lane - r * vpr;
    for (uint32_t v = lane; v < nv; v += 32) {
        asm volatile("cp.async.cg.shared.global [%0], [%1], 16;" ::"r"(stage + 16 * v),
                     "l"(src + r * src_stride + 16ull * c)
                     : "memory");
        c += dr;
        r += dq;
        if (c >= vpr) {
            c -= vpr;
            ++r;
        }
    }
    asm volatile("cp.async.mbarrier.arrive.shared::cta.b64 [%0];" ::"r"(full_bar) : "memory");
}

template <int NPTR>
__device__ __forceinline__ char* bulk_bucket(const BulkArgs<NPTR>& a, uint32_t b, int table_base) {
    return a.bucket_stride ? a.bucket_base + (uint64_t)b * a.bucket_stride
                           : (char*)a.ptr[table_base + (b - a.bucket_lo)];
}

// MODE 0: pack, 1: unpack, 2: unpack with checksum comparison.  CHECK: check
// every item against the plan's buffers first (the check_items option).  F16
// (pack only): the rollout's elements are float16, else bfloat16.
template <int NPTR, int MODE, bool CHECK, bool F16>
__global__ void __launch_bounds__(BulkShape<MODE>::kThreads, 1) rr_bulk_kernel(const __grid_constant__ BulkArgs<NPTR> a) {
    static_assert(MODE == 0 || !F16, "the destination type matters to the pack only");
    using D = DstCast<F16>;
    constexpr int kConsumerWarps = BulkShape<MODE>::kWarps;
    constexpr int kStageBytes = BulkShape<MODE>::kStageBytes;
    constexpr int kStages = BulkShape<MODE>::kStages;
    extern __shared__ __align__(128) char stage_mem[];
    __shared__ __align__(8) uint64_t full[kStages], empty[kStages];
    __shared__ Piece meta[kStages];
    __shared__ rr_pack_item fan_dst[MODE == 0 ? kStages : 1][kMaxFanDst];   // PC_FAN slices
    __shared__ bool last_block;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    constexpr bool kSum = MODE != 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&full[s])) : "memory");
            asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_u32(&empty[s])),
                         "n"(kConsumerWarps)
                         : "memory");
        }
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
        // Programmatic dependent launch: the next kernel on the stream may be
        // scheduled now; it still waits for this grid's completion before it
        // touches memory (its griddepcontrol.wait below).
        asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
    }
    __syncthreads();

    // The plan's tables are immutable: read them before the wait.
    uint32_t i0 = 0, i1 = 0;
    if (!a.claim)
        block_items(a.block_first, a.weight_prefix, a.item_begin, a.item_end, &i0, &i1);
    else if (blockIdx.x < a.n_units) {
        i0 = a.block_first[blockIdx.x];
        i1 = a.block_first[blockIdx.x + 1];
    }
    // Everything else (sources, buckets, tensors, sums, counters) may be the
    // previous kernel's output: wait for it to complete.  A no-op when the
    // launch did not overlap a previous kernel.
    asm volatile("griddepcontrol.wait;" ::: "memory");

    if (warp == 0) {
        // ------------------------------------------------------------ producer
        // The whole warp walks the items in step (every lane decodes the same
        // item).  Each piece completes its stage's full barrier with one
        // arrival by lane 0, made after it wrote the piece's metadata: with the
        // byte count of its bulk copies (expect_tx), or plain.  A gather's lanes
        // have each registered their cp.async copies with the barrier first.
        enum { kMeta = 0, kBulk = 1, kGather = 2 };
        uint32_t count = 0;   // pieces issued
        bool ok = true;
        rr_pack_item fan_mine;   // fan-out head: lane l's destination item (l < its count)
        auto emit = [&](const Piece& p, int how) {
            const int s = (int)(count % kStages);
            if (count >= (uint32_t)kStages &&
                !__all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&empty[s]),
                                                   ((count / kStages) - 1) & 1, a.err))) {
                ok = false;
                return;
            }
            const uint32_t fb = smem_u32(&full[s]);
            if constexpr (MODE == 0) {
                // A fan-out piece carries its destination items in shared memory
                // (each lane's from registers: loaded once per head, not per piece).
                if (p.kind == PC_FAN && lane < p.n) fan_dst[s][lane] = fan_mine;
            }
            const uint32_t stage = smem_u32(stage_mem + s * kStageBytes);
            const uint32_t row_bytes = p.row_len * p.es;
            if (how == kGather) gather_async(stage, fb, p.src, p.src_stride, p.rows, row_bytes, lane);
            __syncwarp();
            if (lane != 0) {
                ++count;
                return;
            }
            meta[s] = p;
            if (how == kBulk) {
                asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(fb),
                             "r"(row_bytes * p.rows)
                             : "memory");
                if (p.rows > 1 && p.src_stride == row_bytes)   // rows back to back: one copy
                    asm volatile(
                        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
                        "[%0], [%1], %2, [%3];" ::"r"(stage),
                        "l"(p.src), "r"(row_bytes * p.rows), "r"(fb)
                        : "memory");
                else
                    for (uint32_t r = 0; r < p.rows; ++r)
                        asm volatile(
                            "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes "
                            "[%0], [%1], %2, [%3];" ::"r"(stage + r * row_bytes),
                            "l"(p.src + r * p.src_stride), "r"(row_bytes), "r"(fb)
                            : "memory");
            } else {
                mbar_arrive(fb);
            }
            ++count;
        };
        // Past its own range a block claims units while any are left, the next
        // claim in flight (lane 0) while the current unit is walked.
        unsigned long long pending = 0;
        bool claimed = false;
        auto next_range = [&](uint32_t* it) -> bool {
            if (!a.claim) return false;
            if (!claimed && lane == 0) pending = atomicAdd(a.claim, 1ull);
            claimed = true;
            const unsigned long long u = gridDim.x + __shfl_sync(0xFFFFFFFFu, pending, 0);
            if (u >= a.n_units) return false;
            if (lane == 0) pending = atomicAdd(a.claim, 1ull);
            *it = a.block_first[u];
            i1 = a.block_first[u + 1];
            return true;
        };
        // Work items pass through a window: lane l holds item win + l (one
        // coalesced 32-byte load per lane) and item win + 32 + l is already in
        // flight, so the walk reads an item with shuffles rather than waiting
        // on a dependent global load for every item.  A jump (a claimed unit)
        // reloads both halves.
        uint32_t win = 0xFFFFFFFFu;
        uint4 w0 = make_uint4(0, 0, 0, 0), w1 = w0, n0 = w0, n1 = w0;
        auto load_words = [&](uint32_t i, uint4& x0, uint4& x1) {
            if (i < a.n_items) {
                const uint4* q = (const uint4*)((const char*)a.items + 32ull * i);
                x0 = __ldg(q);
                x1 = __ldg(q + 1);
            }
        };
        auto window_to = [&](uint32_t at) {   // warp-uniform: win <= at < win + 32
            if (win != 0xFFFFFFFFu && at - win < 32u) return;
            if (win != 0xFFFFFFFFu && at - win < 64u) {
                w0 = n0;
                w1 = n1;
                win += 32;
            } else {
                win = at;
                load_words(win + lane, w0, w1);
            }
            load_words(win + 32 + lane, n0, n1);
        };
        for (uint32_t it = i0; ok; ++it) {
            if (it >= i1) {
                bool more = true;
                while (more && it >= i1) more = next_range(&it);
                if (!more) break;
            }
            window_to(it);
            Piece p;
            p.dst = nullptr;
            p.src_stride = 0;
            if (MODE == 0) {
                ItemWords<rr_pack_item> di;
                shfl_words(w0, w1, (int)(it - win), di.w[0], di.w[1]);
                const rr_pack_item d = di.item;
                if (CHECK && !pack_item_ok(a.chk, d)) {
                    if (d.kind == RR_ITEM_FAN_F32 || d.kind == RR_ITEM_FAN_BF16)
                        it += min(d.dst_off, i1 - 1 - it);   // and its destinations
                    continue;
                }
                char* dst = bulk_bucket(a, d.bucket, a.n_shards) + d.dst_off;
                const char* src = (const char*)a.ptr[d.src >> 48] + (d.src & 0xFFFFFFFFFFFFull);
                p.sum_bucket = d.bucket;
                if (d.kind == RR_ITEM_F32_VEC || d.kind == RR_ITEM_BF16_VEC) {
                    const uint32_t es = d.kind == RR_ITEM_F32_VEC ? 4 : 2;
                    const uint32_t L = d.row_len, R = d.n_rows;
                    const uint64_t sstride = (uint64_t)d.src_stride * es;
                    p.kind = es == 4 ? PC_CAST : PC_COPY;
                    p.es = (uint16_t)es;
                    if (R == 1 || L * es > (uint32_t)kStageBytes) {
                        const uint32_t step = kStageBytes / es;
                        for (uint32_t r = 0; r < R && ok; ++r)
                            for (uint32_t e0 = 0; e0 < L && ok; e0 += step) {
                                p.n = min(step, L - e0);
                                p.rows = 1;
                                p.row_len = p.n;
                                p.src = src + r * sstride + (uint64_t)e0 * es;
                                p.dst = dst + 2ull * ((uint64_t)r * L + e0);
                                p.sum_off = d.dst_off + 2u * (r * L + e0);
                                emit(p, kBulk);
                            }
                    } else {
                        // Whole rows per stage.  Rows under kMinBulkRowBytes are gathered
                        // by the warp's 16-byte cp.async copies (one bulk copy per short
                        // row would leave a single issuing lane the bottleneck).
                        const int how = L * es < kMinBulkRowBytes ? kGather : kBulk;
                        const uint32_t k = kStageBytes / (L * es);
                        for (uint32_t r0 = 0; r0 < R && ok; r0 += k) {
                            p.rows = min(k, R - r0);
                            p.row_len = L;
                            p.n = p.rows * L;
                            p.src_stride = sstride;
                            p.src = src + r0 * sstride;
                            p.dst = dst + 2ull * r0 * L;
                            p.sum_off = d.dst_off + 2u * r0 * L;
                            emit(p, how);
                        }
                    }
                } else if (d.kind == RR_ITEM_FAN_F32 || d.kind == RR_ITEM_FAN_BF16) {
                    // Whole rows of the slices' span, staged once; the destination
                    // items that follow the head are read by the consumers.
                    const uint32_t es = d.kind == RR_ITEM_FAN_F32 ? 4 : 2;
                    const uint32_t rb = d.row_len * es, R = d.n_rows, nd = d.dst_off;
                    const uint64_t sstride = (uint64_t)d.src_stride * es;
                    // The planner guarantees the alignments the vector paths need;
                    // a table that breaks them is refused, not run.
                    bool bad = rb > (uint32_t)kStageBytes || rb % 16 != 0 || nd > kMaxFanDst ||
                               it + 1 + nd > i1 || (uintptr_t)src % 16 != 0 || sstride % 16 != 0;
                    // Lane l's destination is item it + 1 + l: in this window or
                    // the next (it - win < 32 and nd <= kMaxFanDst).
                    {
                        const uint32_t k = it + 1 + min((uint32_t)lane, nd > 0 ? nd - 1 : 0u) - win;
                        ItemWords<rr_pack_item> c, n;
                        shfl_words(w0, w1, (int)(k & 31u), c.w[0], c.w[1]);
                        shfl_words(n0, n1, (int)(k & 31u), n.w[0], n.w[1]);
                        fan_mine = k < 32u ? c.item : n.item;
                    }
                    if (!bad && lane < nd) {
                        const rr_pack_item f = fan_mine;
                        bad = f.kind != RR_ITEM_FAN_DST || f.row_len % 8 != 0 ||
                              f.dst_off % 16 != 0 || (f.src * es) % 16 != 0 ||
                              f.src + f.row_len > d.row_len || f.n_rows != R ||
                              (CHECK && !pack_item_in(a.chk, f));
                    }
                    if (__any_sync(0xFFFFFFFFu, bad)) {
                        if (lane == 0) atomicExch(a.err, kErrBadItem);
                        ok = false;
                        break;
                    }
                    const int how = rb < kMinBulkRowBytes ? kGather : kBulk;
                    const uint32_t k = kStageBytes / rb;
                    p.kind = PC_FAN;
                    p.es = (uint16_t)es;
                    p.row_len = d.row_len;
                    p.src_stride = sstride;
                    p.sum_bucket = it + 1;   // index of the first destination item
                    p.n = nd;
                    for (uint32_t r0 = 0; r0 < R && ok; r0 += k) {
                        p.rows = min(k, R - r0);
                        p.src = src + r0 * sstride;
                        p.sum_off = r0;      // first row of this piece within the item
                        emit(p, how);
                    }
                    it += nd;
                } else if (d.kind == RR_ITEM_ZERO_VEC || d.kind == RR_ITEM_ZERO_SCALAR) {
                    p.kind = d.kind == RR_ITEM_ZERO_VEC ? PC_ZERO_VEC : PC_ZERO_SCALAR;
                    p.dst = dst;
                    p.n = d.row_len;
                    p.rows = 1;
                    p.row_len = d.row_len;
                    p.es = 2;
                    p.src = nullptr;
                    p.sum_off = d.dst_off;
                    emit(p, kMeta);
                } else {
                    p.kind = PC_SCALAR;
                    p.es = d.kind == RR_ITEM_F32_SCALAR ? 4 : 2;
                    p.src = src;
                    p.dst = dst;
                    p.rows = d.n_rows;
                    p.row_len = d.row_len;
                    p.n = d.row_len * d.n_rows;
                    p.src_stride = (uint64_t)d.src_stride * p.es;
                    p.sum_off = d.dst_off;
                    emit(p, kMeta);
                }
            } else {
                ItemWords<rr_unpack_item> di;
                shfl_words(w0, w1, (int)(it - win), di.w[0], di.w[1]);
                const rr_unpack_item d = di.item;
                const bool read_only = d.kind == RR_ITEM_READ_VEC || d.kind == RR_ITEM_READ_SCALAR;
                if (MODE == 1 && read_only) continue;
                if (CHECK && !unpack_item_ok(a.chk, d)) continue;
                const char* src = bulk_bucket(a, d.bucket, 0) + d.src_off;
                char* dst = read_only ? nullptr : (char*)a.ptr[a.dst_base + d.tensor] + d.dst_off;
                p.sum_bucket = d.bucket;
                p.es = 2;
                if (d.kind == RR_ITEM_COPY_VEC || d.kind == RR_ITEM_READ_VEC) {
                    p.kind = read_only ? PC_READ : PC_COPY;
                    for (uint32_t o = 0; o < d.nbytes && ok; o += kStageBytes) {
                        const uint32_t len = min((uint32_t)kStageBytes, d.nbytes - o);
                        p.n = len / 2;
                        p.rows = 1;
                        p.row_len = p.n;
                        p.src = src + o;
                        p.dst = dst ? dst + o : nullptr;
                        p.sum_off = d.src_off + o;
                        emit(p, kBulk);
                    }
                } else {
                    p.kind = PC_SCALAR;
                    p.src = src;
                    p.dst = dst;
                    p.n = d.nbytes / 2;
                    p.rows = 1;
                    p.row_len = p.n;
                    p.sum_off = d.src_off;
                    emit(p, kMeta);
                }
            }
        }
        if (ok) {
            Piece end;
            end.kind = PC_END;
            emit(end, kMeta);
        }
        if (!ok && lane == 0) {
            // Let the bulk loads still in flight land before this block's shared
            // memory goes away.
            const uint32_t from = count > (uint32_t)kStages ? count - kStages : 0;
            for (uint32_t c = from; c < count; ++c)
                mbar_wait(smem_u32(&full[c % kStages]), (c / kStages) & 1, a.err);
        }
        asm volatile("cp.async.wait_all;" ::: "memory");
    } else {

    // ---------------------------------------------------------------- consumers
    const uint32_t ct = threadIdx.x - 32;
    constexpr uint32_t kCT = 32 * kConsumerWarps;
    const uint32_t sum_base = MODE == 2 ? (uint32_t)a.first_bucket : 0u;
    unsigned long long acc = 0;
    uint32_t cur = 0xFFFFFFFFu;
    // Fan-out pieces: a warp serves the same slices (so the same buckets) piece
    // after piece, up to kFanSlots of them per piece.  Each slot keeps its
    // lane-local partial sum and bucket, and goes out only when its bucket
    // changes, instead of one warp reduction and atomic per slice and piece.
    constexpr uint32_t kFanUnitsMax =
        kMaxFanDst > 2 * kConsumerWarps - 1 ? kMaxFanDst : 2 * kConsumerWarps - 1;
    constexpr uint32_t kFanSlots = (kFanUnitsMax + kConsumerWarps - 1) / kConsumerWarps;
    unsigned long long fan_acc[kFanSlots];
    uint32_t fan_bucket[kFanSlots];
#pragma unroll
    for (uint32_t j = 0; j < kFanSlots; ++j) {
        fan_acc[j] = 0;
        fan_bucket[j] = 0xFFFFFFFFu;
    }
    bool ok = true;
    for (uint32_t c = 0;; ++c) {
        const int s = (int)(c % kStages);
        ok = __all_sync(0xFFFFFFFFu, mbar_wait(smem_u32(&full[s]), (c / kStages) & 1, a.err));
        if (!ok) break;
        const Piece p = meta[s];
        if (p.kind == PC_END) break;
        if (kSum && p.kind != PC_FAN && p.sum_bucket != cur) {
            if (cur != 0xFFFFFFFFu) flush(a.sums + (cur - sum_base), acc);
            cur = p.sum_bucket;
            acc = 0;
        }
        const char* st = stage_mem + s * kStageBytes;
        const uint32_t nvec = p.n >> 3;
        switch (p.kind) {
            case PC_CAST:
#pragma unroll 4
                for (uint32_t v = ct; v < nvec; v += kCT) {
                    const uint4 x0 = *(const uint4*)(st + 32ull * v);
                    const uint4 x1 = *(const uint4*)(st + 32ull * v + 16);
                    uint4 o;
                    o.x = D::f32x2(x0.x, x0.y);
                    o.y = D::f32x2(x0.z, x0.w);
                    o.z = D::f32x2(x1.x, x1.y);
                    o.w = D::f32x2(x1.z, x1.w);
                    st_stream(p.dst + 16ull * v, o);
                    acc += words(o);
                }
                break;
            case PC_COPY:
            case PC_READ:
#pragma unroll 4
                for (uint32_t v = ct; v < nvec; v += kCT) {
                    const uint4 x = D::bf16x8(*(const uint4*)(st + 16ull * v));
                    if (p.kind == PC_COPY) st_stream(p.dst + 16ull * v, x);
                    if (kSum) acc += words(x);
                }
                break;
            case PC_SCALAR:
                for (uint32_t e = ct; e < p.n; e += kCT) {
                    const uint32_t r = e / p.row_len, cc = e - r * p.row_len;
                    const char* q = p.src + r * p.src_stride + (uint64_t)cc * p.es;
                    const uint16_t h = p.es == 4 ? D::f32(*(const uint32_t*)q)
                                                 : D::bf16(*(const uint16_t*)q);
                    if (p.dst) *(uint16_t*)(p.dst + 2ull * e) = h;
                    if (kSum) acc += (unsigned long long)h << (8 * ((p.sum_off + 2 * e) & 7));
                }
                break;
            case PC_FAN:   // pack only
                if constexpr (MODE == 0) {
                    // Units of work: each slice's 16-byte output vectors in q parts
                    // (q spreads the slices over all consumer warps, whatever the
                    // number of rows staged); one warp per unit.  nd <= kMaxFanDst
                    // (the producer refuses more), so nd * q <= kFanUnitsMax and a
                    // warp takes at most kFanSlots units: unit j of this warp sums
                    // into slot j.
                    const uint32_t nd = p.n;
                    const uint32_t q = (kConsumerWarps + nd - 1) / nd;
#pragma unroll
                    for (uint32_t j = 0; j < kFanSlots; ++j) {
                        const uint32_t u = warp - 1 + j * kConsumerWarps;
                        if (u >= nd * q) break;
                        const rr_pack_item d = fan_dst[s][u / q];
                        if (d.bucket != fan_bucket[j]) {   // warp-uniform
                            if (fan_bucket[j] != 0xFFFFFFFFu)
                                flush(a.sums + fan_bucket[j], fan_acc[j]);
                            fan_bucket[j] = d.bucket;
                            fan_acc[j] = 0;
                        }
                        const uint32_t part = u % q;
                        const uint32_t vpr = d.row_len >> 3, nv_all = p.rows * vpr;
                        const uint32_t v0 = nv_all * part / q, v1 = nv_all * (part + 1) / q;
                        // Lane l starts at vector v0 + l (row r, vector c of the row)
                        // and steps 32 vectors: dq rows and dr vectors at a time.
                        const uint32_t dq = 32 / vpr, dr = 32 - dq * vpr;
                        const char* base = st + (uint32_t)d.src * p.es;
                        char* out = bulk_bucket(a, d.bucket, a.n_shards) + d.dst_off +
                                    2ull * p.sum_off * d.row_len;
                        uint32_t r = (v0 + lane) / vpr, c = (v0 + lane) - r * vpr;
                        unsigned long long am = 0;
                        for (uint32_t v = v0 + lane; v < v1; v += 32) {
                            const char* q8 = base + ((uint64_t)r * p.row_len + 8u * c) * p.es;
                            uint4 o;
                            if (p.es == 4) {
                                const uint4 x0 = *(const uint4*)q8;
                                const uint4 x1 = *(const uint4*)(q8 + 16);
                                o.x = D::f32x2(x0.x, x0.y);
                                o.y = D::f32x2(x0.z, x0.w);
                                o.z = D::f32x2(x1.x, x1.y);
                                o.w = D::f32x2(x1.z, x1.w);
                            } else {
                                o = D::bf16x8(*(const uint4*)q8);
                            }
                            st_stream(out + 16ull * v, o);
                            am += words(o);
                            c += dr;
                            r += dq;
                            if (c >= vpr) {
                                c -= vpr;
                                ++r;
                            }
                        }
                        fan_acc[j] += am;
                    }
                }
                break;
            case PC_ZERO_VEC:
                for (uint32_t v = ct; v < nvec; v += kCT)
                    st_stream(p.dst + 16ull * v, make_uint4(0, 0, 0, 0));
                break;
            default:  // PC_ZERO_SCALAR
                for (uint32_t e = ct; e < p.n; e += kCT) *(uint16_t*)(p.dst + 2ull * e) = 0;
                break;
        }
        __syncwarp();
        if (lane == 0) mbar_arrive(smem_u32(&empty[s]));
    }
    if (kSum && cur != 0xFFFFFFFFu) flush(a.sums + (cur - sum_base), acc);
    if constexpr (MODE == 0) {
#pragma unroll
        for (uint32_t j = 0; j < kFanSlots; ++j)
            if (fan_bucket[j] != 0xFFFFFFFFu) flush(a.sums + fan_bucket[j], fan_acc[j]);
    }
    }   // consumers

    // ------------------------------------------------------------- epilogue
    // Every warp of the block is done: the producer's claims have returned and
    // the consumers' sums are flushed.  The block that takes the last ticket
    // finishes the launch: the verifying unpack compares the sums (and writes
    // the result); a pack through a slot writes its checksums out of the
    // slot's sums; a launch holding a slot leaves it zeroed.
    if (MODE != 2 && !a.reset_claims) return;
    __syncthreads();
    if (threadIdx.x == 0) {
        __threadfence();
        last_block = atomicAdd(&a.counters[0], 1ull) == gridDim.x - 1;
    }
    __syncthreads();
    if (!last_block) return;
    __threadfence();
    constexpr uint32_t kBT = BulkShape<MODE>::kThreads;
    if constexpr (MODE == 2) {
        for (int32_t i = threadIdx.x; i < a.n_buckets; i += kBT) {
            const int32_t b = a.first_bucket + i;
            const unsigned long long got = __ldcg(a.sums + i);
            const bool differs = got != a.expected[b];
            if (a.bad) a.bad[i] = differs ? 1 : 0;
            if (differs) {
                atomicAdd(&a.counters[1], 1ull);
                atomicMax(&a.counters[2], ULLONG_MAX - (unsigned long long)b);
            }
            if (a.reset_claims) a.sums[i] = 0;
        }
        __syncthreads();
        if (threadIdx.x == 0 && a.result) write_result(a.counters, a.result);
    }
    if constexpr (MODE == 0) {
        if (a.sums_out)
            for (int32_t i = threadIdx.x; i < a.n_buckets; i += kBT) {
                const int32_t b = a.first_bucket + i;
                a.sums_out[b] = __ldcg(a.sums + b);
                a.sums[b] = 0;
            }
    }
    if (a.reset_claims) {
        __syncthreads();
        if (threadIdx.x < 4) atomicExch(&a.counters[threadIdx.x], 0ull);
    }
}

// Self-test of the bounded wait: waits on a barrier phase that nothing
// completes; the wait gives up after its limit and marks the error word.
__global__ void rr_wait_selftest_kernel(unsigned int* err) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        asm volatile("mbarrier.init.shared::cta.b64 [%0], 1;" ::"r"(smem_u32(&bar)) : "memory");
        asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    __syncthreads();
    if (threadIdx.x == 0) mbar_wait(smem_u32(&bar), 0, err);
}

template <int NPTR, int MODE, bool CHECK = false, bool F16 = false>
cudaError_t bulk_prepare() {
    return cudaFuncSetAttribute(rr_bulk_kernel<NPTR, MODE, CHECK, F16>,
                                cudaFuncAttributeMaxDynamicSharedMemorySize,
                                BulkShape<MODE>::kSmem);
}

// ---------------------------------------------------------------------------
// Host helpers
// ---------------------------------------------------------------------------

rr_status cuda_fail(cudaError_t e, const char* what) {
    return rr_fail(RR_ECUDA, "%s: %s", what, cudaGetErrorString(e));
}

#define RR_CUDA(call)                                   \
    do {                                                \
        cudaError_t e_ = (call);                        \
        if (e_ != cudaSuccess) return cuda_fail(e_, #call); \
    } while (0)

bool aligned16(const void* p) { return p && ((uintptr_t)p & 15u) == 0; }

// Equally spaced bucket pointers (one allocation cut into buckets)?
bool uniform(const void* const* ptrs, int32_t n, int64_t min_stride, uint64_t* stride) {
    if (n <= 1) {
        *stride = (uint64_t)min_stride;
        return true;
    }
    const intptr_t s = (const char*)ptrs[1] - (const char*)ptrs[0];
    if (s < min_stride) return false;
    for (int32_t i = 2; i < n; ++i)
        if ((const char*)ptrs[i] - (const char*)ptrs[i - 1] != s) return false;
    *stride = (uint64_t)s;
    return true;
}

rr_status check_plan(const rr_plan* P) {
    if (!P) return rr_fail(RR_EINVAL, "plan is NULL");
    if (P->host_only) return rr_fail(RR_EINVAL, "plan was created host-only");
    int dev = -1;
    RR_CUDA(cudaGetDevice(&dev));
    if (dev != P->device)
        return rr_fail(RR_EINVAL, "plan belongs to device %d, current device is %d", P->device, dev);
    return RR_OK;
}

// Whether a kernel of this library may touch memory at p: the current GPU's
// device (or managed) memory, pinned host memory mapped for the device, or -- on a device
// that reads pageable host memory (address translation over the CPU's page
// tables, as on Grace) -- any host memory.  Pageable memory elsewhere would
// fault the GPU, so it is refused.
bool reachable(const void* p, bool pageable_ok) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return pageable_ok;
    }
    if (at.type == cudaMemoryTypeDevice) {   // this GPU's own memory only
        int dev = -1;
        return cudaGetDevice(&dev) == cudaSuccess && at.device == dev;
    }
    if (at.type == cudaMemoryTypeManaged) return true;
    if (at.type == cudaMemoryTypeHost) return at.devicePointer != nullptr;
    return pageable_ok;
}

// Pointer arrays: every entry 16-byte aligned; the first and the last entry
// reachable from the device (arrays are expected to be of one kind of memory).
rr_status check_ptrs(bool pageable_ok, const void* const* ptrs, int32_t n, const char* what) {
    if (n > 0 && !ptrs) return rr_fail(RR_EINVAL, "%s array is NULL", what);
    for (int32_t i = 0; i < n; ++i)
        if (!aligned16(ptrs[i]))
            return rr_fail(RR_EINVAL, "%s[%d] is NULL or not 16-byte aligned", what, i);
    for (int32_t i : {0, n - 1})
        if (n > 0 && !reachable(ptrs[i], pageable_ok))
            return rr_fail(RR_EINVAL,
                           "%s[%d] is memory this GPU cannot reach (pageable host memory, or "
                           "another GPU's); use this GPU's memory or pinned host memory",
                           what, i);
    return RR_OK;
}

// One buffer a kernel reads or writes (checksums, per-bucket flags): 16-byte
// aligned (when `aligned` is asked) and reachable from the device.
rr_status check_buf(bool pageable_ok, const void* p, const char* what, bool aligned = true) {
    if (!p || (aligned && !aligned16(p)))
        return rr_fail(RR_EINVAL, "%s NULL or not 16-byte aligned", what);
    if (!reachable(p, pageable_ok))
        return rr_fail(RR_EINVAL,
                       "%s is memory this GPU cannot reach (pageable host memory, or another "
                       "GPU's); use this GPU's memory or pinned host memory", what);
    return RR_OK;
}

// A call covers buckets [b0, b1).  The full range uses the plan's balanced
// per-block item ranges; a sub-range splits its items evenly over the grid.
struct Range {
    int32_t b0, b1;
    bool full;
    unsigned long long* scratch;   // verify sums and counters of this call (NULL: the plan's)
    int32_t t_lo, t_hi;            // unpack: the destination tensors its pointer table holds
    int32_t sum_b0, sum_n;         // verify: the whole call's range (sums, flags, counters);
                                   // sum_n == 0: this range itself
};

// Where range S's sums, counters and flags live in its call's scratch.
struct SumSlot {
    unsigned long long* sums;
    unsigned long long* counters;
    uint8_t* bad;
};
SumSlot sum_slot(const rr_plan* P, const Range& S, uint8_t* bad) {
    unsigned long long* sc = S.scratch ? S.scratch : P->d_verify_scratch;
    const int32_t b0 = S.sum_n ? S.sum_b0 : S.b0, n = S.sum_n ? S.sum_n : S.b1 - S.b0;
    return {sc + (S.b0 - b0), sc + n, bad ? bad + (S.b0 - b0) : nullptr};
}

// The bounds the kernels check items against, when the plan asks for checks.
ItemBounds bounds_of(const rr_plan* P) {
    ItemBounds b;
    std::memset(&b, 0, sizeof b);
    if (!P->check_items) return b;
    b.src_bytes = P->d_src_bytes;
    b.tensor_bytes = P->d_tensor_bytes;
    b.bucket_bytes = P->bucket_bytes;
    b.n_src = P->n_shards;
    b.n_buckets = P->n_buckets;
    b.n_tensors = P->n_tensors;
    b.err = P->d_error;
    return b;
}

int32_t take_claim_slot(rr_plan* M, cudaStream_t s);
template <int MODE>
void work_units(const rr_plan* P, const Range& R, const uint32_t** first, uint32_t* n);

// The register-path pack instantiation for a launch: item checks, a source in
// host memory, and the destination type.
template <int NPTR, bool F16>
void pack_kernel_for(bool check, bool host_src, int g, cudaStream_t s, const PackArgs<NPTR>& a) {
    if (check && host_src)
        rr_pack_kernel<NPTR, true, true, F16><<<g, kThreads, 0, s>>>(a);
    else if (check)
        rr_pack_kernel<NPTR, true, false, F16><<<g, kThreads, 0, s>>>(a);
    else if (host_src)
        rr_pack_kernel<NPTR, false, true, F16><<<g, kThreads, 0, s>>>(a);
    else
        rr_pack_kernel<NPTR, false, false, F16><<<g, kThreads, 0, s>>>(a);
}

template <int NPTR>
rr_status launch_pack(const rr_plan* P, Range R, const void* const* src, void* const* buckets,
                      uint64_t* checksums, bool table, uint64_t stride, bool host_src,
                      cudaStream_t s) {
    PackArgs<NPTR> a;
    std::memset(&a, 0, sizeof a);
    a.items = P->d_pack_items;
    a.block_first = R.full ? P->d_pack_block_first : nullptr;
    a.weight_prefix = P->d_pack_weight_prefix;
    a.chk = bounds_of(P);
    a.item_begin = P->pack_bucket_first[R.b0];
    a.item_end = P->pack_bucket_first[R.b1];
    a.checksums = (unsigned long long*)checksums;
    a.n_shards = P->n_shards;
    for (int32_t i = 0; i < P->n_shards; ++i) a.ptr[i] = src[i];
    if (table) {
        a.bucket_lo = R.b0;
        for (int32_t b = R.b0; b < R.b1; ++b) a.ptr[P->n_shards + (b - R.b0)] = buckets[b];
    } else {
        a.bucket_base = (char*)buckets[0];
        a.bucket_stride = stride;
    }
    if (P->dst_f16)
        pack_kernel_for<NPTR, true>(P->check_items != 0, host_src, P->reg_pack_grid, s, a);
    else
        pack_kernel_for<NPTR, false>(P->check_items != 0, host_src, P->reg_pack_grid, s, a);
    RR_CUDA(cudaGetLastError());
    return RR_OK;
}

// Verifying form when checksums != NULL (sums and counters in the plan's scratch).
template <int NPTR>
rr_status launch_unpack(const rr_plan* P, Range R, const void* const* buckets, void* const* dst,
                        const uint64_t* checksums, uint8_t* bad, bool table, uint64_t stride,
                        cudaStream_t s, long long* result = nullptr) {
    UnpackArgs<NPTR> a;
    std::memset(&a, 0, sizeof a);
    a.items = P->d_unpack_items;
    a.block_first = R.full ? P->d_unpack_block_first : nullptr;
    a.weight_prefix = P->d_unpack_weight_prefix;
    a.chk = bounds_of(P);
    a.item_begin = P->unpack_bucket_first[R.b0];
    a.item_end = P->unpack_bucket_first[R.b1];
    if (checksums) {
        const SumSlot q = sum_slot(P, R, bad);
        a.sums = q.sums;
        a.counters = q.counters;
        a.expected = (const unsigned long long*)checksums;
        a.bad = q.bad;
        a.first_bucket = R.b0;
        a.n_buckets = R.b1 - R.b0;
        a.result = result;
    }
    int32_t k = 0;
    if (table) {
        a.bucket_lo = R.b0;
        for (int32_t b = R.b0; b < R.b1; ++b) a.ptr[k++] = buckets[b];
    } else {
        a.bucket_base = (const char*)buckets[0];
        a.bucket_stride = stride;
    }
    a.dst_base = k - R.t_lo;   // ptr[dst_base + tensor] for tensors t_lo .. t_hi
    for (int32_t t = R.t_lo; t <= R.t_hi; ++t) a.ptr[k++] = dst[t];
    // Claimed work units (the per-bucket units of R's buckets): the verifying
    // form through the call's scratch counter, zeroed with its sums; the plain
    // form through a pooled slot when one is free, else the fixed split above.
    rr_plan* M = const_cast<rr_plan*>(P);   // the claim pool is mutable state
    std::unique_lock<std::mutex> lock(M->claim_mutex, std::defer_lock);
    int32_t slot = -1;
    if (checksums) {
        a.claim = a.counters + 3;
        work_units<1>(P, R, &a.unit_first, &a.n_units);
    } else {
        lock.lock();
        if ((slot = take_claim_slot(M, s)) >= 0) {
            a.counters = P->d_slots + size_t(slot) * P->slot_words() + P->n_buckets;
            a.claim = a.counters + 3;
            a.reset_claims = 1;
            work_units<1>(P, R, &a.unit_first, &a.n_units);
        }
    }
    constexpr int VT = RegUnpackShape<true>::kBlock;
    if (checksums && P->check_items)
        rr_unpack_kernel<NPTR, true, true><<<P->reg_vunpack_grid, VT, 0, s>>>(a);
    else if (checksums)
        rr_unpack_kernel<NPTR, true, false><<<P->reg_vunpack_grid, VT, 0, s>>>(a);
    else if (P->check_items)
        rr_unpack_kernel<NPTR, false, true><<<P->reg_unpack_grid, kThreads, 0, s>>>(a);
    else
        rr_unpack_kernel<NPTR, false, false><<<P->reg_unpack_grid, kThreads, 0, s>>>(a);
    RR_CUDA(cudaGetLastError());
    cudaError_t e;
    if (slot >= 0 && (e = cudaEventRecord(P->claim_done[slot], s)) != cudaSuccess) {
        M->claim_retired[slot] = 1;   // its launch's end is unknown: never hand it out again
        return cuda_fail(e, "cudaEventRecord");
    }
    return RR_OK;
}

template <int NPTR>
rr_status launch_verify(const rr_plan* P, Range R, const void* const* buckets,
                        const uint64_t* checksums, uint8_t* bad, bool table, uint64_t stride,
                        cudaStream_t s) {
    VerifyArgs<NPTR> a;
    std::memset(&a, 0, sizeof a);
    const int32_t n = R.b1 - R.b0;
    const SumSlot q = sum_slot(P, R, bad);
    a.sums = q.sums;
    a.counters = q.counters;
    a.expected = (const unsigned long long*)checksums;
    a.bad = q.bad;
    a.first_bucket = R.b0;
    a.bucket_bytes = (uint64_t)P->bucket_bytes;
    a.chunk_bytes = (uint64_t)std::min<int64_t>(kVerifyChunk, P->bucket_bytes);
    a.chunks_per_bucket = (a.bucket_bytes + a.chunk_bytes - 1) / a.chunk_bytes;
    a.total_chunks = a.chunks_per_bucket * (uint64_t)n;
    a.n_buckets = n;
    if (table) {
        a.bucket_lo = R.b0;
        for (int32_t b = R.b0; b < R.b1; ++b) a.ptr[b - R.b0] = buckets[b];
    } else {
        a.bucket_base = (const char*)buckets[0];
        a.bucket_stride = stride;
    }
    rr_verify_kernel<NPTR><<<P->verify_grid_blocks, kThreads, 0, s>>>(a);
    RR_CUDA(cudaGetLastError());
    return RR_OK;
}

// The bulk engine reads and writes device memory only; buffers in host memory
// (a snapshot to pinned host buckets) take the register path.  One call's
// arrays are expected to be all device or all host memory: the first and
// last pointer of each array are checked.
bool device_resident(const void* p) {
    cudaPointerAttributes at;
    if (cudaPointerGetAttributes(&at, p) != cudaSuccess) {
        cudaGetLastError();
        return false;
    }
    return at.type == cudaMemoryTypeDevice;
}

bool all_device(const void* const* ptrs, int32_t n) {
    return n == 0 || (device_resident(ptrs[0]) && device_resident(ptrs[n - 1]));
}

// A pooled slot for a launch on `s`, or -1.  A slot whose last launch has
// completed is free.  When none is, the slot handed out longest ago is taken
// if its last launch ran on `s` itself: `s` then waits (on the GPU) for that
// launch's event, which costs nothing since the stream runs its work in order
// anyway.  Otherwise (every slot held by another stream's launch in flight, or
// `s` capturing a graph -- a captured launch replays whenever the graph does)
// there is none.  The caller holds claim_mutex and records claim_done[slot]
// after the launch.  A slot is all zero when handed out: zeroed once at plan
// creation, then by the last block of each launch that held it.
int32_t take_claim_slot(rr_plan* M, cudaStream_t s) {
    cudaStreamCaptureStatus cs = cudaStreamCaptureStatusNone;
    if (cudaStreamIsCapturing(s, &cs) != cudaSuccess) {
        cudaGetLastError();
        return -1;
    }
    if (cs != cudaStreamCaptureStatusNone) return -1;
    // Querying an event is allowed to this thread even while another thread
    // captures a graph.
    cudaStreamCaptureMode mode = cudaStreamCaptureModeRelaxed;
    cudaThreadExchangeStreamCaptureMode(&mode);
    int32_t slot = -1;
    for (int32_t i = 0; i < rr_plan::kClaimSlots && slot < 0; ++i) {
        const int32_t k = (M->claim_next + i) % rr_plan::kClaimSlots;
        if (M->claim_retired[k]) continue;
        const cudaError_t q = cudaEventQuery(M->claim_done[k]);
        if (q == cudaSuccess)
            slot = k;
        else if (q != cudaErrorNotReady)
            cudaGetLastError();
    }
    for (int32_t i = 0; i < rr_plan::kClaimSlots && slot < 0; ++i) {
        const int32_t k = (M->claim_next + i) % rr_plan::kClaimSlots;
        if (M->claim_retired[k] || M->claim_stream[k] != s) continue;
        if (cudaStreamWaitEvent(s, M->claim_done[k], 0) == cudaSuccess)
            slot = k;
        else
            cudaGetLastError();
    }
    cudaThreadExchangeStreamCaptureMode(&mode);
    if (slot >= 0) {
        M->claim_next = (slot + 1) % rr_plan::kClaimSlots;
        M->claim_stream[slot] = s;
    }
    return slot;
}

// The work units of a bulk launch over range R: for a pack over every bucket
// the whole table's (own shares, then claimed), else the per-bucket units of
// R's buckets (all claimed).  Measured on GB300: the fp32 pack (2 bytes read
// per byte written) runs best with long own runs; the 1:1 unpack passes best
// with every unit claimed.
template <int MODE>
void work_units(const rr_plan* P, const Range& R, const uint32_t** first, uint32_t* n) {
    if (MODE == 0 && R.full) {
        *first = P->d_pack_whole_unit_first;
        *n = uint32_t(P->pack_whole_unit_first.size() - 1);
    } else {
        const std::vector<uint32_t>& bu = MODE == 0 ? P->pack_bucket_unit : P->unpack_bucket_unit;
        *first = (MODE == 0 ? P->d_pack_unit_first : P->d_unpack_unit_first) + bu[R.b0];
        *n = bu[R.b1] - bu[R.b0];
    }
}

// How a bulk launch may use the plan's pooled slots, and what it zeroes itself.
struct BulkOpts {
    bool may_slot = true;                 // try a pooled slot (not for the blocking verifies)
    unsigned long long* zero = nullptr;   // without a slot, zero these words first (pack:
    size_t zero_words = 0;                //   the range's checksums; async verify: scratch)
    long long* result = nullptr;          // verifying unpack: write {n_bad, first_bad} here
};

template <int NPTR, int MODE, bool CHECK, bool F16>
cudaError_t launch_bulk_kernel(int32_t grid, cudaStream_t s, const BulkArgs<NPTR>& a) {
    cudaError_t e = bulk_prepare<NPTR, MODE, CHECK, F16>();
    if (e != cudaSuccess) return e;
    // Programmatic dependent launch: this grid's blocks may be scheduled while
    // the previous kernel on the stream drains (they wait for it to complete
    // before touching memory), so the launch latency and prologue overlap it.
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(BulkShape<MODE>::kThreads);
    cfg.dynamicSmemBytes = BulkShape<MODE>::kSmem;
    cfg.stream = s;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, rr_bulk_kernel<NPTR, MODE, CHECK, F16>, a);
}

template <int NPTR, int MODE>
rr_status launch_bulk(const rr_plan* P, Range R, const void* const* src_shards,
                      const void* const* buckets, void* const* dst, const uint64_t* checksums,
                      uint8_t* bad, bool table, uint64_t stride, cudaStream_t s,
                      const BulkOpts& o = BulkOpts()) {
    BulkArgs<NPTR> a;
    std::memset(&a, 0, sizeof a);
    a.err = P->d_error;
    a.chk = bounds_of(P);
    a.first_bucket = R.b0;
    a.n_buckets = R.b1 - R.b0;
    int32_t k = 0;
    if (MODE == 0) {
        a.items = P->d_pack_items;
        a.block_first = R.full ? P->d_pack_block_first : nullptr;
        a.weight_prefix = P->d_pack_weight_prefix;
        a.item_begin = P->pack_bucket_first[R.b0];
        a.item_end = P->pack_bucket_first[R.b1];
        a.n_items = uint32_t(P->pack_items.size());
        if (R.full && P->d_full_items) {   // every bucket: the table with fan-out groups
            a.items = P->d_full_items;
            a.n_items = uint32_t(P->full_items.size());
            a.block_first = P->d_full_block_first;
            a.item_begin = 0;
            a.item_end = uint32_t(P->full_items.size());
        }
        a.sums = (unsigned long long*)checksums;
        a.n_shards = P->n_shards;
        for (int32_t i = 0; i < P->n_shards; ++i) a.ptr[k++] = src_shards[i];
    } else {
        a.items = P->d_unpack_items;
        a.n_items = uint32_t(P->unpack_items.size());
        a.block_first = R.full ? P->d_unpack_block_first : nullptr;
        a.weight_prefix = P->d_unpack_weight_prefix;
        a.item_begin = P->unpack_bucket_first[R.b0];
        a.item_end = P->unpack_bucket_first[R.b1];
    }
    if (table) {   // the range's buckets (a full-range pack: all of them, for fan-out items)
        a.bucket_lo = R.b0;
        for (int32_t b = R.b0; b < R.b1; ++b) a.ptr[k++] = buckets[b];
    } else {
        a.bucket_base = (char*)buckets[0];
        a.bucket_stride = stride;
    }
    if (MODE != 0) {
        a.dst_base = k - R.t_lo;   // ptr[dst_base + tensor] for tensors t_lo .. t_hi
        for (int32_t t = R.t_lo; t <= R.t_hi; ++t) a.ptr[k++] = dst[t];
    }
    const int32_t grid = MODE == 0 ? P->grid_blocks : P->unpack_grid_blocks;
    // A pooled slot when one is free: the launch claims its units through the
    // slot's counter, and pack and the verifying unpack sum into the slot, so
    // nothing needs zeroing first.  Otherwise pack and plain unpack run the
    // fixed split set above, and the verifying unpack uses the call's scratch.
    rr_plan* M = const_cast<rr_plan*>(P);   // the slot pool is mutable state
    std::unique_lock<std::mutex> lock(M->claim_mutex, std::defer_lock);
    int32_t slot = -1;
    if (o.may_slot) {
        lock.lock();
        slot = take_claim_slot(M, s);
    }
    if (slot >= 0) {
        unsigned long long* area = P->d_slots + size_t(slot) * P->slot_words();
        a.counters = area + P->n_buckets;
        a.claim = a.counters + 3;
        a.reset_claims = 1;
        work_units<MODE>(P, R, &a.block_first, &a.n_units);
        if (MODE == 0 && o.zero) {          // the checksums come out of the slot's sums
            a.sums = area;
            a.sums_out = (unsigned long long*)checksums;
        }
        if (MODE == 2) {
            a.sums = area;                  // indexed from the range's first bucket
            a.bad = bad;
        }
    } else {
        if (o.zero) RR_CUDA(cudaMemsetAsync(o.zero, 0, o.zero_words * 8, s));
        if (MODE == 2) {
            const SumSlot q = sum_slot(P, R, bad);
            a.sums = q.sums;
            a.counters = q.counters;
            a.claim = q.counters + 3;       // the call's work units, claimed through counters[3]
            a.bad = q.bad;
            work_units<MODE>(P, R, &a.block_first, &a.n_units);
        }
    }
    if (MODE == 2) {
        a.expected = (const unsigned long long*)checksums;
        a.result = o.result;
    }
    // The float16 instantiations exist for the pack only (F16 = MODE == 0 there).
    constexpr bool kF16 = MODE == 0;
    const cudaError_t e =
        MODE == 0 && P->dst_f16
            ? (P->check_items ? launch_bulk_kernel<NPTR, MODE, true, kF16>(grid, s, a)
                              : launch_bulk_kernel<NPTR, MODE, false, kF16>(grid, s, a))
            : (P->check_items ? launch_bulk_kernel<NPTR, MODE, true, false>(grid, s, a)
                              : launch_bulk_kernel<NPTR, MODE, false, false>(grid, s, a));
    if (e != cudaSuccess) return cuda_fail(e, "bulk kernel launch");
    cudaError_t er;
    if (slot >= 0 && (er = cudaEventRecord(P->claim_done[slot], s)) != cudaSuccess) {
        M->claim_retired[slot] = 1;   // its launch's end is unknown: never hand it out again
        return cuda_fail(er, "cudaEventRecord");
    }
    return RR_OK;
}

// Synchronises `stream` and reports (then clears) the plan's error word.
rr_status read_error(const rr_plan* P, cudaStream_t stream) {
    unsigned int* h = (unsigned int*)(P->h_verify_result + 4);
    RR_CUDA(cudaMemcpyAsync(h, P->d_error, sizeof(unsigned int), cudaMemcpyDeviceToHost, stream));
    RR_CUDA(cudaStreamSynchronize(stream));
    if (*h) {
        const unsigned int code = *h;
        RR_CUDA(cudaMemsetAsync(P->d_error, 0, sizeof(unsigned int), stream));
        RR_CUDA(cudaStreamSynchronize(stream));
        if (code == kErrBadItem)
            return rr_fail(RR_ECUDA, "a kernel of this plan refused a work item outside the "
                                     "plan's buffers; its output is incomplete");
        return rr_fail(RR_ECUDA, "a kernel of this plan gave up waiting (code %u); its output "
                                 "is incomplete", code);
    }
    return RR_OK;
}

rr_status check_range(const rr_plan* P, int32_t first, int32_t n, Range* R) {
    if (first < 0 || n < 0 || first > P->n_buckets || n > P->n_buckets - first)
        return rr_fail(RR_EINVAL, "bucket range [%d, %d + %d) outside [0, %d)", first, first, n,
                       P->n_buckets);
    *R = Range{first, first + n, first == 0 && n == P->n_buckets};
    return RR_OK;
}

rr_status pack_impl(const rr_plan* P, Range R, const void* const* src_shards, void* const* buckets,
                    uint64_t* checksums, cudaStream_t stream) {
    rr_status st;
    if ((st = check_ptrs(P->pageable_ok != 0, src_shards, P->n_shards, "src_shards"))) return st;
    if ((st = check_ptrs(P->pageable_ok != 0, (const void* const*)buckets, P->n_buckets, "buckets"))) return st;
    if (R.b1 == R.b0) return RR_OK;
    if ((st = check_buf(P->pageable_ok != 0, checksums, "checksums"))) return st;
    uint64_t stride = 0;
    const bool table = !uniform((const void* const*)buckets, P->n_buckets, P->bucket_bytes, &stride);
    // Separately allocated buckets go through the pointer table after the
    // shards: a range with more of them than fit runs as several launches
    // over consecutive bucket ranges (on the bucket-sorted table).
    const int32_t cap = kLargePtrs - P->n_shards;
    if (table && cap < 1)
        return rr_fail(RR_EINVAL,
                       "%d source buffers leave no room for separately allocated buckets in one "
                       "launch's %d pointers; allocate the buckets as one equally spaced block",
                       P->n_shards, kLargePtrs);
    const bool src_device = all_device(src_shards, P->n_shards);
    const bool bulk = P->engine == RR_ENGINE_AUTO && src_device &&
                      all_device((const void* const*)buckets, P->n_buckets);
    const int32_t step = table ? cap : R.b1 - R.b0;
    const bool empty = P->pack_bucket_first[R.b0] == P->pack_bucket_first[R.b1];
    // One bulk launch writes the range's checksums itself (out of a pooled
    // slot's sums, or after zeroing them when no slot is free); otherwise they
    // are zeroed here and every launch adds into them.
    BulkOpts o;
    if (bulk && !empty && step >= R.b1 - R.b0) {
        o.zero = (unsigned long long*)checksums + R.b0;
        o.zero_words = size_t(R.b1 - R.b0);
    } else {
        RR_CUDA(cudaMemsetAsync(checksums + R.b0, 0, size_t(R.b1 - R.b0) * 8, stream));
    }
    if (empty) return RR_OK;
    for (int32_t b = R.b0; b < R.b1; b += step) {
        const int32_t e = std::min(R.b1, b + step);
        const bool whole = R.full && b == R.b0 && e == R.b1;
        const Range S{b, e, whole && (bulk || P->engine == RR_ENGINE_REGISTERS)};
        const int32_t need = P->n_shards + (table ? e - b : 0);
        if (P->pack_bucket_first[b] == P->pack_bucket_first[e]) continue;
        if (bulk)
            st = need <= kSmallPtrs
                     ? launch_bulk<kSmallPtrs, 0>(P, S, src_shards, (const void* const*)buckets,
                                                  nullptr, checksums, nullptr, table, stride, stream,
                                                  o)
                     : launch_bulk<kLargePtrs, 0>(P, S, src_shards, (const void* const*)buckets,
                                                  nullptr, checksums, nullptr, table, stride, stream,
                                                  o);
        else
            st = need <= kSmallPtrs
                     ? launch_pack<kSmallPtrs>(P, S, src_shards, buckets, checksums, table, stride,
                                               !src_device, stream)
                     : launch_pack<kLargePtrs>(P, S, src_shards, buckets, checksums, table, stride,
                                               !src_device, stream);
        if (st) return st;
    }
    return RR_OK;
}

rr_status check_dst(const rr_plan* P, void* const* dst) {
    if (P->n_tensors > 0 && !dst) return rr_fail(RR_EINVAL, "dst array is NULL");
    for (int32_t t = 0; t < P->n_tensors; ++t)
        if (P->tensor_numel[t] > 0 && !aligned16(dst[t]))
            return rr_fail(RR_EINVAL, "dst[%d] is NULL or not 16-byte aligned", t);
    for (int32_t t : {0, P->n_tensors - 1})
        if (P->n_tensors > 0 && P->tensor_numel[t] > 0 && !reachable(dst[t], P->pageable_ok != 0))
            return rr_fail(RR_EINVAL,
                           "dst[%d] is memory this GPU cannot reach (pageable host memory, or "
                           "another GPU's); use this GPU's memory or pinned host memory",
                           t);
    return RR_OK;
}

// The sub-ranges of R that unpack launches take: runs of buckets whose
// destination-tensor window, with the bucket pointers of a table launch, fits
// one launch's pointer table.  Usually R itself.
rr_status unpack_windows(const rr_plan* P, Range R, bool table, std::vector<Range>* out) {
    out->clear();
    for (int32_t b = R.b0; b < R.b1;) {
        int32_t lo = INT32_MAX, hi = -1, e = b;
        for (; e < R.b1; ++e) {
            const int32_t nlo = std::min(lo, P->bucket_tensor_lo[e]);
            const int32_t nhi = std::max(hi, P->bucket_tensor_hi[e]);
            const int32_t need = (table ? e - b + 1 : 0) + (nhi >= nlo ? nhi - nlo + 1 : 0);
            if (need > kLargePtrs) break;
            lo = nlo;
            hi = nhi;
        }
        if (e == b)
            return rr_fail(RR_EINVAL,
                           "bucket %d writes %d destination tensors; one launch addresses at "
                           "most %d pointers",
                           b, P->bucket_tensor_hi[b] - P->bucket_tensor_lo[b] + 1, kLargePtrs);
        if (hi < lo) lo = 0, hi = -1;   // gap and tail bytes only
        out->push_back(Range{b, e, R.full && b == R.b0 && e == R.b1, R.scratch, lo, hi,
                             R.b0, R.b1 - R.b0});
        b = e;
    }
    return RR_OK;
}

// How one unpack-type call addresses its buffers, and the sub-ranges it is
// launched over.
struct UnpackShape {
    bool table;              // buckets through the pointer table (not equally spaced)
    uint64_t stride;         // otherwise bucket b at buckets[0] + b * stride
    std::vector<Range> parts;
};

rr_status unpack_shape(const rr_plan* P, Range R, const void* const* buckets, UnpackShape* sh) {
    sh->stride = 0;
    sh->table = !uniform(buckets, P->n_buckets, P->bucket_bytes, &sh->stride);
    return unpack_windows(P, R, sh->table, &sh->parts);
}

// One unpack launch (MODE 1, or 2 when checksums are given) over sub-range S,
// on the bulk engine or the register path.
rr_status launch_unpack_part(const rr_plan* P, const Range& S, bool bulk,
                             const void* const* buckets, void* const* dst,
                             const uint64_t* checksums, uint8_t* bad, const UnpackShape& sh,
                             cudaStream_t stream, const BulkOpts& o = BulkOpts()) {
    const bool small = (S.t_hi - S.t_lo + 1) + (sh.table ? S.b1 - S.b0 : 0) <= kSmallPtrs;
    if (bulk) {
        if (checksums)
            return small ? launch_bulk<kSmallPtrs, 2>(P, S, nullptr, buckets, dst, checksums, bad,
                                                      sh.table, sh.stride, stream, o)
                         : launch_bulk<kLargePtrs, 2>(P, S, nullptr, buckets, dst, checksums, bad,
                                                      sh.table, sh.stride, stream, o);
        return small ? launch_bulk<kSmallPtrs, 1>(P, S, nullptr, buckets, dst, nullptr, nullptr,
                                                  sh.table, sh.stride, stream)
                     : launch_bulk<kLargePtrs, 1>(P, S, nullptr, buckets, dst, nullptr, nullptr,
                                                  sh.table, sh.stride, stream);
    }
    // The register path's balanced split is the plan's only when it was made for
    // the register grid.
    Range Sr = S;
    Sr.full = S.full && P->engine == RR_ENGINE_REGISTERS;
    return small ? launch_unpack<kSmallPtrs>(P, Sr, buckets, dst, checksums, bad, sh.table,
                                             sh.stride, stream, o.result)
                 : launch_unpack<kLargePtrs>(P, Sr, buckets, dst, checksums, bad, sh.table,
                                             sh.stride, stream, o.result);
}

rr_status unpack_impl(const rr_plan* P, Range R, const void* const* buckets, void* const* dst,
                      cudaStream_t stream) {
    rr_status st;
    if ((st = check_ptrs(P->pageable_ok != 0, buckets, P->n_buckets, "buckets"))) return st;
    if ((st = check_dst(P, dst))) return st;
    if (P->unpack_bucket_first[R.b0] == P->unpack_bucket_first[R.b1]) return RR_OK;
    const bool bulk = P->engine == RR_ENGINE_AUTO && all_device(buckets, P->n_buckets) &&
                      all_device((const void* const*)dst, P->n_tensors);
    UnpackShape sh;
    if ((st = unpack_shape(P, R, buckets, &sh))) return st;
    for (const Range& S : sh.parts)
        if ((st = launch_unpack_part(P, S, bulk, buckets, dst, nullptr, nullptr, sh, stream)))
            return st;
    return RR_OK;
}

rr_status read_error(const rr_plan* P, cudaStream_t stream);

rr_status read_result(const rr_plan* P, int32_t n, int64_t* n_bad, int64_t* first_bad,
                      cudaStream_t stream) {
    RR_CUDA(cudaMemcpyAsync(P->h_verify_result, P->d_verify_scratch + n,
                            4 * sizeof(unsigned long long), cudaMemcpyDeviceToHost, stream));
    rr_status st = read_error(P, stream);
    if (st) return st;
    const unsigned long long nb = P->h_verify_result[1];
    if (n_bad) *n_bad = (int64_t)nb;
    if (first_bad) *first_bad = nb ? (int64_t)(ULLONG_MAX - P->h_verify_result[2]) : -1;
    return nb ? RR_EMISMATCH : RR_OK;
}

// Enqueues the verifying unpack of range R.  The stream-ordered form (R has
// the caller's scratch) in one bulk launch sums into a pooled slot when one is
// free, zeroing nothing first; otherwise the range's sums and counters
// (R.scratch, else the plan's) are zeroed, then one fused launch per sub-range
// (usually one) runs.  Sub-launches share the call's counters; each compares
// its own buckets, and the "last block" ticket and the unit claims are reset
// between them.  `result` (device address or NULL) receives {n_bad,
// first_bad} from the last launch's last block.
rr_status enqueue_unpack_verify(const rr_plan* P, Range R, const void* const* buckets,
                                const uint64_t* checksums, void* const* dst, uint8_t* bad,
                                cudaStream_t stream, long long* result = nullptr) {
    const int32_t n = R.b1 - R.b0;
    unsigned long long* sc = R.scratch ? R.scratch : P->d_verify_scratch;
    UnpackShape sh;
    rr_status st = unpack_shape(P, R, buckets, &sh);
    if (st) return st;
    const bool bulk = P->engine == RR_ENGINE_AUTO && all_device(buckets, P->n_buckets) &&
                      all_device((const void* const*)dst, P->n_tensors);
    if (bulk && R.scratch && sh.parts.size() == 1) {
        BulkOpts o;
        o.zero = sc;
        o.zero_words = size_t(n) + 4;
        o.result = result;
        return launch_unpack_part(P, sh.parts[0], bulk, buckets, dst, checksums, bad, sh, stream,
                                  o);
    }
    RR_CUDA(cudaMemsetAsync(sc, 0, (size_t(n) + 4) * sizeof(unsigned long long), stream));
    for (size_t i = 0; i < sh.parts.size(); ++i) {
        if (i > 0) {   // a fresh "last block" ticket and unit claims
            RR_CUDA(cudaMemsetAsync(sc + n, 0, sizeof(unsigned long long), stream));
            RR_CUDA(cudaMemsetAsync(sc + n + 3, 0, sizeof(unsigned long long), stream));
        }
        BulkOpts o;
        o.may_slot = false;
        o.result = i + 1 == sh.parts.size() ? result : nullptr;
        if ((st = launch_unpack_part(P, sh.parts[i], bulk, buckets, dst, checksums, bad, sh,
                                     stream, o)))
            return st;
    }
    return RR_OK;
}

rr_status check_unpack_verify_args(const rr_plan* P, Range R, const void* const* buckets,
                                   const uint64_t* checksums, void* const* dst,
                                   const uint8_t* bad) {
    rr_status st;
    if ((st = check_ptrs(P->pageable_ok != 0, buckets, P->n_buckets, "buckets"))) return st;
    if ((st = check_dst(P, dst))) return st;
    if (R.b1 > R.b0 && (st = check_buf(P->pageable_ok != 0, checksums, "checksums"))) return st;
    if (R.b1 > R.b0 && bad && (st = check_buf(P->pageable_ok != 0, bad, "bad", false))) return st;
    return RR_OK;
}

rr_status unpack_verify_impl(const rr_plan* P, Range R, const void* const* buckets,
                             const uint64_t* checksums, void* const* dst, uint8_t* bad,
                             int64_t* n_bad, int64_t* first_bad, cudaStream_t stream) {
    rr_status st = check_unpack_verify_args(P, R, buckets, checksums, dst, bad);
    if (st) return st;
    if (n_bad) *n_bad = 0;
    if (first_bad) *first_bad = -1;
    if (R.b1 == R.b0) return RR_OK;
    rr_plan* M = const_cast<rr_plan*>(P);   // the scratch area is the only mutable state
    std::lock_guard<std::mutex> lock(M->verify_mutex);
    if ((st = enqueue_unpack_verify(P, R, buckets, checksums, dst, bad, stream))) return st;
    return read_result(P, R.b1 - R.b0, n_bad, first_bad, stream);
}

// {n_bad, first_bad or -1} from a verifying pass's counters (NULL: an empty range).
__global__ void rr_verify_result_kernel(const unsigned long long* counters, long long* result) {
    const unsigned long long nb = counters ? counters[1] : 0ull;
    result[0] = (long long)nb;
    result[1] = nb ? (long long)(ULLONG_MAX - counters[2]) : -1ll;
}

// The device address of a result buffer: device memory, or pinned (mapped)
// host memory; NULL for anything else (pageable host memory).
long long* result_address(int64_t* result) {
    cudaPointerAttributes at;
    if (!result || (uintptr_t)result % 8 != 0 || cudaPointerGetAttributes(&at, result) != cudaSuccess) {
        cudaGetLastError();
        return nullptr;
    }
    if (at.type == cudaMemoryTypeDevice || at.type == cudaMemoryTypeManaged)
        return (long long*)result;
    if (at.type == cudaMemoryTypeHost && at.devicePointer) return (long long*)at.devicePointer;
    return nullptr;
}

rr_status verify_impl(const rr_plan* P, Range R, const void* const* buckets,
                      const uint64_t* checksums, uint8_t* bad, int64_t* n_bad, int64_t* first_bad,
                      cudaStream_t stream) {
    rr_status st;
    if ((st = check_ptrs(P->pageable_ok != 0, buckets, P->n_buckets, "buckets"))) return st;
    if (R.b1 > R.b0 && (st = check_buf(P->pageable_ok != 0, checksums, "checksums"))) return st;
    if (R.b1 > R.b0 && bad && (st = check_buf(P->pageable_ok != 0, bad, "bad", false))) return st;
    if (n_bad) *n_bad = 0;
    if (first_bad) *first_bad = -1;
    if (R.b1 == R.b0) return RR_OK;
    uint64_t stride = 0;
    const bool table = !uniform(buckets, P->n_buckets, P->bucket_bytes, &stride);

    rr_plan* M = const_cast<rr_plan*>(P);   // the scratch area is the only mutable state
    std::lock_guard<std::mutex> lock(M->verify_mutex);
    const int32_t n = R.b1 - R.b0;
    RR_CUDA(cudaMemsetAsync(P->d_verify_scratch, 0, (size_t(n) + 4) * sizeof(unsigned long long),
                            stream));
    // Separately allocated buckets: one launch per run of buckets that fits the
    // pointer table, sharing the call's counters (ticket reset in between).
    const int32_t step = table ? kLargePtrs : n;
    for (int32_t b = R.b0; b < R.b1; b += step) {
        const int32_t e = std::min(R.b1, b + step);
        if (b > R.b0)
            RR_CUDA(cudaMemsetAsync(P->d_verify_scratch + n, 0, sizeof(unsigned long long), stream));
        const Range S{b, e, false, nullptr, 0, -1, R.b0, n};
        st = (!table || e - b <= kSmallPtrs)
                 ? launch_verify<kSmallPtrs>(P, S, buckets, checksums, bad, table, stride, stream)
                 : launch_verify<kLargePtrs>(P, S, buckets, checksums, bad, table, stride, stream);
        if (st) return st;
    }
    return read_result(P, n, n_bad, first_bad, stream);
}

}  // namespace

// ---------------------------------------------------------------------------
// Plan device state
// ---------------------------------------------------------------------------

rr_status rr_device_default_grid(rr_grids* g) {
    int dev = 0, sms = 0, p = 0, u = 0, vu = 0, v = 0, b = 0;
    RR_CUDA(cudaGetDevice(&dev));
    RR_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&p, rr_pack_kernel<kLargePtrs, false, false, false>, kThreads, 0));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&u, rr_unpack_kernel<kLargePtrs, false, false>, kThreads, 0));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(
        &vu, rr_unpack_kernel<kLargePtrs, true, false>, RegUnpackShape<true>::kBlock, 0));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&v, rr_verify_kernel<kLargePtrs>, kThreads, 0));
    int bp = 0;
    RR_CUDA((bulk_prepare<kLargePtrs, 0>()));
    RR_CUDA((bulk_prepare<kLargePtrs, 2>()));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&bp, rr_bulk_kernel<kLargePtrs, 0, false, false>,
                                                          BulkShape<0>::kThreads,
                                                          BulkShape<0>::kSmem));
    RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(&b, rr_bulk_kernel<kLargePtrs, 2, false, false>,
                                                          BulkShape<2>::kThreads,
                                                          BulkShape<2>::kSmem));
    g->reg_pack = sms * (p > 0 ? p : 1);
    g->reg_unpack = sms * (u > 0 ? u : 1);
    g->reg_vunpack = sms * (vu > 0 ? vu : 1);
    g->verify = sms * (v > 0 ? v : 1);
    g->bulk_pack = sms * (bp > 0 ? bp : 1);
    g->bulk_unpack = sms * (b > 0 ? b : 1);
    return RR_OK;
}

rr_status rr_device_upload(rr_plan* P) {
    RR_CUDA(cudaGetDevice(&P->device));
    int pageable = 0;
    RR_CUDA(cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, P->device));
    P->pageable_ok = pageable;
    auto up = [](void** d, const void* h, size_t bytes) -> cudaError_t {
        cudaError_t e = cudaMalloc(d, bytes ? bytes : 16);
        if (e != cudaSuccess) return e;
        return bytes ? cudaMemcpy(*d, h, bytes, cudaMemcpyHostToDevice) : cudaSuccess;
    };
    std::vector<int64_t> src_bytes(size_t(P->n_shards) + 1, 0), tensor_bytes;
    rr_plan_source_buffers(P, nullptr, src_bytes.data());
    for (int32_t i = 0; i < P->n_tensors; ++i) tensor_bytes.push_back(2 * P->tensor_numel[i]);
    cudaError_t e;
    if ((e = up((void**)&P->d_pack_items, P->pack_items.data(),
                P->pack_items.size() * sizeof(rr_pack_item))) != cudaSuccess ||
        (e = up((void**)&P->d_pack_block_first, P->pack_block_first.data(),
                P->pack_block_first.size() * sizeof(uint32_t))) != cudaSuccess ||
        (e = up((void**)&P->d_unpack_items, P->unpack_items.data(),
                P->unpack_items.size() * sizeof(rr_unpack_item))) != cudaSuccess ||
        (e = up((void**)&P->d_unpack_block_first, P->unpack_block_first.data(),
                P->unpack_block_first.size() * sizeof(uint32_t))) != cudaSuccess ||
        (e = up((void**)&P->d_unpack_unit_first, P->unpack_unit_first.data(),
                P->unpack_unit_first.size() * sizeof(uint32_t))) != cudaSuccess ||
        (e = up((void**)&P->d_pack_unit_first, P->pack_unit_first.data(),
                P->pack_unit_first.size() * sizeof(uint32_t))) != cudaSuccess ||
        (e = up((void**)&P->d_pack_whole_unit_first, P->pack_whole_unit_first.data(),
                P->pack_whole_unit_first.size() * sizeof(uint32_t))) != cudaSuccess ||
        (e = cudaMalloc((void**)&P->d_slots, rr_plan::kClaimSlots * P->slot_words() *
                                                 sizeof(unsigned long long))) != cudaSuccess ||
        (e = cudaMemset(P->d_slots, 0, rr_plan::kClaimSlots * P->slot_words() *
                                           sizeof(unsigned long long))) != cudaSuccess ||
        (e = cudaMalloc((void**)&P->d_verify_scratch,
                        (size_t(P->n_buckets) + 4) * sizeof(unsigned long long))) != cudaSuccess ||
        (e = cudaHostAlloc((void**)&P->h_verify_result, 5 * sizeof(unsigned long long),
                           cudaHostAllocDefault)) != cudaSuccess ||
        (e = cudaMalloc((void**)&P->d_error, sizeof(unsigned int))) != cudaSuccess ||
        (e = cudaMemset(P->d_error, 0, sizeof(unsigned int))) != cudaSuccess ||
        (e = up((void**)&P->d_pack_weight_prefix, P->pack_weight_prefix.data(),
                P->pack_weight_prefix.size() * sizeof(unsigned long long))) != cudaSuccess ||
        (e = up((void**)&P->d_unpack_weight_prefix, P->unpack_weight_prefix.data(),
                P->unpack_weight_prefix.size() * sizeof(unsigned long long))) != cudaSuccess ||
        (P->check_items &&
         ((e = up((void**)&P->d_src_bytes, src_bytes.data(), src_bytes.size() * 8)) != cudaSuccess ||
          (e = up((void**)&P->d_tensor_bytes, tensor_bytes.data(), tensor_bytes.size() * 8)) !=
              cudaSuccess)) ||
        (!P->full_items.empty() &&
         ((e = up((void**)&P->d_full_items, P->full_items.data(),
                  P->full_items.size() * sizeof(rr_pack_item))) != cudaSuccess ||
          (e = up((void**)&P->d_full_block_first, P->full_block_first.data(),
                  P->full_block_first.size() * sizeof(uint32_t))) != cudaSuccess)))
        return e == cudaErrorMemoryAllocation ? rr_fail(RR_ENOMEM, "device allocation failed")
                                              : cuda_fail(e, "plan upload");
    for (cudaEvent_t& ev : P->claim_done)
        RR_CUDA(cudaEventCreateWithFlags(&ev, cudaEventDisableTiming));
    return RR_OK;
}

void rr_device_release(rr_plan* P) {
    if (!P || P->device < 0) return;
    int prev = -1;
    cudaGetDevice(&prev);
    if (prev != P->device) cudaSetDevice(P->device);
    cudaFree(P->d_pack_items);
    cudaFree(P->d_pack_block_first);
    cudaFree(P->d_full_items);
    cudaFree(P->d_full_block_first);
    cudaFree(P->d_pack_weight_prefix);
    cudaFree(P->d_unpack_weight_prefix);
    cudaFree(P->d_src_bytes);
    cudaFree(P->d_tensor_bytes);
    cudaFree(P->d_unpack_items);
    cudaFree(P->d_unpack_block_first);
    cudaFree(P->d_unpack_unit_first);
    cudaFree(P->d_pack_unit_first);
    cudaFree(P->d_pack_whole_unit_first);
    cudaFree(P->d_slots);
    for (cudaEvent_t& ev : P->claim_done) {
        if (ev) cudaEventDestroy(ev);
        ev = nullptr;
    }
    cudaFree(P->d_verify_scratch);
    cudaFreeHost(P->h_verify_result);
    cudaFree(P->d_error);
    P->d_error = nullptr;
    P->d_pack_items = nullptr;
    P->d_pack_block_first = nullptr;
    P->d_full_items = nullptr;
    P->d_full_block_first = nullptr;
    P->d_pack_weight_prefix = nullptr;
    P->d_unpack_weight_prefix = nullptr;
    P->d_src_bytes = nullptr;
    P->d_tensor_bytes = nullptr;
    P->d_unpack_items = nullptr;
    P->d_unpack_block_first = nullptr;
    P->d_unpack_unit_first = nullptr;
    P->d_pack_unit_first = nullptr;
    P->d_pack_whole_unit_first = nullptr;
    P->d_slots = nullptr;
    P->d_verify_scratch = nullptr;
    P->h_verify_result = nullptr;
    if (prev >= 0 && prev != P->device) cudaSetDevice(prev);
    P->device = -1;
}

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

extern "C" rr_status rr_pack(const rr_plan* P, const void* const* src_shards,
                             void* const* buckets, uint64_t* checksums, cudaStream_t stream) {
    RR_TRACE("rr_pack");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    return pack_impl(P, Range{0, P->n_buckets, true}, src_shards, buckets, checksums, stream);
}

extern "C" rr_status rr_unpack(const rr_plan* P, const void* const* buckets, void* const* dst,
                               cudaStream_t stream) {
    RR_TRACE("rr_unpack");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    return unpack_impl(P, Range{0, P->n_buckets, true}, buckets, dst, stream);
}

extern "C" rr_status rr_verify(const rr_plan* P, const void* const* buckets,
                               const uint64_t* checksums, int64_t* n_bad, int64_t* first_bad,
                               cudaStream_t stream) {
    RR_TRACE("rr_verify");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    return verify_impl(P, Range{0, P->n_buckets, true}, buckets, checksums, nullptr, n_bad,
                       first_bad, stream);
}

extern "C" rr_status rr_pack_range(const rr_plan* P, int32_t first_bucket, int32_t n_buckets,
                                   const void* const* src_shards, void* const* buckets,
                                   uint64_t* checksums, cudaStream_t stream) {
    RR_TRACE("rr_pack_range");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    return pack_impl(P, R, src_shards, buckets, checksums, stream);
}

extern "C" rr_status rr_unpack_range(const rr_plan* P, int32_t first_bucket, int32_t n_buckets,
                                     const void* const* buckets, void* const* dst,
                                     cudaStream_t stream) {
    RR_TRACE("rr_unpack_range");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    return unpack_impl(P, R, buckets, dst, stream);
}

extern "C" rr_status rr_verify_range(const rr_plan* P, int32_t first_bucket, int32_t n_buckets,
                                     const void* const* buckets, const uint64_t* checksums,
                                     uint8_t* bad, int64_t* n_bad, int64_t* first_bad,
                                     cudaStream_t stream) {
    RR_TRACE("rr_verify_range");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    return verify_impl(P, R, buckets, checksums, bad, n_bad, first_bad, stream);
}

extern "C" rr_status rr_unpack_verify(const rr_plan* P, const void* const* buckets,
                                      const uint64_t* checksums, void* const* dst, uint8_t* bad,
                                      int64_t* n_bad, int64_t* first_bad, cudaStream_t stream) {
    RR_TRACE("rr_unpack_verify");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    return unpack_verify_impl(P, Range{0, P->n_buckets, true}, buckets, checksums, dst, bad, n_bad,
                              first_bad, stream);
}

extern "C" rr_status rr_unpack_verify_range(const rr_plan* P, int32_t first_bucket,
                                            int32_t n_buckets, const void* const* buckets,
                                            const uint64_t* checksums, void* const* dst,
                                            uint8_t* bad, int64_t* n_bad, int64_t* first_bad,
                                            cudaStream_t stream) {
    RR_TRACE("rr_unpack_verify_range");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    return unpack_verify_impl(P, R, buckets, checksums, dst, bad, n_bad, first_bad, stream);
}

extern "C" rr_status rr_unpack_verify_async(const rr_plan* P, int32_t first_bucket,
                                            int32_t n_buckets, const void* const* buckets,
                                            const uint64_t* checksums, void* const* dst,
                                            uint8_t* bad, uint64_t* scratch, int64_t* result,
                                            cudaStream_t stream) {
    RR_TRACE("rr_unpack_verify_async");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    if ((st = check_unpack_verify_args(P, R, buckets, checksums, dst, bad))) return st;
    long long* res = result_address(result);
    if (!res)
        return rr_fail(RR_EINVAL, "result must be 8-byte aligned device or pinned host memory");
    if (R.b1 > R.b0) {
        if (!aligned16(scratch)) return rr_fail(RR_EINVAL, "scratch NULL or not 16-byte aligned");
        if (!device_resident(scratch)) return rr_fail(RR_EINVAL, "scratch must be device memory");
        R.scratch = (unsigned long long*)scratch;
        // The launch's last block writes the result.
        return enqueue_unpack_verify(P, R, buckets, checksums, dst, bad, stream, res);
    }
    rr_verify_result_kernel<<<1, 1, 0, stream>>>(nullptr, res);   // an empty range
    RR_CUDA(cudaGetLastError());
    return RR_OK;
}

extern "C" rr_status rr_plan_check(const rr_plan* P, cudaStream_t stream) {
    RR_TRACE("rr_plan_check");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    rr_plan* M = const_cast<rr_plan*>(P);   // shares the pinned result buffer with verify
    std::lock_guard<std::mutex> lock(M->verify_mutex);
    return read_error(P, stream);
}

extern "C" rr_status rr_plan_selftest_wait(const rr_plan* P, cudaStream_t stream) {
    RR_TRACE("rr_plan_selftest_wait");
    rr_clear_error();
    rr_status st = check_plan(P);
    if (st) return st;
    rr_wait_selftest_kernel<<<1, 32, 0, stream>>>(P->d_error);
    RR_CUDA(cudaGetLastError());
    return RR_OK;
}

extern "C" rr_status rr_clear_range(const rr_plan* P, int32_t first_bucket, int32_t n_buckets,
                                    void* const* buckets, cudaStream_t stream) {
    RR_TRACE("rr_clear_range");
    rr_clear_error();
    Range R;
    rr_status st = check_plan(P);
    if (st || (st = check_range(P, first_bucket, n_buckets, &R))) return st;
    if ((st = check_ptrs(P->pageable_ok != 0, (const void* const*)buckets, P->n_buckets, "buckets"))) return st;
    if (n_buckets == 0) return RR_OK;
    uint64_t stride = 0;
    if (uniform((const void* const*)buckets, P->n_buckets, P->bucket_bytes, &stride)) {
        RR_CUDA(cudaMemset2DAsync(buckets[R.b0], stride, 0, (size_t)P->bucket_bytes,
                                  (size_t)n_buckets, stream));
    } else {
        for (int32_t b = R.b0; b < R.b1; ++b)
            RR_CUDA(cudaMemsetAsync(buckets[b], 0, (size_t)P->bucket_bytes, stream));
    }
    return RR_OK;
}

// ---------------------------------------------------------------------------
// Allocation-free verify
//
// For callers that must not allocate device memory at the moment they check a
// pull: an inference engine that reserves nearly all device memory up front,
// or a process that runs under a memory pool that refuses cudaMalloc once the
// weights are loaded.  It needs no plan (a plan's creation allocates): the
// caller passes the buckets, their size and the expected checksums.  The
// per-bucket sums and counters live in one file-scope device array, which
// every GPU that loads this library holds until the process exits.
// ---------------------------------------------------------------------------

namespace {

constexpr int32_t kStaticVerifyMaxBuckets = 16384;   // 128 KiB of sums + 4 counters
constexpr int kStaticMaxDevices = 64;

__device__ __align__(256) unsigned long long g_static_verify_scratch[kStaticVerifyMaxBuckets + 4];

struct StaticVerifyDevice {
    bool ready = false;
    int32_t grid = 0;
};

std::mutex g_static_mutex;
StaticVerifyDevice g_static_dev[kStaticMaxDevices];

// With the caller's device current: the array's device address (host code may
// not use the symbol itself as a pointer) and the grid for this device.  The
// grid is sized once per device, on its first call.  The address is looked up
// on every call: a device reset destroys the context that loaded this
// library's module, the next context loads it again, and the array may then
// sit elsewhere.  Neither step allocates.
rr_status static_verify_setup(unsigned long long** scratch, int32_t* grid) {
    int dev = -1;
    RR_CUDA(cudaGetDevice(&dev));
    if (dev < 0 || dev >= kStaticMaxDevices)
        return rr_fail(RR_EINVAL, "device %d beyond the %d devices this entry point serves", dev,
                       kStaticMaxDevices);
    void* p = nullptr;
    RR_CUDA(cudaGetSymbolAddress(&p, g_static_verify_scratch));
    if (!p) return rr_fail(RR_ECUDA, "no device address for the verify scratch array");
    std::lock_guard<std::mutex> lock(g_static_mutex);
    StaticVerifyDevice& d = g_static_dev[dev];
    if (!d.ready) {
        int sms = 0, per_sm = 0;
        RR_CUDA(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev));
        RR_CUDA(cudaOccupancyMaxActiveBlocksPerMultiprocessor(
            &per_sm, rr_verify_kernel<kLargePtrs>, kThreads, 0));
        d.grid = sms * (per_sm > 0 ? per_sm : 1);
        d.ready = true;
    }
    *scratch = (unsigned long long*)p;
    *grid = d.grid;
    return RR_OK;
}

template <int NPTR>
rr_status launch_static_verify(unsigned long long* scratch, int32_t grid, int32_t n_buckets,
                               uint64_t bucket_bytes, const void* const* buckets,
                               const uint64_t* checksums, bool table, uint64_t stride,
                               cudaStream_t s) {
    VerifyArgs<NPTR> a;
    std::memset(&a, 0, sizeof a);
    a.sums = scratch;
    a.counters = scratch + n_buckets;
    a.expected = (const unsigned long long*)checksums;
    a.bucket_bytes = bucket_bytes;
    a.chunk_bytes = std::min<uint64_t>((uint64_t)kVerifyChunk, bucket_bytes);
    a.chunks_per_bucket = (a.bucket_bytes + a.chunk_bytes - 1) / a.chunk_bytes;
    a.total_chunks = a.chunks_per_bucket * (uint64_t)n_buckets;
    a.n_buckets = n_buckets;
    if (table) {
        for (int32_t b = 0; b < n_buckets; ++b) a.ptr[b] = buckets[b];
    } else {
        a.bucket_base = (const char*)buckets[0];
        a.bucket_stride = stride;
    }
    rr_verify_kernel<NPTR><<<grid, kThreads, 0, s>>>(a);
    RR_CUDA(cudaGetLastError());
    return RR_OK;
}

}  // namespace

extern "C" rr_status rr_verify_noalloc(const void* const* buckets, int32_t n_buckets,
                                       size_t bucket_bytes, const uint64_t* checksums,
                                       int64_t* n_bad, int64_t* first_bad, cudaStream_t stream) {
    RR_TRACE("rr_verify_noalloc");
    rr_clear_error();
    if (n_buckets < 0 || n_buckets > kStaticVerifyMaxBuckets)
        return rr_fail(RR_EINVAL,
                       "rr_verify_noalloc checks at most %d buckets per call (got %d); use "
                       "larger buckets, several calls, or rr_verify",
                       kStaticVerifyMaxBuckets, n_buckets);
    if (bucket_bytes < 8 || bucket_bytes % 8 != 0 || bucket_bytes > (size_t(1) << 32) - 16)
        return rr_fail(RR_EINVAL, "bucket_bytes must be a multiple of 8 in [8, 2^32 - 16]");
    int dev = 0, pageable = 0;
    RR_CUDA(cudaGetDevice(&dev));
    RR_CUDA(cudaDeviceGetAttribute(&pageable, cudaDevAttrPageableMemoryAccess, dev));
    rr_status st = check_ptrs(pageable != 0, buckets, n_buckets, "buckets");
    if (st) return st;
    if (n_buckets > 0 && (st = check_buf(pageable != 0, checksums, "checksums"))) return st;
    if (n_bad) *n_bad = 0;
    if (first_bad) *first_bad = -1;
    if (n_buckets == 0) return RR_OK;
    uint64_t stride = 0;
    const bool table = !uniform(buckets, n_buckets, (int64_t)bucket_bytes, &stride);
    if (table && n_buckets > kLargePtrs)
        return rr_fail(RR_EINVAL, "%d separately allocated buckets exceed %d pointers", n_buckets,
                       kLargePtrs);
    unsigned long long* scratch = nullptr;
    int32_t grid = 0;
    if ((st = static_verify_setup(&scratch, &grid))) return st;

    // The array keeps the previous call's contents: clear the sums and counters used here.
    RR_CUDA(cudaMemsetAsync(scratch, 0, (size_t(n_buckets) + 4) * sizeof(unsigned long long),
                            stream));
    st = (!table || n_buckets <= kSmallPtrs)
             ? launch_static_verify<kSmallPtrs>(scratch, grid, n_buckets, bucket_bytes, buckets,
                                                checksums, table, stride, stream)
             : launch_static_verify<kLargePtrs>(scratch, grid, n_buckets, bucket_bytes, buckets,
                                                checksums, table, stride, stream);
    if (st) return st;
    unsigned long long result[4] = {0, 0, 0, 0};   // host stack: no pinned buffer needed
    RR_CUDA(cudaMemcpyAsync(result, scratch + n_buckets, sizeof result, cudaMemcpyDeviceToHost,
                            stream));
    RR_CUDA(cudaStreamSynchronize(stream));
    if (n_bad) *n_bad = (int64_t)result[1];
    if (first_bad) *first_bad = result[1] ? (int64_t)(ULLONG_MAX - result[2]) : -1;
    return result[1] ? RR_EMISMATCH : RR_OK;
}
