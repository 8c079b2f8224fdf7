/*
 * rr.h - C ABI of the trainer -> rollout weight-synchronisation hot path.
 *
 * RobustRL (arXiv 2512.22492), Section 5.2.1 (the UCX-based weight update):
 * after a training step the trainer's weights are (1) resharded to the
 * rollout's sharding and (2) copied, one layer after another, into a transfer buffer
 * that the transport moves to the rollout; Section 5.2.2 has a recovered or
 * resumed rollout pull (part of) that buffer again.  This library is the
 * on-GPU part of that route, for one GPU: gather from flat FSDP-style shards,
 * cast to bfloat16, pack into fixed-size buckets with a 64-bit checksum each,
 * and unpack buckets into the rollout's tensors.  The transport is not here.
 *
 * Definitions (the paper fixes none of these; they are this library's):
 *
 *  Source layout.  Parameters are concatenated in manifest order into one
 *  flat byte buffer, each starting at a multiple of max(align_bytes, element
 *  size) (or at the caller's explicit offsets); the total is padded to a
 *  multiple of 16 * n_shards and cut into n_shards shards of equal size S.
 *  Flat byte f is byte f % S of shard f / S.  A parameter of shape
 *  [d0, d1, ...] is viewed as a matrix [d0, d1 * d2 * ...]; a vector [d0] is
 *  [d0, 1].
 *
 *  Destination.  A destination tensor is a list of blocks; its elements are
 *  the blocks' elements, block after block, each block row-major.  Block
 *  (param, row0, nrows, col0, ncols) covers rows [row0, row0 + nrows) and
 *  columns [col0, col0 + ncols) of the parameter's matrix view.  Fused QKV,
 *  fused gate_up, stacked experts and tensor-parallel slices are all block
 *  lists; the library knows nothing about any model.
 *
 *  Cast.  float32 -> bfloat16 rounds to nearest, ties to even, in integer
 *  arithmetic: +-0, subnormals and +-inf are kept, overflow goes to +-inf,
 *  and a NaN keeps its sign and upper payload with the quiet bit set
 *  ((bits >> 16) | 0x0040).  A bfloat16 source is copied bit for bit.
 *
 *  Stream and buckets.  Each destination rank r has a byte stream holding
 *  its tensors in the order given, each starting at the next multiple of
 *  tensor_align_bytes, elements little-endian.  The stream is cut into
 *  buckets of exactly bucket_bytes; alignment gaps and the last bucket's
 *  tail are zero.  Buckets are numbered rank-major: rank 0's first.
 *
 *  Checksum.  checksums[b] = sum of the little-endian 64-bit words of
 *  bucket b, modulo 2^64.  The sum is order-independent, so the GPU may
 *  accumulate in any grouping and still match exactly.
 *
 * Memory.  Every pointer argument named "device" is CUDA device memory of
 * the device the plan was created on, owned by the caller; every device
 * pointer must be 16-byte aligned.  Where a call says so, a buffer may
 * instead be host memory this GPU reads (pinned, or any host memory on a
 * device with pageable memory access, as on Grace); memory it cannot reach
 * is refused with RR_EINVAL before anything is launched.  The plan owns its device segment tables,
 * a small verify scratch area and 16 work-unit counters (rr_plan_work_units);
 * rr_pack and rr_unpack allocate nothing.
 *
 * Errors.  Every call returns rr_status.  Argument and layout errors are
 * reported synchronously and leave outputs untouched; RR_ECUDA means a CUDA
 * call failed (rr_last_error() has the CUDA message).  rr_last_error()
 * returns a per-thread description of the most recent failure.
 *
 * Threads and streams.  A plan's tables are immutable after creation; rr_pack
 * and rr_unpack may run on it concurrently on different streams, and from
 * different threads, as long as their outputs are distinct (each launch
 * takes its own work-unit counter, under a lock).  rr_verify serialises on
 * the plan.  The stream-ordered calls (rr_pack(_range), rr_unpack(_range),
 * rr_clear_range, rr_unpack_verify_async) may be captured into a CUDA graph;
 * the blocking ones (rr_verify(_range), rr_unpack_verify(_range),
 * rr_plan_check) may not, and rr_unpack_verify_async takes their place in a
 * graph.
 */
#ifndef RR_H
#define RR_H

#include <stddef.h>
#include <stdint.h>

#include <cuda_runtime_api.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    RR_OK = 0,
    RR_EINVAL = 1,    /* bad argument: null pointer, bad size, misaligned pointer        */
    RR_ENOMEM = 2,    /* host or device allocation failed (plan creation only)           */
    RR_ECUDA = 3,     /* a CUDA call failed                                              */
    RR_ELAYOUT = 4,   /* the layout description is inconsistent or out of range          */
    RR_EMISMATCH = 5  /* rr_verify: at least one bucket's checksum differs               */
} rr_status;

typedef enum { RR_F32 = 0, RR_BF16 = 1 } rr_dtype;

/* One trainer parameter (manifest entry). */
typedef struct {
    const char* name;   /* informational, may be NULL                              */
    int32_t ndim;       /* 0..4                                                    */
    int64_t shape[4];   /* sizes of the first ndim dimensions                      */
    rr_dtype dtype;     /* dtype of the trainer's copy: RR_F32 or RR_BF16          */
} rr_param;

/* How the trainer's parameters are cut into shards.
 *  RR_SHARD_FLAT: one flat buffer cut into equal shards (FSDP1 FlatParameter),
 *                 as defined at the top of this file.
 *  RR_SHARD_ROWS: every parameter is cut on dim 0 separately (FSDP2 Shard(0),
 *                 torch.chunk rule): with c = ceil(rows / n_shards), shard s
 *                 holds rows [s*c, min((s+1)*c, rows)), padded to c rows.
 *                 Within each shard the parameters' chunks follow one another
 *                 in manifest order, each starting at a multiple of
 *                 max(align_bytes, element size); all shards share that local
 *                 layout and are S = (end of the last chunk rounded up to 16)
 *                 bytes.  Padding rows are never read.
 *  RR_SHARD_TENSORS: every parameter is its own buffer: "shard" p is
 *                 parameter p, row-major from byte 0 (n_shards must equal the
 *                 number of parameters).  This is how a relay re-packs from
 *                 the rollout tensors it has loaded.
 *  RR_SHARD_UNITS: FSDP1 with one FlatParameter per wrapped module (a
 *                 "unit": typically one per decoder layer, plus the root
 *                 holding what no layer wraps).  param_unit[p] names the unit
 *                 of parameter p.  Each unit is laid out exactly like the
 *                 RR_SHARD_FLAT buffer above, on its own: its parameters in
 *                 manifest order from offset 0, padded to a multiple of
 *                 16 * n_shards, cut into n_shards shards of S_u bytes.  The
 *                 calls then take n_units * n_shards source buffers,
 *                 unit-major: buffer u * n_shards + s is shard s of unit u.
 *                 No explicit offsets or shard size. */
typedef enum {
    RR_SHARD_FLAT = 0,
    RR_SHARD_ROWS = 1,
    RR_SHARD_TENSORS = 2,
    RR_SHARD_UNITS = 3
} rr_sharding;

/* Trainer side. */
typedef struct {
    int32_t n_shards;                 /* 1..65535                                      */
    int64_t align_bytes;              /* parameter start alignment, >= 1 (16 typical)  */
    const int64_t* param_flat_offset; /* FLAT only, optional: [n_params] explicit flat
                                         byte offsets (each a multiple of the element
                                         size, non-overlapping); NULL = computed      */
    int32_t sharding;                 /* rr_sharding; 0 = RR_SHARD_FLAT                */
    int64_t shard_bytes;              /* FLAT only, optional: shard size S, a multiple
                                         of 16 with n_shards * S covering every
                                         parameter; 0 = computed                      */
    int32_t n_units;                  /* UNITS only: number of FSDP units, >= 1;
                                         0 for the other shardings                    */
    const int32_t* param_unit;        /* UNITS only: [n_params] unit of each parameter,
                                         in [0, n_units), every unit used; NULL
                                         otherwise                                    */
} rr_src_layout;

/* A 2-D block of a parameter's matrix view. */
typedef struct {
    int32_t param;
    int64_t row0, nrows, col0, ncols;
} rr_block;

/* One rollout tensor. */
typedef struct {
    const char* name;        /* informational, may be NULL                          */
    int32_t rank;            /* destination rank, 0 .. tp-1                         */
    int64_t numel;           /* must equal the sum of the blocks' nrows * ncols     */
    int32_t n_blocks;
    const rr_block* blocks;
} rr_dst_tensor;

/* The rollout's 16-bit element type.  bfloat16 is the default (zero); a
 * float16 rollout takes IEEE binary16 (Section 7.4 counts the transferred
 * model as FP16): round to nearest, ties to even, subnormals kept, overflow to
 * +-inf, and a NaN kept as a quiet NaN with its sign and top payload bits
 * (sign | 0x7E00 | ((b >> 13) & 0x1FF) for float32 bits b).  A bfloat16
 * source is widened exactly and rounded the same way. */
typedef enum { RR_DST_BF16 = 0, RR_DST_F16 = 1 } rr_dst_dtype;

/* Rollout side. */
typedef struct {
    int32_t tp;                   /* number of destination ranks (tensor parallel)     */
    int32_t n_tensors;
    const rr_dst_tensor* tensors; /* order within a rank = order in its stream         */
    int64_t tensor_align_bytes;   /* power of two >= 2; 256 typical                    */
    int32_t dtype;                /* rr_dst_dtype; 0 (bfloat16) by default             */
    int32_t reserved;             /* 0                                                 */
} rr_dst_layout;

typedef struct rr_plan rr_plan;

/* Which kernels move the data.  RR_ENGINE_AUTO (default): the bulk-copy
 * engine (cp.async.bulk into shared-memory stages, consumer warps cast/copy
 * and sum) when every buffer of the call is device memory, otherwise the
 * register path (16-byte loads and stores).  RR_ENGINE_REGISTERS: always the
 * register path.  Both produce identical bytes. */
typedef enum { RR_ENGINE_AUTO = 0, RR_ENGINE_REGISTERS = 1 } rr_engine;

/* Tuning / inspection options for rr_plan_create_ex.  Zero means default. */
typedef struct {
    int32_t host_only;   /* 1: build the tables on the host only and touch no GPU; such
                            a plan can be queried and exported but not executed       */
    int32_t grid_blocks; /* persistent grid size; default: SMs x resident blocks      */
    int64_t chunk_bytes; /* largest destination bytes per work item; default 64 KiB   */
    int32_t engine;      /* rr_engine                                                 */
    int32_t check_items; /* 1: every kernel checks each work item against the source,
                            bucket and tensor sizes of the plan before touching
                            memory; an item outside them is skipped and marks the
                            plan's error word (rr_plan_check then reports RR_ECUDA).
                            A debugging aid in place of a memory-checking tool; costs a
                            little producer time                                    */
} rr_plan_options;

/* Compiles manifest + source layout + destination layout + bucket size into
 * device-resident segment tables (Section 5.2.1 step 1: the weights are
 * re-laid out in the rollout's sharding).  bucket_bytes: a multiple of 8, at most
 * 2^32 - 16.  Uses the current CUDA device.  *out is valid only on RR_OK. */
rr_status rr_plan_create(const rr_param* manifest, int32_t n_params, const rr_src_layout* src,
                         const rr_dst_layout* dst, size_t bucket_bytes, rr_plan** out);
/* rr_plan_create with tuning options (opts may be NULL).  The options have no
 * counterpart in the paper; the plan they build computes the same bytes. */
rr_status rr_plan_create_ex(const rr_param* manifest, int32_t n_params,
                            const rr_src_layout* src, const rr_dst_layout* dst,
                            size_t bucket_bytes, const rr_plan_options* opts, rr_plan** out);

/* Frees the plan's device tables, scratch and events.  Section 5.2.1 reserves
 * the transfer's memory ahead of the transfer so that it cannot run out of GPU
 * memory mid-sync; a plan is that reservation for the work tables, held from
 * creation until this call.  NULL is ignored.  No call of this plan may still
 * be running on any stream. */
void rr_plan_destroy(rr_plan* plan);

/* Bucket geometry: the size of the transfer buffer (Section 5.2.1: a buffer
 * reserved up front, large enough to keep the RDMA links busy), so that the
 * caller can allocate every bucket before the first sync.  Any output pointer
 * may be NULL.  stream_bytes_per_rank has tp entries; first_bucket_of_rank has
 * tp + 1 (the last is n_buckets).  RR_EINVAL for a NULL plan. */
rr_status rr_plan_query(const rr_plan* plan, int32_t* n_buckets, int64_t* stream_bytes_per_rank,
                        int32_t* first_bucket_of_rank);

/* Source geometry (the trainer's FSDP shards, Section 7.1): shard size S, end of the last parameter, and per-parameter
 * byte offsets ([n_params]): flat offsets for RR_SHARD_FLAT, offsets within
 * each shard for RR_SHARD_ROWS, 0 for RR_SHARD_TENSORS (whose S is the size of
 * the largest parameter), offsets within the parameter's unit for
 * RR_SHARD_UNITS (whose S is the largest S_u; flat_bytes is then the end of
 * the largest unit).  Any output pointer may be NULL. */
rr_status rr_plan_source(const rr_plan* plan, int64_t* shard_bytes, int64_t* flat_bytes,
                         int64_t* param_flat_offset);

/* The source buffers the calls take (the trainer's shards, Section 7.1): their number (the length of every
 * src_shards array) and the bytes each must hold ([*n_buffers]).  FLAT and
 * ROWS: n_shards buffers of S bytes; TENSORS: one per parameter, of its size;
 * UNITS: n_units * n_shards, unit-major, each of its unit's S_u.  Pass
 * buffer_bytes = NULL to learn the count first.  Any output pointer may be NULL. */
rr_status rr_plan_source_buffers(const rr_plan* plan, int32_t* n_buffers, int64_t* buffer_bytes);

/* Destination geometry (the rollout's sharding that Section 5.2.1 step 1
 * reshards into): per tensor numel and byte offset within its rank's stream
 * ([n_tensors] each).  Any output pointer may be NULL. */
rr_status rr_plan_tensors(const rr_plan* plan, int64_t* tensor_numel,
                          int64_t* tensor_stream_offset);

typedef struct {
    int64_t n_pack_items;
    int64_t n_unpack_items;
    int32_t grid_blocks;         /* pack kernel grid (blocks)                          */
    int32_t unpack_grid_blocks;
    int32_t verify_grid_blocks;
    int32_t n_buckets;
    int32_t n_shards;
    int32_t n_tensors;
    int64_t bucket_bytes;
    int64_t pack_bytes_read;     /* source bytes read by one rr_pack                    */
    int64_t pack_bytes_written;  /* bucket bytes written by one rr_pack (all buckets)   */
    int64_t unpack_bytes_read;   /* bucket bytes read by one rr_unpack                  */
    int64_t unpack_bytes_written;/* destination bytes written by one rr_unpack          */
    int64_t verify_bytes_read;   /* bucket bytes read by one rr_verify                  */
    int64_t n_pack_full_items;   /* items of the whole-sync pack table (see
                                    rr_plan_export_pack_full); equals n_pack_items
                                    when no fan-out groups were found                  */
} rr_plan_stats;

/* Table sizes, grids and the algorithmic bytes each call moves.  No
 * counterpart in the paper: it serves measurement against the HBM roofline. */
rr_status rr_plan_get_stats(const rr_plan* plan, rr_plan_stats* stats);

/* Work items of the segment tables, as the kernels read them (exported for
 * inspection and host-side tests; no counterpart in the paper). */
enum {
    RR_ITEM_F32_VEC = 0,    /* fp32 -> bf16, 8 elements per 16-byte store            */
    RR_ITEM_F32_SCALAR = 1, /* fp32 -> bf16, one element at a time (ragged/misaligned)*/
    RR_ITEM_BF16_VEC = 2,   /* bf16 -> bf16                                          */
    RR_ITEM_BF16_SCALAR = 3,
    RR_ITEM_ZERO_VEC = 4,   /* zero fill of alignment gaps / bucket tails            */
    RR_ITEM_ZERO_SCALAR = 5,
    RR_ITEM_COPY_VEC = 6,   /* unpack: 16-byte copies                                */
    RR_ITEM_COPY_SCALAR = 7, /* unpack: 2-byte copies                                */
    RR_ITEM_READ_VEC = 8,    /* unpack table: alignment gap / tail, read only by the    */
    RR_ITEM_READ_SCALAR = 9, /*   verifying unpack (their bytes count in the checksum)  */
    RR_ITEM_FAN_F32 = 10,    /* whole-sync table only: fan-out head (see below)         */
    RR_ITEM_FAN_BF16 = 11,
    RR_ITEM_FAN_DST = 12     /* one destination of the fan-out head before it           */
};

/* Pack work item: n_rows rows of row_len elements; row i starts at source
 * element offset i * src_stride from the first; the destination is the
 * contiguous range [dst_off, dst_off + 2 * n_rows * row_len) of one bucket. */
typedef struct {
    uint64_t src;        /* bits 0..47: byte offset in the shard; bits 48..63: shard   */
    uint32_t dst_off;    /* byte offset in the bucket                                   */
    uint32_t bucket;     /* global bucket index                                         */
    uint32_t row_len;    /* elements per row                                            */
    uint32_t n_rows;
    uint32_t src_stride; /* elements between consecutive row starts                     */
    uint16_t kind;       /* RR_ITEM_F32_* / BF16_* / ZERO_*                            */
    uint16_t reserved;
} rr_pack_item;

/* Unpack work item: copy nbytes from bucket `bucket` at src_off to tensor
 * `tensor` at dst_off (READ items: bucket bytes outside every tensor; tensor
 * and dst_off unused). */
typedef struct {
    uint64_t dst_off;
    uint32_t src_off;
    uint32_t bucket;
    uint32_t tensor;
    uint32_t nbytes;
    uint32_t kind;       /* RR_ITEM_COPY_*                                             */
    uint32_t reserved;
} rr_unpack_item;

/* Copies up to cap items (and, if block_first is not NULL, the per-block item
 * ranges: grid_blocks + 1 entries for pack, unpack_grid_blocks + 1 for
 * unpack) into caller memory.  No counterpart in the paper (inspection). */
rr_status rr_plan_export_pack(const rr_plan* plan, rr_pack_item* items, int64_t cap,
                              uint32_t* block_first);

/* The whole-sync pack table: what rr_pack runs on the bulk-copy engine when it
 * packs every bucket.  It holds the items of rr_plan_export_pack (bucket-sorted,
 * used by the range calls and the register path) except where several rollout
 * ranks take narrow column slices (under 1 KiB of source per row) of the same
 * parameter rows -- a row-parallel weight under tensor parallelism.  Those
 * slices become fan-out groups that read each source row once:
 *   head (RR_ITEM_FAN_F32 / RR_ITEM_FAN_BF16): n_rows rows of row_len source
 *        elements (the slices' joint column span) at src, src_stride elements
 *        apart; dst_off = the number of RR_ITEM_FAN_DST items that follow;
 *   each RR_ITEM_FAN_DST: src = the slice's first column within the span,
 *        row_len = its width, and the slice of row i goes to bucket `bucket`
 *        at dst_off + 2 * i * row_len.
 * Every slice is 16-byte aligned in source and destination and a multiple of 8
 * elements wide; no destination run crosses a bucket.  The per-block ranges
 * never separate a head from its destinations. */
rr_status rr_plan_export_pack_full(const rr_plan* plan, rr_pack_item* items, int64_t cap,
                                   uint32_t* block_first);
rr_status rr_plan_export_unpack(const rr_plan* plan, rr_unpack_item* items, int64_t cap,
                                uint32_t* block_first);

/* Reshard + cast + pack + checksum, fused in one persistent kernel launch
 * (Section 5.2.1 steps 1-2: the resharded model fills a transfer buffer; the
 * checksums serve the reconnect cases of Section 5.2.2).
 *   src_shards: host array of n_shards pointers, S bytes each: device
 *               memory, or host memory this GPU reads (pinned; any host
 *               memory where the device has pageable memory access).  A
 *               host-memory source is read by the pack's own loads over the
 *               host link, with nothing copied to the device first; its fp32
 *               vectors are 4 elements wide, so that every warp load uses
 *               whole 32-byte sectors of host memory.
 *   buckets:    host array of n_buckets pointers, bucket_bytes each (device
 *               memory, or host memory as above: a snapshot); equally spaced
 *               pointers (one allocation cut into buckets) lift the limit on
 *               how many buckets a launch can address.
 *   checksums:  device array of n_buckets uint64, overwritten.
 * Any host-memory array runs the call on the register path.  Stream-ordered
 * and asynchronous: returns after enqueueing one kernel on `stream`, preceded
 * by a memset of the checksums unless the launch holds a pooled work-unit
 * slot (the bulk-copy engine outside graph capture). */
rr_status rr_pack(const rr_plan* plan, const void* const* src_shards, void* const* buckets,
                  uint64_t* checksums, cudaStream_t stream);

/* Buckets -> rollout tensors (Section 5.2.1: the receiving rollout completes
 * its weight update from what it pulled).
 *   buckets: host array of n_buckets pointers (device memory, or host memory
 *            this GPU reads: restoring a snapshot);
 *   dst:     host array of n_tensors pointers, numel * 2 bytes each.
 * Stream-ordered and asynchronous (one kernel launch). */
rr_status rr_unpack(const rr_plan* plan, const void* const* buckets, void* const* dst,
                    cudaStream_t stream);

/* Recomputes every bucket's checksum on the GPU and compares it with
 * checksums (device, n_buckets).  Section 5.2.2: a rollout that reconnects
 * after a relay or trainer failure, or resumes a pull, must know which of the
 * buckets it holds are intact before it completes its update.
 *   buckets:   host array of n_buckets pointers (device or pinned host),
 *              bucket_bytes each, 16-byte aligned; read only.
 *   checksums: device (or pinned host) array of n_buckets uint64, read only.
 *   stream:    where the check runs.  This argument extends the four-call
 *              interface: the check is ordered after the caller's own work
 *              (the pull that filled the buckets) without a device-wide sync.
 * Blocks the calling thread until `stream` has finished the check.  *n_bad =
 * number of mismatching buckets, *first_bad = lowest such index or -1 (either
 * pointer may be NULL).  Returns RR_EMISMATCH when n_bad > 0, RR_ECUDA when a
 * kernel of this plan gave up a bounded wait (see rr_plan_check), RR_EINVAL
 * for bad pointers (nothing is launched then).  Serialises on the plan. */
rr_status rr_verify(const rr_plan* plan, const void* const* buckets, const uint64_t* checksums,
                    int64_t* n_bad, int64_t* first_bad, cudaStream_t stream);

/* Resumable sync (Section 5.2.2): when a relay fails mid-pull, the rollout
 * keeps what it already pulled and fetches the rest elsewhere; when the trainer
 * fails mid-pull, the partial update is cleared and the pull starts again.
 * These calls act on buckets [first_bucket, first_bucket + n_buckets) only.
 * The pointer arrays are the full ones (all n_buckets buckets, all tensors,
 * as for the full calls); only the range is read or written.  A range outside
 * [0, n_buckets) is RR_EINVAL.
 *
 * rr_pack_range:   writes those buckets and checksums[first .. first+n) and
 *                  nothing else; its output equals the full rr_pack's there.
 * rr_unpack_range: writes exactly the destination bytes that lie in those
 *                  buckets (a tensor that straddles the range's edge is
 *                  written in part).
 * rr_verify_range: as rr_verify over the range; if `bad` (device, n_buckets
 *                  bytes) is not NULL, bad[i] = 1 when bucket first+i differs,
 *                  else 0.  *first_bad is a global bucket index.
 * rr_clear_range:  zero-fills those buckets (the "clear partial" path: a
 *                  cleared bucket fails verify unless its checksum is 0).
 * All four are stream-ordered; rr_verify_range blocks like rr_verify. */
rr_status rr_pack_range(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                        const void* const* src_shards, void* const* buckets, uint64_t* checksums,
                        cudaStream_t stream);
rr_status rr_unpack_range(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                          const void* const* buckets, void* const* dst, cudaStream_t stream);
rr_status rr_verify_range(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                          const void* const* buckets, const uint64_t* checksums, uint8_t* bad,
                          int64_t* n_bad, int64_t* first_bad, cudaStream_t stream);
rr_status rr_clear_range(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                         void* const* buckets, cudaStream_t stream);

/* Receiver side, fused: rr_unpack and rr_verify in one pass over the buckets
 * (every bucket byte is read once, for the copy and for the checksum).
 * Sections 5.2.1 and 5.2.2: the rollout completes its update from what it
 * pulled, and must know which of the buckets it holds are intact.
 * Writes every destination byte of the range, as rr_unpack / rr_unpack_range
 * would, whether or not its bucket verifies; the caller re-pulls the flagged
 * buckets and unpacks them again (for example with this call on a range).
 * bad, n_bad, first_bad and the return value are those of rr_verify_range.
 * Blocks the calling thread until `stream` has finished, like rr_verify. */
rr_status rr_unpack_verify(const rr_plan* plan, const void* const* buckets,
                           const uint64_t* checksums, void* const* dst, uint8_t* bad,
                           int64_t* n_bad, int64_t* first_bad, cudaStream_t stream);
rr_status rr_unpack_verify_range(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                                 const void* const* buckets, const uint64_t* checksums,
                                 void* const* dst, uint8_t* bad, int64_t* n_bad,
                                 int64_t* first_bad, cudaStream_t stream);

/* Per-bucket item index of the two work tables (n_buckets + 1 entries each,
 * either pointer may be NULL): the pack items of bucket b are
 * [pack_first[b], pack_first[b + 1]); likewise for unpack.  Inspection only;
 * no counterpart in the paper. */
rr_status rr_plan_bucket_items(const rr_plan* plan, uint32_t* pack_first, uint32_t* unpack_first);

/* Work units of the bulk-copy engine (inspection; no counterpart in the
 * paper, whose reshard is plain framework kernels).  Blocks drain HBM at unequal rates, so
 * a launch does not fix each block's whole share: block g takes the launch's
 * unit g, then claims the next unclaimed unit (an atomic counter) until none
 * are left, and all blocks finish together.
 *   which:
 *   RR_UNITS_PACK, RR_UNITS_UNPACK: the units of a bucket-range pack, and of
 *     every unpack and verifying unpack (on either engine).  Each bucket's
 *     items are cut into units of at most about 1 MiB of traffic (less on
 *     small plans, so that a block of the grid has a few dozen), none empty,
 *     none spanning two buckets; toward the end of the table units get
 *     smaller (about the weight left over twice the grid, down to 64 KiB), so
 *     that the last blocks to finish stop close together.  A range's units
 *     are the run of its buckets' units.
 *   RR_UNITS_PACK_FULL: the units of a pack over every bucket, over the table
 *     rr_plan_export_pack_full gives.  Units 0 .. grid - 1 are equal
 *     contiguous shares of 85% of the table's weight, one per block; the
 *     units after them cut the rest to the sizes above, smaller toward the
 *     end.  A cut never falls before a fan-out destination item.  Own units
 *     may be empty.
 *   *n_units: the number of units.
 *   unit_first (NULL, or n_units + 1 entries): unit u holds items
 *     [unit_first[u], unit_first[u + 1]) of that table.
 *   bucket_unit (NULL, or n_buckets + 1 entries; must be NULL for
 *     RR_UNITS_PACK_FULL): the units of bucket b are [bucket_unit[b],
 *     bucket_unit[b + 1]).
 * Call with both arrays NULL to learn n_units.  Host-only plans have units
 * too.  Errors: RR_EINVAL for a NULL plan or n_units, an unknown `which`, or
 * a bucket_unit array with RR_UNITS_PACK_FULL; nothing is written then.
 * Which launches claim: every verifying unpack (either engine), its counter
 * kept in the call's scratch (the plan's for the blocking forms, the
 * caller's for rr_unpack_verify_async) or in a pooled slot; rr_unpack (either
 * engine) and rr_pack (bulk-copy engine) when they get one of the plan's 16
 * pooled slots.  A slot is free once the launch that last held it has
 * completed; when none is, a launch takes the slot handed out longest ago if
 * that slot's launch ran on the same stream, and the stream waits on the GPU
 * for that launch (which it would anyway).  A launch gets no slot when every
 * slot is held by another stream's launch still in flight, or when its stream
 * is capturing a graph; it then splits its items evenly over the grid, as the
 * register path's pack always does.  Which of these runs changes no output
 * byte. */
enum { RR_UNITS_PACK = 0, RR_UNITS_PACK_FULL = 1, RR_UNITS_UNPACK = 2 };
rr_status rr_plan_work_units(const rr_plan* plan, int32_t which, int32_t* n_units,
                             uint32_t* unit_first, uint32_t* bucket_unit);

/* Stream-ordered form of rr_unpack_verify(_range), for a receiver that unpacks
 * and checks piece after piece without waiting on the host (Sections 5.2.1 and
 * 5.2.2: the pull completes, and a resumed pull checks what it holds).
 *   first_bucket, n_buckets: the range (0 and the plan's count for all).
 *   scratch: caller device memory of n_buckets + 4 uint64, 16-byte aligned;
 *            zeroed and used by the call, free again once `result` is written.
 *            Calls that overlap in time need distinct scratch.
 *   result:  two int64 in device memory or pinned (mapped) host memory, 8-byte
 *            aligned; when the call's work is done on `stream` they hold
 *            {number of bad buckets, first bad bucket or -1}.
 * Returns after enqueueing; argument errors come back at once.  A kernel that
 * gave up a bounded wait is reported by rr_plan_check, not in `result`. */
rr_status rr_unpack_verify_async(const rr_plan* plan, int32_t first_bucket, int32_t n_buckets,
                                 const void* const* buckets, const uint64_t* checksums,
                                 void* const* dst, uint8_t* bad, uint64_t* scratch,
                                 int64_t* result, cudaStream_t stream);

/* Allocation-free form of rr_verify.  The paper has no counterpart: this
 * entry point exists for callers that cannot allocate device memory when they
 * check a pull, such as an inference engine that has reserved nearly all
 * device memory for its weights and cache, or code running under a memory
 * pool that refuses new cudaMalloc calls.  It takes no plan, because creating
 * one allocates; the caller passes the buckets (host array of n_buckets device
 * pointers, bucket_bytes each), the expected checksums (device) and host
 * outputs as for rr_verify, and the result and blocking behaviour are those
 * of rr_verify.
 *   Scratch: one file-scope device array of 16384 + 4 64-bit words (128 KiB),
 *   which every GPU that loads this library keeps until the process exits.
 *   n_buckets above 16384 is rejected with RR_EINVAL.  Buckets that are not
 *   equally spaced (separately allocated, passed as a pointer table in the
 *   kernel's parameters) are limited to 3968 per call, RR_EINVAL beyond;
 *   equally spaced buckets (one allocation cut into buckets) have only the
 *   16384 limit.  The first call on a device sizes the grid for that device;
 *   make that first call before any stream capture.  Every call looks up the
 *   array's device address again (a device reset may move it).  Each call
 *   clears the part of the array it uses before its kernel runs; calls that
 *   overlap on the GPU (on different streams, or from different threads)
 *   share the array and race, so serialise them.  Calls no cudaMalloc or
 *   cudaFree. */
rr_status rr_verify_noalloc(const void* const* buckets, int32_t n_buckets, size_t bucket_bytes,
                            const uint64_t* checksums, int64_t* n_bad, int64_t* first_bad,
                            cudaStream_t stream);

/* Section 5.2.2: a role must know whether what it holds is whole.  Waits
 * for `stream`, then reports whether a kernel of this plan gave up on
 * a wait (the bulk-copy engine bounds every wait; one that runs out marks the
 * plan and its output is incomplete): RR_ECUDA if so (and clears the mark),
 * RR_OK otherwise.  rr_verify and rr_unpack_verify check this themselves. */
rr_status rr_plan_check(const rr_plan* plan, cudaStream_t stream);

/* Test hook for the bounded waits (no counterpart in the paper): enqueues on `stream` one small kernel that
 * waits on a barrier nothing completes.  The wait gives up after its limit
 * (about a second) and marks the plan, so the next rr_plan_check (or
 * rr_verify / rr_unpack_verify) reports RR_ECUDA while the CUDA context stays
 * usable.  It touches no buffer. */
rr_status rr_plan_selftest_wait(const rr_plan* plan, cudaStream_t stream);

/* A static description of a status code ("RR_OK", "RR_EINVAL: invalid
 * argument", ...; "unknown rr_status" otherwise), and this thread's
 * description of its most recent failure ("" if none).  The
 * returned strings are owned by the library.  No counterpart in the paper. */
const char* rr_status_str(rr_status status);
const char* rr_last_error(void);

#ifdef __cplusplus
}
#endif

#endif /* RR_H */
