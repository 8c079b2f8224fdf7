// Internal plan representation shared by the host planner (rr_plan.cpp) and
// the device code (rr_device.cu).  Not part of the public ABI.
#pragma once

#include <mutex>
#include <string>
#include <vector>

#include <nvtx3/nvToolsExt.h>

#include "rr.h"

// A scoped NVTX range named after a C-ABI call: visible on the timeline of an
// Nsight tool attached to the process, close to free when none is.
struct RrTraceRange {
    explicit RrTraceRange(const char* name) { nvtxRangePushA(name); }
    ~RrTraceRange() { nvtxRangePop(); }
    RrTraceRange(const RrTraceRange&) = delete;
    RrTraceRange& operator=(const RrTraceRange&) = delete;
};
#define RR_TRACE(name) RrTraceRange rr_trace_range_(name)

struct rr_plan {
    // ---- source ---------------------------------------------------------
    int32_t n_params = 0;
    std::vector<int64_t> rows, cols;   // matrix view of each parameter
    std::vector<int32_t> es;           // element bytes (4 or 2)
    std::vector<int64_t> param_off;    // flat byte offsets (FLAT), in-shard offsets (ROWS),
                                       // offsets within the unit (UNITS)
    std::vector<int64_t> chunk_rows;   // ROWS: rows per shard, ceil(rows / n_shards)
    int32_t sharding = RR_SHARD_FLAT;
    int32_t n_shards = 0;              // source buffers the calls take
    int64_t shard_bytes = 0;           // S (UNITS: the largest S_u)
    int64_t flat_bytes = 0;
    int32_t unit_shards = 0;           // UNITS: shards per unit
    std::vector<int32_t> unit_of;      // UNITS: unit of each parameter
    std::vector<int64_t> unit_shard_bytes;  // UNITS: S_u

    // ---- destination ----------------------------------------------------
    int32_t tp = 0;
    int32_t n_tensors = 0;
    std::vector<int32_t> tensor_rank;
    std::vector<int64_t> tensor_numel;
    std::vector<int64_t> tensor_off;   // byte offset in its rank's stream
    int64_t tensor_align = 0;
    int64_t bucket_bytes = 0;
    std::vector<int64_t> rank_stream_bytes;
    std::vector<int32_t> rank_first_bucket;  // tp + 1
    int32_t n_buckets = 0;

    // ---- work tables ----------------------------------------------------
    int32_t grid_blocks = 0;          // pack kernel grid (the partition's block count)
    int32_t unpack_grid_blocks = 0;   // unpack kernel grid (likewise)
    int32_t verify_grid_blocks = 0;
    int32_t reg_pack_grid = 0;        // register-path grids when the bulk engine is the default
    int32_t reg_unpack_grid = 0;
    int32_t reg_vunpack_grid = 0;     // the register path's verifying unpack (its own block size)
    int32_t engine = RR_ENGINE_AUTO;
    int32_t dst_f16 = 0;              // the rollout's elements are float16 (else bfloat16)
    int64_t chunk_bytes = 0;
    bool host_only = false;
    std::vector<rr_pack_item> pack_items;
    std::vector<uint32_t> pack_block_first;     // grid_blocks + 1
    std::vector<rr_unpack_item> unpack_items;
    std::vector<uint32_t> unpack_block_first;   // grid_blocks + 1
    // Claimed work units of the bulk-copy engine: first item of each unit (+ 1
    // past the last); per bucket, its first unit (n_buckets + 1).
    std::vector<uint32_t> unpack_unit_first;
    std::vector<uint32_t> unpack_bucket_unit;
    std::vector<uint32_t> pack_unit_first;
    std::vector<uint32_t> pack_bucket_unit;
    std::vector<uint32_t> pack_whole_unit_first;   // a pack over every bucket: own units
                                                   //   (one per block), then claimed ones
    std::vector<uint32_t> pack_bucket_first;    // n_buckets + 1: first pack item of bucket b
    std::vector<unsigned long long> pack_weight_prefix;    // items + 1: balancing weights,
    std::vector<unsigned long long> unpack_weight_prefix;  // summed (bucket-range calls)
    std::vector<rr_pack_item> full_items;       // whole-sync table with fan-out groups;
                                                // empty when it would equal pack_items
    std::vector<uint32_t> full_block_first;     // grid_blocks + 1
    std::vector<uint32_t> unpack_bucket_first;  // n_buckets + 1: first unpack item of bucket b
    std::vector<int32_t> bucket_tensor_lo;      // n_buckets: lowest / highest destination
    std::vector<int32_t> bucket_tensor_hi;      //   tensor a bucket's unpack items write
    rr_plan_stats stats{};

    // ---- device state (owned) -------------------------------------------
    int device = -1;
    rr_pack_item* d_pack_items = nullptr;
    uint32_t* d_pack_block_first = nullptr;
    rr_pack_item* d_full_items = nullptr;
    uint32_t* d_full_block_first = nullptr;
    unsigned long long* d_pack_weight_prefix = nullptr;
    unsigned long long* d_unpack_weight_prefix = nullptr;
    int32_t check_items = 0;                 // kernels check every item's bounds
    int32_t pageable_ok = 0;                 // the device can read pageable host memory
    int64_t* d_src_bytes = nullptr;          // check_items: bytes of each source buffer
    int64_t* d_tensor_bytes = nullptr;       //              and of each destination tensor
    rr_unpack_item* d_unpack_items = nullptr;
    uint32_t* d_unpack_block_first = nullptr;
    uint32_t* d_unpack_unit_first = nullptr;
    uint32_t* d_pack_unit_first = nullptr;
    uint32_t* d_pack_whole_unit_first = nullptr;
    // Pooled scratch of launches that need no per-call scratch: a slot is
    // handed to a launch only once the event recorded after its previous
    // launch has completed, and that launch's last block left it zeroed.  Slot
    // k is slot_words() words at d_slots + k * slot_words(): per-bucket sums
    // [n_buckets], then counters {ticket, n_bad, max(~0 - bad index), claim}.
    static constexpr int kClaimSlots = 16;
    unsigned long long* d_slots = nullptr;
    size_t slot_words() const { return size_t(n_buckets) + 4; }
    cudaEvent_t claim_done[kClaimSlots] = {};
    cudaStream_t claim_stream[kClaimSlots] = {};   // the stream of the slot's last launch
    char claim_retired[kClaimSlots] = {};
    int32_t claim_next = 0;
    std::mutex claim_mutex;
    unsigned long long* d_verify_scratch = nullptr;  // n_buckets sums + 4 counters
    unsigned long long* h_verify_result = nullptr;   // pinned, 5 words (4 counters + error)
    unsigned int* d_error = nullptr;                 // set by a kernel whose wait ran out
    std::mutex verify_mutex;
};

// Records a per-thread error message and returns s.
rr_status rr_fail(rr_status s, const char* fmt, ...);
void rr_clear_error();

// Device side (rr_device.cu).
struct rr_grids {
    int32_t bulk_pack, bulk_unpack, reg_pack, reg_unpack, verify, reg_vunpack;
};
rr_status rr_device_default_grid(rr_grids* g);
rr_status rr_device_upload(rr_plan* p);
void rr_device_release(rr_plan* p);
