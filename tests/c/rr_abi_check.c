/*
 * The C ABI of include/rr.h used from plain C11, with no Python in between.
 *
 * A two-parameter model is synced to a TP=2 rollout and compared with bytes
 * worked out by hand from the definitions at the top of rr.h:
 *
 *   A [4, 16] fp32, A[i][j] = i * 16 + j + 1 (integers up to 64, exact in
 *     bf16, so the bf16 bits are the upper half of the fp32 bits);
 *   B [8] bf16, B[k] = 0x4000 + k (copied bit for bit).
 *   Source: one flat buffer, A at byte 0 (256 B), B at byte 256 (16 B); the
 *     272 bytes pad to 288 = a multiple of 16 * 2 shards, so S = 144.
 *   Rank r: tensor "a" = A's columns [8r, 8r + 8) of all 4 rows (32 elements,
 *     stream bytes [0, 64)), tensor "b" = all of B (stream bytes [256, 272));
 *     272 stream bytes in buckets of 128 bytes: 3 per rank, 6 in all.
 *
 * Without arguments only host-side calls run (a host-only plan); with "gpu"
 * the plan runs: pack, verify, unpack, pack again from a source in pinned
 * host memory, and verify again after one byte of one bucket is damaged.
 * Exit status 0 means every check passed.
 */
#include <stdint.h>
#include <stdio.h>
#include <stdlib.h>
#include <string.h>

#include <cuda_runtime_api.h>

#include "rr.h"

#define CHECK(cond, what)                                                     \
    do {                                                                      \
        if (!(cond)) {                                                        \
            fprintf(stderr, "FAIL %s (line %d): %s\n", what, __LINE__,        \
                    rr_last_error());                                         \
            return 1;                                                         \
        }                                                                     \
    } while (0)

#define CUDA(call)                                                            \
    do {                                                                      \
        cudaError_t e_ = (call);                                              \
        if (e_ != cudaSuccess) {                                              \
            fprintf(stderr, "FAIL %s: %s\n", #call, cudaGetErrorString(e_));  \
            return 1;                                                         \
        }                                                                     \
    } while (0)

enum { BUCKET = 128, N_BUCKETS = 6, STREAM = 272, S = 144 };

static float a_value(int i, int j) { return (float)(i * 16 + j + 1); }

static uint16_t bf16_of(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    return (uint16_t)(u >> 16);
}

/* The 768 bucket bytes and 6 checksums, from the definitions. */
static void expected(uint8_t buckets[N_BUCKETS][BUCKET], uint64_t sums[N_BUCKETS]) {
    memset(buckets, 0, (size_t)N_BUCKETS * BUCKET);
    for (int r = 0; r < 2; ++r) {
        uint8_t stream[3 * BUCKET];
        memset(stream, 0, sizeof stream);
        for (int i = 0; i < 4; ++i)
            for (int j = 0; j < 8; ++j) {
                const uint16_t h = bf16_of(a_value(i, 8 * r + j));
                stream[2 * (i * 8 + j)] = (uint8_t)(h & 0xFF);
                stream[2 * (i * 8 + j) + 1] = (uint8_t)(h >> 8);
            }
        for (int k = 0; k < 8; ++k) {
            const uint16_t h = (uint16_t)(0x4000 + k);
            stream[256 + 2 * k] = (uint8_t)(h & 0xFF);
            stream[256 + 2 * k + 1] = (uint8_t)(h >> 8);
        }
        memcpy(buckets[3 * r], stream, 3 * BUCKET);
    }
    for (int b = 0; b < N_BUCKETS; ++b) {
        uint64_t s = 0;
        for (int w = 0; w < BUCKET / 8; ++w) {
            uint64_t word = 0;
            for (int i = 0; i < 8; ++i) word |= (uint64_t)buckets[b][8 * w + i] << (8 * i);
            s += word;
        }
        sums[b] = s;
    }
}

int main(int argc, char** argv) {
    const int gpu = argc > 1 && strcmp(argv[1], "gpu") == 0;
    rr_param man[2] = {{"A", 2, {4, 16, 0, 0}, RR_F32}, {"B", 1, {8, 0, 0, 0}, RR_BF16}};
    rr_src_layout src;
    memset(&src, 0, sizeof src);
    src.n_shards = 2;
    src.align_bytes = 16;
    src.sharding = RR_SHARD_FLAT;
    rr_block blocks[4] = {{0, 0, 4, 0, 8}, {1, 0, 8, 0, 1}, {0, 0, 4, 8, 8}, {1, 0, 8, 0, 1}};
    rr_dst_tensor tensors[4] = {{"a", 0, 32, 1, &blocks[0]}, {"b", 0, 8, 1, &blocks[1]},
                                {"a", 1, 32, 1, &blocks[2]}, {"b", 1, 8, 1, &blocks[3]}};
    rr_dst_layout dst = {2, 4, tensors, 256, RR_DST_BF16, 0};
    rr_plan_options opt;
    memset(&opt, 0, sizeof opt);
    opt.host_only = !gpu;

    /* Refusals come back as status codes with a message. */
    rr_plan* bad = NULL;
    CHECK(rr_plan_create_ex(man, 2, &src, &dst, 12, &opt, &bad) == RR_EINVAL && bad == NULL,
          "bucket size not a multiple of 8 refused");
    CHECK(strlen(rr_last_error()) > 0 && strcmp(rr_status_str(RR_EINVAL), "") != 0,
          "error text");
    rr_block off_end = {0, 3, 2, 0, 8};
    rr_dst_tensor t_bad = {"x", 0, 16, 1, &off_end};
    rr_dst_layout d_bad = {1, 1, &t_bad, 256, RR_DST_BF16, 0};
    CHECK(rr_plan_create_ex(man, 2, &src, &d_bad, 128, &opt, &bad) == RR_ELAYOUT,
          "rows past the parameter refused");
    rr_dst_layout d_type = {2, 4, tensors, 256, 7, 0};
    CHECK(rr_plan_create_ex(man, 2, &src, &d_type, 128, &opt, &bad) == RR_EINVAL,
          "unknown destination dtype refused");

    rr_plan* plan = NULL;
    CHECK(rr_plan_create_ex(man, 2, &src, &dst, BUCKET, &opt, &plan) == RR_OK, "plan");

    int32_t nb = 0, first[3] = {0, 0, 0};
    int64_t stream_bytes[2] = {0, 0};
    CHECK(rr_plan_query(plan, &nb, stream_bytes, first) == RR_OK, "query");
    CHECK(nb == N_BUCKETS && stream_bytes[0] == STREAM && stream_bytes[1] == STREAM &&
              first[0] == 0 && first[1] == 3 && first[2] == 6,
          "bucket geometry");
    int64_t shard = 0, flat = 0, offs[2] = {-1, -1};
    CHECK(rr_plan_source(plan, &shard, &flat, offs) == RR_OK, "source");
    CHECK(shard == S && flat == 272 && offs[0] == 0 && offs[1] == 256, "source geometry");
    int32_t n_buf = 0;
    int64_t buf_bytes[2] = {0, 0};
    CHECK(rr_plan_source_buffers(plan, &n_buf, buf_bytes) == RR_OK && n_buf == 2 &&
              buf_bytes[0] == S && buf_bytes[1] == S,
          "source buffers");
    int64_t numel[4], toff[4];
    CHECK(rr_plan_tensors(plan, numel, toff) == RR_OK, "tensors");
    CHECK(numel[0] == 32 && numel[1] == 8 && toff[0] == 0 && toff[1] == 256 && toff[3] == 256,
          "tensor geometry");
    int32_t n_units = -1;
    uint32_t unit_first[64], bucket_unit[N_BUCKETS + 1];
    CHECK(rr_plan_work_units(plan, RR_UNITS_UNPACK, &n_units, NULL, NULL) == RR_OK &&
              n_units >= N_BUCKETS && n_units < 64,
          "unit count");
    CHECK(rr_plan_work_units(plan, RR_UNITS_UNPACK, &n_units, unit_first, bucket_unit) == RR_OK &&
              unit_first[0] == 0 && bucket_unit[0] == 0 && bucket_unit[N_BUCKETS] == (uint32_t)n_units,
          "unit tables");
    CHECK(rr_plan_work_units(plan, 7, &n_units, NULL, NULL) == RR_EINVAL, "unknown unit table");
    CHECK(rr_plan_work_units(plan, RR_UNITS_PACK_FULL, &n_units, NULL, bucket_unit) == RR_EINVAL,
          "no bucket index for the whole-sync units");
    rr_plan_stats st;
    CHECK(rr_plan_get_stats(plan, &st) == RR_OK, "stats");
    CHECK(st.pack_bytes_read == 2 * (32 * 4 + 8 * 2) && st.pack_bytes_written == 6 * BUCKET,
          "algorithmic bytes");

    if (!gpu) {
        rr_plan_destroy(plan);
        printf("host ok\n");
        return 0;
    }

    /* The source, two shards of one allocation. */
    uint8_t host_flat[2 * S];
    memset(host_flat, 0, sizeof host_flat);
    for (int i = 0; i < 4; ++i)
        for (int j = 0; j < 16; ++j) {
            const float v = a_value(i, j);
            memcpy(host_flat + 4 * (i * 16 + j), &v, 4);
        }
    for (int k = 0; k < 8; ++k) {
        const uint16_t h = (uint16_t)(0x4000 + k);
        memcpy(host_flat + 256 + 2 * k, &h, 2);
    }
    uint8_t *d_flat = NULL, *d_buckets = NULL, *d_dst = NULL;
    uint64_t* d_sums = NULL;
    CUDA(cudaMalloc((void**)&d_flat, sizeof host_flat));
    CUDA(cudaMalloc((void**)&d_buckets, N_BUCKETS * BUCKET));
    CUDA(cudaMalloc((void**)&d_sums, N_BUCKETS * sizeof(uint64_t)));
    CUDA(cudaMalloc((void**)&d_dst, 4 * 256));
    CUDA(cudaMemcpy(d_flat, host_flat, sizeof host_flat, cudaMemcpyHostToDevice));
    CUDA(cudaMemset(d_buckets, 0xAB, N_BUCKETS * BUCKET));
    const void* shards[2] = {d_flat, d_flat + S};
    void* bucket_ptrs[N_BUCKETS];
    for (int b = 0; b < N_BUCKETS; ++b) bucket_ptrs[b] = d_buckets + b * BUCKET;
    void* dst_ptrs[4];
    for (int t = 0; t < 4; ++t) dst_ptrs[t] = d_dst + 256 * t;

    CHECK(rr_pack(plan, shards, bucket_ptrs, d_sums, 0) == RR_OK, "pack");
    CUDA(cudaDeviceSynchronize());
    uint8_t got[N_BUCKETS][BUCKET], want[N_BUCKETS][BUCKET];
    uint64_t got_sums[N_BUCKETS], want_sums[N_BUCKETS];
    expected(want, want_sums);
    CUDA(cudaMemcpy(got, d_buckets, sizeof got, cudaMemcpyDeviceToHost));
    CUDA(cudaMemcpy(got_sums, d_sums, sizeof got_sums, cudaMemcpyDeviceToHost));
    CHECK(memcmp(got, want, sizeof got) == 0, "bucket bytes");
    CHECK(memcmp(got_sums, want_sums, sizeof got_sums) == 0, "checksums");

    int64_t n_bad = -1, first_bad = -2;
    CHECK(rr_verify(plan, (const void* const*)bucket_ptrs, d_sums, &n_bad, &first_bad, 0) ==
                  RR_OK &&
              n_bad == 0 && first_bad == -1,
          "verify clean");
    CHECK(rr_unpack(plan, (const void* const*)bucket_ptrs, dst_ptrs, 0) == RR_OK, "unpack");
    CUDA(cudaDeviceSynchronize());
    uint8_t t_a1[64], t_b0[16];
    CUDA(cudaMemcpy(t_a1, d_dst + 256 * 2, 64, cudaMemcpyDeviceToHost));
    CUDA(cudaMemcpy(t_b0, d_dst + 256 * 1, 16, cudaMemcpyDeviceToHost));
    CHECK(memcmp(t_a1, want[3], 64) == 0 && memcmp(t_b0, want[2] + 0, 16) == 0,
          "unpacked tensors");

    /* The same pack with the source left in pinned host memory: the pack's own
     * loads read it over the host link; the bytes are the same. */
    uint8_t* h_flat = NULL;
    uint8_t* d_buckets2 = NULL;
    uint64_t* d_sums2 = NULL;
    CUDA(cudaMallocHost((void**)&h_flat, sizeof host_flat));
    memcpy(h_flat, host_flat, sizeof host_flat);
    CUDA(cudaMalloc((void**)&d_buckets2, N_BUCKETS * BUCKET));
    CUDA(cudaMalloc((void**)&d_sums2, N_BUCKETS * sizeof(uint64_t)));
    CUDA(cudaMemset(d_buckets2, 0xAB, N_BUCKETS * BUCKET));
    const void* h_shards[2] = {h_flat, h_flat + S};
    void* bucket_ptrs2[N_BUCKETS];
    for (int b = 0; b < N_BUCKETS; ++b) bucket_ptrs2[b] = d_buckets2 + b * BUCKET;
    CHECK(rr_pack(plan, h_shards, bucket_ptrs2, d_sums2, 0) == RR_OK, "pack from host memory");
    CUDA(cudaDeviceSynchronize());
    CUDA(cudaMemcpy(got, d_buckets2, sizeof got, cudaMemcpyDeviceToHost));
    CUDA(cudaMemcpy(got_sums, d_sums2, sizeof got_sums, cudaMemcpyDeviceToHost));
    CHECK(memcmp(got, want, sizeof got) == 0, "bucket bytes, host source");
    CHECK(memcmp(got_sums, want_sums, sizeof got_sums) == 0, "checksums, host source");
    cudaFreeHost(h_flat);
    cudaFree(d_buckets2);
    cudaFree(d_sums2);

    CUDA(cudaMemset(d_buckets + 4 * BUCKET + 7, 0x5A, 1));   /* one damaged byte */
    CHECK(rr_verify(plan, (const void* const*)bucket_ptrs, d_sums, &n_bad, &first_bad, 0) ==
                  RR_EMISMATCH &&
              n_bad == 1 && first_bad == 4,
          "verify finds the damaged bucket");

    rr_plan_destroy(plan);
    cudaFree(d_flat);
    cudaFree(d_buckets);
    cudaFree(d_sums);
    cudaFree(d_dst);
    printf("gpu ok\n");
    return 0;
}
