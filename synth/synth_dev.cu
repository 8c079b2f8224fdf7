/*
 * Seeded synthetic parameter generator, device side.
 *
 * Input generation only: the same counter-based definition as synth_host.c
 * (SplitMix64 -> Irwin-Hall of four 16-bit fields -> one binary32 multiply,
 * optional 1% special bit patterns), evaluated on the GPU so that tens of GB
 * of model-shaped source can be produced in HBM without a host copy.  It
 * shares no code with the weight-sync kernels.
 */
#include <cuda_runtime.h>
#include <stdint.h>

#include "synth_specials.h"

__constant__ uint32_t d_special_f32[SYNTH_N_SPECIAL];

__device__ __forceinline__ uint64_t splitmix64(uint64_t x) {
    uint64_t z = x + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ uint32_t f32_bits(uint64_t seed, int64_t idx, int specials) {
    uint64_t h = splitmix64((seed << 40) ^ (uint64_t)idx);
    if (specials) {
        uint64_t h2 = splitmix64(h);
        if (h2 % 100u == 0u) return d_special_f32[(h2 >> 32) % SYNTH_N_SPECIAL];
    }
    int32_t s = (int32_t)(h & 0xFFFFu) + (int32_t)((h >> 16) & 0xFFFFu) +
                (int32_t)((h >> 32) & 0xFFFFu) + (int32_t)((h >> 48) & 0xFFFFu);
    float x = __fmul_rn((float)(s - 131070), __uint_as_float(SYNTH_SCALE_BITS));
    return __float_as_uint(x);
}

__global__ void synth_fill_kernel(void* out, int64_t n, int elem_bytes, uint64_t seed,
                                  int64_t first_idx, int specials) {
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    if (elem_bytes == 4) {
        uint32_t* o = (uint32_t*)out;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
            o[i] = f32_bits(seed, first_idx + i, specials);
    } else {
        uint16_t* o = (uint16_t*)out;
        for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
            o[i] = (uint16_t)(f32_bits(seed, first_idx + i, specials) >> 16);
    }
}

__global__ void synth_gather_kernel(void* out, const int64_t* idx, int64_t n, int elem_bytes,
                                    uint64_t seed, int specials) {
    int64_t stride = (int64_t)gridDim.x * blockDim.x;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride) {
        uint32_t b = f32_bits(seed, idx[i], specials);
        if (elem_bytes == 4) ((uint32_t*)out)[i] = b;
        else ((uint16_t*)out)[i] = (uint16_t)(b >> 16);
    }
}

static int ensure_table(void) {
    /* The table is per device; copy it each time (a few dozen bytes). */
    return cudaMemcpyToSymbol(d_special_f32, SPECIAL_F32, sizeof(SPECIAL_F32)) == cudaSuccess ? 0 : -1;
}

static int grid_for(int64_t n) {
    int dev = 0, sms = 0;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int64_t want = (n + 255) / 256;
    int64_t cap = (int64_t)(sms > 0 ? sms : 1) * 8;
    if (want > cap) want = cap;
    return (int)(want < 1 ? 1 : want);
}

/* Fill n elements of `out` (device) with the values of indices first_idx..first_idx+n-1.
 * Returns 0, or a CUDA error code. */
extern "C" int synth_fill_dev(void* out, int64_t n, int elem_bytes, uint64_t seed,
                              int64_t first_idx, int specials, cudaStream_t stream) {
    if (n <= 0) return 0;
    if (elem_bytes != 2 && elem_bytes != 4) return -2;
    if (ensure_table()) return (int)cudaGetLastError();
    synth_fill_kernel<<<grid_for(n), 256, 0, stream>>>(out, n, elem_bytes, seed, first_idx,
                                                        specials);
    return (int)cudaGetLastError();
}

/* out[i] = value at element index idx[i] (idx on the device). */
extern "C" int synth_gather_dev(void* out, const int64_t* idx, int64_t n, int elem_bytes,
                                uint64_t seed, int specials, cudaStream_t stream) {
    if (n <= 0) return 0;
    if (elem_bytes != 2 && elem_bytes != 4) return -2;
    if (ensure_table()) return (int)cudaGetLastError();
    synth_gather_kernel<<<grid_for(n), 256, 0, stream>>>(out, idx, n, elem_bytes, seed, specials);
    return (int)cudaGetLastError();
}
