/*
 * Seeded synthetic parameter generator, host side.
 *
 * This file is input generation only: it holds none of the weight-sync
 * method's arithmetic (no layout, no cast, no packing, no checksum).  The
 * same counter-based definition is implemented on the device in
 * synth_dev.cu; a GPU test checks that both produce identical bits.
 *
 * Definition (one value per element index `idx` of the unsharded flat
 * parameter buffer, i.e. flat byte offset / element size):
 *
 *   key = (seed << 40) ^ idx
 *   h   = splitmix64(key)                     SplitMix64 finaliser
 *                                             (Steele, Lea, Flood, OOPSLA 2014)
 *   s   = sum of the four 16-bit fields of h  Irwin-Hall of 4 uniforms on
 *                                             [0, 65535]: mean 131070,
 *                                             sd 37837.2
 *   x   = float(s - 131070) * SCALE           one IEEE binary32 multiply,
 *                                             SCALE = binary32 nearest to
 *                                             0.02 / 37837 (bits 0x350DE3F5)
 *
 * so x approximates N(0, 0.02), the spread of freshly initialised LLM
 * weights.  With `specials` set, h2 = splitmix64(h) replaces about 1% of
 * the values (h2 % 100 == 0) by SPECIAL_F32[(h2 >> 32) % SYNTH_N_SPECIAL]: bit
 * patterns that stress a float32 -> bfloat16 round-to-nearest-even cast.
 * A bf16 source takes the upper 16 bits of x's binary32 pattern.
 */
#include <stdint.h>
#include <string.h>

#include "synth_specials.h"


uint64_t synth_splitmix64(uint64_t x) {
    uint64_t z = x + 0x9E3779B97F4A7C15ull;
    z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
    z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
    return z ^ (z >> 31);
}

static float bits_to_float(uint32_t u) {
    float f;
    memcpy(&f, &u, 4);
    return f;
}

static uint32_t float_to_bits(float f) {
    uint32_t u;
    memcpy(&u, &f, 4);
    return u;
}

uint32_t synth_f32_bits(uint64_t seed, int64_t idx, int specials) {
    uint64_t h = synth_splitmix64((seed << 40) ^ (uint64_t)idx);
    if (specials) {
        uint64_t h2 = synth_splitmix64(h);
        if (h2 % 100u == 0u) return SPECIAL_F32[(h2 >> 32) % SYNTH_N_SPECIAL];
    }
    int32_t s = (int32_t)(h & 0xFFFFu) + (int32_t)((h >> 16) & 0xFFFFu) +
                (int32_t)((h >> 32) & 0xFFFFu) + (int32_t)((h >> 48) & 0xFFFFu);
    float centred = (float)(s - 131070);   /* exact: |s - 131070| < 2^24 */
    float x = centred * bits_to_float(SYNTH_SCALE_BITS);
    return float_to_bits(x);
}

uint16_t synth_bf16_bits(uint64_t seed, int64_t idx, int specials) {
    return (uint16_t)(synth_f32_bits(seed, idx, specials) >> 16);
}

/* Fill out[0..n) with the values of element indices first_idx .. first_idx+n-1.
 * elem_bytes is 4 (float32 bits) or 2 (bf16 bits). */
void synth_fill_host(void* out, int64_t n, int elem_bytes, uint64_t seed, int64_t first_idx,
                     int specials) {
    if (elem_bytes == 4) {
        uint32_t* o = (uint32_t*)out;
        for (int64_t i = 0; i < n; ++i) o[i] = synth_f32_bits(seed, first_idx + i, specials);
    } else {
        uint16_t* o = (uint16_t*)out;
        for (int64_t i = 0; i < n; ++i) o[i] = synth_bf16_bits(seed, first_idx + i, specials);
    }
}

/* Gather form: out[i] = value at element index idx[i]. */
void synth_gather_host(void* out, const int64_t* idx, int64_t n, int elem_bytes, uint64_t seed,
                       int specials) {
    if (elem_bytes == 4) {
        uint32_t* o = (uint32_t*)out;
        for (int64_t i = 0; i < n; ++i) o[i] = synth_f32_bits(seed, idx[i], specials);
    } else {
        uint16_t* o = (uint16_t*)out;
        for (int64_t i = 0; i < n; ++i) o[i] = synth_bf16_bits(seed, idx[i], specials);
    }
}

/* Context-taking form, so that a consumer written in C can draw source values
 * through a plain function pointer without linking this file. */
typedef struct {
    uint64_t seed;
    int32_t specials;
} synth_ctx;

uint32_t synth_value_fn(const void* ctx, int64_t idx, int32_t elem_bytes) {
    const synth_ctx* c = (const synth_ctx*)ctx;
    uint32_t b = synth_f32_bits(c->seed, idx, c->specials);
    return elem_bytes == 4 ? b : (b >> 16);
}

int synth_n_special(void) { return (int)SYNTH_N_SPECIAL; }

void synth_special_table(uint32_t* out) {
    for (uint64_t i = 0; i < SYNTH_N_SPECIAL; ++i) out[i] = SPECIAL_F32[i];
}
