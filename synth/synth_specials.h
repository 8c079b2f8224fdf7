/*
 * Bit patterns (float32) that the seeded generator injects when `specials` is
 * set: rounding ties of both parities, overflow into infinity, subnormals,
 * signed zeros, infinities and NaNs with assorted payloads.  Shared by the
 * host and device generators; input generation only.
 */
#pragma once
#include <stdint.h>

static const uint32_t SPECIAL_F32[] = {
    0x3F808000u, /* tie, kept bf16 mantissa even: stays 0x3F80            */
    0x3F818000u, /* tie, bf16 mantissa odd: rounds up to 0x3F82           */
    0xBF838000u, /* negative tie, odd: rounds away from zero to 0xBF84    */
    0x3F80FFFFu, /* just below a tie: rounds down                          */
    0x3F808001u, /* just above a tie: rounds up                            */
    0x7F7F8000u, /* tie at the largest bf16 finite, odd: overflows to +inf */
    0x7F7FFFFFu, /* largest binary32 finite: rounds to +inf               */
    0xFF7F7FFFu, /* below the overflow tie: stays finite (0xFF7F)          */
    0x00000001u, /* smallest subnormal: rounds to +0                       */
    0x00008000u, /* subnormal tie, even: rounds to 0x0000                  */
    0x00018000u, /* subnormal tie, odd: rounds up to 0x0002                */
    0x007FFFFFu, /* largest subnormal: carries into the smallest normal    */
    0x80000000u, /* -0                                                     */
    0x00000000u, /* +0                                                     */
    0x7F800000u, /* +inf                                                   */
    0xFF800000u, /* -inf                                                   */
    0x7FC00000u, /* canonical quiet NaN                                    */
    0x7FA00000u, /* signalling NaN                                         */
    0x7F800001u, /* NaN whose payload sits only in the low 16 bits         */
    0xFFC12345u, /* negative quiet NaN with payload                        */
};
#define SYNTH_N_SPECIAL ((uint64_t)(sizeof(SPECIAL_F32) / sizeof(SPECIAL_F32[0])))
#define SYNTH_SCALE_BITS 0x350DE3F5u
