// quant_math.cuh -- the per-element arithmetic of the blockwise FP8 cast
// (section "FP8 Mixed-Precision Training"): the E8M0 scale exponent of a
// group from its BF16 amax, the saturating round-to-nearest-even FP8
// encoding of x * 2^(127-g), and the tensor-core layout of the scale
// vectors.  Shared by the quantiser kernels and the GEMM epilogue that
// quantises its own output, so both produce the same bytes from the same
// BF16 values.
#pragma once

#include <cfloat>
#include <cstdint>

#include "ptx.cuh"

namespace puro {

// Smallest power of two 2^(g-127) with amax <= fmt_max * 2^(g-127), from
// the bf16 bit fields of amax = 1.m x 2^(E-127): fmt_max = 1.75 x 2^P with
// P = 8 (E4M3) or 15 (E5M2), so g = E - P, plus one when 1.m > 1.75
// (m > 96/128).  bf16 subnormals and tiny values clamp at g = 0; zero gives
// g = 127; a non-finite amax gives 0xFF.
template <int FMT>
PURO_DEV uint32_t e8m0_exponent(uint32_t amax_bits) {
    constexpr int P = (FMT == 0) ? 8 : 15;
    if (amax_bits == 0) return 127u;
    if (amax_bits >= 0x7F80u) return 0xFFu;
    const int E = static_cast<int>(amax_bits >> 7);
    if (E == 0) return 0u;
    const int g = E - P + (((amax_bits & 0x7Fu) > 96u) ? 1 : 0);
    return g < 0 ? 0u : static_cast<uint32_t>(g);
}

template <int FMT>
PURO_DEV uint32_t cvt_pair(float lo, float hi) {  // -> 16 bits, lo in the low byte
    uint16_t r;
    if constexpr (FMT == 0)
        asm("cvt.rn.satfinite.e4m3x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
    else
        asm("cvt.rn.satfinite.e5m2x2.f32 %0, %1, %2;" : "=h"(r) : "f"(hi), "f"(lo));
    return r;
}

PURO_DEV float bf16_lo(uint32_t w) { return __uint_as_float(w << 16); }
PURO_DEV float bf16_hi(uint32_t w) { return __uint_as_float(w & 0xFFFF0000u); }

PURO_DEV uint64_t f32x2(float lo, float hi) {
    uint64_t r;
    asm("mov.b64 %0, {%1, %2};" : "=l"(r) : "f"(lo), "f"(hi));
    return r;
}

// Two IEEE round-to-nearest fp32 products in one packed instruction.
PURO_DEV uint64_t mul_f32x2(uint64_t a, uint64_t b) {
    uint64_t r;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(r) : "l"(a), "l"(b));
    return r;
}

template <int FMT>
PURO_DEV uint32_t cvt_f32x2(uint64_t v) {
    float lo, hi;
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
    return cvt_pair<FMT>(lo, hi);
}

// Codes of four values a, b, c, d (exact fp32 widenings of bf16) as four
// bytes, a in the low byte.  `mul2` holds the multiplier twice: the exact
// power of two 2^(127-g) (BLOCK) or the fp32 tensor scale (TENSOR).  A
// non-finite group gives NaN codes that keep each value's sign.
template <int FMT>
PURO_DEV uint32_t quant4(float a, float b, float c, float d, uint64_t mul2, bool nan_group) {
    if (__builtin_expect(nan_group, 0)) {
        const uint32_t s = ((__float_as_uint(a) >> 24) & 0x80u) | (((__float_as_uint(b) >> 24) & 0x80u) << 8) |
                           (((__float_as_uint(c) >> 24) & 0x80u) << 16) | (((__float_as_uint(d) >> 24) & 0x80u) << 24);
        return s | 0x7F7F7F7Fu;
    }
    return cvt_f32x2<FMT>(mul_f32x2(f32x2(a, b), mul2)) | (cvt_f32x2<FMT>(mul_f32x2(f32x2(c, d), mul2)) << 16);
}

// Exact 2^(127 - g) as fp32 for g in [0, 247] (always a normal number).
PURO_DEV float pow2_inv_scale(uint32_t g) { return __uint_as_float((254u - g) << 23); }

template <int FMT>
PURO_DEV float tensor_scale(uint32_t amax_bits) {
    constexpr float kMax = (FMT == 0) ? 448.0f : 57344.0f;
    if (amax_bits == 0) return 1.0f;
    float s = __fdiv_rn(kMax, __uint_as_float(amax_bits << 16));
    return isinf(s) ? FLT_MAX : s;
}

// Tensor-core scale-vector layout of an FP8 operand [R, red] (see the
// public header): 512-byte chunks per (128-row block, group of four
// k-blocks); byte 16*l + 4*j + b of chunk (rb, kg) is the exponent of row
// 128*rb + 32*j + l for k-block 4*kg + b.  The tile that owns the last
// k-block also fills the group's unused bytes with 127 (scale 1).
PURO_DEV void store_scale_vec(uint8_t *__restrict__ base, int64_t row, int64_t kb, int64_t kblocks, uint8_t g) {
    const int64_t groups = (kblocks + 3) / 4;
    const int64_t rb = row / 128;
    const int i = static_cast<int>(row & 127);
    uint8_t *chunk = base + (rb * groups + kb / 4) * 512 + 16 * (i & 31) + 4 * (i >> 5);
    const int b = static_cast<int>(kb & 3);
    chunk[b] = g;
    if (kb == kblocks - 1)
        for (int pb = b + 1; pb < 4; ++pb) chunk[pb] = 127;
}

// 2^(127-g) for a scale exponent, NaN for the non-finite marker 0xFF.
PURO_DEV float mul_of(uint32_t g) { return g == 0xFFu ? __uint_as_float(0x7FC00000u) : pow2_inv_scale(g); }

}  // namespace puro
