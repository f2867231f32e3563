// quantize.cu -- amax reduction and the fused BF16 -> FP8 cast(+transpose)
// kernels of the FP8 linear path (Puro-2B, section "FP8 Mixed-Precision
// Training": scales computed online per local group -- 1x128 groups along
// the GEMM reduction dimension for activations and activation gradients,
// 128x128 blocks for weights -- each a power of two).
//
// Both kernels are HBM-bandwidth bound.  The cast kernel reads each 128x128
// BF16 tile once (cp.async, double buffered), computes the row-group and the
// column-group scales from the same shared-memory copy, and writes the
// rowwise codes and the transposed codes through shared memory with TMA
// stores (the transposed staging tile uses the 128-byte swizzle so the
// column pass stores without bank conflicts).  The arithmetic per value is
// kept to a widening shift, half a packed fp32 multiply and half a paired
// cvt, since at HBM rates the kernel is otherwise instruction bound.
#include <cfloat>
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace puro {

// --------------------------------------------------------------- amax
// Integer max of (bits & 0x7FFF) over bf16 values: exact for finite values,
// +inf sorts above them and NaN above +inf.
__global__ void __launch_bounds__(256) amax_kernel(const uint4 *__restrict__ x, int64_t nvec,
                                                   const uint16_t *__restrict__ tail, int ntail,
                                                   uint32_t *__restrict__ out) {
    uint32_t m2 = 0;  // two packed 16-bit running maxima
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    for (; i + 3 * stride < nvec; i += 4 * stride) {
        uint4 v0 = __ldg(x + i), v1 = __ldg(x + i + stride), v2 = __ldg(x + i + 2 * stride),
              v3 = __ldg(x + i + 3 * stride);
        m2 = __vmaxu2(m2, __vmaxu2(__vmaxu2(v0.x & 0x7FFF7FFFu, v0.y & 0x7FFF7FFFu),
                                   __vmaxu2(v0.z & 0x7FFF7FFFu, v0.w & 0x7FFF7FFFu)));
        m2 = __vmaxu2(m2, __vmaxu2(__vmaxu2(v1.x & 0x7FFF7FFFu, v1.y & 0x7FFF7FFFu),
                                   __vmaxu2(v1.z & 0x7FFF7FFFu, v1.w & 0x7FFF7FFFu)));
        m2 = __vmaxu2(m2, __vmaxu2(__vmaxu2(v2.x & 0x7FFF7FFFu, v2.y & 0x7FFF7FFFu),
                                   __vmaxu2(v2.z & 0x7FFF7FFFu, v2.w & 0x7FFF7FFFu)));
        m2 = __vmaxu2(m2, __vmaxu2(__vmaxu2(v3.x & 0x7FFF7FFFu, v3.y & 0x7FFF7FFFu),
                                   __vmaxu2(v3.z & 0x7FFF7FFFu, v3.w & 0x7FFF7FFFu)));
    }
    for (; i < nvec; i += stride) {
        uint4 v = __ldg(x + i);
        m2 = __vmaxu2(m2, __vmaxu2(__vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu),
                                   __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu)));
    }
    if (blockIdx.x == 0 && threadIdx.x < ntail) m2 = __vmaxu2(m2, tail[threadIdx.x] & 0x7FFFu);
    uint32_t m = max(m2 & 0xFFFFu, m2 >> 16);
    m = __reduce_max_sync(0xFFFFFFFFu, m);
    __shared__ uint32_t warp_max[8];
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) warp_max[warp] = m;
    __syncthreads();
    if (warp == 0) {
        m = (threadIdx.x < 8) ? warp_max[threadIdx.x] : 0u;
        m = __reduce_max_sync(0xFFFFFFFFu, m);
        if (threadIdx.x == 0 && m != 0) atomicMax(out, m);
    }
}

cudaError_t launch_amax(const uint16_t *x, int64_t n, uint32_t *amax, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(amax, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess || n == 0) return e;
    const int64_t nvec = n / 8;
    const int ntail = static_cast<int>(n - nvec * 8);
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    int64_t want = (nvec + 255) / 256;
    int64_t cap = static_cast<int64_t>(sms) * 8;
    int grid = static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
    amax_kernel<<<grid, 256, 0, s>>>(reinterpret_cast<const uint4 *>(x), nvec, x + nvec * 8, ntail, amax);
    return cudaGetLastError();
}

// ------------------------------------------------------ scale helpers
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

// max of the bf16 magnitudes in each 16-bit half, over four words
PURO_DEV uint32_t max_abs4(uint4 v) {
    return __vmaxu2(__vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu), __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu));
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

// ------------------------------------------------------ cast kernel
constexpr int kQT = 128;          // tile edge
constexpr int kQThreads = 256;

struct QuantSmem {
    alignas(1024) uint8_t qt_stage[kQT * kQT];    // transposed codes, 128B-swizzled rows
    alignas(1024) uint8_t q_stage[kQT * kQT];     // rowwise codes, plain rows
    alignas(128) uint16_t in[2][kQT * kQT];       // bf16 tile, double buffered
    uint32_t col_amax2[4][kQT / 2];  // per row quarter, two columns per word
    uint32_t red[8];
    alignas(16) uint8_t row_g[kQT];
    alignas(16) uint8_t col_g[kQT];
};

PURO_DEV void load_tile_async(uint16_t *dst, const uint16_t *__restrict__ x, int64_t rows, int64_t cols,
                              int64_t r0, int64_t c0) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        const int k = threadIdx.x + kQThreads * i;  // 16-byte chunk id in the tile
        const int r = k >> 4, cc = (k & 15) * 8;
        const int64_t gr = r0 + r, gc = c0 + cc;
        const bool ok = (gr < rows) && (gc < cols);
        const uint16_t *src = ok ? x + gr * cols + gc : x;
        cp_async_16(dst + r * kQT + cc, src, ok ? 16u : 0u);
    }
    cp_async_commit();
}

template <int FMT, int KIND, bool HAS_T>
__global__ void __launch_bounds__(kQThreads, 2)
    quant_tile_kernel(const __grid_constant__ CUtensorMap tm_q, const __grid_constant__ CUtensorMap tm_qt,
                      const uint16_t *__restrict__ x, int64_t rows, int64_t cols,
                      uint8_t *__restrict__ scale_u8, uint8_t *__restrict__ scale_t_u8, float *scale_f,
                      float *scale_t_f, const uint32_t *__restrict__ amax_bits, int tiles_n, int ntiles) {
    extern __shared__ uint8_t smem_raw[];
    QuantSmem &sm = *reinterpret_cast<QuantSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                   ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;

    // Per-tensor mode: the one scale, from the device amax.
    float t_scale = 1.0f;
    bool t_nan = false;
    if constexpr (KIND == kQuantTensor) {
        const uint32_t a = *amax_bits & 0xFFFFu;
        t_nan = a >= 0x7F80u;
        t_scale = tensor_scale<FMT>(a);
        if (blockIdx.x == 0 && tid == 0) {
            const float si = t_nan ? __uint_as_float(0x7FC00000u) : __fdiv_rn(1.0f, t_scale);
            *scale_f = si;
            if (scale_t_f) *scale_t_f = si;
        }
    }
    if (tid == 0) {
        tma_prefetch_desc(&tm_q);
        if (HAS_T) tma_prefetch_desc(&tm_qt);
    }

    int tile = blockIdx.x;
    if (tile < ntiles)
        load_tile_async(sm.in[0], x, rows, cols, static_cast<int64_t>(tile / tiles_n) * kQT,
                        static_cast<int64_t>(tile % tiles_n) * kQT);
    for (int it = 0; tile < ntiles; ++it, tile += gridDim.x) {
        const int buf = it & 1;
        const int64_t r0 = static_cast<int64_t>(tile / tiles_n) * kQT;
        const int64_t c0 = static_cast<int64_t>(tile % tiles_n) * kQT;
        const int next = tile + gridDim.x;
        if (next < ntiles)
            load_tile_async(sm.in[buf ^ 1], x, rows, cols, static_cast<int64_t>(next / tiles_n) * kQT,
                            static_cast<int64_t>(next % tiles_n) * kQT);
        else
            cp_async_commit();
        cp_async_wait<1>();
        if (tid == 0) bulk_wait_group_read0();  // previous tile's stores have read the staging
        __syncthreads();                         // (S1) tile visible, staging free

        const uint16_t *in = sm.in[buf];

        // ---- 128x128 block scale (weights): amax over the whole tile
        uint32_t blk_g = 0;
        if constexpr (KIND == kQuantBlockWeight) {
            uint32_t m = 0;
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint4 v = *reinterpret_cast<const uint4 *>(in + (tid + kQThreads * i) * 8);
                m = __vmaxu2(m, max_abs4(v));
            }
            m = max(m & 0xFFFFu, m >> 16);
            m = __reduce_max_sync(0xFFFFFFFFu, m);
            if (lane == 0) sm.red[warp] = m;
            __syncthreads();
            m = sm.red[lane & 7];
            m = __reduce_max_sync(0xFFFFFFFFu, m);
            blk_g = e8m0_exponent<FMT>(m);
        }

        // ---- row pass: 1x128 groups along cols -> q.  A half-warp per row,
        // eight values per thread.
        {
            const int h = lane >> 4, j = lane & 15;
#pragma unroll 2
            for (int i = 0; i < 8; ++i) {
                const int r = 16 * warp + 2 * i + h;
                const uint4 v = *reinterpret_cast<const uint4 *>(in + r * kQT + 8 * j);
                float mul;
                bool nan_group;
                uint32_t g = 0;
                if constexpr (KIND == kQuantBlockAct) {
                    const uint32_t m2 = max_abs4(v);
                    const uint32_t m = max(m2 & 0xFFFFu, m2 >> 16);
                    const uint32_t m_lo = __reduce_max_sync(0xFFFFFFFFu, h == 0 ? m : 0u);
                    const uint32_t m_hi = __reduce_max_sync(0xFFFFFFFFu, h == 1 ? m : 0u);
                    g = e8m0_exponent<FMT>(h ? m_hi : m_lo);
                    nan_group = (g == 0xFFu);
                    mul = pow2_inv_scale(nan_group ? 0u : g);
                } else if constexpr (KIND == kQuantBlockWeight) {
                    nan_group = (blk_g == 0xFFu);
                    mul = pow2_inv_scale(nan_group ? 0u : blk_g);
                } else {
                    nan_group = t_nan;
                    mul = t_scale;
                }
                const uint64_t mul2 = f32x2(mul, mul);
                uint2 out;
                out.x = quant4<FMT>(bf16_lo(v.x), bf16_hi(v.x), bf16_lo(v.y), bf16_hi(v.y), mul2, nan_group);
                out.y = quant4<FMT>(bf16_lo(v.z), bf16_hi(v.z), bf16_lo(v.w), bf16_hi(v.w), mul2, nan_group);
                *reinterpret_cast<uint2 *>(sm.q_stage + r * kQT + 8 * j) = out;
                if (KIND == kQuantBlockAct && j == 0) sm.row_g[r] = static_cast<uint8_t>(g);
            }
        }

        // ---- column pass: 128x1 groups along rows -> q_t (transposed).
        // Thread t owns columns 2cp, 2cp+1 (cp = t % 64) over the 32 rows of
        // quarter rq = t / 64: one 4-byte load per row feeds both columns.
        if constexpr (HAS_T) {
            const int cp = tid & 63, rq = tid >> 6;
            uint32_t w[32];
#pragma unroll
            for (int k = 0; k < 32; ++k) w[k] = *reinterpret_cast<const uint32_t *>(in + (32 * rq + k) * kQT + 2 * cp);
            float mul_lo, mul_hi;
            bool nan_lo, nan_hi;
            if constexpr (KIND == kQuantBlockAct) {
                uint32_t m2 = 0;
#pragma unroll
                for (int k = 0; k < 32; ++k) m2 = __vmaxu2(m2, w[k] & 0x7FFF7FFFu);
                sm.col_amax2[rq][cp] = m2;
                __syncthreads();  // (S2)
                m2 = __vmaxu2(__vmaxu2(sm.col_amax2[0][cp], sm.col_amax2[1][cp]),
                              __vmaxu2(sm.col_amax2[2][cp], sm.col_amax2[3][cp]));
                const uint32_t g_lo = e8m0_exponent<FMT>(m2 & 0xFFFFu), g_hi = e8m0_exponent<FMT>(m2 >> 16);
                nan_lo = (g_lo == 0xFFu);
                nan_hi = (g_hi == 0xFFu);
                mul_lo = pow2_inv_scale(nan_lo ? 0u : g_lo);
                mul_hi = pow2_inv_scale(nan_hi ? 0u : g_hi);
                if (rq == 0) {
                    sm.col_g[2 * cp] = static_cast<uint8_t>(g_lo);
                    sm.col_g[2 * cp + 1] = static_cast<uint8_t>(g_hi);
                }
            } else if constexpr (KIND == kQuantBlockWeight) {
                nan_lo = nan_hi = (blk_g == 0xFFu);
                mul_lo = mul_hi = pow2_inv_scale(nan_lo ? 0u : blk_g);
            } else {
                nan_lo = nan_hi = t_nan;
                mul_lo = mul_hi = t_scale;
            }
            const uint64_t m2lo = f32x2(mul_lo, mul_lo), m2hi = f32x2(mul_hi, mul_hi);
            uint32_t c_lo[8], c_hi[8];  // 32 codes of each column, rows 32rq .. 32rq+31
#pragma unroll
            for (int q4 = 0; q4 < 8; ++q4) {
                const uint32_t a = w[4 * q4], b = w[4 * q4 + 1], c = w[4 * q4 + 2], d = w[4 * q4 + 3];
                c_lo[q4] = quant4<FMT>(bf16_lo(a), bf16_lo(b), bf16_lo(c), bf16_lo(d), m2lo, nan_lo);
                c_hi[q4] = quant4<FMT>(bf16_hi(a), bf16_hi(b), bf16_hi(c), bf16_hi(d), m2hi, nan_hi);
            }
            // Store the two transposed rows; lanes with cp bit 2 set store the
            // odd row first, so each 8-lane phase touches 8 distinct rows mod 8
            // (distinct swizzled chunks: no bank conflicts).
            const int sel = (cp >> 2) & 1;
#pragma unroll
            for (int pass = 0; pass < 2; ++pass) {
                const int which = sel ^ pass;  // 0: column 2cp, 1: column 2cp+1
                const int row = 2 * cp + which;
                uint8_t *dst = sm.qt_stage + row * kQT;
#pragma unroll
                for (int i = 0; i < 2; ++i) {
                    const uint4 o = which ? make_uint4(c_hi[4 * i], c_hi[4 * i + 1], c_hi[4 * i + 2], c_hi[4 * i + 3])
                                          : make_uint4(c_lo[4 * i], c_lo[4 * i + 1], c_lo[4 * i + 2], c_lo[4 * i + 3]);
                    *reinterpret_cast<uint4 *>(dst + 16 * ((2 * rq + i) ^ (row & 7))) = o;
                }
            }
        }

        fence_proxy_async_smem();
        __syncthreads();  // (S3) staging complete
        if (tid == 0) {
            tma_store_2d(&tm_q, sm.q_stage, static_cast<int32_t>(c0), static_cast<int32_t>(r0));
            if (HAS_T) tma_store_2d(&tm_qt, sm.qt_stage, static_cast<int32_t>(r0), static_cast<int32_t>(c0));
            bulk_commit_group();
        }
        if constexpr (KIND != kQuantTensor) {
            // Scale vectors in the tensor-core layout: thread i < 128 writes
            // row i of the rowwise operand (k-block c0/128), thread 128 + i
            // writes row i of the transposed operand (k-block r0/128).
            const bool col = tid >= kQT;
            if (!col || HAS_T) {
                const int i = tid & (kQT - 1);
                const int64_t op_rows0 = col ? c0 : r0;       // first operand row of this tile
                const int64_t kb = (col ? r0 : c0) / kQT;     // k-block of this tile
                const int64_t kblocks = (col ? rows : cols) / kQT;
                uint8_t g;
                if constexpr (KIND == kQuantBlockAct)
                    g = col ? sm.col_g[i] : sm.row_g[i];
                else
                    g = static_cast<uint8_t>(blk_g);
                store_scale_vec(col ? scale_t_u8 : scale_u8, op_rows0 + i, kb, kblocks, g);
            }
        }
    }
    cp_async_wait<0>();
    if (tid == 0) bulk_wait_group0();
}

// Per-tensor scale only (empty tensors: amax = 0 gives scale_inv = 1).
template <int FMT>
__global__ void tensor_scale_only_kernel(const uint32_t *amax_bits, float *scale_f, float *scale_t_f) {
    const uint32_t a = *amax_bits & 0xFFFFu;
    const float si = (a >= 0x7F80u) ? __uint_as_float(0x7FC00000u) : __fdiv_rn(1.0f, tensor_scale<FMT>(a));
    *scale_f = si;
    if (scale_t_f) *scale_t_f = si;
}

cudaError_t launch_tensor_scale_only(const QuantArgs &a, cudaStream_t s) {
    if (a.fmt == 0)
        tensor_scale_only_kernel<0><<<1, 1, 0, s>>>(a.amax, a.scale_f, a.scale_t_f);
    else
        tensor_scale_only_kernel<1><<<1, 1, 0, s>>>(a.amax, a.scale_f, a.scale_t_f);
    return cudaGetLastError();
}

template <int FMT, int KIND, bool HAS_T>
static cudaError_t launch_quant_t(const QuantArgs &a, const CUtensorMap &tm_q, const CUtensorMap &tm_qt,
                                  cudaStream_t s) {
    auto kern = quant_tile_kernel<FMT, KIND, HAS_T>;
    const size_t smem = sizeof(QuantSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int tiles_m = static_cast<int>((a.rows + kQT - 1) / kQT);
    const int tiles_n = static_cast<int>((a.cols + kQT - 1) / kQT);
    const int ntiles = tiles_m * tiles_n;
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    const int grid = ntiles < 2 * sms ? ntiles : 2 * sms;  // persistent: two CTAs per SM
    kern<<<grid, kQThreads, smem, s>>>(tm_q, tm_qt, a.x, a.rows, a.cols, a.scale_u8, a.scale_t_u8, a.scale_f,
                                       a.scale_t_f, a.amax, tiles_n, ntiles);
    return cudaGetLastError();
}

template <int FMT, int KIND>
static cudaError_t launch_quant_k(const QuantArgs &a, const CUtensorMap &tm_q, const CUtensorMap &tm_qt,
                                  cudaStream_t s) {
    return a.has_t ? launch_quant_t<FMT, KIND, true>(a, tm_q, tm_qt, s)
                   : launch_quant_t<FMT, KIND, false>(a, tm_q, tm_qt, s);
}

template <int FMT>
static cudaError_t launch_quant_f(const QuantArgs &a, const CUtensorMap &tm_q, const CUtensorMap &tm_qt,
                                  cudaStream_t s) {
    switch (a.kind) {
        case kQuantBlockAct: return launch_quant_k<FMT, kQuantBlockAct>(a, tm_q, tm_qt, s);
        case kQuantBlockWeight: return launch_quant_k<FMT, kQuantBlockWeight>(a, tm_q, tm_qt, s);
        default: return launch_quant_k<FMT, kQuantTensor>(a, tm_q, tm_qt, s);
    }
}

cudaError_t launch_quantize(const QuantArgs &a, const CUtensorMap &tm_q, const CUtensorMap &tm_qt,
                            cudaStream_t s) {
    return a.fmt == 0 ? launch_quant_f<0>(a, tm_q, tm_qt, s) : launch_quant_f<1>(a, tm_q, tm_qt, s);
}

}  // namespace puro
