// quantize.cu -- amax reduction and the fused BF16 -> FP8 cast(+transpose)
// kernels of the FP8 linear path (Puro-2B, section "FP8 Mixed-Precision
// Training": scales computed online per local group -- 1x128 groups along
// the GEMM reduction dimension for activations and activation gradients,
// 128x128 blocks for weights -- each a power of two).
//
// The kernels are HBM-bandwidth bound.  The cast kernels read each 128x128
// BF16 tile once (one TMA load per tile, double buffered), compute the
// scales from the same shared-memory copy, and write the rowwise codes and
// the transposed codes through shared memory with TMA stores (the
// transposed staging tile uses the 128-byte swizzle so the column pass
// stores without bank conflicts).  Activations and gradients (1x128 groups
// both ways, optionally behind a fused RMSNorm or SwiGLU producer) use a
// 512-thread kernel; weights (128x128 blocks) and per-tensor scaling use a
// 256-thread one.  The arithmetic per value is kept to a widening shift,
// half a packed fp32 multiply and half a paired cvt, since at HBM rates the
// kernels are otherwise instruction bound.
#include <cfloat>
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"
#include "quant_math.cuh"

namespace puro {

static int sm_count_here() {
    int dev = 0, sms = 148;
    cudaGetDevice(&dev);
    cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
    return sms;
}

// --------------------------------------------------------------- amax
// Integer max of (bits & 0x7FFF) over bf16 values: exact for finite values,
// +inf sorts above them and NaN above +inf.  A read-only stream: every
// thread keeps eight 16-byte loads in flight (the remainder, fewer than
// eight per thread, also in one batch), and the grid is the number of blocks
// that are resident at once (four per SM at 64 registers), so the
// grid-stride loop runs in one wave with about 20 MB in flight.
constexpr int kAmaxThreads = 256;
constexpr int kAmaxBlocksPerSm = 4;
constexpr int kAmaxUnroll = 8;

PURO_DEV uint32_t max_abs8(uint32_t m2, const uint4 &v) {
    return __vmaxu2(m2, __vmaxu2(__vmaxu2(v.x & 0x7FFF7FFFu, v.y & 0x7FFF7FFFu),
                                 __vmaxu2(v.z & 0x7FFF7FFFu, v.w & 0x7FFF7FFFu)));
}

__global__ void __launch_bounds__(kAmaxThreads, kAmaxBlocksPerSm)
    amax_kernel(const uint4 *__restrict__ x, int64_t nvec, const uint16_t *__restrict__ tail, int ntail,
                uint32_t *__restrict__ out) {
    pdl_wait();
    pdl_launch_dependents();
    uint32_t m2 = 0;  // two packed 16-bit running maxima
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x;
    for (; i + (kAmaxUnroll - 1) * stride < nvec; i += kAmaxUnroll * stride) {
        uint4 v[kAmaxUnroll];
#pragma unroll
        for (int k = 0; k < kAmaxUnroll; ++k) v[k] = __ldg(x + i + k * stride);
#pragma unroll
        for (int k = 0; k < kAmaxUnroll; ++k) m2 = max_abs8(m2, v[k]);
    }
    {  // fewer than kAmaxUnroll vectors remain per thread: load them together
        uint4 v[kAmaxUnroll - 1];
#pragma unroll
        for (int k = 0; k < kAmaxUnroll - 1; ++k) {
            const int64_t j = i + k * stride;
            v[k] = j < nvec ? __ldg(x + j) : make_uint4(0u, 0u, 0u, 0u);
        }
#pragma unroll
        for (int k = 0; k < kAmaxUnroll - 1; ++k) m2 = max_abs8(m2, v[k]);
    }
    if (blockIdx.x == 0 && threadIdx.x < ntail) m2 = __vmaxu2(m2, tail[threadIdx.x] & 0x7FFFu);
    uint32_t m = max(m2 & 0xFFFFu, m2 >> 16);
    m = __reduce_max_sync(0xFFFFFFFFu, m);
    __shared__ uint32_t warp_max[kAmaxThreads / 32];
    const int warp = threadIdx.x >> 5;
    if ((threadIdx.x & 31) == 0) warp_max[warp] = m;
    __syncthreads();
    if (warp == 0) {
        m = (threadIdx.x < kAmaxThreads / 32) ? warp_max[threadIdx.x] : 0u;
        m = __reduce_max_sync(0xFFFFFFFFu, m);
        if (threadIdx.x == 0 && m != 0) atomicMax(out, m);
    }
}

cudaError_t launch_amax(const uint16_t *x, int64_t n, uint32_t *amax, cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(amax, 0, sizeof(uint32_t), s);
    if (e != cudaSuccess || n == 0) return e;
    const int64_t nvec = n / 8;
    const int ntail = static_cast<int>(n - nvec * 8);
    const int sms = sm_count_here();
    const int64_t want = (nvec + kAmaxThreads - 1) / kAmaxThreads;
    const int64_t cap = static_cast<int64_t>(sms) * kAmaxBlocksPerSm;
    const int grid = static_cast<int>(want < cap ? (want > 0 ? want : 1) : cap);
    return launch_pdl(amax_kernel, dim3(grid), dim3(kAmaxThreads), 0, s, reinterpret_cast<const uint4 *>(x), nvec,
                      x + nvec * 8, ntail, amax);
}

// ------------------------------------------------------ RMSNorm producer
// RMSNorm of the activation the quantiser receives (the model's
// normalisation ahead of the attention and MLP projections): per row
// rstd = 1 / sqrt(mean(h^2) + eps), then y = bf16((h * rstd) * gamma).

// rstd of each row of h [rows, cols] (cols a multiple of 8), one warp per
// row: fp32 sums of squares in a fixed order (lane-strided 8-value chunks,
// then a butterfly), then an IEEE division and square root.  A lane loads
// up to eight of its chunks before it adds any (in chunk order), so a
// row's loads are in flight together.
__global__ void __launch_bounds__(256) rmsnorm_rstd_kernel(const uint16_t *__restrict__ h, int64_t rows, int64_t cols,
                                                           float eps, float *__restrict__ rstd) {
    pdl_wait();
    pdl_launch_dependents();
    constexpr int kBatch = 8;
    const int lane = threadIdx.x & 31;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * (blockDim.x >> 5);
    const int64_t n8 = cols / 8;
    for (int64_t r = static_cast<int64_t>(blockIdx.x) * (blockDim.x >> 5) + (threadIdx.x >> 5); r < rows; r += nwarps) {
        const uint4 *row = reinterpret_cast<const uint4 *>(h + r * cols);
        float a = 0.0f, b = 0.0f;
        for (int64_t c0 = lane; c0 < n8; c0 += 32 * kBatch) {
            uint4 w[kBatch];
#pragma unroll
            for (int k = 0; k < kBatch; ++k)
                w[k] = c0 + 32 * k < n8 ? __ldg(row + c0 + 32 * k) : make_uint4(0u, 0u, 0u, 0u);
#pragma unroll
            for (int k = 0; k < kBatch; ++k) {
                if (c0 + 32 * k >= n8) break;
                const uint32_t ws[4] = {w[k].x, w[k].y, w[k].z, w[k].w};
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const float lo = __uint_as_float(ws[j] << 16), hi = __uint_as_float(ws[j] & 0xFFFF0000u);
                    a = __fmaf_rn(lo, lo, a);
                    b = __fmaf_rn(hi, hi, b);
                }
            }
        }
        float ss = a + b;
#pragma unroll
        for (int off = 16; off > 0; off >>= 1) ss += __shfl_xor_sync(0xFFFFFFFFu, ss, off);
        if (lane == 0) rstd[r] = __fdiv_rn(1.0f, __fsqrt_rn(__fdiv_rn(ss, static_cast<float>(cols)) + eps));
    }
}

// y = bf16((h * rstd) * gamma) for an 8-value chunk (gm unused without gamma).
PURO_DEV uint4 rmsnorm_chunk(uint4 w, float rs, const float (&gm)[8], bool has_gamma) {
    uint32_t ws[4] = {w.x, w.y, w.z, w.w};
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        float lo = __fmul_rn(__uint_as_float(ws[j] << 16), rs), hi = __fmul_rn(__uint_as_float(ws[j] & 0xFFFF0000u), rs);
        if (has_gamma) {
            lo = __fmul_rn(lo, gm[2 * j]);
            hi = __fmul_rn(hi, gm[2 * j + 1]);
        }
        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        ws[j] = *reinterpret_cast<uint32_t *>(&v);
    }
    return make_uint4(ws[0], ws[1], ws[2], ws[3]);
}

PURO_DEV void load_gamma8(const uint16_t *gamma, int64_t c, int64_t cols, float (&gm)[8]) {
    if (c + 8 <= cols) {
        const uint4 g = __ldg(reinterpret_cast<const uint4 *>(gamma + c));
        const uint32_t gw[4] = {g.x, g.y, g.z, g.w};
#pragma unroll
        for (int j = 0; j < 4; ++j) {
            gm[2 * j] = __uint_as_float(gw[j] << 16);
            gm[2 * j + 1] = __uint_as_float(gw[j] & 0xFFFF0000u);
        }
    } else {
#pragma unroll
        for (int j = 0; j < 8; ++j) gm[j] = 0.0f;  // columns past the end hold zeros
    }
}

// Unfused comparison: y = bf16((h * rstd) * gamma), one 8-value chunk per
// thread and step.
__global__ void __launch_bounds__(256) rmsnorm_apply_kernel(const uint16_t *__restrict__ h, int64_t rows, int64_t cols,
                                                            const float *__restrict__ rstd,
                                                            const uint16_t *__restrict__ gamma, uint16_t *__restrict__ y) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t per_row = cols / 8;
    const int64_t chunks = rows * per_row;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < chunks; i += stride) {
        const int64_t r = i / per_row, c = (i - r * per_row) * 8;
        float gm[8];
        if (gamma) load_gamma8(gamma, c, cols, gm);
        reinterpret_cast<uint4 *>(y)[i] =
            rmsnorm_chunk(__ldg(reinterpret_cast<const uint4 *>(h) + i), __ldg(rstd + r), gm, gamma != nullptr);
    }
}

cudaError_t launch_rmsnorm_rstd(const uint16_t *h, int64_t rows, int64_t cols, float eps, float *rstd, cudaStream_t s) {
    const int sms = sm_count_here();
    const int64_t want = (rows + 7) / 8;
    const int grid = static_cast<int>(want < 8 * sms ? want : 8 * sms);
    return launch_pdl(rmsnorm_rstd_kernel, dim3(grid > 0 ? grid : 1), dim3(256), 0, s, h, rows, cols, eps, rstd);
}

cudaError_t launch_rmsnorm_apply(const uint16_t *h, int64_t rows, int64_t cols, const float *rstd,
                                 const uint16_t *gamma, uint16_t *y, cudaStream_t s) {
    const int sms = sm_count_here();
    const int64_t want = (rows * (cols / 8) + 255) / 256;
    const int grid = static_cast<int>(want < 8 * sms ? want : 8 * sms);
    return launch_pdl(rmsnorm_apply_kernel, dim3(grid > 0 ? grid : 1), dim3(256), 0, s, h, rows, cols, rstd, gamma, y);
}

// ------------------------------------------------------ SwiGLU producer
// 2^x and 1/x by the special-function unit (PTX ex2.approx / rcp.approx:
// relative error around 2^-22; subnormal results flush to zero).
PURO_DEV float ex2_approx(float x) {
    float y;
    asm("ex2.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}
PURO_DEV float rcp_approx(float x) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return y;
}

// silu(g) = g * sigmoid(g) in fp32, with sigmoid from t = e^-|g| (in (0, 1],
// so nothing overflows): sigmoid(g) = r = 1 / (1 + t) for g >= 0, t * r
// otherwise.  t = 2^(64 - |g| log2 e) * 2^-64: the special-function
// exponent stays in the normal range for |g| < 131.7, and the exact IEEE
// scaling by 2^-64 (and t * r) keep subnormal values of e^-|g|.  The
// special-function forms cost one instruction each; their few-ulp fp32
// error is far below the bf16 rounding that follows (with correctly rounded
// exp and division the fused kernel is bound by those instructions, not by
// memory).  Below g ~ -131.7 t is zero, where the exact product
// silu(g) * u is below 1e-55 |u|.  NaN stays NaN; -inf gives NaN (-inf * 0).
PURO_DEV float silu_f32(float g) {
    const float a = fabsf(g);
    const float t = __fmul_rn(ex2_approx(fmaf(a, -1.44269504f, 64.0f)), 0x1p-64f);
    const float r = rcp_approx(__fadd_rn(1.0f, t));
    return __fmul_rn(g, g >= 0.0f ? r : __fmul_rn(t, r));
}

// y = bf16(silu(g) * u) for an 8-value chunk.
PURO_DEV uint4 swiglu_chunk(uint4 g, uint4 u) {
    const uint32_t gw[4] = {g.x, g.y, g.z, g.w}, uw[4] = {u.x, u.y, u.z, u.w};
    uint32_t out[4];
#pragma unroll
    for (int j = 0; j < 4; ++j) {
        const float lo = __fmul_rn(silu_f32(__uint_as_float(gw[j] << 16)), __uint_as_float(uw[j] << 16));
        const float hi = __fmul_rn(silu_f32(__uint_as_float(gw[j] & 0xFFFF0000u)), __uint_as_float(uw[j] & 0xFFFF0000u));
        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        out[j] = *reinterpret_cast<uint32_t *>(&v);
    }
    return make_uint4(out[0], out[1], out[2], out[3]);
}

// Unfused comparison: y = bf16(silu(gate) * up), one 8-value chunk per thread
// and step; gate and up rows ld elements apart, y contiguous.
__global__ void __launch_bounds__(256) swiglu_apply_kernel(const uint16_t *__restrict__ gate,
                                                           const uint16_t *__restrict__ up, int64_t rows,
                                                           int64_t cols, int64_t ld, uint16_t *__restrict__ y) {
    pdl_wait();
    pdl_launch_dependents();
    const int64_t per_row = cols / 8;
    const int64_t chunks = rows * per_row;
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < chunks; i += stride) {
        const int64_t r = i / per_row, c = (i - r * per_row) * 8;
        const uint4 g = __ldg(reinterpret_cast<const uint4 *>(gate + r * ld + c));
        const uint4 u = __ldg(reinterpret_cast<const uint4 *>(up + r * ld + c));
        reinterpret_cast<uint4 *>(y)[i] = swiglu_chunk(g, u);
    }
}

cudaError_t launch_swiglu_apply(const uint16_t *gate, const uint16_t *up, int64_t rows, int64_t cols, int64_t ld,
                                uint16_t *y, cudaStream_t s) {
    const int sms = sm_count_here();
    const int64_t want = (rows * (cols / 8) + 255) / 256;
    const int grid = static_cast<int>(want < 8 * sms ? want : 8 * sms);
    return launch_pdl(swiglu_apply_kernel, dim3(grid > 0 ? grid : 1), dim3(256), 0, s, gate, up, rows, cols, ld, y);
}

// ------------------------------------------------------ cast kernel
constexpr int kQT = 128;          // tile edge
// Threads of the single-scale cast kernels (weights, per-tensor): thread t
// owns the 8x4 block of rows 8*(t/32) .. +7 and columns 4*(t%32) .. +3 of
// the 128x128 tile, the layout of the activation kernel below.
constexpr int kQThreads = 512;

// Shared memory of one CTA.  Both staging tiles are TMA store sources and
// so 1024-byte aligned; the transposed tile uses the 128-byte swizzle
// (16-byte chunk k of row r at k ^ (r % 8)).
struct QuantSmem {
    alignas(1024) uint8_t q_stage[kQT * kQT];    // rowwise codes, plain rows
    alignas(1024) uint8_t qt_stage[kQT * kQT];   // transposed codes, 128B-swizzled rows
    alignas(128) uint16_t in[2][kQT * kQT];      // bf16 tile, double buffered
    uint32_t red[kQThreads / 32];                // weight kind: per-warp block maxima
    uint64_t full[2];                            // TMA tile loads into in[0], in[1]
};

constexpr uint64_t kQuantDrainNs = 2000000000ull;  // after an abort: bound on the loads still in flight
constexpr uint64_t kPollBelowNs = 100000ull;       // shorter bounds are polled without suspending
constexpr int32_t kQuantStatusTimeout = 4;         // PURO_ERR_TIMEOUT

// Wait for a tile load, bounded by the library's wait bound
// (puro_set_wait_timeout_ns).  A bound under 100 us is polled with the
// non-blocking test, so that a short bound is kept even where one
// suspending try_wait would sleep until the copy lands; a zero bound is a
// single test (it does not depend on the timer's resolution).
PURO_DEV bool tile_landed(uint64_t *bar, uint32_t parity, uint64_t wait_ns) {
    if (wait_ns >= kPollBelowNs) return mbar_wait_bounded(bar, parity, wait_ns);
    if (mbar_test_wait(bar, parity)) return true;
    const uint64_t t0 = global_timer_ns();
    while (global_timer_ns() - t0 < wait_ns)
        if (mbar_test_wait(bar, parity)) return true;
    return false;
}

// A CTA gave up on the load of its tile `it` (every thread leaves the tile
// loop together, after a block-wide vote): record the time-out, then let
// the loads it still has in flight (this tile's and, when issued, the next
// one's) land before it exits, since they write into its shared memory.
// The drain is bounded too.  One thread.
PURO_DEV void quant_abort(uint64_t *full, int it, bool next_issued, int32_t *status) {
    if (status) atomicExch(status, kQuantStatusTimeout);
    const int buf = it & 1;
    mbar_wait_bounded(&full[buf], static_cast<uint32_t>(it >> 1) & 1u, kQuantDrainNs);
    if (next_issued) mbar_wait_bounded(&full[buf ^ 1], static_cast<uint32_t>((it + 1) >> 1) & 1u, kQuantDrainNs);
}


// The transposed codes of one thread's 8x4 block (rows 8br .. 8br+7,
// columns 4bc .. 4bc+3 of a 128x128 tile) into the transposed staging tile.
// rw[i] holds row 8br+i's four codes, byte j for column 4bc+j.  Column j's
// eight codes (rows 8br .. 8br+7) belong in transposed row 4bc + j, bytes
// 8br .. 8br+7, whose 16-byte chunk is (br / 2) ^ ((4bc + j) % 8) under the
// 128-byte swizzle.  All 32 lanes of a warp share br, so storing the same j
// together would put them in two chunks; lane bc stores column
// (s + bc / 2) % 4 at step s instead, which spreads them over all eight.
// Two 4x4 byte transposes per four rows gather the columns, and the first
// stage's selectors (per-lane constants) already put column (s + rot) % 4
// in output word s, so the rotation costs no instruction.
PURO_DEV void stage_transposed_8x4(uint8_t *qt_stage, const uint32_t (&rw)[8], int br, int bc) {
    const uint32_t rot = static_cast<uint32_t>(bc >> 1) & 3u;
    const uint32_t a = rot, b = (rot + 1u) & 3u, c = (rot + 2u) & 3u, d = (rot + 3u) & 3u;
    const uint32_t sel_ab = a | ((4u + a) << 4) | (b << 8) | ((4u + b) << 12);
    const uint32_t sel_cd = c | ((4u + c) << 4) | (d << 8) | ((4u + d) << 12);
    uint32_t wt[2][4];  // [rows 0-3 / 4-7][step s]: column (s + rot) mod 4
#pragma unroll
    for (int h = 0; h < 2; ++h) {
        const uint32_t x0 = __byte_perm(rw[4 * h], rw[4 * h + 1], sel_ab);
        const uint32_t x1 = __byte_perm(rw[4 * h], rw[4 * h + 1], sel_cd);
        const uint32_t x2 = __byte_perm(rw[4 * h + 2], rw[4 * h + 3], sel_ab);
        const uint32_t x3 = __byte_perm(rw[4 * h + 2], rw[4 * h + 3], sel_cd);
        wt[h][0] = __byte_perm(x0, x2, 0x5410);
        wt[h][1] = __byte_perm(x0, x2, 0x7632);
        wt[h][2] = __byte_perm(x1, x3, 0x5410);
        wt[h][3] = __byte_perm(x1, x3, 0x7632);
    }
#pragma unroll
    for (int st = 0; st < 4; ++st) {
        const int r = 4 * bc + ((st + static_cast<int>(rot)) & 3);  // transposed row (tile column)
        *reinterpret_cast<uint2 *>(qt_stage + r * kQT + 16 * ((br >> 1) ^ (r & 7)) + 8 * (br & 1)) =
            make_uint2(wt[0][st], wt[1][st]);
    }
}

// Rowwise and transposed codes of one thread's 8x4 block v (rows 8br ..
// 8br+7, columns 4bc .. 4bc+3) into the staging tiles, for a tile with one
// multiplier (m2: it twice; nan_all: a non-finite tile).  With a single
// scale the transposed codes are the rowwise codes transposed, so each
// value is converted once.
template <int FMT, bool HAS_T>
PURO_DEV void tile_codes_to_stage(QuantSmem &sm, const uint2 (&v)[8], int br, int bc, uint64_t m2, bool nan_all) {
    uint32_t rw[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) {
        rw[i] = quant4<FMT>(bf16_lo(v[i].x), bf16_hi(v[i].x), bf16_lo(v[i].y), bf16_hi(v[i].y), m2, nan_all);
        *reinterpret_cast<uint32_t *>(sm.q_stage + (8 * br + i) * kQT + 4 * bc) = rw[i];  // a warp: one 128-byte row
    }
    if constexpr (HAS_T) stage_transposed_8x4(sm.qt_stage, rw, br, bc);
}

// Row and column block of a persistent CTA's tiles t, t + step, t + 2 step,
// ... in a grid of tiles_n column blocks, advanced without a division.
struct TileWalk {
    int r, c, dr, dc, n;
    PURO_DEV TileWalk(int t, int step, int tiles_n)
        : r(t / tiles_n), c(t % tiles_n), dr(step / tiles_n), dc(step % tiles_n), n(tiles_n) {}
    PURO_DEV void advance() {
        r += dr;
        c += dc;
        if (c >= n) {
            c -= n;
            ++r;
        }
    }
};

// Maximum |bf16| of a thread's 8x4 block in both halves of a word.
PURO_DEV uint32_t block_max_8x4(const uint2 (&v)[8]) {
    uint32_t m = 0;
#pragma unroll
    for (int i = 0; i < 8; ++i) m = __vmaxu2(m, __vmaxu2(v[i].x & 0x7FFF7FFFu, v[i].y & 0x7FFF7FFFu));
    return __vmaxu2(m, __byte_perm(m, 0u, 0x1032));
}

// Weight (128x128 blocks) and per-tensor cast kernel: one scale per tile
// (the block's or the tensor's), so the transposed codes (q_t) are the
// rowwise codes (q) transposed.  Thread t owns the 8x4 block of rows
// 8*(t/32) .. +7 and columns 4*(t%32) .. +3.  The weight kind reduces the
// block maximum through the warps (one barrier); the per-tensor kind reads
// its scale from the device amax.
template <int FMT, int KIND, bool HAS_T>
__global__ void __launch_bounds__(kQThreads, 2)
    quant_tile_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_q,
                      const __grid_constant__ CUtensorMap tm_qt, int64_t rows, int64_t cols,
                      uint8_t *__restrict__ scale_u8, uint8_t *__restrict__ scale_t_u8, float *scale_f,
                      float *scale_t_f, const uint32_t *__restrict__ amax_bits, int tiles_n, int ntiles,
                      int32_t *status, uint64_t wait_ns) {
    static_assert(KIND == kQuantBlockWeight || KIND == kQuantTensor, "activations use quant_act_kernel");
    extern __shared__ uint8_t smem_raw[];
    QuantSmem &sm = *reinterpret_cast<QuantSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                   ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int br = warp;  // block row: tile rows 8br .. 8br+7
    const int bc = lane;  // block column: tile columns 4bc .. 4bc+3
    pdl_wait();
    pdl_launch_dependents();

    // Per-tensor mode: the one scale, from the device amax.
    float t_mul = 1.0f;
    if constexpr (KIND == kQuantTensor) {
        const uint32_t a = *amax_bits & 0xFFFFu;
        const bool t_nan = a >= 0x7F80u;
        const float t_scale = tensor_scale<FMT>(a);
        t_mul = t_nan ? __uint_as_float(0x7FC00000u) : t_scale;
        if (blockIdx.x == 0 && tid == 0) {
            const float si = t_nan ? __uint_as_float(0x7FC00000u) : __fdiv_rn(1.0f, t_scale);
            *scale_f = si;
            if (scale_t_f) *scale_t_f = si;
        }
    }
    if (tid == 0) {
        mbar_init(&sm.full[0], 1);
        mbar_init(&sm.full[1], 1);
        fence_mbarrier_init();
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_q);
        if (HAS_T) tma_prefetch_desc(&tm_qt);
    }
    __syncthreads();

    // One TMA load per 128x128 bf16 tile (out-of-range parts read as zero),
    // double buffered: tile it+1 streams in while tile it is processed.
    auto issue_load = [&](const TileWalk &t, int b) {
        mbar_arrive_expect_tx(&sm.full[b], kQT * kQT * 2);
        tma_load_2d(sm.in[b], &tm_x, &sm.full[b], t.c * kQT, t.r * kQT);
    };
    int tile = blockIdx.x;
    TileWalk cur(tile, gridDim.x, tiles_n), nxt = cur;
    nxt.advance();
    if (tid == 0 && tile < ntiles) issue_load(cur, 0);
    for (int it = 0; tile < ntiles; ++it, tile += gridDim.x, cur = nxt, nxt.advance()) {
        const int buf = it & 1;
        const int64_t r0 = static_cast<int64_t>(cur.r) * kQT;
        const int64_t c0 = static_cast<int64_t>(cur.c) * kQT;
        if (tid == 0) {
            const int next = tile + gridDim.x;
            if (next < ntiles) issue_load(nxt, buf ^ 1);  // its buffer was last read before (S3) of it-1
            // The previous tile's TMA stores must have read the staging tiles
            // before they are rewritten: per-tensor mode writes them right
            // after (S1); the weight kind waits just before (S2).
            if constexpr (KIND == kQuantTensor) bulk_wait_group_read0();
        }
        // Every thread waits on the tile's barrier itself, which makes the
        // TMA-written tile visible to it.  A wait that runs out is voted on
        // at the next barrier, where every thread leaves together.
        const bool landed = tile_landed(&sm.full[buf], static_cast<uint32_t>(it >> 1) & 1u, wait_ns);
        if constexpr (KIND == kQuantTensor) {
            if (__syncthreads_or(!landed)) {  // (S1) staging free
                if (tid == 0) quant_abort(sm.full, it, tile + static_cast<int>(gridDim.x) < ntiles, status);
                break;
            }
        }

        // ---- the thread's 8x4 block: v[i] = row 8br+i, columns 4bc .. 4bc+3
        const uint16_t *in = sm.in[buf];
        uint2 v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = *reinterpret_cast<const uint2 *>(in + (8 * br + i) * kQT + 4 * bc);

        // ---- the tile's scale
        float mul = t_mul;
        uint32_t blk_g = 0;
        if constexpr (KIND == kQuantBlockWeight) {
            const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, block_max_8x4(v));
            if (lane == 0) sm.red[warp] = m;
            if (tid == 0) bulk_wait_group_read0();  // staging free (see above)
            if (__syncthreads_or(!landed)) {         // (S2) block maxima written, staging free
                if (tid == 0) quant_abort(sm.full, it, tile + static_cast<int>(gridDim.x) < ntiles, status);
                break;
            }
            blk_g = e8m0_exponent<FMT>(__reduce_max_sync(0xFFFFFFFFu, sm.red[lane & 15]) & 0xFFFFu);
            mul = mul_of(blk_g);
        }
        const uint64_t m2 = f32x2(mul, mul);
        const bool nan_all = isnan(mul);

        tile_codes_to_stage<FMT, HAS_T>(sm, v, br, bc, m2, nan_all);

        fence_proxy_async_smem();
        __syncthreads();  // (S3) staging complete
        if (tid == 0) {
            tma_store_2d(&tm_q, sm.q_stage, static_cast<int32_t>(c0), static_cast<int32_t>(r0));
            if (HAS_T) tma_store_2d(&tm_qt, sm.qt_stage, static_cast<int32_t>(r0), static_cast<int32_t>(c0));
            bulk_commit_group();
        }
        if constexpr (KIND == kQuantBlockWeight) {
            // Scale vectors in the tensor-core layout: thread i < 128 writes
            // row i of the rowwise operand (k-block c0/128), thread 128 + i
            // writes row i of the transposed operand (k-block r0/128); the
            // block's exponent repeats over its 128 rows.
            const bool col = tid >= kQT;
            if (tid < 2 * kQT && (!col || HAS_T)) {
                const int i = tid & (kQT - 1);
                const int64_t op_rows0 = col ? c0 : r0;
                const int64_t kb = (col ? r0 : c0) / kQT;
                const int64_t kblocks = (col ? rows : cols) / kQT;
                store_scale_vec(col ? scale_t_u8 : scale_u8, op_rows0 + i, kb, kblocks, static_cast<uint8_t>(blk_g));
            }
        }
    }
    if (tid == 0) bulk_wait_group0();
}

// ------------------------------------------- activation cast kernel (512)
// The 1x128 activation / gradient quantiser (optionally fed by a producer)
// with 512 threads per 128x128 tile: thread t owns the 8x4 block of rows
// 8*br .. 8*br+7 and columns 4*bc .. 4*bc+3, br = warp (0..15), bc = lane.
// A warp thus holds eight whole rows, so a row's group maximum is one
// warp-wide redux per row and needs no shared memory; the column maxima go
// through shared memory as before.  Compared with 256 threads on 8x8
// blocks, twice the warps per SM hide the latency of each phase (the
// kernel is latency bound at two 256-thread CTAs per SM), at about half the
// registers per thread.  Rows and columns are whole tiles (the blockwise
// entry points require multiples of 128).
constexpr int kQAThreads = 512;

struct QuantActSmem {
    alignas(1024) uint8_t q_stage[kQT * kQT];    // rowwise codes, plain rows
    alignas(1024) uint8_t qt_stage[kQT * kQT];   // transposed codes, 128B-swizzled rows
    alignas(128) uint16_t in[2][kQT * kQT];      // bf16 tile, double buffered
    alignas(16) uint32_t col_part[16][kQT / 2];  // [row block][column pair]: 16-bit column maxima, two per word
    alignas(16) float col_mul[kQT];
    alignas(16) uint8_t row_g[kQT];
    alignas(16) uint8_t col_g[kQT];
    uint64_t full[2];
};

// y = bf16((h * rstd) * gamma) for a 4-value chunk.
PURO_DEV uint2 rmsnorm_chunk4(uint2 w, float rs, const float (&gm)[4], bool has_gamma) {
    uint32_t ws[2] = {w.x, w.y};
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        float lo = __fmul_rn(__uint_as_float(ws[j] << 16), rs), hi = __fmul_rn(__uint_as_float(ws[j] & 0xFFFF0000u), rs);
        if (has_gamma) {
            lo = __fmul_rn(lo, gm[2 * j]);
            hi = __fmul_rn(hi, gm[2 * j + 1]);
        }
        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        ws[j] = *reinterpret_cast<uint32_t *>(&v);
    }
    return make_uint2(ws[0], ws[1]);
}

// y = bf16(silu(g) * u) for a 4-value chunk.
PURO_DEV uint2 swiglu_chunk4(uint2 g, uint2 u) {
    const uint32_t gw[2] = {g.x, g.y}, uw[2] = {u.x, u.y};
    uint32_t out[2];
#pragma unroll
    for (int j = 0; j < 2; ++j) {
        const float lo = __fmul_rn(silu_f32(__uint_as_float(gw[j] << 16)), __uint_as_float(uw[j] << 16));
        const float hi = __fmul_rn(silu_f32(__uint_as_float(gw[j] & 0xFFFF0000u)), __uint_as_float(uw[j] & 0xFFFF0000u));
        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
        out[j] = *reinterpret_cast<uint32_t *>(&v);
    }
    return make_uint2(out[0], out[1]);
}

template <int FMT, bool HAS_T, int PROD>
__global__ void __launch_bounds__(kQAThreads, 2)
    quant_act_kernel(const __grid_constant__ CUtensorMap tm_x, const __grid_constant__ CUtensorMap tm_q,
                     const __grid_constant__ CUtensorMap tm_qt, const __grid_constant__ CUtensorMap tm_y,
                     int64_t rows, int64_t cols, uint8_t *__restrict__ scale_u8, uint8_t *__restrict__ scale_t_u8,
                     ProdArgs prod, int tiles_n, int ntiles, int32_t *status, uint64_t wait_ns) {
    extern __shared__ uint8_t smem_raw[];
    QuantActSmem &sm = *reinterpret_cast<QuantActSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                         ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, lane = tid & 31;
    const int br = tid >> 5;  // block row: tile rows 8br .. 8br+7 (the warp)
    const int bc = lane;      // block column: tile columns 4bc .. 4bc+3
    if (tid == 0) {
        mbar_init(&sm.full[0], 1);
        mbar_init(&sm.full[1], 1);
        fence_mbarrier_init();
        tma_prefetch_desc(&tm_x);
        tma_prefetch_desc(&tm_q);
        if (HAS_T) tma_prefetch_desc(&tm_qt);
    }
    __syncthreads();
    pdl_wait();
    pdl_launch_dependents();

    auto issue_load = [&](const TileWalk &t, int b) {
        mbar_arrive_expect_tx(&sm.full[b], kQT * kQT * 2);
        tma_load_2d(sm.in[b], &tm_x, &sm.full[b], t.c * kQT, t.r * kQT);
    };
    int tile = blockIdx.x;
    TileWalk cur(tile, gridDim.x, tiles_n), nxt = cur;  // this tile and the CTA's next one
    nxt.advance();
    if (tid == 0 && tile < ntiles) issue_load(cur, 0);
    uint2 un[8];  // kProdSwiGlu: this thread's block of u for the current tile
    auto load_up = [&](const TileWalk &t) {
        const int64_t row0 = static_cast<int64_t>(t.r) * kQT + 8 * br;
        const int64_t col0 = static_cast<int64_t>(t.c) * kQT + 4 * bc;
        const uint16_t *p = prod.up + row0 * prod.ld + col0;
#pragma unroll
        for (int i = 0; i < 8; ++i) un[i] = __ldg(reinterpret_cast<const uint2 *>(p + i * prod.ld));
    };
    if constexpr (PROD == kProdSwiGlu) {
        if (tile < ntiles) load_up(cur);
    }
    for (int it = 0; tile < ntiles; ++it, tile += gridDim.x, cur = nxt, nxt.advance()) {
        const int buf = it & 1;
        const int64_t r0 = static_cast<int64_t>(cur.r) * kQT;
        const int64_t c0 = static_cast<int64_t>(cur.c) * kQT;
        if (tid == 0) {
            const int next = tile + gridDim.x;
            // with a y output, the buffer's last reader was the y store of
            // tile it-1: all but the newest bulk group (its code stores) done
            if (PROD != kProdNone && prod.write_y) bulk_wait_group_read<1>();
            if (next < ntiles) issue_load(nxt, buf ^ 1);  // its buffer was last read before (S4) of it-1
        }
        // Every thread waits on the tile's barrier itself (which makes the
        // TMA-written tile visible to it); the shared buffers written before
        // (S2) were last read before (S4) of the previous tile.  A wait that
        // runs out is voted on at (S2): nothing global is written before it.
        const bool landed = tile_landed(&sm.full[buf], static_cast<uint32_t>(it >> 1) & 1u, wait_ns);

        uint16_t *in = sm.in[buf];
        uint2 v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = *reinterpret_cast<const uint2 *>(in + (8 * br + i) * kQT + 4 * bc);
        if constexpr (PROD == kProdRmsNorm) {
            float gm[4] = {0.0f, 0.0f, 0.0f, 0.0f};
            const bool has_gamma = prod.gamma != nullptr;
            if (has_gamma) {
                const uint2 g = __ldg(reinterpret_cast<const uint2 *>(prod.gamma + c0 + 4 * bc));
                gm[0] = __uint_as_float(g.x << 16);
                gm[1] = __uint_as_float(g.x & 0xFFFF0000u);
                gm[2] = __uint_as_float(g.y << 16);
                gm[3] = __uint_as_float(g.y & 0xFFFF0000u);
            }
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                v[i] = rmsnorm_chunk4(v[i], __ldg(prod.rstd + r0 + 8 * br + i), gm, has_gamma);
                *reinterpret_cast<uint2 *>(in + (8 * br + i) * kQT + 4 * bc) = v[i];
            }
            if (prod.write_y) fence_proxy_async_smem();
        } else if constexpr (PROD == kProdSwiGlu) {
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                v[i] = swiglu_chunk4(v[i], un[i]);
                *reinterpret_cast<uint2 *>(in + (8 * br + i) * kQT + 4 * bc) = v[i];
            }
            if (prod.write_y) fence_proxy_async_smem();
            if (tile + static_cast<int>(gridDim.x) < ntiles) load_up(nxt);
        }

        // ---- A: row groups (a warp holds its eight rows whole) and column partials
        float rmul[8];
        {
            // each row's maximum in both halves of a word (the halves swapped
            // and maxed), so one redux gives it without splitting the halves
            uint32_t rmax[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint32_t m = __vmaxu2(v[i].x & 0x7FFF7FFFu, v[i].y & 0x7FFF7FFFu);
                rmax[i] = __reduce_max_sync(0xFFFFFFFFu, __vmaxu2(m, __byte_perm(m, 0u, 0x1032)));
            }
            // lane l takes row (l mod 8)'s maximum by a three-level select
            const bool b0 = lane & 1, b1 = lane & 2, b2 = lane & 4;
            const uint32_t s01 = b0 ? rmax[1] : rmax[0], s23 = b0 ? rmax[3] : rmax[2];
            const uint32_t s45 = b0 ? rmax[5] : rmax[4], s67 = b0 ? rmax[7] : rmax[6];
            const uint32_t mine = (b2 ? (b1 ? s67 : s45) : (b1 ? s23 : s01)) & 0xFFFFu;
            // lane i < 8 derives row 8br+i's scale; every lane then takes the
            // eight multipliers from those lanes
            const uint32_t g = e8m0_exponent<FMT>(mine);
            const float mul = mul_of(g);
            if (lane < 8) sm.row_g[8 * br + lane] = static_cast<uint8_t>(g);
#pragma unroll
            for (int i = 0; i < 8; ++i) rmul[i] = __shfl_sync(0xFFFFFFFFu, mul, i);
        }
        if constexpr (HAS_T) {
            uint2 cm = make_uint2(0u, 0u);  // columns (4bc, 4bc+1), (4bc+2, 4bc+3): max over the 8 rows
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                cm.x = __vmaxu2(cm.x, v[i].x & 0x7FFF7FFFu);
                cm.y = __vmaxu2(cm.y, v[i].y & 0x7FFF7FFFu);
            }
            *reinterpret_cast<uint2 *>(&sm.col_part[br][2 * bc]) = cm;
        }
        if (__syncthreads_or(!landed)) {  // (S2) partials and row scales written
            if (tid == 0) quant_abort(sm.full, it, tile + static_cast<int>(gridDim.x) < ntiles, status);
            break;
        }
        if constexpr (PROD != kProdNone) {
            if (prod.write_y && tid == 0) {  // every block's y is in shared memory
                tma_store_2d(&tm_y, sm.in[buf], static_cast<int32_t>(c0), static_cast<int32_t>(r0));
                bulk_commit_group();
            }
        }

        // ---- B: column scales, two threads per column (eight row blocks each)
        if constexpr (HAS_T) {
            if (tid < 2 * kQT) {
                const int c = tid >> 1, h = tid & 1;
                uint32_t m = 0;
#pragma unroll
                for (int b = 0; b < 8; ++b) m = __vmaxu2(m, sm.col_part[8 * h + b][c >> 1]);
                m = __vmaxu2(m, __shfl_xor_sync(0xFFFFFFFFu, m, 1));
                if (h == 0) {
                    const uint32_t g = e8m0_exponent<FMT>((c & 1) ? (m >> 16) : (m & 0xFFFFu));
                    sm.col_mul[c] = mul_of(g);
                    sm.col_g[c] = static_cast<uint8_t>(g);
                }
            }
        }
        if (tid == 0) {  // staging free; a y store issued after (S2) may still run
            if (PROD != kProdNone && prod.write_y)
                bulk_wait_group_read<1>();
            else
                bulk_wait_group_read0();
        }
        __syncthreads();  // (S3) column scales ready, staging free

        // Scale vectors: thread i < 128 writes row i of the rowwise operand
        // (k-block c0/128), thread 128 + i row i of the transposed operand
        // (k-block r0/128).  They read the exponents before (S4), so the next
        // tile's row exponents (written before its (S2), after (S4) here)
        // cannot overtake them.
        if (tid < 2 * kQT) {
            const bool col = tid >= kQT;
            if (!col || HAS_T) {
                const int i = tid & (kQT - 1);
                const int64_t op_rows0 = col ? c0 : r0;
                const int64_t kb = (col ? r0 : c0) / kQT;
                const int64_t kblocks = (col ? rows : cols) / kQT;
                store_scale_vec(col ? scale_t_u8 : scale_u8, op_rows0 + i, kb, kblocks, col ? sm.col_g[i] : sm.row_g[i]);
            }
        }

        // ---- C: rowwise codes (row i, 4 columns) and transposed codes
        // (column j, 8 rows) from the block, re-read from shared memory.
        // Every multiplier of the thread's rows and columns finite: the
        // common path.  (A NaN multiplier -- a non-finite group -- makes the
        // sum NaN; large finite ones can only overflow it to infinity.)
        float4 cmv = make_float4(1.0f, 1.0f, 1.0f, 1.0f);
        float msum = rmul[0];
#pragma unroll
        for (int i = 1; i < 8; ++i) msum += rmul[i];
        if constexpr (HAS_T) {
            cmv = *reinterpret_cast<const float4 *>(&sm.col_mul[4 * bc]);
            msum += (cmv.x + cmv.y) + (cmv.z + cmv.w);
        }
        if (!isnan(msum)) {
            // Each row's four values are widened to fp32 once and give both
            // copies: the rowwise codes (the row's multiplier) and, packed
            // into one word per row (byte j: column 4bc+j), the transposed
            // codes (the columns' multipliers), which byte transposes then
            // gather by column (stage_transposed_8x4).
            const uint64_t cm01 = f32x2(cmv.x, cmv.y), cm23 = f32x2(cmv.z, cmv.w);
            uint32_t rw[8];
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint2 w = *reinterpret_cast<const uint2 *>(in + (8 * br + i) * kQT + 4 * bc);
                const uint64_t p0 = f32x2(bf16_lo(w.x), bf16_hi(w.x)), p1 = f32x2(bf16_lo(w.y), bf16_hi(w.y));
                const uint64_t rr = f32x2(rmul[i], rmul[i]);
                *reinterpret_cast<uint32_t *>(sm.q_stage + (8 * br + i) * kQT + 4 * bc) =
                    cvt_f32x2<FMT>(mul_f32x2(p0, rr)) | (cvt_f32x2<FMT>(mul_f32x2(p1, rr)) << 16);
                if constexpr (HAS_T)
                    rw[i] = cvt_f32x2<FMT>(mul_f32x2(p0, cm01)) | (cvt_f32x2<FMT>(mul_f32x2(p1, cm23)) << 16);
            }
            if constexpr (HAS_T) stage_transposed_8x4(sm.qt_stage, rw, br, bc);
        } else {
            // General path (a group of the tile held Inf or NaN): codes one by
            // one with the NaN handling of quant4, the transposed ones rotated
            // by register selects.
#pragma unroll
            for (int i = 0; i < 8; ++i) v[i] = *reinterpret_cast<const uint2 *>(in + (8 * br + i) * kQT + 4 * bc);
#pragma unroll
            for (int i = 0; i < 8; ++i) {
                const uint64_t m2 = f32x2(rmul[i], rmul[i]);
                const uint32_t o = quant4<FMT>(bf16_lo(v[i].x), bf16_hi(v[i].x), bf16_lo(v[i].y), bf16_hi(v[i].y), m2,
                                               isnan(rmul[i]));
                *reinterpret_cast<uint32_t *>(sm.q_stage + (8 * br + i) * kQT + 4 * bc) = o;  // a warp: one 128-byte row
            }
            if constexpr (HAS_T) {
                const float4 cmv = *reinterpret_cast<const float4 *>(&sm.col_mul[4 * bc]);
                const float cmul[4] = {cmv.x, cmv.y, cmv.z, cmv.w};
                uint2 cc[4];
#pragma unroll
                for (int j = 0; j < 4; ++j) {
                    const uint64_t m2 = f32x2(cmul[j], cmul[j]);
                    const bool nan_col = isnan(cmul[j]);
                    float c[8];
#pragma unroll
                    for (int i = 0; i < 8; ++i) {
                        const uint32_t w = (j >> 1) ? v[i].y : v[i].x;
                        c[i] = (j & 1) ? bf16_hi(w) : bf16_lo(w);
                    }
                    cc[j].x = quant4<FMT>(c[0], c[1], c[2], c[3], m2, nan_col);
                    cc[j].y = quant4<FMT>(c[4], c[5], c[6], c[7], m2, nan_col);
                }
                // Column j's 8 codes (rows 8br .. 8br+7) go to transposed row
                // 4bc + j, bytes 8br .. 8br+7, whose 16-byte chunk is
                // (br / 2) ^ ((4bc + j) % 8) under the 128-byte swizzle.  All 32
                // lanes of a warp share br, so storing the same j together would
                // put them in two chunks; lane bc stores column (s + bc / 2) % 4 at
                // step s, which spreads them over all eight (a rotation of cc).
                const int rot = (bc >> 1) & 3;
#pragma unroll
                for (int b = 1; b < 4; b <<= 1) {  // cc[s] <- cc[(s + rot) % 4], one rotate-by-b stage per bit
                    const bool on = (rot & b) != 0;
                    uint2 t[4];
#pragma unroll
                    for (int k = 0; k < 4; ++k) t[k] = on ? cc[(k + b) & 3] : cc[k];
#pragma unroll
                    for (int k = 0; k < 4; ++k) cc[k] = t[k];
                }
#pragma unroll
                for (int st = 0; st < 4; ++st) {
                    const int r = 4 * bc + ((st + rot) & 3);  // transposed row (tile column)
                    *reinterpret_cast<uint2 *>(sm.qt_stage + r * kQT + 16 * ((br >> 1) ^ (r & 7)) + 8 * (br & 1)) = cc[st];
                }
            }
        }

        fence_proxy_async_smem();
        __syncthreads();  // (S4) staging complete
        if (tid == 0) {
            tma_store_2d(&tm_q, sm.q_stage, static_cast<int32_t>(c0), static_cast<int32_t>(r0));
            if (HAS_T) tma_store_2d(&tm_qt, sm.qt_stage, static_cast<int32_t>(r0), static_cast<int32_t>(c0));
            bulk_commit_group();
        }
    }
    if (tid == 0) bulk_wait_group0();
}

// ------------------------------------------------------ grouped weight cast
// The weights of a model are quantised once per optimizer step (section "FP8
// Mixed-Precision Training": 128x128 blocks), so all of them can go through
// one launch: the persistent CTAs take the 128x128 tiles of every weight in
// one sequence, weight after weight, and treat each exactly as
// quant_tile_kernel<FMT, kQuantBlockWeight, HAS_T> does.  Small weights then
// share waves instead of each paying a launch, a ramp and a tail.
template <int FMT, bool HAS_T>
__global__ void __launch_bounds__(kQThreads, 2) quant_weight_group_kernel(const __grid_constant__ WeightGroup g) {
    extern __shared__ uint8_t smem_raw[];
    QuantSmem &sm = *reinterpret_cast<QuantSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                   ~static_cast<uintptr_t>(1023));
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int br = warp;  // block row: tile rows 8br .. 8br+7
    const int bc = lane;  // block column: tile columns 4bc .. 4bc+3
    pdl_wait();
    pdl_launch_dependents();
    if (tid == 0) {
        mbar_init(&sm.full[0], 1);
        mbar_init(&sm.full[1], 1);
        fence_mbarrier_init();
    }
    __syncthreads();

    const int ntiles = g.tile_start[g.count];
    // the weight of tile t, scanning forward from w (tiles only increase)
    auto locate = [&](int t, int w) {
        while (t >= g.tile_start[w + 1]) ++w;
        return w;
    };
    auto issue_load = [&](int t, int w, int b) {
        const int lt = t - g.tile_start[w];
        mbar_arrive_expect_tx(&sm.full[b], kQT * kQT * 2);
        tma_load_2d(sm.in[b], &g.x[w], &sm.full[b], (lt % g.tiles_n[w]) * kQT, (lt / g.tiles_n[w]) * kQT);
    };
    int tile = blockIdx.x;
    int w = 0;
    if (tile < ntiles) {
        w = locate(tile, 0);
        if (tid == 0) issue_load(tile, w, 0);
    }
    for (int it = 0; tile < ntiles; ++it, tile += gridDim.x) {
        w = locate(tile, w);
        const int buf = it & 1;
        const int lt = tile - g.tile_start[w];
        const int64_t r0 = static_cast<int64_t>(lt / g.tiles_n[w]) * kQT;
        const int64_t c0 = static_cast<int64_t>(lt % g.tiles_n[w]) * kQT;
        if (tid == 0) {
            const int next = tile + gridDim.x;
            if (next < ntiles) issue_load(next, locate(next, w), buf ^ 1);  // buffer last read before (S3) of it-1
        }
        const bool landed = tile_landed(&sm.full[buf], static_cast<uint32_t>(it >> 1) & 1u, g.wait_ns);

        const uint16_t *in = sm.in[buf];
        uint2 v[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) v[i] = *reinterpret_cast<const uint2 *>(in + (8 * br + i) * kQT + 4 * bc);
        const uint32_t m = __reduce_max_sync(0xFFFFFFFFu, block_max_8x4(v));
        if (lane == 0) sm.red[warp] = m;
        if (tid == 0) bulk_wait_group_read0();  // the previous tile's stores have read the staging
        if (__syncthreads_or(!landed)) {         // (S2) block maxima written, staging free
            if (tid == 0) quant_abort(sm.full, it, tile + static_cast<int>(gridDim.x) < ntiles, g.status);
            break;
        }
        const uint32_t blk_g = e8m0_exponent<FMT>(__reduce_max_sync(0xFFFFFFFFu, sm.red[lane & 15]) & 0xFFFFu);
        const float mul = mul_of(blk_g);
        tile_codes_to_stage<FMT, HAS_T>(sm, v, br, bc, f32x2(mul, mul), isnan(mul));

        fence_proxy_async_smem();
        __syncthreads();  // (S3) staging complete
        if (tid == 0) {
            tma_store_2d(&g.q[w], sm.q_stage, static_cast<int32_t>(c0), static_cast<int32_t>(r0));
            if (HAS_T) tma_store_2d(&g.qt[w], sm.qt_stage, static_cast<int32_t>(r0), static_cast<int32_t>(c0));
            bulk_commit_group();
        }
        // scale vectors: thread i < 128 row i of the rowwise copy, 128 + i row
        // i of the transposed copy (the block's exponent over its 128 rows)
        const bool col = tid >= kQT;
        if (tid < 2 * kQT && (!col || HAS_T)) {
            const int i = tid & (kQT - 1);
            store_scale_vec(col ? g.scale_t[w] : g.scale[w], (col ? c0 : r0) + i, (col ? r0 : c0) / kQT,
                            col ? g.kb_rows[w] : g.tiles_n[w], static_cast<uint8_t>(blk_g));
        }
    }
    if (tid == 0) bulk_wait_group0();
}

cudaError_t launch_quantize_weights(const WeightGroup &g, int fmt, bool has_t, cudaStream_t s) {
    const int ntiles = g.tile_start[g.count];
    if (ntiles == 0) return cudaSuccess;
    auto kern = fmt == 0 ? (has_t ? quant_weight_group_kernel<0, true> : quant_weight_group_kernel<0, false>)
                         : (has_t ? quant_weight_group_kernel<1, true> : quant_weight_group_kernel<1, false>);
    const size_t smem = sizeof(QuantSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int sms = sm_count_here();
    const int grid = ntiles < 2 * sms ? ntiles : 2 * sms;  // persistent: two CTAs per SM
    return launch_pdl(kern, dim3(grid), dim3(kQThreads), smem, s, g);
}

// Per-tensor scale only (empty tensors: amax = 0 gives scale_inv = 1).
template <int FMT>
__global__ void tensor_scale_only_kernel(const uint32_t *amax_bits, float *scale_f, float *scale_t_f) {
    pdl_wait();
    pdl_launch_dependents();
    const uint32_t a = *amax_bits & 0xFFFFu;
    const float si = (a >= 0x7F80u) ? __uint_as_float(0x7FC00000u) : __fdiv_rn(1.0f, tensor_scale<FMT>(a));
    *scale_f = si;
    if (scale_t_f) *scale_t_f = si;
}

cudaError_t launch_tensor_scale_only(const QuantArgs &a, cudaStream_t s) {
    return launch_pdl(a.fmt == 0 ? tensor_scale_only_kernel<0> : tensor_scale_only_kernel<1>, dim3(1), dim3(1), 0, s,
                      a.amax, a.scale_f, a.scale_t_f);
}

template <int FMT, int KIND, bool HAS_T, int PROD = kProdNone>
static cudaError_t launch_quant_t(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                  const CUtensorMap &tm_qt, cudaStream_t s, const CUtensorMap *tm_y = nullptr,
                                  ProdArgs prod = ProdArgs{}) {
    if constexpr (KIND == kQuantBlockAct) {  // the 512-thread activation kernel (whole tiles)
        auto kern = quant_act_kernel<FMT, HAS_T, PROD>;
        const size_t smem = sizeof(QuantActSmem) + 1024;
        cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
        if (e != cudaSuccess) return e;
        const int tiles_n = static_cast<int>(a.cols / kQT);
        const int ntiles = static_cast<int>(a.rows / kQT) * tiles_n;
        int dev = 0, sms = 148;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        const int grid = ntiles < 2 * sms ? ntiles : 2 * sms;  // persistent: two CTAs per SM
        return launch_pdl(kern, dim3(grid), dim3(kQAThreads), smem, s, tm_x, tm_q, tm_qt, tm_y ? *tm_y : tm_x, a.rows,
                          a.cols, a.scale_u8, a.scale_t_u8, prod, tiles_n, ntiles, a.status, a.wait_ns);
    } else {
        static_assert(PROD == kProdNone, "producers feed the activation quantiser");
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
        return launch_pdl(kern, dim3(grid), dim3(kQThreads), smem, s, tm_x, tm_q, tm_qt, a.rows, a.cols, a.scale_u8,
                          a.scale_t_u8, a.scale_f, a.scale_t_f, a.amax, tiles_n, ntiles, a.status, a.wait_ns);
    }
}

template <int FMT, int KIND>
static cudaError_t launch_quant_k(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                  const CUtensorMap &tm_qt, cudaStream_t s) {
    return a.has_t ? launch_quant_t<FMT, KIND, true>(a, tm_x, tm_q, tm_qt, s)
                   : launch_quant_t<FMT, KIND, false>(a, tm_x, tm_q, tm_qt, s);
}

template <int FMT>
static cudaError_t launch_quant_f(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                  const CUtensorMap &tm_qt, cudaStream_t s) {
    switch (a.kind) {
        case kQuantBlockAct: return launch_quant_k<FMT, kQuantBlockAct>(a, tm_x, tm_q, tm_qt, s);
        case kQuantBlockWeight: return launch_quant_k<FMT, kQuantBlockWeight>(a, tm_x, tm_q, tm_qt, s);
        default: return launch_quant_k<FMT, kQuantTensor>(a, tm_x, tm_q, tm_qt, s);
    }
}

cudaError_t launch_quantize(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                            const CUtensorMap &tm_qt, cudaStream_t s) {
    return a.fmt == 0 ? launch_quant_f<0>(a, tm_x, tm_q, tm_qt, s) : launch_quant_f<1>(a, tm_x, tm_q, tm_qt, s);
}

template <int FMT>
static cudaError_t launch_rms_f(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                cudaStream_t s) {
    return a.has_t ? launch_quant_t<FMT, kQuantBlockAct, true, kProdRmsNorm>(a, tm_x, tm_q, tm_qt, s, &tm_y, prod)
                   : launch_quant_t<FMT, kQuantBlockAct, false, kProdRmsNorm>(a, tm_x, tm_q, tm_qt, s, &tm_y, prod);
}

cudaError_t launch_quantize_rmsnorm(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                    const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                    cudaStream_t s) {
    return a.fmt == 0 ? launch_rms_f<0>(a, tm_x, tm_q, tm_qt, tm_y, prod, s)
                      : launch_rms_f<1>(a, tm_x, tm_q, tm_qt, tm_y, prod, s);
}

template <int FMT>
static cudaError_t launch_swiglu_f(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                   const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                   cudaStream_t s) {
    return a.has_t ? launch_quant_t<FMT, kQuantBlockAct, true, kProdSwiGlu>(a, tm_x, tm_q, tm_qt, s, &tm_y, prod)
                   : launch_quant_t<FMT, kQuantBlockAct, false, kProdSwiGlu>(a, tm_x, tm_q, tm_qt, s, &tm_y, prod);
}

cudaError_t launch_quantize_swiglu(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                   const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                   cudaStream_t s) {
    return a.fmt == 0 ? launch_swiglu_f<0>(a, tm_x, tm_q, tm_qt, tm_y, prod, s)
                      : launch_swiglu_f<1>(a, tm_x, tm_q, tm_qt, tm_y, prod, s);
}

}  // namespace puro
