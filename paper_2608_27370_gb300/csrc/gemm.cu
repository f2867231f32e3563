// gemm.cu -- tcgen05 tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T (both
// operands K-major, "TN") with FP32 accumulation in tensor memory and a BF16
// output, for the three GEMMs of an FP8 linear layer (Puro-2B, appendix
// "Production Training Details", paragraph "FP8 implementation pipeline":
// Fprop, Dgrad and Wgrad all from E4M3 operands, BF16 output).
//
// One persistent, warp-specialised CTA per SM:
//   warp 0      TMA producer: A/B tiles (128-byte swizzle) and, for the
//               block-scaled kind, the raw E8M0 row scales, into a
//               STAGES-deep shared-memory ring gated by mbarriers;
//   warp 1      MMA issuer: allocates tensor memory, copies the staged
//               block scales into tensor memory (tcgen05.cp), issues
//               tcgen05.mma (kind::f16 / kind::f8f6f4 /
//               kind::mxf8f6f4.block_scale) and commits stage releases and
//               accumulator hand-offs;
//   warp 2      (block-scaled kind) scale staging: rearranges each stage's
//               E8M0 exponents into the tcgen05.cp source layout, off the
//               MMA issuer's critical path;
//   warps 4..7  epilogue: tcgen05.ld the 128x256 FP32 accumulator (one
//               32-lane quarter per warp), release it, convert to BF16
//               (times scale_inv_a * scale_inv_b for the per-tensor kind)
//               and TMA-store it through a swizzled staging tile.
// Every mbarrier wait is bounded in wall time; on expiry the CTA records
// PURO_ERR_TIMEOUT in the caller's status word, drains its own in-flight
// copies and MMAs (with a fixed bound), frees tensor memory and returns.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace puro {

constexpr int kBM = kGemmBM;       // rows of A per tile (= TMEM lanes)
constexpr int kBN = kGemmBN;       // rows of B per tile (= accumulator columns)
constexpr int kBKBytes = 128;      // bytes of K per pipeline stage (one swizzle row)
constexpr int kStages = 4;
constexpr int kThreads = 256;
constexpr int kTmemCols = 512;
constexpr int kSfColsPerStage = 12;  // 4 for A (128 rows) + 8 for B (256 rows)
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;
constexpr int32_t kStatusTimeout = 4;  // PURO_ERR_TIMEOUT

struct GemmSmem {
    alignas(1024) uint8_t a[kStages][kBM * kBKBytes];
    alignas(1024) uint8_t b[kStages][kBN * kBKBytes];
    alignas(1024) uint8_t epi[4][32 * 128];          // per epilogue warp: 32 rows x 64 bf16
    alignas(128) uint8_t sf_utccp_a[kStages][512];   // 32 lines x 16 B
    alignas(128) uint8_t sf_utccp_b[kStages][1024];  // 2 x (32 lines x 16 B)
    alignas(16) uint8_t sf_raw_a[kStages][kBM];
    alignas(16) uint8_t sf_raw_b[kStages][kBN];
    uint64_t full[kStages];
    uint64_t sf_ready[kStages];  // block-scaled kind: scale vectors staged for tcgen05.cp
    uint64_t empty[kStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    volatile int abort_flag;
};

struct GemmParams {
    int M, N, K;
    int num_n, num_kb, num_tiles;
    uint32_t idesc;
    const uint8_t *sfa;
    const uint8_t *sfb;
    int sfb_blk;
    int sfb_kb;  // K / 128 (row length of the 128x128 grid)
    const float *sia;
    const float *sib;
    int32_t *status;
    uint64_t wait_ns;
};

// Instruction descriptors (tcgen05.mma), both operands K-major.
//   kind::f16 / kind::f8f6f4: [4,6) D format (1 = F32), [7,10) A type,
//     [10,13) B type, [17,23) N >> 3, [24,29) M >> 4.
//   kind::mxf8f6f4: [4,6) B scale id, [7,10) A type, [10,13) B type,
//     [17,23) N >> 3, [23] scale type (1 = UE8M0), [24,29) M >> 4,
//     [29,31) A scale id.
__host__ __device__ constexpr uint32_t idesc_dense(uint32_t atype, uint32_t btype) {
    return (1u << 4) | (atype << 7) | (btype << 10) | (static_cast<uint32_t>(kBN >> 3) << 17) |
           (static_cast<uint32_t>(kBM >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_mx(uint32_t atype, uint32_t btype) {
    return (atype << 7) | (btype << 10) | (static_cast<uint32_t>(kBN >> 3) << 17) | (1u << 23) |
           (static_cast<uint32_t>(kBM >> 4) << 24);
}

PURO_DEV void record_timeout(GemmSmem &sm, int32_t *status) {
    sm.abort_flag = 1;
    if (status) atomicExch(status, kStatusTimeout);
}

template <int KIND>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tn_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                   const __grid_constant__ CUtensorMap tm_d, const GemmParams p) {
    constexpr bool kMX = (KIND == kGemmFP8Block);
    constexpr int kAccBufs = kMX ? 1 : 2;              // accumulators of kBN columns
    constexpr int kSfBase = kAccBufs * kBN;            // first scale-factor column (MX)
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;         // elements of K per stage
    constexpr int kKSteps = kBKBytes / 32;             // MMAs per stage (32 bytes of K each)
    static_assert(!kMX || kSfBase + kStages * kSfColsPerStage <= kTmemCols, "TMEM budget");

    extern __shared__ uint8_t smem_raw[];
    GemmSmem &sm = *reinterpret_cast<GemmSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                 ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.sf_ready[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sm.tfull[b], 1);
            mbar_init(&sm.tempty[b], 4);
        }
        mbar_init(&sm.drain, 1);
        sm.abort_flag = 0;
        fence_mbarrier_init();
        tma_prefetch_desc(&tm_a);
        tma_prefetch_desc(&tm_b);
        tma_prefetch_desc(&tm_d);
    }
    if (warp == 1) {
        tmem_alloc(&sm.tmem_base, kTmemCols);
        tmem_relinquish_alloc_permit();
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            uint32_t stage = 0, phase = 0;
            uint32_t issued = 0;  // stage fills started by this thread
            bool aborted = false;
            for (int tile = blockIdx.x; tile < p.num_tiles && !aborted; tile += gridDim.x) {
                const int m0 = (tile / p.num_n) * kBM;
                const int n0 = (tile % p.num_n) * kBN;
                const uint32_t sfb_bytes = static_cast<uint32_t>(min(kBN, p.N - n0));
                for (int kb = 0; kb < p.num_kb; ++kb) {
                    if (sm.abort_flag || !mbar_wait_bounded(&sm.empty[stage], phase ^ 1u, p.wait_ns)) {
                        record_timeout(sm, p.status);
                        aborted = true;
                        break;
                    }
                    uint32_t bytes = (kBM + kBN) * kBKBytes;
                    if (kMX) bytes += kBM + (p.sfb_blk ? 0u : sfb_bytes);
                    mbar_arrive_expect_tx(&sm.full[stage], bytes);
                    tma_load_2d(sm.a[stage], &tm_a, &sm.full[stage], kb * kBK, m0);
                    tma_load_2d(sm.b[stage], &tm_b, &sm.full[stage], kb * kBK, n0);
                    if (kMX) {
                        bulk_load(sm.sf_raw_a[stage], p.sfa + static_cast<int64_t>(kb) * p.M + m0, kBM,
                                  &sm.full[stage]);
                        if (!p.sfb_blk)
                            bulk_load(sm.sf_raw_b[stage], p.sfb + static_cast<int64_t>(kb) * p.N + n0, sfb_bytes,
                                      &sm.full[stage]);
                    }
                    ++issued;
                    if (++stage == kStages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            // Every copy this thread started must land before the CTA exits:
            // wait for the latest fill of each stage (fills go round-robin).
            for (uint32_t s = 0; s < kStages; ++s) {
                const uint32_t fills = issued / kStages + (s < issued % kStages ? 1u : 0u);
                if (fills > 0) mbar_wait_bounded(&sm.full[s], (fills - 1u) & 1u, kDrainTimeoutNs);
            }
        }
    } else if (warp == 1) {
        // ------------------------------------------------ MMA issuer
        uint32_t stage = 0, phase = 0;
        bool aborted = false;
        int local = 0;
        for (int tile = blockIdx.x; tile < p.num_tiles && !aborted; tile += gridDim.x, ++local) {
            const int buf = local % kAccBufs;
            const uint32_t acc_phase = static_cast<uint32_t>(local / kAccBufs) & 1u;
            bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tempty[buf], acc_phase ^ 1u, p.wait_ns);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                if (lane == 0) record_timeout(sm, p.status);
                aborted = true;
                break;
            }
            tc_fence_after_sync();
            const uint32_t d_tmem = tmem + static_cast<uint32_t>(buf * kBN);

            for (int kb = 0; kb < p.num_kb; ++kb) {
                // block-scaled: the scale warp has staged this stage's scale
                // vectors (and has itself seen the operands land)
                ok = (sm.abort_flag == 0) &&
                     mbar_wait_bounded(kMX ? &sm.sf_ready[stage] : &sm.full[stage], phase, p.wait_ns) &&
                     (!kMX || mbar_wait_bounded(&sm.full[stage], phase, p.wait_ns));
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    if (lane == 0) record_timeout(sm, p.status);
                    aborted = true;
                    break;
                }
                tc_fence_after_sync();
                if (lane == 0) {
                    const uint32_t sfa_col = kSfBase + stage * kSfColsPerStage;
                    const uint32_t sfb_col = sfa_col + 4;
                    if constexpr (kMX) {
                        tmem_cp_32x128b_warpx4(tmem + sfa_col, smem_desc_plain_16B_rows(smem_u32(sm.sf_utccp_a[stage])));
                        tmem_cp_32x128b_warpx4(tmem + sfb_col, smem_desc_plain_16B_rows(smem_u32(sm.sf_utccp_b[stage])));
                        tmem_cp_32x128b_warpx4(tmem + sfb_col + 4,
                                               smem_desc_plain_16B_rows(smem_u32(sm.sf_utccp_b[stage] + 512)));
                    }
                    const uint32_t a_addr = smem_u32(sm.a[stage]);
                    const uint32_t b_addr = smem_u32(sm.b[stage]);
#pragma unroll
                    for (int k = 0; k < kKSteps; ++k) {
                        const uint64_t ad = smem_desc_k_sw128(a_addr + 32 * k);
                        const uint64_t bd = smem_desc_k_sw128(b_addr + 32 * k);
                        const uint32_t acc = (kb > 0 || k > 0) ? 1u : 0u;
                        if constexpr (KIND == kGemmBF16)
                            mma_f16(d_tmem, ad, bd, p.idesc, acc);
                        else if constexpr (KIND == kGemmFP8Tensor)
                            mma_f8(d_tmem, ad, bd, p.idesc, acc);
                        else
                            mma_mxf8(d_tmem, ad, bd, p.idesc, tmem + sfa_col, tmem + sfb_col, acc);
                    }
                    tc_commit(&sm.empty[stage]);  // stage reusable once these MMAs finish
                }
                __syncwarp();
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (aborted) break;
            if (lane == 0) tc_commit(&sm.tfull[buf]);  // accumulator complete
            __syncwarp();
        }
        // All MMAs and copies issued by this warp complete before teardown.
        if (lane == 0) {
            tc_commit(&sm.drain);
            mbar_wait_bounded(&sm.drain, 0, kDrainTimeoutNs);
        }
        __syncwarp();
    } else if (kMX && warp == 2) {
        // ------------------------------------------------ scale staging
        // Turns each stage's raw E8M0 exponents into the tcgen05.cp source
        // layout: row r of a 128-row operand block goes to line r % 32, word
        // r / 32, all four bytes of the word carrying the exponent (one 1x128
        // group spans four K=32 MMAs, each reading one scale per row).
        uint32_t stage = 0, phase = 0;
        bool aborted = false;
        // 128x128 weight-block scales of the current / next tile: lane j
        // holds k-blocks 8j .. 8j+7 of n-block 0 (words 0,1) and 1 (2,3).
        uint32_t blk_cur[4] = {0, 0, 0, 0}, blk_nxt[4] = {0, 0, 0, 0};
        auto load_blk = [&](int tile, uint32_t (&r)[4]) {
            const int nb0 = (tile % p.num_n) * (kBN / 128);
#pragma unroll
            for (int h = 0; h < 2; ++h) {
                const int nb = nb0 + h;
                const bool nb_ok = nb * 128 < p.N;
#pragma unroll
                for (int w = 0; w < 2; ++w) {
                    uint32_t word = 0;
#pragma unroll
                    for (int i = 0; i < 4; ++i) {
                        const int kb = 8 * lane + 4 * w + i;
                        uint32_t v = 127u;
                        if (nb_ok && kb < p.sfb_kb) v = p.sfb[static_cast<int64_t>(nb) * p.sfb_kb + kb];
                        word |= v << (8 * i);
                    }
                    r[2 * h + w] = word;
                }
            }
        };
        if (p.sfb_blk && static_cast<int>(blockIdx.x) < p.num_tiles) load_blk(blockIdx.x, blk_cur);
        for (int tile = blockIdx.x; tile < p.num_tiles && !aborted; tile += gridDim.x) {
            const int n0 = (tile % p.num_n) * kBN;
            if (p.sfb_blk && tile + static_cast<int>(gridDim.x) < p.num_tiles) load_blk(tile + gridDim.x, blk_nxt);
            for (int kb = 0; kb < p.num_kb; ++kb) {
                bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.full[stage], phase, p.wait_ns);
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    if (lane == 0) record_timeout(sm, p.status);
                    aborted = true;
                    break;
                }
                const uint8_t *ra = sm.sf_raw_a[stage];
                uint4 la;
                la.x = ra[lane] * 0x01010101u;
                la.y = ra[lane + 32] * 0x01010101u;
                la.z = ra[lane + 64] * 0x01010101u;
                la.w = ra[lane + 96] * 0x01010101u;
                *reinterpret_cast<uint4 *>(sm.sf_utccp_a[stage] + 16 * lane) = la;
                uint32_t wb[8];
                if (p.sfb_blk) {
                    const int src = kb >> 3, wsel = (kb >> 2) & 1, sh = 8 * (kb & 3);
                    const uint32_t w00 = __shfl_sync(0xFFFFFFFFu, blk_cur[0], src);
                    const uint32_t w01 = __shfl_sync(0xFFFFFFFFu, blk_cur[1], src);
                    const uint32_t w10 = __shfl_sync(0xFFFFFFFFu, blk_cur[2], src);
                    const uint32_t w11 = __shfl_sync(0xFFFFFFFFu, blk_cur[3], src);
                    const uint32_t s0 = ((wsel ? w01 : w00) >> sh) & 0xFFu;
                    const uint32_t s1 = ((wsel ? w11 : w10) >> sh) & 0xFFu;
#pragma unroll
                    for (int j = 0; j < 8; ++j) wb[j] = (j < 4 ? s0 : s1) * 0x01010101u;
                } else {
                    const uint8_t *rb = sm.sf_raw_b[stage];
                    const int valid = p.N - n0;
#pragma unroll
                    for (int j = 0; j < 8; ++j) {
                        const int r = lane + 32 * j;
                        wb[j] = (r < valid ? static_cast<uint32_t>(rb[r]) : 127u) * 0x01010101u;
                    }
                }
                *reinterpret_cast<uint4 *>(sm.sf_utccp_b[stage] + 16 * lane) = make_uint4(wb[0], wb[1], wb[2], wb[3]);
                *reinterpret_cast<uint4 *>(sm.sf_utccp_b[stage] + 512 + 16 * lane) =
                    make_uint4(wb[4], wb[5], wb[6], wb[7]);
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sm.sf_ready[stage]);
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (p.sfb_blk) {
#pragma unroll
                for (int i = 0; i < 4; ++i) blk_cur[i] = blk_nxt[i];
            }
        }
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lane quarter of this warp
        float sab = 1.0f;
        if constexpr (KIND == kGemmFP8Tensor) sab = __fmul_rn(*p.sia, *p.sib);
        uint8_t *stage_buf = sm.epi[q];
        int local = 0;
        for (int tile = blockIdx.x; tile < p.num_tiles; tile += gridDim.x, ++local) {
            const int m0 = (tile / p.num_n) * kBM;
            const int n0 = (tile % p.num_n) * kBN;
            const int buf = local % kAccBufs;
            const uint32_t acc_phase = static_cast<uint32_t>(local / kAccBufs) & 1u;
            bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tfull[buf], acc_phase, p.wait_ns);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                if (lane == 0) record_timeout(sm, p.status);
                break;
            }
            tc_fence_after_sync();
            const uint32_t t_row = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(buf * kBN);
            uint32_t packed[kBN / 2];  // the whole 256-column row as bf16 pairs
#pragma unroll
            for (int h = 0; h < kBN / 128; ++h) {
                uint32_t r[4][32];
#pragma unroll
                for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(t_row + 128 * h + 32 * c, r[c]);
                tmem_ld_wait();
#pragma unroll
                for (int c = 0; c < 4; ++c) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) {
                        float lo = __uint_as_float(r[c][2 * i]), hi = __uint_as_float(r[c][2 * i + 1]);
                        if constexpr (KIND == kGemmFP8Tensor) {
                            lo = __fmul_rn(lo, sab);
                            hi = __fmul_rn(hi, sab);
                        }
                        __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
                        packed[64 * h + 16 * c + i] = *reinterpret_cast<uint32_t *>(&v);
                    }
                }
            }
            tc_fence_before_sync();
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.tempty[buf]);  // accumulator free for the next tile
            // Store 4 chunks of 64 columns (128 bytes per row) through the
            // per-warp staging tile, 16-byte chunk i of row l at i ^ (l % 8).
#pragma unroll
            for (int ch = 0; ch < kBN / 64; ++ch) {
                if (n0 + 64 * ch >= p.N) break;
                if (lane == 0) bulk_wait_group_read0();
                __syncwarp();
                uint8_t *row = stage_buf + 128 * lane;
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    const uint4 v = make_uint4(packed[32 * ch + 4 * i], packed[32 * ch + 4 * i + 1],
                                               packed[32 * ch + 4 * i + 2], packed[32 * ch + 4 * i + 3]);
                    *reinterpret_cast<uint4 *>(row + 16 * (i ^ (lane & 7))) = v;
                }
                fence_proxy_async_smem();
                __syncwarp();
                if (lane == 0) {
                    tma_store_2d(&tm_d, stage_buf, n0 + 64 * ch, m0 + 32 * q);
                    bulk_commit_group();
                }
            }
        }
        if (lane == 0) bulk_wait_group0();
        __syncwarp();
    }

    tc_fence_before_sync();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after_sync();
        tmem_dealloc(tmem, kTmemCols);
    }
}

template <int KIND>
static cudaError_t launch_kind(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                               const CUtensorMap &tm_d, cudaStream_t s) {
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;
    GemmParams p{};
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.K = static_cast<int>(g.K);
    p.num_n = static_cast<int>((g.N + kBN - 1) / kBN);
    const int num_m = static_cast<int>((g.M + kBM - 1) / kBM);
    p.num_kb = static_cast<int>((g.K + kBK - 1) / kBK);
    p.num_tiles = num_m * p.num_n;
    if (KIND == kGemmBF16)
        p.idesc = idesc_dense(1u, 1u);
    else if (KIND == kGemmFP8Tensor)
        p.idesc = idesc_dense(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt));
    else
        p.idesc = idesc_mx(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt));
    p.sfa = g.sfa;
    p.sfb = g.sfb;
    p.sfb_blk = g.sfb_blk;
    p.sfb_kb = static_cast<int>(g.K / 128);
    p.sia = g.sia;
    p.sib = g.sib;
    p.status = g.status;
    p.wait_ns = g.wait_timeout_ns;

    auto kern = gemm_tn_kernel<KIND>;
    const size_t smem = sizeof(GemmSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int grid = p.num_tiles < g.num_sms ? p.num_tiles : g.num_sms;
    kern<<<grid, kThreads, smem, s>>>(tm_a, tm_b, tm_d, p);
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                        const CUtensorMap &tm_d, cudaStream_t s) {
    switch (g.kind) {
        case kGemmBF16: return launch_kind<kGemmBF16>(g, tm_a, tm_b, tm_d, s);
        case kGemmFP8Tensor: return launch_kind<kGemmFP8Tensor>(g, tm_a, tm_b, tm_d, s);
        default: return launch_kind<kGemmFP8Block>(g, tm_a, tm_b, tm_d, s);
    }
}

}  // namespace puro
