// gemm.cu -- tcgen05 tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T (both
// operands K-major, "TN") with FP32 accumulation in tensor memory and a BF16
// output, for the three GEMMs of an FP8 linear layer (Puro-2B, appendix
// "Production Training Details", paragraph "FP8 implementation pipeline":
// Fprop, Dgrad and Wgrad all from E4M3 operands, BF16 output).
//
// One persistent, warp-specialised CTA per SM:
//   warp 0      TMA producer: A/B tiles (128-byte swizzle) and, for the
//               block-scaled kind, the E8M0 scale vectors (already in the
//               tensor-core layout, 512 bytes per 128 rows and four
//               k-blocks), into a STAGES-deep shared-memory ring gated by
//               mbarriers;
//   warp 1      MMA issuer: allocates tensor memory, copies the scale
//               vectors into tensor memory (tcgen05.cp, once per four
//               k-blocks), issues tcgen05.mma (kind::f16 / kind::f8f6f4 /
//               kind::mxf8f6f4.block_scale, the scale id picking the
//               k-block's byte) and commits stage releases and accumulator
//               hand-offs;
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
constexpr int kBKBytes = kGemmBKBytes;             // bytes of K per pipeline stage (one swizzle row)
constexpr int kStages = kBKBytes == 128 ? 4 : 8;   // ~192 KB of operand ring either way
constexpr int kStagesPerKBlock = 128 / kBKBytes;   // stages per 128-byte k-block (one FP8 scale group)
constexpr int kStagesPerGroup = 512 / kBKBytes;    // stages per group of four k-blocks (one scale chunk)
constexpr int kThreads = 256;
constexpr int kTmemCols = 512;
constexpr int kSfColsPerSet = 12;  // 4 for A (128 rows) + 8 for B (256 rows)
constexpr int kSfSets = 2;         // double-buffered across groups of four k-blocks
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;
constexpr int32_t kStatusTimeout = 4;  // PURO_ERR_TIMEOUT
constexpr int64_t kSplitRefSms = 152;  // SM count the split heuristic plans for (GB300)

struct GemmSmem {
    alignas(1024) uint8_t a[kStages][kBM * kBKBytes];
    alignas(1024) uint8_t b[kStages][kBN * kBKBytes];
    alignas(1024) uint8_t epi[4][32 * 128];          // per epilogue warp: 32 rows x 64 bf16
    alignas(128) uint8_t sf_a[kStages][512];   // scale vectors of A: 32 lines x 16 B
    alignas(128) uint8_t sf_b[kStages][1024];  // scale vectors of B: 2 x (32 lines x 16 B)
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t tfull[2];
    uint64_t tempty[2];
    uint64_t drain;
    uint32_t tmem_base;
    volatile int abort_flag;
};

struct GemmParams {
    int M, N, K;
    int num_m, num_n, num_kb, num_tiles;
    int splits;        // reduction split into this many chunks (1: no split)
    int kb_per_split;  // stages per chunk (a whole number of scale groups)
    int num_units;     // num_tiles * splits
    int m_fastest;     // tile order: 1 = row blocks of A vary fastest
    uint32_t idesc;
    const uint8_t *sfa;  // scale vectors of A, [M/128][kgroups][512]
    const uint8_t *sfb;  // scale vectors of B, [N/128][kgroups][512]
    int kgroups;         // ceil(K / 512)
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
//     [29,31) A scale id.  The scale id selects the byte of the 32-bit
//     tensor-memory scale word: here the k-block within its group of four.
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

// One unit of work: an output tile and a chunk of the reduction.  Units of
// the same chunk are consecutive; within a chunk the tile order iterates the
// blocks of the smaller operand fastest, so the CTAs of a wave share (and
// read once) the blocks of the larger one.
struct WorkUnit {
    int m0, n0, kb0, kb1, split;
};

PURO_DEV WorkUnit work_unit(const GemmParams &p, int u) {
    WorkUnit w;
    w.split = u / p.num_tiles;
    const int tile = u - w.split * p.num_tiles;
    const int mb = p.m_fastest ? tile % p.num_m : tile / p.num_n;
    const int nb = p.m_fastest ? tile / p.num_m : tile % p.num_n;
    w.m0 = mb * kBM;
    w.n0 = nb * kBN;
    w.kb0 = w.split * p.kb_per_split;
    w.kb1 = min(p.num_kb, w.kb0 + p.kb_per_split);
    return w;
}

// OUT_F32: write FP32 partial tiles of a split reduction to the workspace
// [splits * Mp, N], Mp = M rounded up to 128 (rows split * Mp + m), instead
// of the BF16 output; a ragged last row tile then stays inside its chunk.
template <int KIND, bool OUT_F32>
__global__ void __launch_bounds__(kThreads, 1)
    gemm_tn_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                   const __grid_constant__ CUtensorMap tm_d, const GemmParams p) {
    constexpr bool kMX = (KIND == kGemmFP8Block);
    constexpr int kAccBufs = kMX ? 1 : 2;              // accumulators of kBN columns
    constexpr int kSfBase = kAccBufs * kBN;            // first scale-vector column (MX)
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;         // elements of K per stage
    constexpr int kKSteps = kBKBytes / 32;             // MMAs per stage (32 bytes of K each)
    static_assert(!kMX || kSfBase + kSfSets * kSfColsPerSet <= kTmemCols, "TMEM budget");

    extern __shared__ uint8_t smem_raw[];
    GemmSmem &sm = *reinterpret_cast<GemmSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                 ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
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
            for (int u = blockIdx.x; u < p.num_units && !aborted; u += gridDim.x) {
                const WorkUnit wu = work_unit(p, u);
                const int m0 = wu.m0, n0 = wu.n0;
                const bool b_second = n0 + 128 < p.N;  // second 128-row block of B in range
                for (int kb = wu.kb0; kb < wu.kb1; ++kb) {
                    if (sm.abort_flag || !mbar_wait_bounded(&sm.empty[stage], phase ^ 1u, p.wait_ns)) {
                        record_timeout(sm, p.status);
                        aborted = true;
                        break;
                    }
                    const bool sf_load = kMX && (kb % kStagesPerGroup) == 0;
                    const uint32_t bytes = (kBM + kBN) * kBKBytes + (sf_load ? 512u + 1024u : 0u);
                    mbar_arrive_expect_tx(&sm.full[stage], bytes);
                    tma_load_2d(sm.a[stage], &tm_a, &sm.full[stage], kb * kBK, m0);
                    tma_load_2d(sm.b[stage], &tm_b, &sm.full[stage], kb * kBK, n0);
                    if (sf_load) {
                        const int64_t kg = kb / kStagesPerGroup;
                        bulk_load(sm.sf_a[stage], p.sfa + ((m0 / 128) * static_cast<int64_t>(p.kgroups) + kg) * 512, 512,
                                  &sm.full[stage]);
                        const uint8_t *b0 = p.sfb + ((n0 / 128) * static_cast<int64_t>(p.kgroups) + kg) * 512;
                        bulk_load(sm.sf_b[stage], b0, 512, &sm.full[stage]);
                        // beyond N the B rows are zero-filled; any finite scale will do
                        bulk_load(sm.sf_b[stage] + 512, b_second ? b0 + static_cast<int64_t>(p.kgroups) * 512 : b0, 512,
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
        for (int u = blockIdx.x; u < p.num_units && !aborted; u += gridDim.x, ++local) {
            const WorkUnit wu = work_unit(p, u);
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

            for (int kb = wu.kb0; kb < wu.kb1; ++kb) {
                ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.full[stage], phase, p.wait_ns);
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    if (lane == 0) record_timeout(sm, p.status);
                    aborted = true;
                    break;
                }
                tc_fence_after_sync();
                if (lane == 0) {
                    const uint32_t sfa_col = kSfBase + ((kb / kStagesPerGroup) & 1) * kSfColsPerSet;
                    const uint32_t sfb_col = sfa_col + 4;
                    uint32_t idesc = p.idesc;
                    if constexpr (kMX) {
                        if (kb % kStagesPerGroup == 0) {  // new group of four k-blocks: its scale vectors
                            tmem_cp_32x128b_warpx4(tmem + sfa_col, smem_desc_plain_16B_rows(smem_u32(sm.sf_a[stage])));
                            tmem_cp_32x128b_warpx4(tmem + sfb_col, smem_desc_plain_16B_rows(smem_u32(sm.sf_b[stage])));
                            tmem_cp_32x128b_warpx4(tmem + sfb_col + 4,
                                                   smem_desc_plain_16B_rows(smem_u32(sm.sf_b[stage] + 512)));
                        }
                        const uint32_t sf_id = static_cast<uint32_t>((kb / kStagesPerKBlock) & 3);
                        idesc |= (sf_id << 29) | (sf_id << 4);
                    }
                    const uint32_t a_addr = smem_u32(sm.a[stage]);
                    const uint32_t b_addr = smem_u32(sm.b[stage]);
#pragma unroll
                    for (int k = 0; k < kKSteps; ++k) {
                        const uint64_t ad = smem_desc_k_swizzled<kBKBytes>(a_addr + 32 * k);
                        const uint64_t bd = smem_desc_k_swizzled<kBKBytes>(b_addr + 32 * k);
                        const uint32_t acc = (kb > wu.kb0 || k > 0) ? 1u : 0u;
                        if constexpr (KIND == kGemmBF16)
                            mma_f16(d_tmem, ad, bd, idesc, acc);
                        else if constexpr (KIND == kGemmFP8Tensor)
                            mma_f8(d_tmem, ad, bd, idesc, acc);
                        else
                            mma_mxf8(d_tmem, ad, bd, idesc, tmem + sfa_col, tmem + sfb_col, acc);
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
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue
        const int q = warp & 3;  // TMEM lane quarter of this warp
        float sab = 1.0f;
        if constexpr (KIND == kGemmFP8Tensor) sab = __fmul_rn(*p.sia, *p.sib);
        uint8_t *stage_buf = sm.epi[q];
        int local = 0;
        for (int u = blockIdx.x; u < p.num_units; u += gridDim.x, ++local) {
            const WorkUnit wu = work_unit(p, u);
            const int m0 = wu.m0, n0 = wu.n0;
            const int buf = local % kAccBufs;
            const uint32_t acc_phase = static_cast<uint32_t>(local / kAccBufs) & 1u;
            bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tfull[buf], acc_phase, p.wait_ns);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                if (lane == 0) record_timeout(sm, p.status);
                break;
            }
            tc_fence_after_sync();
            const uint32_t t_row = tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>(buf * kBN);
            if constexpr (OUT_F32) {
                // FP32 partial tile: 8 chunks of 32 columns (128 bytes per row)
                const int row0 = wu.split * p.num_m * kBM + m0 + 32 * q;  // chunks 128-row aligned
#pragma unroll
                for (int h = 0; h < kBN / 128; ++h) {
                    uint32_t r[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(t_row + 128 * h + 32 * c, r[c]);
                    tmem_ld_wait();
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int col = n0 + 128 * h + 32 * c;
                        if (col >= p.N) break;
                        if (lane == 0) bulk_wait_group_read0();
                        __syncwarp();
                        uint8_t *row = stage_buf + 128 * lane;
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            uint4 v = make_uint4(r[c][4 * i], r[c][4 * i + 1], r[c][4 * i + 2], r[c][4 * i + 3]);
                            if constexpr (KIND == kGemmFP8Tensor) {
                                v.x = __float_as_uint(__fmul_rn(__uint_as_float(v.x), sab));
                                v.y = __float_as_uint(__fmul_rn(__uint_as_float(v.y), sab));
                                v.z = __float_as_uint(__fmul_rn(__uint_as_float(v.z), sab));
                                v.w = __float_as_uint(__fmul_rn(__uint_as_float(v.w), sab));
                            }
                            *reinterpret_cast<uint4 *>(row + 16 * (i ^ (lane & 7))) = v;
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tm_d, stage_buf, col, row0);
                            bulk_commit_group();
                        }
                    }
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive(&sm.tempty[buf]);
            } else {
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

// Split-K reduction: out[i] = bf16(sum_s ws[s][i]) in fixed order s = 0, 1, ...
// (chunk s starts split_stride4 float4s after chunk s-1).
__global__ void __launch_bounds__(256) splitk_reduce_kernel(const float4 *__restrict__ ws, int splits, int64_t n4,
                                                            int64_t split_stride4, uint2 *__restrict__ out) {
    const int64_t stride = static_cast<int64_t>(gridDim.x) * blockDim.x;
    for (int64_t i = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; i < n4; i += stride) {
        float4 a = ws[i];
        for (int sp = 1; sp < splits; ++sp) {
            const float4 b = ws[sp * split_stride4 + i];
            a.x += b.x;
            a.y += b.y;
            a.z += b.z;
            a.w += b.w;
        }
        __nv_bfloat162 lo = __floats2bfloat162_rn(a.x, a.y), hi = __floats2bfloat162_rn(a.z, a.w);
        out[i] = make_uint2(*reinterpret_cast<uint32_t *>(&lo), *reinterpret_cast<uint32_t *>(&hi));
    }
}

int choose_splits(int64_t M, int64_t N, int64_t K, bool bf16) {
    if (bf16) return 1;
    const int64_t tiles = ((M + kBM - 1) / kBM) * ((N + kBN - 1) / kBN);
    const int64_t kblocks = (K + 127) / 128;  // 128-byte k-blocks (independent of the stage size)
    if (tiles >= kSplitRefSms) return 1;
    // Modelled time = waves x k-blocks per chunk; chunks keep >= 16 k-blocks
    // (whole groups of four).  Split only for a >= 15% modelled gain.
    auto cost = [&](int64_t sp) {
        const int64_t chunk = ((kblocks + sp - 1) / sp + 3) / 4 * 4;
        const int64_t chunks = (kblocks + chunk - 1) / chunk;
        return ((tiles * chunks + kSplitRefSms - 1) / kSplitRefSms) * chunk;
    };
    const int64_t base = cost(1);
    int best = 1;
    int64_t best_cost = base;
    for (int sp = 2; sp <= 8; ++sp) {
        if (kblocks / sp < 16) break;
        const int64_t c = cost(sp);
        if (c < best_cost) {
            best = sp;
            best_cost = c;
        }
    }
    return (best_cost * 100 <= base * 85) ? best : 1;
}

size_t splitk_workspace_bytes(int64_t M, int64_t N, int64_t K, bool bf16) {
    const int sp = choose_splits(M, N, K, bf16);
    const int64_t m_pad = (M + kBM - 1) / kBM * kBM;
    return sp > 1 ? static_cast<size_t>(sp) * static_cast<size_t>(m_pad) * static_cast<size_t>(N) * sizeof(float) : 0;
}

template <int KIND, bool OUT_F32>
static cudaError_t launch_kind(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                               const CUtensorMap &tm_d, int splits, cudaStream_t s) {
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;
    GemmParams p{};
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.K = static_cast<int>(g.K);
    p.num_m = static_cast<int>((g.M + kBM - 1) / kBM);
    p.num_n = static_cast<int>((g.N + kBN - 1) / kBN);
    p.num_kb = static_cast<int>((g.K + kBK - 1) / kBK);
    p.num_tiles = p.num_m * p.num_n;
    p.splits = splits;
    p.kb_per_split = ((p.num_kb + splits - 1) / splits + kStagesPerGroup - 1) / kStagesPerGroup * kStagesPerGroup;
    p.splits = (p.num_kb + p.kb_per_split - 1) / p.kb_per_split;  // no empty chunk
    p.num_units = p.num_tiles * p.splits;
    p.m_fastest = g.M < g.N ? 1 : 0;  // re-read the smaller operand, stream the larger once
    if (KIND == kGemmBF16)
        p.idesc = idesc_dense(1u, 1u);
    else if (KIND == kGemmFP8Tensor)
        p.idesc = idesc_dense(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt));
    else
        p.idesc = idesc_mx(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt));
    p.sfa = g.sfa;
    p.sfb = g.sfb;
    p.kgroups = static_cast<int>((g.K / 128 + 3) / 4);
    p.sia = g.sia;
    p.sib = g.sib;
    p.status = g.status;
    p.wait_ns = g.wait_timeout_ns;

    auto kern = gemm_tn_kernel<KIND, OUT_F32>;
    const size_t smem = sizeof(GemmSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int grid = p.num_units < g.num_sms ? p.num_units : g.num_sms;
    kern<<<grid, kThreads, smem, s>>>(tm_a, tm_b, tm_d, p);
    return cudaGetLastError();
}

template <int KIND>
static cudaError_t launch_split_or_not(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                                       const CUtensorMap &tm_d, const CUtensorMap &tm_ws, cudaStream_t s) {
    if (g.splits <= 1) return launch_kind<KIND, false>(g, tm_a, tm_b, tm_d, 1, s);
    cudaError_t e = launch_kind<KIND, true>(g, tm_a, tm_b, tm_ws, g.splits, s);
    if (e != cudaSuccess) return e;
    const int64_t n4 = g.M * g.N / 4;
    const int64_t stride4 = (g.M + kBM - 1) / kBM * kBM * g.N / 4;
    int64_t want = (n4 + 255) / 256;
    const int64_t cap = static_cast<int64_t>(g.num_sms) * 8;
    const int grid = static_cast<int>(want < cap ? want : cap);
    splitk_reduce_kernel<<<grid, 256, 0, s>>>(reinterpret_cast<const float4 *>(g.workspace), g.splits, n4, stride4,
                                              reinterpret_cast<uint2 *>(g.out));
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                        const CUtensorMap &tm_d, const CUtensorMap &tm_ws, cudaStream_t s) {
    switch (g.kind) {
        case kGemmBF16: return launch_kind<kGemmBF16, false>(g, tm_a, tm_b, tm_d, 1, s);
        case kGemmFP8Tensor: return launch_split_or_not<kGemmFP8Tensor>(g, tm_a, tm_b, tm_d, tm_ws, s);
        default: return launch_split_or_not<kGemmFP8Block>(g, tm_a, tm_b, tm_d, tm_ws, s);
    }
}

}  // namespace puro
