// gemm.cu -- tcgen05 tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T (both
// operands K-major, "TN") with FP32 accumulation in tensor memory and a BF16
// output, for the three GEMMs of an FP8 linear layer (Puro-2B, appendix
// "Production Training Details", paragraph "FP8 implementation pipeline":
// Fprop, Dgrad and Wgrad all from E4M3 operands, BF16 output).
//
// Persistent, warp-specialised CTA pairs: each 2-CTA cluster (one pair of
// SMs) computes 256x256 output tiles with pair MMAs (tcgen05 cta_group::2,
// M = 256): CTA r of the pair holds rows 128r..128r+127 of the A tile and
// rows 128r..128r+127 of the B tile in its shared memory, and receives its
// 128 rows x 256 columns of D in its own tensor memory.  Per SM this halves
// the B bytes moved and read per MMA against a one-SM 128x256 tile, which is
// what bounds the one-SM form's tensor-pipe utilisation.
//   warp 0      TMA producer (both CTAs): A/B tiles (128-byte swizzle) and,
//               for the block-scaled kind, the E8M0 scale vectors (already
//               in the tensor-core layout: 512 bytes per 128 rows and four
//               k-blocks; the CTA's own 128 rows of A, all 256 rows of B)
//               into a 3-deep ring of 256-byte K stages (two k-blocks, two
//               swizzle atoms each).  Both CTAs' copies of a stage count on
//               the even CTA's `full` barrier.  Stages of two k-blocks (eight
//               MMAs per stage hand-off) rather than one keep the tensor pipe
//               busy across the per-stage barrier round trip.
//   warp 1      even CTA: MMA issuer -- copies scale vectors into tensor
//               memory (tcgen05.cp, once per four k-blocks), issues the pair
//               MMAs (kind::f16 / kind::f8f6f4 / kind::mxf8f6f4.block_scale,
//               the scale id picking the k-block's byte), and releases each
//               stage to both CTAs' producers and each accumulator to both
//               CTAs' epilogues with multicast commits.  Both CTAs: tensor
//               memory allocation (collective over the pair).
//   warps 4..7  epilogue (both CTAs): tcgen05.ld the CTA's 128x256 FP32
//               accumulator (one 32-lane quarter per warp) in two 128-column
//               halves, release it to the even CTA's MMA warp, convert to
//               BF16 (times scale_inv_a * scale_inv_b for the per-tensor
//               kind) and TMA-store it through a swizzled staging tile.
// Accumulators in tensor memory (512 columns):
//   dense kinds  two 256-column buffers, tiles alternate between them;
//   block kind   the scale vectors need 24 columns, so two whole buffers do
//               not fit: tiles alternate between columns [0, 256) and
//               [128, 384), sharing [128, 256).  The epilogue reads the
//               shared half first and releases the accumulator as soon as
//               that half is in registers, so the next tile's MMAs wait for
//               one half of the drain instead of all of it.
// Every mbarrier wait is bounded in wall time; on expiry the CTA records
// PURO_ERR_TIMEOUT in the caller's status word, drains its own in-flight
// copies and MMAs (with a fixed bound), and both CTAs meet at a cluster
// barrier before tensor memory is freed.
#include <cuda_bf16.h>

#include "internal.h"
#include "ptx.cuh"

namespace puro {

constexpr int kBM = kGemmBM;       // rows of A per CTA (= TMEM lanes); a pair tile has 2 * kBM rows
constexpr int kPairM = 2 * kBM;    // rows of A per pair tile
constexpr int kBN = kGemmBN;       // columns of a tile (= accumulator columns)
constexpr int kBNHalf = kBN / 2;   // rows of B per CTA
constexpr int kAtomBytes = kGemmBKBytes;       // one 128-byte swizzle row of K: one k-block of FP8
constexpr int kAtoms = 2;                      // k-blocks per pipeline stage
constexpr int kBKBytes = kAtoms * kAtomBytes;  // bytes of K per pipeline stage
constexpr int kStages = 3;                     // 3 x 64 KB operand ring
constexpr int kStagesPerGroup = 512 / kBKBytes;  // stages per group of four k-blocks (one scale chunk)
constexpr int kThreads = 256;
constexpr int kTmemCols = 512;
constexpr int kSfColsPerSet = 12;  // 4 for A (128 rows) + 8 for B (256 rows)
constexpr int kSfSets = 2;         // double-buffered across groups of four k-blocks
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;
constexpr uint64_t kSettleNs = 200000ull;  // after an abort: let the peer-counted copies land
constexpr int32_t kStatusTimeout = 4;  // PURO_ERR_TIMEOUT
constexpr int64_t kSplitRefPairs = 76;  // SM pairs the split heuristic plans for (GB300: 152 SMs)
static_assert(kAtomBytes == 128 && kStagesPerGroup * kBKBytes == 512, "whole k-blocks per stage, whole stages per group");

struct GemmSmem {
    alignas(1024) uint8_t a[kStages][kAtoms][kBM * kAtomBytes];
    alignas(1024) uint8_t b[kStages][kAtoms][kBNHalf * kAtomBytes];
    alignas(1024) uint8_t epi[4][32 * 128];    // per epilogue warp: 32 rows x 64 bf16
    alignas(128) uint8_t sf_a[kStages][512];   // scale vectors of this CTA's 128 rows of A
    alignas(128) uint8_t sf_b[kStages][1024];  // scale vectors of the tile's 256 rows of B
    uint64_t full[kStages];   // even CTA: both CTAs' copies of a stage landed
    uint64_t empty[kStages];  // both CTAs: the pair MMAs reading a stage are done
    uint64_t tfull[2];        // both CTAs: accumulator complete
    uint64_t tempty[2];       // even CTA: both CTAs' epilogues released the accumulator
    uint64_t drain;
    uint32_t tmem_base;
    volatile int abort_flag;
};

struct GemmParams {
    int M, N, K;
    int num_m, num_n, num_kb, num_tiles;  // num_m counts 256-row pair tiles
    int splits;        // reduction split into this many chunks (1: no split)
    int kb_per_split;  // stages per chunk (a whole number of scale groups)
    int num_units;     // num_tiles * splits
    int m_fastest;     // tile order: 1 = row blocks of A vary fastest
    int kgroups;       // ceil(K / 512): scale-vector chunks per 128 rows
    uint32_t idesc;
    const float *sia;
    const float *sib;
    int32_t *status;
    uint64_t wait_ns;
};

// Instruction descriptors (tcgen05.mma), both operands K-major, M = 256
// (a pair MMA), N = kBN.
//   kind::f16 / kind::f8f6f4: [4,6) D format (1 = F32), [7,10) A type,
//     [10,13) B type, [17,23) N >> 3, [24,29) M >> 4.
//   kind::mxf8f6f4: [4,6) B scale id, [7,10) A type, [10,13) B type,
//     [17,23) N >> 3, [23] scale type (1 = UE8M0), [24,29) M >> 4,
//     [29,31) A scale id.  The scale id selects the byte of the 32-bit
//     tensor-memory scale word: here the k-block within its group of four.
__host__ __device__ constexpr uint32_t idesc_dense(uint32_t atype, uint32_t btype) {
    return (1u << 4) | (atype << 7) | (btype << 10) | (static_cast<uint32_t>(kBN >> 3) << 17) |
           (static_cast<uint32_t>(kPairM >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_mx(uint32_t atype, uint32_t btype) {
    return (atype << 7) | (btype << 10) | (static_cast<uint32_t>(kBN >> 3) << 17) | (1u << 23) |
           (static_cast<uint32_t>(kPairM >> 4) << 24);
}

PURO_DEV void record_timeout(GemmSmem &sm, int32_t *status) {
    sm.abort_flag = 1;
    if (status) atomicExch(status, kStatusTimeout);
}

// One unit of work: a 256x256 pair tile and a chunk of the reduction.  Units
// of the same chunk are consecutive; within a chunk the tile order iterates
// the blocks of the smaller operand fastest, so the pairs of a wave share
// (and read once) the blocks of the larger one.
struct WorkUnit {
    int m0, n0, kb0, kb1, split;  // m0: first row of the pair tile
};

PURO_DEV WorkUnit work_unit(const GemmParams &p, int u) {
    WorkUnit w;
    w.split = u / p.num_tiles;
    const int tile = u - w.split * p.num_tiles;
    const int mb = p.m_fastest ? tile % p.num_m : tile / p.num_n;
    const int nb = p.m_fastest ? tile / p.num_m : tile % p.num_n;
    w.m0 = mb * kPairM;
    w.n0 = nb * kBN;
    w.kb0 = w.split * p.kb_per_split;
    w.kb1 = min(p.num_kb, w.kb0 + p.kb_per_split);
    return w;
}

// OUT_F32: write FP32 partial tiles of a split reduction to the workspace
// [splits * Mp, N], Mp = num_m * 256 (rows split * Mp + m), instead of the
// BF16 output; a ragged last pair tile then stays inside its chunk.
// tm_sfa / tm_sfb (block kind only): the scale vectors of A / B viewed as
// uint32 [chunks, 128] (one 512-byte chunk per row), box {128, 1}.
template <int KIND, bool OUT_F32>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(kThreads, 1)
    gemm_tn_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                   const __grid_constant__ CUtensorMap tm_d, const __grid_constant__ CUtensorMap tm_sfa,
                   const __grid_constant__ CUtensorMap tm_sfb, const GemmParams p) {
    constexpr bool kMX = (KIND == kGemmFP8Block);
    constexpr int kAccBufs = kMX ? 1 : 2;              // hand-off barrier pairs (tfull / tempty)
    constexpr int kAccShift = kMX ? kBN / 2 : kBN;     // column offset between consecutive tiles' accumulators
    constexpr int kSfBase = kBN + kAccShift;           // first scale-vector column (MX)
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;         // elements of K per stage
    constexpr int kAtomK = kAtomBytes / kElemBytes;    // elements of K per 128-byte atom
    constexpr int kKSteps = kAtomBytes / 32;           // MMAs per atom (32 bytes of K each)
    constexpr uint32_t kStageBytes = (kBM + kBNHalf) * kBKBytes;  // one CTA's operand bytes per stage
    constexpr uint32_t kSfBytes = 512 + 1024;                     // one CTA's scale-vector bytes per group
    static_assert(!kMX || kSfBase + kSfSets * kSfColsPerSet <= kTmemCols, "TMEM budget");

    extern __shared__ uint8_t smem_raw[];
    GemmSmem &sm = *reinterpret_cast<GemmSmem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                                 ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();  // 0: even CTA (issues the MMAs), 1: its peer
    const int pair = blockIdx.x >> 1;
    const int num_pairs = gridDim.x >> 1;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int b = 0; b < 2; ++b) {
            mbar_init(&sm.tfull[b], 1);
            mbar_init(&sm.tempty[b], 8);  // four epilogue warps in each CTA
        }
        mbar_init(&sm.drain, 1);
        sm.abort_flag = 0;
        fence_mbarrier_init();
        tma_prefetch_desc(&tm_a);
        tma_prefetch_desc(&tm_b);
        tma_prefetch_desc(&tm_d);
        if (kMX) {
            tma_prefetch_desc(&tm_sfa);
            tma_prefetch_desc(&tm_sfb);
        }
    }
    if (warp == 1) {
        tmem_alloc_pair(&sm.tmem_base, kTmemCols);
        tmem_relinquish_alloc_permit_pair();
    }
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers exist before any copy or arrival targets them
    tc_fence_after_sync();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t full0 = mapa_shared(smem_u32(&sm.full[0]), 0);  // the even CTA's ring
            uint32_t stage = 0, phase = 0;
            uint32_t issued = 0;  // stage fills started by this thread
            bool aborted = false;
            for (int u = pair; u < p.num_units && !aborted; u += num_pairs) {
                const WorkUnit wu = work_unit(p, u);
                const int a_row = wu.m0 + kBM * static_cast<int>(rank);
                const int b_row = wu.n0 + kBNHalf * static_cast<int>(rank);
                for (int kb = wu.kb0; kb < wu.kb1; ++kb) {
                    if (sm.abort_flag || !mbar_wait_bounded(&sm.empty[stage], phase ^ 1u, p.wait_ns)) {
                        record_timeout(sm, p.status);
                        aborted = true;
                        break;
                    }
                    const bool sf_load = kMX && (kb % kStagesPerGroup) == 0;
                    const uint32_t full_bar = full0 + 8u * stage;
                    if (rank == 0)
                        mbar_arrive_expect_tx(&sm.full[stage], 2u * (kStageBytes + (sf_load ? kSfBytes : 0u)));
#pragma unroll
                    for (int at = 0; at < kAtoms; ++at) {
                        tma_load_2d_pair(sm.a[stage][at], &tm_a, full_bar, kb * kBK + at * kAtomK, a_row);
                        tma_load_2d_pair(sm.b[stage][at], &tm_b, full_bar, kb * kBK + at * kAtomK, b_row);
                    }
                    if (sf_load) {
                        // chunks beyond the operand's rows read as zero (their rows are zero too)
                        const int kg = kb / kStagesPerGroup;
                        tma_load_2d_pair(sm.sf_a[stage], &tm_sfa, full_bar, 0, (a_row / 128) * p.kgroups + kg);
                        tma_load_2d_pair(sm.sf_b[stage], &tm_sfb, full_bar, 0, (wu.n0 / 128) * p.kgroups + kg);
                        tma_load_2d_pair(sm.sf_b[stage] + 512, &tm_sfb, full_bar, 0,
                                         (wu.n0 / 128 + 1) * p.kgroups + kg);
                    }
                    ++issued;
                    if (++stage == kStages) {
                        stage = 0;
                        phase ^= 1u;
                    }
                }
            }
            if (rank == 0) {
                // Every fill of the ring (both CTAs' copies) lands before the
                // pair exits: wait for the latest fill of each stage.
                for (uint32_t s = 0; s < kStages; ++s) {
                    const uint32_t fills = issued / kStages + (s < issued % kStages ? 1u : 0u);
                    if (fills > 0) mbar_wait_bounded(&sm.full[s], (fills - 1u) & 1u, kDrainTimeoutNs);
                }
            }
            if (aborted) {
                // This CTA's copies count on the even CTA's barriers, so it
                // cannot wait for them itself: give any still in flight a
                // fixed time to land.
                const uint64_t t0 = global_timer_ns();
                while (global_timer_ns() - t0 < kSettleNs) {
                }
            }
        }
    } else if (warp == 1 && rank == 0) {
        // ------------------------------------------------ MMA issuer (even CTA)
        uint32_t stage = 0, phase = 0;
        bool aborted = false;
        int local = 0;
        for (int u = pair; u < p.num_units && !aborted; u += num_pairs, ++local) {
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
            const uint32_t d_tmem = tmem + static_cast<uint32_t>((local & 1) * kAccShift);

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
                    if constexpr (kMX) {
                        if (kb % kStagesPerGroup == 0) {  // new group of four k-blocks: its scale vectors
                            tmem_cp_pair_32x128b_warpx4(tmem + sfa_col,
                                                        smem_desc_plain_16B_rows(smem_u32(sm.sf_a[stage])));
                            tmem_cp_pair_32x128b_warpx4(tmem + sfb_col,
                                                        smem_desc_plain_16B_rows(smem_u32(sm.sf_b[stage])));
                            tmem_cp_pair_32x128b_warpx4(tmem + sfb_col + 4,
                                                        smem_desc_plain_16B_rows(smem_u32(sm.sf_b[stage] + 512)));
                        }
                    }
#pragma unroll
                    for (int at = 0; at < kAtoms; ++at) {
                        uint32_t idesc = p.idesc;
                        if constexpr (kMX) {
                            const uint32_t sf_id = static_cast<uint32_t>((kb * kAtoms + at) & 3);  // k-block in its group
                            idesc |= (sf_id << 29) | (sf_id << 4);
                        }
                        const uint32_t a_addr = smem_u32(sm.a[stage][at]);
                        const uint32_t b_addr = smem_u32(sm.b[stage][at]);
#pragma unroll
                        for (int k = 0; k < kKSteps; ++k) {
                            const uint64_t ad = smem_desc_k_sw128(a_addr + 32 * k);
                            const uint64_t bd = smem_desc_k_sw128(b_addr + 32 * k);
                            const uint32_t acc = (kb > wu.kb0 || at > 0 || k > 0) ? 1u : 0u;
                            if constexpr (KIND == kGemmBF16)
                                mma_pair_f16(d_tmem, ad, bd, idesc, acc);
                            else if constexpr (KIND == kGemmFP8Tensor)
                                mma_pair_f8(d_tmem, ad, bd, idesc, acc);
                            else
                                mma_pair_mxf8(d_tmem, ad, bd, idesc, tmem + sfa_col, tmem + sfb_col, acc);
                        }
                    }
                    tc_commit_pair_multicast(&sm.empty[stage], 0x3);  // stage reusable in both CTAs
                }
                __syncwarp();
                if (++stage == kStages) {
                    stage = 0;
                    phase ^= 1u;
                }
            }
            if (aborted) break;
            if (lane == 0) tc_commit_pair_multicast(&sm.tfull[buf], 0x3);  // accumulator complete in both CTAs
            __syncwarp();
        }
        // All MMAs and copies issued by this warp complete before teardown.
        if (lane == 0) {
            tc_commit_pair(&sm.drain);
            mbar_wait_bounded(&sm.drain, 0, kDrainTimeoutNs);
        }
        __syncwarp();
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue (both CTAs)
        const int q = warp & 3;  // TMEM lane quarter of this warp
        float sab = 1.0f;
        if constexpr (KIND == kGemmFP8Tensor) sab = __fmul_rn(*p.sia, *p.sib);
        uint8_t *stage_buf = sm.epi[q];
        const uint32_t tempty0 = mapa_shared(smem_u32(&sm.tempty[0]), 0);  // the even CTA's
        int local = 0;
        for (int u = pair; u < p.num_units; u += num_pairs, ++local) {
            const WorkUnit wu = work_unit(p, u);
            const int m0 = wu.m0 + kBM * static_cast<int>(rank), n0 = wu.n0;  // this CTA's rows
            const int buf = local % kAccBufs;
            const uint32_t acc_phase = static_cast<uint32_t>(local / kAccBufs) & 1u;
            bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tfull[buf], acc_phase, p.wait_ns);
            if (!__all_sync(0xFFFFFFFFu, ok)) {
                if (lane == 0) record_timeout(sm, p.status);
                break;
            }
            tc_fence_after_sync();
            const uint32_t t_row =
                tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>((local & 1) * kAccShift);
            if constexpr (OUT_F32) {
                // FP32 partial tile: 8 chunks of 32 columns (128 bytes per row)
                const int row0 = wu.split * p.num_m * kPairM + m0 + 32 * q;  // chunks pair-tile aligned
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
                if (lane == 0) mbar_arrive_cluster(tempty0 + 8u * buf);
            } else {
                // Block kind: the half in the columns the next tile's
                // accumulator shares ([128, 256) of tensor memory) first, and
                // the accumulator released once it is in registers.  Dense
                // kinds: halves in order, released after the second load.
                const int h_first = kMX ? ((local & 1) ? 0 : 1) : 0;
#pragma unroll 1
                for (int hh = 0; hh < 2; ++hh) {
                    const int h = hh ^ h_first;
                    uint32_t r[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(t_row + 128 * h + 32 * c, r[c]);
                    tmem_ld_wait();
                    if (hh == (kMX ? 0 : 1)) {
                        tc_fence_before_sync();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_cluster(tempty0 + 8u * buf);  // accumulator free for the next tile
                    }
                    // Two chunks of 64 columns (128 bytes per row) through the
                    // per-warp staging tile, 16-byte unit i of row l at i ^ (l % 8).
#pragma unroll
                    for (int ch = 0; ch < 2; ++ch) {
                        const int col = n0 + 128 * h + 64 * ch;
                        if (col >= p.N) break;
                        if (lane == 0) bulk_wait_group_read0();
                        __syncwarp();
                        uint8_t *row = stage_buf + 128 * lane;
#pragma unroll
                        for (int i = 0; i < 8; ++i) {
                            const uint32_t *src = &r[2 * ch + (i >> 2)][8 * (i & 3)];
                            uint32_t w[4];
#pragma unroll
                            for (int j = 0; j < 4; ++j) {
                                float lo = __uint_as_float(src[2 * j]), hi = __uint_as_float(src[2 * j + 1]);
                                if constexpr (KIND == kGemmFP8Tensor) {
                                    lo = __fmul_rn(lo, sab);
                                    hi = __fmul_rn(hi, sab);
                                }
                                __nv_bfloat162 v = __floats2bfloat162_rn(lo, hi);
                                w[j] = *reinterpret_cast<uint32_t *>(&v);
                            }
                            *reinterpret_cast<uint4 *>(row + 16 * (i ^ (lane & 7))) = make_uint4(w[0], w[1], w[2], w[3]);
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(&tm_d, stage_buf, col, m0 + 32 * q);
                            bulk_commit_group();
                        }
                    }
                }
            }
        }
        if (lane == 0) bulk_wait_group0();
        __syncwarp();
    }

    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // the pair's MMAs into both CTAs' tensor memory are complete
    tc_fence_after_sync();
    if (warp == 1) tmem_dealloc_pair(tmem, kTmemCols);
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
    const int64_t tiles = ((M + kPairM - 1) / kPairM) * ((N + kBN - 1) / kBN);
    const int64_t kblocks = (K + 127) / 128;  // 128-byte k-blocks
    if (tiles >= kSplitRefPairs) return 1;
    // Modelled time = waves x k-blocks per chunk; chunks keep >= 16 k-blocks
    // (whole groups of four).  Split only for a >= 15% modelled gain.
    auto cost = [&](int64_t sp) {
        const int64_t chunk = ((kblocks + sp - 1) / sp + 3) / 4 * 4;
        const int64_t chunks = (kblocks + chunk - 1) / chunk;
        return ((tiles * chunks + kSplitRefPairs - 1) / kSplitRefPairs) * chunk;
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

int64_t splitk_rows_per_chunk(int64_t M) { return (M + kPairM - 1) / kPairM * kPairM; }

size_t splitk_workspace_bytes(int64_t M, int64_t N, int64_t K, bool bf16) {
    const int sp = choose_splits(M, N, K, bf16);
    return sp > 1 ? static_cast<size_t>(sp) * static_cast<size_t>(splitk_rows_per_chunk(M)) * static_cast<size_t>(N) *
                        sizeof(float)
                  : 0;
}

// Pairs that can be resident at once for this kernel (the persistent grid
// size), cached per device and kernel.
template <int KIND, bool OUT_F32>
static int max_resident_pairs(int num_sms, size_t smem) {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return num_sms / 2;
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(num_sms / 2 * 2), 1, 1);
    cfg.blockDim = dim3(kThreads, 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tn_kernel<KIND, OUT_F32>, &cfg) != cudaSuccess || n <= 0) {
        (void)cudaGetLastError();
        n = num_sms / 2;
    }
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

template <int KIND, bool OUT_F32>
static cudaError_t launch_kind(const GemmArgs &g, const GemmMaps &m, int splits, cudaStream_t s) {
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;
    GemmParams p{};
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.K = static_cast<int>(g.K);
    p.num_m = static_cast<int>((g.M + kPairM - 1) / kPairM);
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
    p.kgroups = static_cast<int>((g.K / 128 + 3) / 4);
    p.sia = g.sia;
    p.sib = g.sib;
    p.status = g.status;
    p.wait_ns = g.wait_timeout_ns;

    auto kern = gemm_tn_kernel<KIND, OUT_F32>;
    const size_t smem = sizeof(GemmSmem) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int pairs_max = max_resident_pairs<KIND, OUT_F32>(g.num_sms, smem);
    const int pairs = p.num_units < pairs_max ? p.num_units : pairs_max;
    kern<<<2 * pairs, kThreads, smem, s>>>(m.a, m.b, OUT_F32 ? m.ws : m.d, m.sfa, m.sfb, p);
    return cudaGetLastError();
}

template <int KIND>
static cudaError_t launch_split_or_not(const GemmArgs &g, const GemmMaps &m, cudaStream_t s) {
    if (g.splits <= 1) return launch_kind<KIND, false>(g, m, 1, s);
    cudaError_t e = launch_kind<KIND, true>(g, m, g.splits, s);
    if (e != cudaSuccess) return e;
    const int64_t n4 = g.M * g.N / 4;
    const int64_t stride4 = splitk_rows_per_chunk(g.M) * g.N / 4;
    int64_t want = (n4 + 255) / 256;
    const int64_t cap = static_cast<int64_t>(g.num_sms) * 8;
    const int grid = static_cast<int>(want < cap ? want : cap);
    splitk_reduce_kernel<<<grid, 256, 0, s>>>(reinterpret_cast<const float4 *>(g.workspace), g.splits, n4, stride4,
                                              reinterpret_cast<uint2 *>(g.out));
    return cudaGetLastError();
}

cudaError_t launch_gemm(const GemmArgs &g, const GemmMaps &m, cudaStream_t s) {
    switch (g.kind) {
        case kGemmBF16: return launch_kind<kGemmBF16, false>(g, m, 1, s);
        case kGemmFP8Tensor: return launch_split_or_not<kGemmFP8Tensor>(g, m, s);
        default: return launch_split_or_not<kGemmFP8Block>(g, m, s);
    }
}

}  // namespace puro
