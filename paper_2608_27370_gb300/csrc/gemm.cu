// gemm.cu -- tcgen05 tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T (both
// operands K-major, "TN") with FP32 accumulation in tensor memory and a BF16
// output, for the three GEMMs of an FP8 linear layer (Puro-2B, appendix
// "Production Training Details", paragraph "FP8 implementation pipeline":
// Fprop, Dgrad and Wgrad all from E4M3 operands, BF16 output).
//
// Persistent, warp-specialised CTA pairs: each 2-CTA cluster (one pair of
// SMs) computes 256 x BN output tiles with pair MMAs (tcgen05 cta_group::2,
// M = 256, N = BN): CTA r of the pair holds rows 128r..128r+127 of the A
// tile and rows (BN/2)r..(BN/2)r+BN/2-1 of the B tile in its shared memory,
// and receives its 128 rows x BN columns of D in its own tensor memory.  Per
// SM this halves the B bytes moved and read per MMA against a one-SM tile.
//   warp 0      TMA producer (both CTAs): A/B tiles (128-byte swizzle) into
//               a 3-deep ring of 256-byte K stages (two k-blocks, two swizzle
//               atoms each), and the E8M0 scale vectors of the CTA's 128 rows
//               of A (already in the tensor-core layout: 512 bytes per 128
//               rows and four k-blocks); with BN = 256 also those of the
//               tile's 256 rows of B.  Both CTAs' copies of a stage count on
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
//   warp 2      BN = 224 only (both CTAs): builds the tensor-core image of
//               the B scale vectors for tiles that start at any 32-row
//               offset, which no TMA box can gather (see below).
//   warps 4..7  epilogue (both CTAs): tcgen05.ld the CTA's 128 x BN FP32
//               accumulator (one 32-lane quarter per warp), release it to
//               the even CTA's MMA warp, convert to BF16 (times scale_inv_a *
//               scale_inv_b for the per-tensor kind) and TMA-store it through
//               a swizzled staging tile.
// Accumulators in tensor memory (512 columns):
//   dense kinds       two 256-column buffers, tiles alternate between them;
//   block, BN = 256   the scale vectors need 24 columns, so two whole
//                     buffers do not fit: tiles alternate between columns
//                     [0, 256) and [128, 384), sharing [128, 256).  The
//                     epilogue reads the shared half first and releases the
//                     accumulator as soon as that half is in registers, so
//                     the next tile's MMAs wait for half a drain.
//   block, BN = 224   two independent buffers at columns 0 and 256 (scale
//                     vectors at 480): the next tile never waits for a drain.
//                     The host picks this form where the per-tile hand-off
//                     of the 256 form would cost more than its narrower MMAs.
// Every mbarrier wait is bounded in wall time; on expiry the CTA records
// PURO_ERR_TIMEOUT in the caller's status word, drains its own in-flight
// copies and MMAs (with a fixed bound), and both CTAs meet at a cluster
// barrier before tensor memory is freed.
#include <cuda_bf16.h>

#include <algorithm>
#include <type_traits>

#include "internal.h"
#include "ptx.cuh"
#include "quant_math.cuh"

namespace puro {

constexpr int kBM = kGemmBM;       // rows of A per CTA (= TMEM lanes); a pair tile has 2 * kBM rows
constexpr int kPairM = 2 * kBM;    // rows of A per pair tile
constexpr int kAtomBytes = kGemmBKBytes;       // one 128-byte swizzle row of K: one k-block of FP8
constexpr int kAtoms = 2;                      // k-blocks per pipeline stage
constexpr int kBKBytes = kAtoms * kAtomBytes;  // bytes of K per pipeline stage
constexpr int kStages = 3;                     // 3-deep operand ring (64 KB / 60 KB per stage)
constexpr int kStagesPerGroup = 512 / kBKBytes;  // stages per group of four k-blocks (one scale chunk)
constexpr int kThreads = 256;
constexpr int kTmemCols = 512;
constexpr int kSfColsPerSet = 12;  // 4 for A (128 rows) + 8 for B (up to 256 rows)
constexpr int kSfSets = 2;         // double-buffered across groups of four k-blocks
constexpr int kSfbSlots = 4;       // BN = 224: ring of helper-built B scale images
constexpr uint64_t kDrainTimeoutNs = 2000000000ull;
constexpr uint64_t kSettleNs = 200000ull;  // after an abort: let the peer-counted copies land
constexpr int32_t kStatusTimeout = 4;  // PURO_ERR_TIMEOUT
constexpr int64_t kSplitRefPairs = 76;  // SM pairs the split heuristic plans for (GB300: 152 SMs)
static_assert(kAtomBytes == 128 && kStagesPerGroup * kBKBytes == 512, "whole k-blocks per stage, whole stages per group");
static_assert(kAtoms == 2 && kStagesPerGroup == 2, "a stage holds k-blocks 2j, 2j+1 of a group of four");

// Shared memory of the quantising epilogue (kGemmOutQuant), per column
// quarter j of the tile (64 columns, four epilogue warps q = 0..3): the row
// maxima each warp found over its 64 columns (its partner quarter j ^ 1
// covers the rest of the rows' 1x128 groups), the column maxima over each
// warp's 32 rows, and the 64 column multipliers.
struct QuantEpiSmem {
    uint32_t rowmax[4][4][32];        // [quarter][warp][lane]: max |bf16| of the lane's row over the quarter
    uint32_t colmax[4][4][32];        // [quarter][warp][column pair]: packed max |bf16| over the warp's rows
    alignas(16) float colmul[4][64];  // [quarter][column]: 2^(127 - g), NaN for a non-finite column
};
struct NoQuantEpiSmem {};

template <int BN, bool QOUT = false>
struct GemmSmem {
    static constexpr int kBNHalf = BN / 2;                 // rows of B per CTA
    static constexpr bool kSfbByHelper = (BN != 256);      // B scale images built by warp 2
    alignas(1024) uint8_t a[kStages][kAtoms][kBM * kAtomBytes];
    alignas(1024) uint8_t b[kStages][kAtoms][kBNHalf * kAtomBytes];
    alignas(1024) uint8_t epi[4][32 * 128];    // per epilogue warp: 32 rows x 128 bytes
    alignas(128) uint8_t sf_a[kStages][512];   // scale vectors of this CTA's 128 rows of A
    // scale vectors of the tile's rows of B: per stage (TMA, BN = 256) or per
    // slot of the helper's ring (BN = 224); 2 x 512 bytes = two tcgen05.cp images
    alignas(128) uint8_t sf_b[kSfbByHelper ? kSfbSlots : kStages][1024];
    uint64_t full[kStages];   // even CTA: both CTAs' copies of a stage landed
    uint64_t empty[kStages];  // both CTAs: the pair MMAs reading a stage are done
    uint64_t tfull[2];        // both CTAs: accumulator complete
    uint64_t tempty[2];       // even CTA: both CTAs' epilogues released the accumulator
    uint64_t sfb_full[kSfbSlots];   // even CTA (BN = 224): both CTAs' B scale images built
    uint64_t sfb_empty[kSfbSlots];  // both CTAs (BN = 224): the copies reading an image are done
    uint64_t drain;
    uint32_t tmem_base;
    volatile int abort_flag;
    std::conditional_t<QOUT, QuantEpiSmem, NoQuantEpiSmem> qe;
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
    const uint8_t *sfb;  // scale vectors of B (BN = 224: read by the helper warp)
    const float *sia;
    const float *sib;
    int32_t *status;
    uint64_t wait_ns;
    // kGemmOutQuant: the rowwise copy Dq [M, N] and its scale vectors, the
    // transposed copy Dq^T [N, M] and its scale vectors (both null: none),
    // the BF16 D (null: not stored), and the FP8 format of the copies
    uint8_t *q, *q_scale, *qt, *qt_scale;
    uint16_t *d_bf16;
    int q_fmt;
    // A second problem in the same launch (the grouped backward pass: Dgrad
    // and Wgrad of one linear; block kind, BF16 output, 256-wide, unsplit):
    // units units0 .. num_units-1 are its whole tiles, read and written
    // through tm_a1 .. tm_sfb1.  units0 == num_units: one problem.
    int units0;
    int N1, num_m1, num_n1, num_kb1, m_fastest1, kgroups1;
    uint32_t idesc1;
    // Grouped launch: short (second-problem) units the pairs with one long
    // unit fewer take first (see PairUnits); 0: plain round-robin.
    int lead;
};

// Instruction descriptors (tcgen05.mma), both operands K-major, M = 256
// (a pair MMA), N = bn.
//   kind::f16 / kind::f8f6f4: [4,6) D format (1 = F32), [7,10) A type,
//     [10,13) B type, [17,23) N >> 3, [24,29) M >> 4.
//   kind::mxf8f6f4: [4,6) B scale id, [7,10) A type, [10,13) B type,
//     [17,23) N >> 3, [23] scale type (1 = UE8M0), [24,29) M >> 4,
//     [29,31) A scale id.  The scale id selects the byte of the 32-bit
//     tensor-memory scale word: here the k-block within its group of four.
__host__ __device__ constexpr uint32_t idesc_dense(uint32_t atype, uint32_t btype, int bn) {
    return (1u << 4) | (atype << 7) | (btype << 10) | (static_cast<uint32_t>(bn >> 3) << 17) |
           (static_cast<uint32_t>(kPairM >> 4) << 24);
}
__host__ __device__ constexpr uint32_t idesc_mx(uint32_t atype, uint32_t btype, int bn) {
    return (atype << 7) | (btype << 10) | (static_cast<uint32_t>(bn >> 3) << 17) | (1u << 23) |
           (static_cast<uint32_t>(kPairM >> 4) << 24);
}

template <class Smem>
PURO_DEV void record_timeout(Smem &sm, int32_t *status) {
    sm.abort_flag = 1;
    if (status) atomicExch(status, kStatusTimeout);
}

// One unit of work: a 256 x BN pair tile and a chunk of the reduction.
// Units of the same chunk are consecutive; within a chunk the tile order
// iterates the blocks of the smaller operand fastest, so the pairs of a wave
// share (and read once) the blocks of the larger one.
struct WorkUnit {
    int m0, n0, kb0, kb1, split;  // m0: first row of the pair tile
    int problem;                  // 0, or 1 for the second problem of a grouped launch
};

// The work units of one CTA pair, in the order it takes them.  A launch
// hands them out round-robin over its P pairs: pair p takes units p, p + P,
// p + 2P, ...  A grouped launch puts the problem with the longer reduction
// first (units [0, units0)), so its long units go round-robin and the short
// ones follow in the same global order, which lets the pairs that got one
// long unit fewer start on the short ones first.  Where there are fewer long
// units than pairs (a small Wgrad output grouped with its Dgrad), the pairs
// without one would idle through most of the launch, so they first take
// `lead` short units among themselves (about one long unit's worth of
// work), and then every pair goes on round-robin over the rest.  The
// sequence is a function of (params, pair, P) alone: the producer, the MMA
// issuer, the helpers and the epilogue of both CTAs walk the same one.
struct PairUnits {
    int p, P, units0, u1, plong, pshort, lead, rank, nh, k;
    PURO_DEV PairUnits(const GemmParams &gp, int pair, int num_pairs)
        : p(pair), P(num_pairs), units0(gp.units0), u1(gp.num_units - gp.units0), k(0) {
        plong = units0 % P;                    // pairs [0, plong) take one long unit more
        pshort = P - plong;
        rank = (p - plong + P) % P;            // the pair's turn in the short units' round-robin
        lead = (units0 < P && u1 > 0) ? gp.lead : 0;
        nh = units0 / P + (p < plong ? 1 : 0);
    }
    // The next unit, or -1 when the pair is done.
    PURO_DEV int next() {
        if (k < nh) return p + P * k++;
        int kk = k++ - nh;
        if (lead > 0 && rank < pshort) {
            if (kk < lead) {
                const int j = rank + pshort * kk;
                return j < u1 ? units0 + j : -1;
            }
            kk -= lead;
        }
        const int j = pshort * lead + rank + P * kk;
        return j < u1 ? units0 + j : -1;
    }
};

template <int BN>
PURO_DEV WorkUnit work_unit(const GemmParams &p, int u) {
    WorkUnit w;
    if (u >= p.units0) {  // the second problem: whole tiles
        const int tile = u - p.units0;
        const int mb = p.m_fastest1 ? tile % p.num_m1 : tile / p.num_n1;
        const int nb = p.m_fastest1 ? tile / p.num_m1 : tile % p.num_n1;
        w.m0 = mb * kPairM;
        w.n0 = nb * BN;
        w.split = 0;
        w.kb0 = 0;
        w.kb1 = p.num_kb1;
        w.problem = 1;
        return w;
    }
    w.problem = 0;
    w.split = u / p.num_tiles;
    const int tile = u - w.split * p.num_tiles;
    const int mb = p.m_fastest ? tile % p.num_m : tile / p.num_n;
    const int nb = p.m_fastest ? tile / p.num_m : tile % p.num_n;
    w.m0 = mb * kPairM;
    w.n0 = nb * BN;
    w.kb0 = w.split * p.kb_per_split;
    w.kb1 = min(p.num_kb, w.kb0 + p.kb_per_split);
    return w;
}

// Convert 32 FP32 accumulator columns of this thread's row to BF16 (times sab
// for the per-tensor kind) into four 16-byte units.
template <int KIND>
PURO_DEV void pack_bf16x8(const uint32_t *src, float sab, uint32_t (&w)[4]) {
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
}

// p ? a : b as one selp on registers.
PURO_DEV uint32_t sel_u32(bool p, uint32_t a, uint32_t b) {
    uint32_t r;
    asm("{\n\t.reg .pred q;\n\tsetp.ne.u32 q, %3, 0;\n\tselp.b32 %0, %1, %2, q;\n\t}"
        : "=r"(r)
        : "r"(a), "r"(b), "r"(static_cast<uint32_t>(p)));
    return r;
}

// Codes of two values of one row that belong to two columns with their own
// multipliers m0, m1 (transposed copy); a non-finite column gives NaN codes
// that keep each value's sign, as in quant4.
template <int FMT>
PURO_DEV uint32_t quant2_cols(float x0, float x1, float m0, float m1) {
    uint32_t r = cvt_f32x2<FMT>(mul_f32x2(f32x2(x0, x1), f32x2(m0, m1)));
    if (__builtin_expect(isnan(m0), 0)) r = (r & 0xFF00u) | ((__float_as_uint(x0) >> 24) & 0x80u) | 0x7Fu;
    if (__builtin_expect(isnan(m1), 0)) r = (r & 0x00FFu) | ((((__float_as_uint(x1) >> 24) & 0x80u) | 0x7Fu) << 8);
    return r;
}

// 4x4 transpose of 16-byte chunks within each quad of lanes: on entry
// x[4k .. 4k+3] is chunk k of this lane's row; on exit lane c of the quad
// holds, in x[4r .. 4r+3], chunk c of the quad's row r.  A warp's store of
// x[4r .. 4r+3] then writes whole 64-byte row segments (eight rows per
// instruction) instead of a 16-byte piece of each of 32 rows.
PURO_DEV void quad_transpose_chunks(uint32_t (&x)[16], int lane) {
    const int qi = lane & 3;
#pragma unroll
    for (int b = 1; b <= 2; b <<= 1) {
        const bool up = (qi & b) != 0;
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if (k & b) continue;  // chunk pairs (k, k | b): the lower lane sends k | b, the upper k
#pragma unroll
            for (int w = 0; w < 4; ++w) {
                const uint32_t got = __shfl_xor_sync(0xFFFFFFFFu, sel_u32(up, x[4 * k + w], x[4 * (k | b) + w]), b);
                if (up)
                    x[4 * k + w] = got;
                else
                    x[4 * (k | b) + w] = got;
            }
        }
    }
}

// Quantising epilogue (kGemmOutQuant), run by warps 4..19 of both CTAs of
// a pair.  Warp 4 + 4j + q takes column quarter j (columns 64j .. 64j+63 of
// every tile; half h = j / 2) and, as its tensor-memory lane quarter q, the
// rows m0 + 32q .. m0 + 32q + 31, one per lane; four warps per SM
// sub-partition keep the conversion chains overlapped.  Each thread rounds
// its row's 64 accumulators to BF16 (the values the BF16 output has) and
// produces the codes and scales the blockwise activation quantiser produces
// from them (section "FP8 Mixed-Precision Training": 1x128 groups along the
// row for the rowwise copy -- a row's group spans quarters 2h and 2h+1,
// whose warps exchange row maxima at the half's named barrier; 128x1 groups
// along M -- exactly this CTA's 128 rows, the quarter's four warps -- for
// the transposed copy).  All outputs leave by plain global stores from
// registers: a row's 64 codes (and its 64 BF16 values, when asked for)
// after a transpose of 16-byte chunks within each quad of lanes, so that a
// store instruction writes eight whole 64-byte row segments; the transposed codes
// after a 4x4 byte transpose within each quad of lanes, as 4-byte stores
// that fill a 32-byte sector per column and warp.  The accumulator is
// released once every quarter is in registers (32 arrivals), so no warp can
// fall a tile behind the MMAs.
template <int FMT, class Smem>
PURO_DEV void quant_epilogue(Smem &sm, const GemmParams &p, uint32_t tmem, int warp, int lane, int pair,
                             int num_pairs, int rank) {
    const int j = (warp - 4) >> 2, q = warp & 3, h = j >> 1;
    const uint32_t bar_half = 1u + static_cast<uint32_t>(h);  // the half's eight warps
    const uint32_t bar_quarter = 3u + static_cast<uint32_t>(j);  // the quarter's four warps
    const uint32_t tempty0 = mapa_shared(smem_u32(&sm.tempty[0]), 0);  // the even CTA's
    QuantEpiSmem &qe = sm.qe;
    // quad byte transpose selectors (lane p of each quad of lanes)
    const uint32_t sel1 = (lane & 1) ? 0x3715u : 0x6240u;
    const uint32_t sel2 = (lane & 2) ? 0x3276u : 0x5410u;
    int local = 0;
    PairUnits units(p, pair, num_pairs);
    for (int u = units.next(); u >= 0; u = units.next(), ++local) {
        const WorkUnit wu = work_unit<256>(p, u);
        const int m0 = wu.m0 + kBM * rank;
        const int nq = wu.n0 + 64 * j;  // first column of the quarter
        bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tfull[0], static_cast<uint32_t>(local & 1), p.wait_ns);
        // the half's warps meet at named barriers, so they leave together;
        // each reaches this one after its own bounded wait
        ok = named_bar_and(bar_half, 256, __all_sync(0xFFFFFFFFu, ok));
        if (!ok) {
            if (lane == 0) record_timeout(sm, p.status);
            break;
        }
        tc_fence_after_sync();
        // consecutive tiles' accumulators at columns 0 / 128 (shifted scheme)
        const uint32_t t_row = tmem + (static_cast<uint32_t>(32 * q) << 16) +
                               static_cast<uint32_t>((local & 1) * 128 + 64 * j);
        uint32_t v[32];  // the row's quarter in BF16, columns 2k / 2k+1 in the low / high half of v[k]
#pragma unroll
        for (int c = 0; c < 2; ++c) {
            uint32_t r[32];
            tmem_ld_32x32b_x32(t_row + 32 * c, r);
            tmem_ld_wait();
#pragma unroll
            for (int i = 0; i < 16; ++i) {
                __nv_bfloat162 b2 = __floats2bfloat162_rn(__uint_as_float(r[2 * i]), __uint_as_float(r[2 * i + 1]));
                v[16 * c + i] = *reinterpret_cast<uint32_t *>(&b2);
            }
        }
        tc_fence_before_sync();
        __syncwarp();
        if (lane == 0) mbar_arrive_cluster_cta_scope(tempty0);  // this warp's quarter is in registers
        if (wu.n0 + 128 * h >= p.N) continue;  // a half past the last column (uniform over the half)
        const bool rows_in = m0 < p.M;  // the CTA's 128 rows
        const int64_t row = static_cast<int64_t>(m0 + 32 * q + lane);

        // rows of the quad of lanes this lane stores for (quad_transpose_chunks)
        const int64_t quad_row = static_cast<int64_t>(m0 + 32 * q + (lane & ~3));
        const int qc = lane & 3;
        if (p.d_bf16 && rows_in) {  // the row's 64 BF16 values: two groups of four 16-byte chunks
#pragma unroll
            for (int h2 = 0; h2 < 2; ++h2) {
                uint32_t x[16];
#pragma unroll
                for (int i = 0; i < 16; ++i) x[i] = v[16 * h2 + i];
                quad_transpose_chunks(x, lane);
#pragma unroll
                for (int r = 0; r < 4; ++r)
                    *reinterpret_cast<uint4 *>(p.d_bf16 + (quad_row + r) * p.N + nq + 32 * h2 + 8 * qc) =
                        make_uint4(x[4 * r], x[4 * r + 1], x[4 * r + 2], x[4 * r + 3]);
            }
        }

        // ---- rowwise copy: the row's 1x128 group is this quarter and its partner
        {
            uint32_t m2 = 0;
#pragma unroll
            for (int k = 0; k < 32; ++k) m2 = __vmaxu2(m2, v[k] & 0x7FFF7FFFu);
            const uint32_t mine = max(m2 & 0xFFFFu, m2 >> 16);
            qe.rowmax[j][q][lane] = mine;
            named_bar_sync(bar_half, 256);  // both quarters' row maxima written
            const uint32_t g = e8m0_exponent<FMT>(max(mine, qe.rowmax[j ^ 1][q][lane]));
            const float rmul = mul_of(g);
            const uint64_t rm2 = f32x2(rmul, rmul);
            const bool rnan = isnan(rmul);
            if (rows_in) {
                uint32_t x[16];  // x[4i .. 4i+3]: codes of columns 16i .. 16i+15 of the quarter
#pragma unroll
                for (int i = 0; i < 4; ++i) {
#pragma unroll
                    for (int k = 0; k < 4; ++k) {
                        const uint32_t a = v[8 * i + 2 * k], b = v[8 * i + 2 * k + 1];
                        x[4 * i + k] = quant4<FMT>(bf16_lo(a), bf16_hi(a), bf16_lo(b), bf16_hi(b), rm2, rnan);
                    }
                }
                quad_transpose_chunks(x, lane);
#pragma unroll
                for (int r = 0; r < 4; ++r)
                    *reinterpret_cast<uint4 *>(p.q + (quad_row + r) * p.N + nq + 16 * qc) =
                        make_uint4(x[4 * r], x[4 * r + 1], x[4 * r + 2], x[4 * r + 3]);
                if ((j & 1) == 0)  // one scale per row and group
                    store_scale_vec(p.q_scale, row, (wu.n0 + 128 * h) / 128, p.N / 128, static_cast<uint8_t>(g));
            }
        }
        if (p.qt == nullptr) continue;  // uniform

        // ---- transposed copy: column c's group is its 128 rows in this CTA.
        // Column maxima over the warp's 32 rows by a reduce-scatter butterfly
        // on the packed |bf16| pairs: at the step with lane bit b the lane
        // keeps the half of its words that bit selects and takes the max with
        // the other half from lane ^ b; after five steps lane l holds word l
        // (columns 2l and 2l + 1 of the quarter).
        {
            uint32_t a[32];
#pragma unroll
            for (int k = 0; k < 32; ++k) a[k] = v[k] & 0x7FFF7FFFu;
#pragma unroll
            for (int st = 0; st < 5; ++st) {
                const int half = 16 >> st;  // words kept after this step = lane bit of this step
                const bool upper = (lane & half) != 0;
#pragma unroll
                for (int i = 0; i < half; ++i) {
                    const uint32_t keep = sel_u32(upper, a[i + half], a[i]);
                    const uint32_t send = sel_u32(upper, a[i], a[i + half]);
                    a[i] = __vmaxu2(keep, __shfl_xor_sync(0xFFFFFFFFu, send, half));
                }
            }
            qe.colmax[j][q][lane] = a[0];
        }
        named_bar_sync(bar_quarter, 128);  // the quarter's column maxima written
        bool col_ok = true;
        {
            const int t = 32 * q + lane;  // t < 64: this thread's column
            if (t < 64) {
                const uint32_t m2c = __vmaxu2(__vmaxu2(qe.colmax[j][0][t >> 1], qe.colmax[j][1][t >> 1]),
                                              __vmaxu2(qe.colmax[j][2][t >> 1], qe.colmax[j][3][t >> 1]));
                const uint32_t gc = e8m0_exponent<FMT>((t & 1) ? (m2c >> 16) : (m2c & 0xFFFFu));
                const float cmul = mul_of(gc);
                qe.colmul[j][t] = cmul;
                col_ok = !isnan(cmul);
                if (rows_in) store_scale_vec(p.qt_scale, nq + t, m0 / 128, p.M / 128, static_cast<uint8_t>(gc));
            }
        }
        // column multipliers ready; any non-finite column in the quarter?
        const bool any_nan = !named_bar_and(bar_quarter, 128, col_ok);
        uint8_t *qt_base = p.qt + static_cast<int64_t>(nq + (lane & 3)) * p.M + m0 + 32 * q + 4 * (lane >> 2);
#pragma unroll
        for (int w = 0; w < 16; ++w) {  // columns 4w .. 4w+3 of the quarter
            const float4 cm = *reinterpret_cast<const float4 *>(&qe.colmul[j][4 * w]);
            const uint32_t a = v[2 * w], b = v[2 * w + 1];
            uint32_t lo, hi;
            if (any_nan) {
                lo = quant2_cols<FMT>(bf16_lo(a), bf16_hi(a), cm.x, cm.y);
                hi = quant2_cols<FMT>(bf16_lo(b), bf16_hi(b), cm.z, cm.w);
            } else {
                lo = cvt_f32x2<FMT>(mul_f32x2(f32x2(bf16_lo(a), bf16_hi(a)), f32x2(cm.x, cm.y)));
                hi = cvt_f32x2<FMT>(mul_f32x2(f32x2(bf16_lo(b), bf16_hi(b)), f32x2(cm.z, cm.w)));
            }
            // this row's codes of columns 4w .. 4w+3 -> (4x4 transpose in the
            // quad) rows 4k .. 4k+3 of column 4w + (lane & 3)
            uint32_t x = lo | (hi << 16);
            x = __byte_perm(x, __shfl_xor_sync(0xFFFFFFFFu, x, 1), sel1);
            x = __byte_perm(x, __shfl_xor_sync(0xFFFFFFFFu, x, 2), sel2);
            if (rows_in) *reinterpret_cast<uint32_t *>(qt_base + static_cast<int64_t>(4 * w) * p.M) = x;
        }
    }
}

// OUT: kGemmOutBF16 writes D in BF16; kGemmOutF32Partial writes FP32
// partial tiles of a split reduction to the workspace [splits * Mp, N],
// Mp = num_m * 256 (rows split * Mp + m), so that a ragged last pair tile
// stays inside its chunk; kGemmOutF32Add adds the FP32 tile to D (an FP32
// main-grad, one TMA reduce-add per element, so the result is deterministic).
// The FP32 forms are BN = 256 only.  tm_d: BF16 D with box {32, 32} and the
// 64-byte swizzle, or FP32 D / workspace with box {32, 32} and the 128-byte
// swizzle.
// tm_sfa / tm_sfb (block kind only): the scale vectors of A / B viewed as
// uint32 [chunks, 128] (one 512-byte chunk per row), box {128, 1}; tm_sfb is
// read only with BN = 256.  kGemmOutQuant (block kind, BN = 256, 640
// threads) quantises the BF16-rounded tile in the epilogue (quant_epilogue)
// and does not use tm_d.
template <int OUT>
constexpr int gemm_threads() { return OUT == kGemmOutQuant ? kThreads + 384 : kThreads; }

template <int KIND, int OUT, int BN>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(gemm_threads<OUT>(), 1)
    gemm_tn_kernel(const __grid_constant__ CUtensorMap tm_a, const __grid_constant__ CUtensorMap tm_b,
                   const __grid_constant__ CUtensorMap tm_d, const __grid_constant__ CUtensorMap tm_sfa,
                   const __grid_constant__ CUtensorMap tm_sfb, const __grid_constant__ CUtensorMap tm_a1,
                   const __grid_constant__ CUtensorMap tm_b1, const __grid_constant__ CUtensorMap tm_d1,
                   const __grid_constant__ CUtensorMap tm_sfa1, const __grid_constant__ CUtensorMap tm_sfb1,
                   const GemmParams p) {
    using Smem = GemmSmem<BN, OUT == kGemmOutQuant>;
    constexpr int kBNHalf = Smem::kBNHalf;
    constexpr bool kMX = (KIND == kGemmFP8Block);
    constexpr bool kHelper = kMX && Smem::kSfbByHelper;
    constexpr bool kShifted = kMX && BN == 256;         // shared-half accumulators
    constexpr int kAccBufs = kShifted ? 1 : 2;          // hand-off barrier pairs (tfull / tempty)
    constexpr int kAccShift = kShifted ? 128 : 256;     // column offset between consecutive tiles' accumulators
    constexpr int kSfBase = kShifted ? 384 : 480;       // first scale-vector column (MX)
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;          // elements of K per stage
    constexpr int kAtomK = kAtomBytes / kElemBytes;     // elements of K per 128-byte atom
    constexpr int kKSteps = kAtomBytes / 32;            // MMAs per atom (32 bytes of K each)
    constexpr uint32_t kStageBytes = (kBM + kBNHalf) * kBKBytes;  // one CTA's operand bytes per stage
    constexpr uint32_t kSfBytes = kHelper ? 512u : 512u + 1024u;  // one CTA's TMA scale bytes per group
    constexpr bool OUT_F32 = (OUT == kGemmOutF32Partial || OUT == kGemmOutF32Add);
    constexpr bool OUT_Q = (OUT == kGemmOutQuant);
    static_assert(BN == 256 || (BN == 224 && kMX && OUT == kGemmOutBF16), "the 224-wide form is block-scaled, BF16 out");
    static_assert(!OUT_Q || (kMX && BN == 256), "the quantising epilogue is block-scaled and 256-wide");
    static_assert(!kMX || kSfBase + kSfSets * kSfColsPerSet <= kTmemCols, "TMEM budget");
    static_assert(kAccShift + BN <= (kMX ? kSfBase : kTmemCols), "accumulators clear of the scale columns");

    extern __shared__ uint8_t smem_raw[];
    Smem &sm = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
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
            mbar_init(&sm.tempty[b], OUT_Q ? 32 : 8);  // the epilogue warps of both CTAs
        }
        for (int s = 0; s < kSfbSlots; ++s) {
            mbar_init(&sm.sfb_full[s], 2);  // the helper warp of each CTA
            mbar_init(&sm.sfb_empty[s], 1);
        }
        mbar_init(&sm.drain, 1);
        sm.abort_flag = 0;
        fence_mbarrier_init();
        tma_prefetch_desc(&tm_a);
        tma_prefetch_desc(&tm_b);
        tma_prefetch_desc(&tm_d);
        if (kMX) {
            tma_prefetch_desc(&tm_sfa);
            if (!kHelper) tma_prefetch_desc(&tm_sfb);
        }
        if (p.units0 < p.num_units) {  // grouped launch: the second problem's maps
            tma_prefetch_desc(&tm_a1);
            tma_prefetch_desc(&tm_b1);
            tma_prefetch_desc(&tm_d1);
            tma_prefetch_desc(&tm_sfa1);
            tma_prefetch_desc(&tm_sfb1);
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
    pdl_wait();  // the set-up above overlaps the previous kernel's tail
    pdl_launch_dependents();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ------------------------------------------------ TMA producer
        if (lane == 0) {
            const uint32_t full0 = mapa_shared(smem_u32(&sm.full[0]), 0);  // the even CTA's ring
            uint32_t stage = 0, phase = 0;
            uint32_t issued = 0;  // stage fills started by this thread
            bool aborted = false;
            PairUnits units(p, pair, num_pairs);
            for (int u = units.next(); u >= 0 && !aborted; u = units.next()) {
                const WorkUnit wu = work_unit<BN>(p, u);
                const int a_row = wu.m0 + kBM * static_cast<int>(rank);
                const int b_row = wu.n0 + kBNHalf * static_cast<int>(rank);
                const CUtensorMap *ma = wu.problem ? &tm_a1 : &tm_a;
                const CUtensorMap *mb = wu.problem ? &tm_b1 : &tm_b;
                const CUtensorMap *msfa = wu.problem ? &tm_sfa1 : &tm_sfa;
                const CUtensorMap *msfb = wu.problem ? &tm_sfb1 : &tm_sfb;
                const int kgroups = wu.problem ? p.kgroups1 : p.kgroups;
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
                        tma_load_2d_pair(sm.a[stage][at], ma, full_bar, kb * kBK + at * kAtomK, a_row);
                        tma_load_2d_pair(sm.b[stage][at], mb, full_bar, kb * kBK + at * kAtomK, b_row);
                    }
                    if (sf_load) {
                        // chunks beyond the operand's rows read as zero (their rows are zero too)
                        const int kg = kb / kStagesPerGroup;
                        tma_load_2d_pair(sm.sf_a[stage], msfa, full_bar, 0, (a_row / 128) * kgroups + kg);
                        if constexpr (!kHelper) {
                            tma_load_2d_pair(sm.sf_b[stage], msfb, full_bar, 0, (wu.n0 / 128) * kgroups + kg);
                            tma_load_2d_pair(sm.sf_b[stage] + 512, msfb, full_bar, 0,
                                             (wu.n0 / 128 + 1) * kgroups + kg);
                        }
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
        uint32_t gseq = 0;  // groups of four k-blocks started (BN = 224: slot of the scale ring)
        bool aborted = false;
        int local = 0;
        PairUnits units(p, pair, num_pairs);
        for (int u = units.next(); u >= 0 && !aborted; u = units.next(), ++local) {
            const WorkUnit wu = work_unit<BN>(p, u);
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
                const bool group_start = kMX && (kb % kStagesPerGroup) == 0;
                const uint32_t slot = gseq % kSfbSlots;
                ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.full[stage], phase, p.wait_ns);
                if (kHelper && group_start)
                    ok = ok && mbar_wait_bounded(&sm.sfb_full[slot], (gseq / kSfbSlots) & 1u, p.wait_ns);
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
                        if (group_start) {  // new group of four k-blocks: its scale vectors
                            const uint8_t *sfb_src = kHelper ? sm.sf_b[slot] : sm.sf_b[stage];
                            tmem_cp_pair_32x128b_warpx4(tmem + sfa_col,
                                                        smem_desc_plain_16B_rows(smem_u32(sm.sf_a[stage])));
                            tmem_cp_pair_32x128b_warpx4(tmem + sfb_col, smem_desc_plain_16B_rows(smem_u32(sfb_src)));
                            tmem_cp_pair_32x128b_warpx4(tmem + sfb_col + 4,
                                                        smem_desc_plain_16B_rows(smem_u32(sfb_src + 512)));
                        }
                    }
#pragma unroll
                    for (int at = 0; at < kAtoms; ++at) {
                        uint32_t idesc = wu.problem ? p.idesc1 : p.idesc;
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
                    // the scale image is free once its copies (issued above) are done
                    if (kHelper && group_start) tc_commit_pair_multicast(&sm.sfb_empty[slot], 0x3);
                }
                __syncwarp();
                if (group_start) ++gseq;
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
    } else if ((warp == 2 || warp == 3) && kHelper) {
        // ------------------------------------------------ B scale images (BN = 224, both CTAs)
        // A tile's rows of B start at a multiple of 32 that need not be a
        // multiple of 128, so the 512-byte chunks of the scale-vector layout
        // do not line up with the tile.  For each group of four k-blocks a
        // helper warp gathers the words the MMA needs -- lane l, column j:
        // row n0 + 32j + l -- into two 512-byte tcgen05.cp images.  Warps 2
        // and 3 take alternate groups, so the L2 round trip of one group's
        // loads overlaps the next.
        const uint32_t sfb_full0 = mapa_shared(smem_u32(&sm.sfb_full[0]), 0);  // the even CTA's
        const uint32_t *sfb_words = reinterpret_cast<const uint32_t *>(p.sfb);
        const uint32_t mine = static_cast<uint32_t>(warp - 2);
        uint32_t gseq = 0;
        bool aborted = false;
        PairUnits units(p, pair, num_pairs);
        for (int u = units.next(); u >= 0 && !aborted; u = units.next()) {
            const WorkUnit wu = work_unit<BN>(p, u);
            for (int kb = wu.kb0; kb < wu.kb1; kb += kStagesPerGroup, ++gseq) {
                if ((gseq & 1u) != mine) continue;
                const uint32_t slot = gseq % kSfbSlots;
                const bool ok = (sm.abort_flag == 0) &&
                                mbar_wait_bounded(&sm.sfb_empty[slot], ((gseq / kSfbSlots) & 1u) ^ 1u, p.wait_ns);
                if (!__all_sync(0xFFFFFFFFu, ok)) {
                    if (lane == 0) record_timeout(sm, p.status);
                    aborted = true;
                    break;
                }
                const int kg = kb / kStagesPerGroup;
                uint32_t words[8];
#pragma unroll
                for (int j = 0; j < 8; ++j) {
                    const int grp = wu.n0 / 32 + j;  // 32-row group of B
                    // rows past N (and the eighth column) hold no data: 2^0
                    words[j] = (j < BN / 32 && 32 * grp < p.N)
                                   ? __ldg(sfb_words + ((static_cast<int64_t>(grp / 4) * p.kgroups + kg) * 128 +
                                                        4 * lane + (grp % 4)))
                                   : 0x7F7F7F7Fu;
                }
                uint8_t *img = sm.sf_b[slot];
#pragma unroll
                for (int h = 0; h < 2; ++h)
                    *reinterpret_cast<uint4 *>(img + 512 * h + 16 * lane) =
                        make_uint4(words[4 * h], words[4 * h + 1], words[4 * h + 2], words[4 * h + 3]);
                fence_proxy_async_smem();  // generic writes -> the tensor core's copy
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster(sfb_full0 + 8u * slot);
            }
        }
    } else if constexpr (OUT_Q) {
        // ------------------------------------------------ quantising epilogue (both CTAs)
        if (warp >= 4) {
            if (p.q_fmt == 0)
                quant_epilogue<0>(sm, p, tmem, warp, lane, pair, num_pairs, static_cast<int>(rank));
            else
                quant_epilogue<1>(sm, p, tmem, warp, lane, pair, num_pairs, static_cast<int>(rank));
        }
    } else if (warp >= 4) {
        // ------------------------------------------------ epilogue (both CTAs)
        const int q = warp & 3;  // TMEM lane quarter of this warp
        float sab = 1.0f;
        if constexpr (KIND == kGemmFP8Tensor) sab = __fmul_rn(*p.sia, *p.sib);
        uint8_t *stage_buf = sm.epi[q];
        const uint32_t tempty0 = mapa_shared(smem_u32(&sm.tempty[0]), 0);  // the even CTA's
        int local = 0;
        uint32_t pieces = 0;  // BF16 output: 32-column pieces stored, alternating staging halves
        PairUnits units(p, pair, num_pairs);
        for (int u = units.next(); u >= 0; u = units.next(), ++local) {
            const WorkUnit wu = work_unit<BN>(p, u);
            const int m0 = wu.m0 + kBM * static_cast<int>(rank), n0 = wu.n0;  // this CTA's rows
            const int buf = local % kAccBufs;
            const uint32_t acc_phase = static_cast<uint32_t>(local / kAccBufs) & 1u;
            bool ok = (sm.abort_flag == 0) && mbar_wait_bounded(&sm.tfull[buf], acc_phase, p.wait_ns);
            ok = __all_sync(0xFFFFFFFFu, ok);
            if (!ok) {
                if (lane == 0) record_timeout(sm, p.status);
                break;
            }
            tc_fence_after_sync();
            const uint32_t t_row =
                tmem + (static_cast<uint32_t>(32 * q) << 16) + static_cast<uint32_t>((local & 1) * kAccShift);
            const int n_out = wu.problem ? p.N1 : p.N;  // columns of this unit's output
            const CUtensorMap *md = wu.problem ? &tm_d1 : &tm_d;
            if constexpr (OUT_F32) {
                // FP32 tile: 8 chunks of 32 columns (128 bytes per row), stored
                // as a split partial or added to D
                const int row0 = (OUT == kGemmOutF32Partial ? wu.split * p.num_m * kPairM : 0) + m0 + 32 * q;
#pragma unroll
                for (int h = 0; h < BN / 128; ++h) {
                    uint32_t r[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c) tmem_ld_32x32b_x32(t_row + 128 * h + 32 * c, r[c]);
                    tmem_ld_wait();
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int col = n0 + 128 * h + 32 * c;
                        if (col >= n_out) break;
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
                            if constexpr (OUT == kGemmOutF32Add)
                                tma_reduce_add_2d(md, stage_buf, col, row0);
                            else
                                tma_store_2d(md, stage_buf, col, row0);
                            bulk_commit_group();
                        }
                    }
                }
                tc_fence_before_sync();
                __syncwarp();
                if (lane == 0) mbar_arrive_cluster_cta_scope(tempty0 + 8u * buf);
            } else {
                // BF16 tile in two halves of 128 columns (BN = 224: 128 + 96).
                // Shifted (block kind, BN = 256): the half in the columns the
                // next tile's accumulator shares ([128, 256) of tensor
                // memory) first, and the accumulator released once it is in
                // registers; otherwise halves in order, released after the
                // second load.  Each half leaves in 32-column pieces (64
                // bytes per row, 64-byte swizzle: 16-byte unit i of row l at
                // i ^ ((l / 2) % 4)) that alternate between the two 2 KB
                // halves of the staging tile, so a piece is written while the
                // previous one is still being stored.
                const int h_first = kShifted ? ((local & 1) ? 0 : 1) : 0;
                constexpr int kReleaseAt = kShifted ? 0 : 1;
#pragma unroll 1
                for (int hh = 0; hh < 2; ++hh) {
                    const int h = hh ^ h_first;
                    const int nc = h == 0 ? 4 : (BN - 128) / 32;
                    uint32_t r[4][32];
#pragma unroll
                    for (int c = 0; c < 4; ++c)
                        if (c < nc) tmem_ld_32x32b_x32(t_row + 128 * h + 32 * c, r[c]);
                    tmem_ld_wait();
                    if (hh == kReleaseAt) {
                        tc_fence_before_sync();
                        __syncwarp();
                        if (lane == 0) mbar_arrive_cluster_cta_scope(tempty0 + 8u * buf);  // accumulator free for the next tile
                    }
#pragma unroll
                    for (int c = 0; c < 4; ++c) {
                        const int col = n0 + 128 * h + 32 * c;
                        if (c >= nc || col >= n_out) break;
                        uint8_t *half = stage_buf + 2048 * (pieces & 1u);
                        if (lane == 0) bulk_wait_group_read<1>();  // the store that last read this half is done
                        __syncwarp();
                        uint8_t *row = half + 64 * lane;
#pragma unroll
                        for (int i = 0; i < 4; ++i) {
                            uint32_t w[4];
                            pack_bf16x8<KIND>(&r[c][8 * i], sab, w);
                            *reinterpret_cast<uint4 *>(row + 16 * (i ^ ((lane >> 1) & 3))) = make_uint4(w[0], w[1], w[2], w[3]);
                        }
                        fence_proxy_async_smem();
                        __syncwarp();
                        if (lane == 0) {
                            tma_store_2d(md, half, col, m0 + 32 * q);
                            bulk_commit_group();
                        }
                        ++pieces;
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
    pdl_wait();
    pdl_launch_dependents();
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

// The same sum added to an FP32 main-grad: out[i] += sum_s ws[s][i] (one
// add per element, fixed order).
__global__ void __launch_bounds__(256) splitk_reduce_add_f32_kernel(const float4 *__restrict__ ws, int splits,
                                                                    int64_t n4, int64_t split_stride4,
                                                                    float4 *__restrict__ out) {
    pdl_wait();
    pdl_launch_dependents();
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
        float4 o = out[i];
        o.x += a.x;
        o.y += a.y;
        o.z += a.z;
        o.w += a.w;
        out[i] = o;
    }
}

int choose_splits(int64_t M, int64_t N, int64_t K, bool bf16) {
    if (bf16) return 1;
    const int64_t tiles = ((M + kPairM - 1) / kPairM) * ((N + 255) / 256);
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

// Tile width of an unsplit block-scaled GEMM.  Modelled pair time = waves x
// per-tile cycles, with constants fitted to measured GB300 times of both
// forms over the C5 and C6 linear shapes: about 163 cycles per pair MMA plus
// a 600-cycle accumulator hand-off per tile for the 256-wide form, 176 cycles
// per MMA plus 350 per tile for the 224-wide one (its helpers' scale images
// slow the issue).  The narrower form has more tiles, so it pays off only
// where the 256-wide tiles leave a much worse last wave; it is taken only for
// a modelled gain above 5.5%.  (With the hand-off at 600 cycles the 256-wide
// form measured faster on every shape of both models.)
int choose_tile_n(int64_t M, int64_t N, int64_t K) {
    const int64_t stages = (K + kBKBytes - 1) / kBKBytes;
    const int64_t m_tiles = (M + kPairM - 1) / kPairM;
    auto waves = [&](int64_t bn) { return (m_tiles * ((N + bn - 1) / bn) + kSplitRefPairs - 1) / kSplitRefPairs; };
    const int64_t c256 = waves(256) * (stages * kAtoms * 4 * 163 + 600);
    const int64_t c224 = waves(224) * (stages * kAtoms * 4 * 176 + 350);
    return c224 * 1000 < c256 * 945 ? 224 : 256;
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
template <int KIND, int OUT, int BN>
static int max_resident_pairs(int num_sms, size_t smem) {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return num_sms / 2;
    if (dev >= 0 && dev < 64 && cache[dev] > 0) return cache[dev];
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3(static_cast<unsigned>(num_sms / 2 * 2), 1, 1);
    cfg.blockDim = dim3(gemm_threads<OUT>(), 1, 1);
    cfg.dynamicSmemBytes = smem;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeClusterDimension;
    attr.val.clusterDim.x = 2;
    attr.val.clusterDim.y = 1;
    attr.val.clusterDim.z = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    int n = 0;
    if (cudaOccupancyMaxActiveClusters(&n, gemm_tn_kernel<KIND, OUT, BN>, &cfg) != cudaSuccess || n <= 0) {
        (void)cudaGetLastError();
        n = num_sms / 2;
    }
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

template <int KIND, int OUT, int BN>
static GemmParams make_params(const GemmArgs &g, int splits) {
    constexpr int kElemBytes = (KIND == kGemmBF16) ? 2 : 1;
    constexpr int kBK = kBKBytes / kElemBytes;
    GemmParams p{};
    p.M = static_cast<int>(g.M);
    p.N = static_cast<int>(g.N);
    p.K = static_cast<int>(g.K);
    p.num_m = static_cast<int>((g.M + kPairM - 1) / kPairM);
    p.num_n = static_cast<int>((g.N + BN - 1) / BN);
    p.num_kb = static_cast<int>((g.K + kBK - 1) / kBK);
    p.num_tiles = p.num_m * p.num_n;
    p.splits = splits;
    p.kb_per_split = ((p.num_kb + splits - 1) / splits + kStagesPerGroup - 1) / kStagesPerGroup * kStagesPerGroup;
    p.splits = (p.num_kb + p.kb_per_split - 1) / p.kb_per_split;  // no empty chunk
    p.num_units = p.num_tiles * p.splits;
    p.m_fastest = g.M < g.N ? 1 : 0;  // re-read the smaller operand, stream the larger once
    if (KIND == kGemmBF16)
        p.idesc = idesc_dense(1u, 1u, BN);
    else if (KIND == kGemmFP8Tensor)
        p.idesc = idesc_dense(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt), BN);
    else
        p.idesc = idesc_mx(static_cast<uint32_t>(g.a_fmt), static_cast<uint32_t>(g.b_fmt), BN);
    p.kgroups = static_cast<int>((g.K / 128 + 3) / 4);
    p.sfb = g.sfb;
    p.sia = g.sia;
    p.sib = g.sib;
    p.status = g.status;
    p.wait_ns = g.wait_timeout_ns;

    p.q = g.q;
    p.q_scale = g.q_scale;
    p.qt = g.qt;
    p.qt_scale = g.qt_scale;
    p.d_bf16 = static_cast<uint16_t *>(g.d_bf16);
    p.q_fmt = g.q_fmt;
    p.units0 = p.num_units;  // one problem unless a grouped launch adds a second
    p.lead = 0;
    return p;
}

// Launch with the parameters p; m1: the second problem's maps of a grouped
// launch (unused otherwise).
template <int KIND, int OUT, int BN>
static cudaError_t launch_params(const GemmParams &p, const GemmArgs &g, const GemmMaps &m, const GemmMaps &m1,
                                 cudaStream_t s) {
    auto kern = gemm_tn_kernel<KIND, OUT, BN>;
    const size_t smem = sizeof(GemmSmem<BN, OUT == kGemmOutQuant>) + 1024;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    const int pairs_max = max_resident_pairs<KIND, OUT, BN>(g.num_sms, smem);
    const int pairs = p.num_units < pairs_max ? p.num_units : pairs_max;
    return launch_pdl(kern, dim3(2 * pairs), dim3(gemm_threads<OUT>()), smem, s, m.a, m.b,
                      OUT == kGemmOutF32Partial ? m.ws : m.d, m.sfa, m.sfb, m1.a, m1.b, m1.d, m1.sfa, m1.sfb, p);
}

template <int KIND, int OUT, int BN>
static cudaError_t launch_kind(const GemmArgs &g, const GemmMaps &m, int splits, cudaStream_t s) {
    return launch_params<KIND, OUT, BN>(make_params<KIND, OUT, BN>(g, splits), g, m, m, s);
}

template <int KIND>
static cudaError_t launch_split_or_not(const GemmArgs &g, const GemmMaps &m, cudaStream_t s) {
    if constexpr (KIND == kGemmFP8Block)
        if (g.quant_out) return launch_kind<KIND, kGemmOutQuant, 256>(g, m, 1, s);
    if (g.splits <= 1) {
        if (g.accumulate_f32) return launch_kind<KIND, kGemmOutF32Add, 256>(g, m, 1, s);
        if constexpr (KIND == kGemmFP8Block)
            if (g.tile_n == 224) return launch_kind<KIND, kGemmOutBF16, 224>(g, m, 1, s);
        return launch_kind<KIND, kGemmOutBF16, 256>(g, m, 1, s);
    }
    cudaError_t e = launch_kind<KIND, kGemmOutF32Partial, 256>(g, m, g.splits, s);
    if (e != cudaSuccess) return e;
    const int64_t n4 = g.M * g.N / 4;
    const int64_t stride4 = splitk_rows_per_chunk(g.M) * g.N / 4;
    int64_t want = (n4 + 255) / 256;
    const int64_t cap = static_cast<int64_t>(g.num_sms) * 8;
    const int grid = static_cast<int>(want < cap ? want : cap);
    const float4 *ws = reinterpret_cast<const float4 *>(g.workspace);
    if (g.accumulate_f32)
        return launch_pdl(splitk_reduce_add_f32_kernel, dim3(grid), dim3(256), 0, s, ws, g.splits, n4, stride4,
                          reinterpret_cast<float4 *>(g.out));
    return launch_pdl(splitk_reduce_kernel, dim3(grid), dim3(256), 0, s, ws, g.splits, n4, stride4,
                      reinterpret_cast<uint2 *>(g.out));
}

// Two block-scaled GEMMs (BF16 output, 256-wide, unsplit) in one persistent
// launch: g0's tiles first, then g1's (the caller puts the problem with the
// longer reductions first, so the shorter tiles fill the last round).
cudaError_t launch_gemm_grouped(const GemmArgs &g0, const GemmMaps &m0, const GemmArgs &g1, const GemmMaps &m1,
                                cudaStream_t s) {
    GemmParams p = make_params<kGemmFP8Block, kGemmOutBF16, 256>(g0, 1);
    const GemmParams q = make_params<kGemmFP8Block, kGemmOutBF16, 256>(g1, 1);
    p.units0 = p.num_units;
    p.N1 = q.N;
    p.num_m1 = q.num_m;
    p.num_n1 = q.num_n;
    p.num_kb1 = q.num_kb;
    p.m_fastest1 = q.m_fastest;
    p.kgroups1 = q.kgroups;
    p.idesc1 = q.idesc;
    p.num_units += q.num_units;
    // the pairs with one long unit fewer first take about a long unit's
    // worth of short ones (rounded)
    p.lead = q.num_kb > 0 ? (2 * p.num_kb + q.num_kb) / (2 * q.num_kb) : 0;
    return launch_params<kGemmFP8Block, kGemmOutBF16, 256>(p, g0, m0, m1, s);
}

// Modelled time, in pipeline stages of one pair, of a linear's Dgrad and
// Wgrad as one grouped launch with the balanced schedule (the longer
// reduction's tiles first), against separate launches where the Wgrad
// splits its reduction into `w_splits` chunks (plus its reduction kernel and
// launch, about 20 stages).  Host-only, shape-only.
bool grouped_backward_faster(int64_t M, int64_t N, int64_t K, int w_splits) {
    const int64_t P = kSplitRefPairs;
    auto tiles = [](int64_t r, int64_t c) { return ((r + kPairM - 1) / kPairM) * ((c + 255) / 256); };
    auto stages = [](int64_t red) { return (red + kBKBytes - 1) / kBKBytes; };
    const int64_t ud = tiles(M, K), ld = stages(N);  // Dgrad: dX [M, K], reduction N
    const int64_t uw = tiles(N, K), lw = stages(M);  // Wgrad: dW [N, K], reduction M
    const int64_t u0 = ld >= lw ? ud : uw, l0 = ld >= lw ? ld : lw;
    const int64_t u1 = ld >= lw ? uw : ud, l1 = ld >= lw ? lw : ld;
    const int64_t grouped = std::max((u0 + P - 1) / P * l0, (u0 * l0 + u1 * l1 + P - 1) / P + l1);
    if (w_splits <= 1) return true;  // both unsplit: one launch, no worse than two
    const int64_t chunk = ((lw + w_splits - 1) / w_splits + kStagesPerGroup - 1) / kStagesPerGroup * kStagesPerGroup;
    const int64_t separate = (ud + P - 1) / P * ld + (uw * w_splits + P - 1) / P * chunk + 20;
    return grouped < separate;
}

cudaError_t launch_gemm(const GemmArgs &g, const GemmMaps &m, cudaStream_t s) {
    switch (g.kind) {
        case kGemmBF16: return launch_kind<kGemmBF16, kGemmOutBF16, 256>(g, m, 1, s);
        case kGemmFP8Tensor: return launch_split_or_not<kGemmFP8Tensor>(g, m, s);
        default: return launch_split_or_not<kGemmFP8Block>(g, m, s);
    }
}

}  // namespace puro
