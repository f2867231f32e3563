// tcgen05_issue_rate.cu -- stand-alone probe of how fast one thread can keep
// the tensor pipe busy with tcgen05.mma (cta_group::1, M = 128, K = 32 bytes
// of FP8 per instruction) on GB300, and of what each per-stage extra of a
// pipelined GEMM main loop costs.  One CTA per SM issues MMAs from a fixed
// shared-memory stage (its contents only matter for power), so the numbers
// are free of any load latency.  Not part of the library: the design of the
// GEMM's main loop (256-wide MMAs, two k-blocks per pipeline stage) rests on
// what it measures.
//
// Build and run (one GPU, about ten seconds):
//   nvcc -gencode arch=compute_103a,code=sm_103a -O3 -std=c++17 \
//        -I paper_2608_27370_gb300/csrc -o /tmp/tcgen05_issue_rate \
//        paper_2608_27370_gb300/microbench/tcgen05_issue_rate.cu && /tmp/tcgen05_issue_rate
//
// Every wait is bounded; the kernels allocate 512 tensor-memory columns and
// free them before they return (the pair kernel after a cluster barrier).
#include <cuda.h>
#include <cuda_runtime.h>

#include <cstdint>
#include <cstdio>

#include "ptx.cuh"

using namespace puro;

namespace {

PURO_DEV void tmem_alloc1(uint32_t *dst, uint32_t n) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(smem_u32(dst)), "r"(n)
                 : "memory");
}
PURO_DEV void tmem_relinquish1() { asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory"); }
PURO_DEV void tmem_dealloc1(uint32_t t, uint32_t n) {
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(t), "r"(n) : "memory");
}
PURO_DEV void commit1(uint64_t *bar) {
    asm volatile("tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(smem_u32(bar))
                 : "memory");
}
PURO_DEV void cp1(uint32_t taddr, uint64_t sdesc) {
    asm volatile("tcgen05.cp.cta_group::1.32x128b.warpx4 [%0], %1;" ::"r"(taddr), "l"(sdesc) : "memory");
}
PURO_DEV void mma1_f8(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\ttcgen05.mma.cta_group::1.kind::f8f6f4 [%0], %1, %2, %3, p;\n\t}\n" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(acc)
        : "memory");
}
PURO_DEV void mma1_mx(uint32_t d, uint64_t a, uint64_t b, uint32_t idesc, uint32_t sfa, uint32_t sfb, uint32_t acc) {
    asm volatile(
        "{\n\t.reg .pred p;\n\tsetp.ne.b32 p, %4, 0;\n\t"
        "tcgen05.mma.cta_group::1.kind::mxf8f6f4.block_scale.scale_vec::1X [%0], %1, %2, %3, [%5], [%6], p;\n\t}\n" ::"r"(d),
        "l"(a), "l"(b), "r"(idesc), "r"(acc), "r"(sfa), "r"(sfb)
        : "memory");
}

constexpr int kRing = 8;             // barrier ring (>= the dependency distance)
constexpr uint64_t kBound = 2000000000ull;

struct Smem {
    alignas(1024) uint8_t a[4][16384];  // 128 rows x 128 bytes of K
    alignas(1024) uint8_t b[4][32768];  // up to 256 rows x 128 bytes of K
    alignas(128) uint8_t sf[2][1536];   // scale-vector images: 512 B (A) + 1024 B (B)
    uint64_t done_bar[kRing];           // commit of stage s lands on done_bar[s % DIST]
    uint64_t go_bar[kRing];             // relay's arrival that stage s + DIST may start
    uint64_t fin;
    uint32_t tmem;
};

// The variant is compile-time: the issuing loop's own instruction count is
// part of what is measured, so it carries no run-time switches.
//   MX        kind::mxf8f6f4.block_scale (else kind::f8f6f4)
//   COMMIT    tcgen05.commit per stage
//   READY     a wait per stage on a barrier that is already complete
//   DIST      > 0: stage s waits until the MMAs of stage s - DIST completed,
//             through a relay warp (the shape of a pipelined main loop)
//   CP_EVERY  > 0: three scale-vector copies every CP_EVERY stages (MX only)
template <int N, int MMAS, bool MX, bool COMMIT, bool READY, int DIST, int CP_EVERY>
__global__ void __launch_bounds__(128, 1) issue_rate(int stages, uint32_t seed, uint64_t *cycles) {
    constexpr int kDist = DIST > 0 ? DIST : 1;       // divisors for the branches a variant compiles out
    constexpr int kCpEvery = CP_EVERY > 0 ? CP_EVERY : 1;
    static_assert(DIST <= kRing, "dependency distance within the barrier ring");
    extern __shared__ uint8_t raw[];
    Smem &sm = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&sm.done_bar[i], 1);
            mbar_init(&sm.go_bar[i], 1);
        }
        mbar_init(&sm.fin, 1);
        fence_mbarrier_init();
    }
    // seed 0: every FP8 byte 1.0 (0x38); otherwise pseudo-random finite E4M3 bytes
    for (int i = threadIdx.x; i < 4 * 16384 / 4; i += blockDim.x) {
        uint32_t h = (i + 1) * 2654435761u ^ seed * 40503u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        reinterpret_cast<uint32_t *>(sm.a)[i] = seed ? (h & 0xF6F6F6F6u) : 0x38383838u;
    }
    for (int i = threadIdx.x; i < 4 * 32768 / 4; i += blockDim.x) {
        uint32_t h = (i + 7) * 2246822519u ^ seed * 3266489917u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        reinterpret_cast<uint32_t *>(sm.b)[i] = seed ? (h & 0xF6F6F6F6u) : 0x38383838u;
    }
    for (int i = threadIdx.x; i < 2 * 1536; i += blockDim.x) (&sm.sf[0][0])[i] = static_cast<uint8_t>(124 + i % 7);
    fence_proxy_async_smem();
    if (warp == 0) {
        tmem_alloc1(&sm.tmem, 512);
        tmem_relinquish1();
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    const uint32_t tmem = sm.tmem;
    const uint32_t idesc_f8 = (1u << 4) | (static_cast<uint32_t>(N >> 3) << 17) | ((128u >> 4) << 24);
    const uint32_t idesc_mx = (static_cast<uint32_t>(N >> 3) << 17) | (1u << 23) | ((128u >> 4) << 24);
    if (MX && warp == 1 && lane == 0) {  // scale vectors in place once (columns 256..267)
        cp1(tmem + 256, smem_desc_plain_16B_rows(smem_u32(sm.sf[0])));
        cp1(tmem + 260, smem_desc_plain_16B_rows(smem_u32(sm.sf[0] + 512)));
        cp1(tmem + 264, smem_desc_plain_16B_rows(smem_u32(sm.sf[0] + 1024)));
    }

    if (DIST > 0 && warp == 2 && lane == 0) {
        // relay: stage s's MMAs completed (commit) -> stage s + dist may start
        for (int s = 0; s + kDist < stages; ++s) {
            if (!mbar_wait_bounded(&sm.done_bar[s % kDist], (s / kDist) & 1, kBound)) break;
            mbar_arrive(&sm.go_bar[s % kDist]);
        }
    }
    if (warp == 1) {
        const uint64_t t0 = clock64();
        for (int s = 0; s < stages; ++s) {
            bool ok = true;
            if (DIST > 0) {
                if (s >= kDist) ok = mbar_wait_bounded(&sm.go_bar[s % kDist], ((s / kDist) - 1) & 1, kBound);
            } else if (READY) {
                ok = mbar_try_wait(&sm.fin, 1);  // the phase before the first: complete
            }
            if (!__all_sync(0xFFFFFFFFu, ok)) break;
            tc_fence_after_sync();
            if (lane == 0) {
                uint32_t sf_col = 256;
                if (MX && CP_EVERY > 0) {
                    const int grp = s / kCpEvery;
                    sf_col = 256 + 12 * (grp & 1);
                    if (s % kCpEvery == 0) {
                        const uint32_t src = smem_u32(sm.sf[grp & 1]);
                        cp1(tmem + sf_col, smem_desc_plain_16B_rows(src));
                        cp1(tmem + sf_col + 4, smem_desc_plain_16B_rows(src + 512));
                        cp1(tmem + sf_col + 8, smem_desc_plain_16B_rows(src + 1024));
                    }
                }
                const uint32_t a = smem_u32(sm.a[s & 3]), b = smem_u32(sm.b[s & 3]);
#pragma unroll
                for (int k = 0; k < MMAS; ++k) {
                    const uint64_t ad = smem_desc_k_sw128(a + 32 * (k & 3)), bd = smem_desc_k_sw128(b + 32 * (k & 3));
                    const uint32_t acc = (s > 0 || k > 0) ? 1u : 0u;
                    if (MX)
                        mma1_mx(tmem, ad, bd, idesc_mx | (static_cast<uint32_t>(k & 3) << 29) | (static_cast<uint32_t>(k & 3) << 4),
                                tmem + sf_col, tmem + sf_col + 4, acc);
                    else
                        mma1_f8(tmem, ad, bd, idesc_f8, acc);
                }
                if (COMMIT || DIST > 0) commit1(&sm.done_bar[DIST > 0 ? s % kDist : s & (kRing - 1)]);
            }
            __syncwarp();
        }
        if (lane == 0) commit1(&sm.fin);
        __syncwarp();
        mbar_wait_bounded(&sm.fin, 0, kBound);
        if (lane == 0) cycles[blockIdx.x] = clock64() - t0;
    }
    tc_fence_before_sync();
    __syncthreads();
    tc_fence_after_sync();
    if (warp == 0) tmem_dealloc1(tmem, 512);
}

// The same loop with pair MMAs (tcgen05 cta_group::2, M = 256 over a 2-CTA
// cluster): the even CTA issues, each CTA holds its 128 rows of A and half
// of B's rows at the same shared-memory offsets, commits arrive in both CTAs
// (multicast), and the relay runs in the even CTA.  "cycles" is per cluster.
template <int N, int MMAS, bool MX, bool COMMIT, int DIST, int CP_EVERY>
__global__ void __cluster_dims__(2, 1, 1) __launch_bounds__(128, 1)
    issue_rate_pair(int stages, uint32_t seed, uint64_t *cycles) {
    constexpr int kDist = DIST > 0 ? DIST : 1;
    constexpr int kCpEvery = CP_EVERY > 0 ? CP_EVERY : 1;
    static_assert(DIST <= kRing, "dependency distance within the barrier ring");
    extern __shared__ uint8_t raw[];
    Smem &sm = *reinterpret_cast<Smem *>((reinterpret_cast<uintptr_t>(raw) + 1023) & ~uintptr_t(1023));
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    if (threadIdx.x == 0) {
        for (int i = 0; i < kRing; ++i) {
            mbar_init(&sm.done_bar[i], 1);
            mbar_init(&sm.go_bar[i], 1);
        }
        mbar_init(&sm.fin, 1);
        fence_mbarrier_init();
    }
    for (int i = threadIdx.x; i < 4 * 16384 / 4; i += blockDim.x) {
        uint32_t h = (i + 1 + 977 * rank) * 2654435761u ^ seed * 40503u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        reinterpret_cast<uint32_t *>(sm.a)[i] = seed ? (h & 0xF6F6F6F6u) : 0x38383838u;
    }
    for (int i = threadIdx.x; i < 4 * 32768 / 4; i += blockDim.x) {
        uint32_t h = (i + 7 + 131 * rank) * 2246822519u ^ seed * 3266489917u;
        h ^= h >> 13;
        h *= 0x5bd1e995u;
        h ^= h >> 15;
        reinterpret_cast<uint32_t *>(sm.b)[i] = seed ? (h & 0xF6F6F6F6u) : 0x38383838u;
    }
    for (int i = threadIdx.x; i < 2 * 1536; i += blockDim.x) (&sm.sf[0][0])[i] = static_cast<uint8_t>(124 + i % 7);
    fence_proxy_async_smem();
    if (warp == 0) {
        tmem_alloc_pair(&sm.tmem, 512);
        tmem_relinquish_alloc_permit_pair();
    }
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // both CTAs' barriers, operands and tensor memory ready
    tc_fence_after_sync();
    const uint32_t tmem = sm.tmem;
    const uint32_t idesc_f8 = (1u << 4) | (static_cast<uint32_t>(N >> 3) << 17) | ((256u >> 4) << 24);
    const uint32_t idesc_mx = (static_cast<uint32_t>(N >> 3) << 17) | (1u << 23) | ((256u >> 4) << 24);
    if (rank == 0 && MX && warp == 1 && lane == 0) {  // scale vectors in place once (columns 256..267)
        tmem_cp_pair_32x128b_warpx4(tmem + 256, smem_desc_plain_16B_rows(smem_u32(sm.sf[0])));
        tmem_cp_pair_32x128b_warpx4(tmem + 260, smem_desc_plain_16B_rows(smem_u32(sm.sf[0] + 512)));
        tmem_cp_pair_32x128b_warpx4(tmem + 264, smem_desc_plain_16B_rows(smem_u32(sm.sf[0] + 1024)));
    }
    if (rank == 0 && DIST > 0 && warp == 2 && lane == 0) {
        for (int s = 0; s + kDist < stages; ++s) {
            if (!mbar_wait_bounded(&sm.done_bar[s % kDist], (s / kDist) & 1, kBound)) break;
            mbar_arrive(&sm.go_bar[s % kDist]);
        }
    }
    if (rank == 0 && warp == 1) {
        const uint64_t t0 = clock64();
        for (int s = 0; s < stages; ++s) {
            bool ok = true;
            if (DIST > 0 && s >= kDist) ok = mbar_wait_bounded(&sm.go_bar[s % kDist], ((s / kDist) - 1) & 1, kBound);
            if (!__all_sync(0xFFFFFFFFu, ok)) break;
            tc_fence_after_sync();
            if (lane == 0) {
                uint32_t sf_col = 256;
                if (MX && CP_EVERY > 0) {
                    const int grp = s / kCpEvery;
                    sf_col = 256 + 12 * (grp & 1);
                    if (s % kCpEvery == 0) {
                        const uint32_t src = smem_u32(sm.sf[grp & 1]);
                        tmem_cp_pair_32x128b_warpx4(tmem + sf_col, smem_desc_plain_16B_rows(src));
                        tmem_cp_pair_32x128b_warpx4(tmem + sf_col + 4, smem_desc_plain_16B_rows(src + 512));
                        tmem_cp_pair_32x128b_warpx4(tmem + sf_col + 8, smem_desc_plain_16B_rows(src + 1024));
                    }
                }
                const uint32_t a = smem_u32(sm.a[s & 3]), b = smem_u32(sm.b[s & 3]);
#pragma unroll
                for (int k = 0; k < MMAS; ++k) {
                    const uint64_t ad = smem_desc_k_sw128(a + 32 * (k & 3)), bd = smem_desc_k_sw128(b + 32 * (k & 3));
                    const uint32_t acc = (s > 0 || k > 0) ? 1u : 0u;
                    if (MX)
                        mma_pair_mxf8(tmem, ad, bd,
                                      idesc_mx | (static_cast<uint32_t>(k & 3) << 29) | (static_cast<uint32_t>(k & 3) << 4),
                                      tmem + sf_col, tmem + sf_col + 4, acc);
                    else
                        mma_pair_f8(tmem, ad, bd, idesc_f8, acc);
                }
                if (COMMIT || DIST > 0) tc_commit_pair_multicast(&sm.done_bar[DIST > 0 ? s % kDist : s & (kRing - 1)], 0x3);
            }
            __syncwarp();
        }
        if (lane == 0) tc_commit_pair_multicast(&sm.fin, 0x3);
        __syncwarp();
        mbar_wait_bounded(&sm.fin, 0, kBound);
        if (lane == 0) cycles[blockIdx.x / 2] = clock64() - t0;
    } else if (rank == 1 && warp == 1) {
        mbar_wait_bounded(&sm.fin, 0, 4 * kBound);  // the pair's MMAs into this CTA's tensor memory are done
    }
    tc_fence_before_sync();
    __syncthreads();
    cluster_sync();  // no pair MMA can still write either CTA's tensor memory
    tc_fence_after_sync();
    if (warp == 0) tmem_dealloc_pair(tmem, 512);
}

#define CK(x)                                                                         \
    do {                                                                              \
        cudaError_t e_ = (x);                                                         \
        if (e_ != cudaSuccess) {                                                      \
            std::printf("CUDA error %s at line %d\n", cudaGetErrorString(e_), __LINE__); \
            return 1;                                                                 \
        }                                                                             \
    } while (0)

template <int N, int MMAS, bool MX, bool COMMIT, bool READY, int DIST, int CP_EVERY>
int run(const char *name, uint32_t seed, int reps, int sms, uint64_t *d_cycles) {
    auto k = issue_rate<N, MMAS, MX, COMMIT, READY, DIST, CP_EVERY>;
    const int smem = static_cast<int>(sizeof(Smem)) + 1024;
    CK(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    const int total_mmas = 16384;
    const int stages = total_mmas / MMAS;
    k<<<sms, 128, smem>>>(64, seed, d_cycles);  // warm-up
    CK(cudaGetLastError());
    CK(cudaDeviceSynchronize());
    cudaEvent_t e0, e1;
    CK(cudaEventCreate(&e0));
    CK(cudaEventCreate(&e1));
    CK(cudaEventRecord(e0));
    for (int r = 0; r < reps; ++r) k<<<sms, 128, smem>>>(stages, seed, d_cycles);
    CK(cudaEventRecord(e1));
    CK(cudaDeviceSynchronize());
    float ms = 0;
    CK(cudaEventElapsedTime(&ms, e0, e1));
    ms /= reps;
    uint64_t cyc[512];
    CK(cudaMemcpy(cyc, d_cycles, sms * sizeof(uint64_t), cudaMemcpyDeviceToHost));
    double avg = 0;
    for (int i = 0; i < sms; ++i) avg += static_cast<double>(cyc[i]);
    avg /= sms;
    const double ideal = 2.0 * 128 * N * 32 / 16384.0;  // cycles per MMA at 16384 flop/clk/SM
    const double per_mma = avg / total_mmas;
    const double tflops = 2.0 * 128 * N * 32 * total_mmas * sms / (ms * 1e-3) / 1e12;
    std::printf("| %-44s | %3d | %2d | %6.1f | %5.1f | %5.1f %% | %7.0f |\n", name, N, MMAS, per_mma, ideal,
                100.0 * ideal / per_mma, tflops);
    return 0;
}

template <int N, int MMAS, bool MX, bool COMMIT, int DIST, int CP_EVERY>
int run_pair(const char *name, uint32_t seed, int reps, int sms, uint64_t *d_cycles) {
    auto k = issue_rate_pair<N, MMAS, MX, COMMIT, DIST, CP_EVERY>;
    const int smem = static_cast<int>(sizeof(Smem)) + 1024;
    CK(cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem));
    const int total_mmas = 16384;
    const int stages = total_mmas / MMAS;
    const int grid = sms / 2 * 2;
    k<<<grid, 128, smem>>>(64, seed, d_cycles);  // warm-up
    CK(cudaGetLastError());
    CK(cudaDeviceSynchronize());
    cudaEvent_t e0, e1;
    CK(cudaEventCreate(&e0));
    CK(cudaEventCreate(&e1));
    CK(cudaEventRecord(e0));
    for (int r = 0; r < reps; ++r) k<<<grid, 128, smem>>>(stages, seed, d_cycles);
    CK(cudaEventRecord(e1));
    CK(cudaDeviceSynchronize());
    float ms = 0;
    CK(cudaEventElapsedTime(&ms, e0, e1));
    ms /= reps;
    uint64_t cyc[512];
    CK(cudaMemcpy(cyc, d_cycles, grid / 2 * sizeof(uint64_t), cudaMemcpyDeviceToHost));
    double avg = 0;
    for (int i = 0; i < grid / 2; ++i) avg += static_cast<double>(cyc[i]);
    avg /= grid / 2;
    const double ideal = 2.0 * 128 * N * 32 / 16384.0;  // cycles per pair MMA at 16384 flop/clk/SM on each SM
    const double per_mma = avg / total_mmas;
    const double tflops = 2.0 * 256 * N * 32 * total_mmas * (grid / 2) / (ms * 1e-3) / 1e12;
    std::printf("| pair: %-38s | %3d | %2d | %6.1f | %5.1f | %5.1f %% | %7.0f |\n", name, N, MMAS, per_mma, ideal,
                100.0 * ideal / per_mma, tflops);
    return 0;
}

}  // namespace

int main() {
    int sms = 0;
    CK(cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, 0));
    uint64_t *d_cycles = nullptr;
    CK(cudaMalloc(&d_cycles, 512 * sizeof(uint64_t)));
    const uint32_t rnd = 12345;
    std::printf("| variant | N | MMAs/stage | cycles/MMA | ideal | pipe busy | TFLOP/s |\n|---|---|---|---|---|---|---|\n");
    // issue cost of the loop (N = 64: the pipe needs only 32 cycles per MMA)
    run<64, 8, false, false, false, 0, 0>("f8, bare", rnd, 3, sms, d_cycles);
    run<64, 8, false, true, false, 0, 0>("f8, + commit per stage", rnd, 3, sms, d_cycles);
    run<64, 8, false, true, true, 0, 0>("f8, + commit + ready wait", rnd, 3, sms, d_cycles);
    run<64, 8, true, false, false, 0, 0>("mx, bare", rnd, 3, sms, d_cycles);
    run<64, 8, true, false, false, 0, 2>("mx, + 3 scale copies per 2 stages", rnd, 3, sms, d_cycles);
    // the pipelined main loop: stage s waits for stage s - DIST through a relay
    run<256, 4, true, true, false, 6, 4>("mx, dependent loop, copies every 4 stages", rnd, 3, sms, d_cycles);
    run<256, 8, true, true, false, 3, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    run<224, 8, true, true, false, 3, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    run<192, 8, true, true, false, 3, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    run<128, 8, true, true, false, 4, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    // pair MMAs (cta_group::2, M = 256): the issue cost and the dependent loop
    run_pair<64, 8, true, false, 0, 0>("mx, bare", rnd, 3, sms, d_cycles);
    run_pair<64, 8, true, true, 0, 2>("mx, + commit + copies per 2 stages", rnd, 3, sms, d_cycles);
    run_pair<256, 8, true, true, 3, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    run_pair<224, 8, true, true, 3, 2>("mx, dependent loop, copies every 2 stages", rnd, 3, sms, d_cycles);
    run_pair<256, 8, false, true, 3, 0>("f8, dependent loop", rnd, 3, sms, d_cycles);
    // power: constant vs random operands over about 2 s
    run<256, 4, false, false, false, 0, 0>("f8, bare, operands all 1.0, ~2 s", 0, 1500, sms, d_cycles);
    run<256, 4, false, false, false, 0, 0>("f8, bare, random operands, ~2 s", rnd, 1500, sms, d_cycles);
    CK(cudaFree(d_cycles));
    return 0;
}
