// muonh.cu -- the MuonH hyperball step (section "Hyperball Optimization",
// Eq. hyperball-update) for an FP32 master weight W and its Muon direction u:
//     u_hat = u / ||u||_F,   W~ = W - eta R u_hat,   W <- R W~ / ||W~||_F,
// with R = ||W_0||_F fixed for the matrix.
//
// Two passes over HBM, because the projection needs ||W~||_F before any
// element can be written.  The norm comes from one reduction pass:
//     ||W~||^2 = S_ww - 2 c S_wu + c^2 S_uu,   c = eta R / sqrt(S_uu),
// with S_ww = sum W^2, S_wu = sum W u, S_uu = sum u^2 (all three additive
// over shards of the matrix).  The update pass then writes
//     W <- s (W - c u),   s = R / ||W~||_F,
// and optionally the BF16 copy the next forward pass quantises.
//
// Many matrices go through one launch of each kernel (a grouped, "multi-
// tensor" step): every matrix is cut into chunks of C float4 values, C a
// function of its size alone (n/4096 elements, clamped to [4096, 65536]),
// and each CTA takes one chunk of one matrix.  So small matrices still fill
// the GPU, the three launches serve the whole model, and a matrix's result
// does not depend on what it is grouped with.
//
// Reductions are deterministic: each thread sums a fixed set of at most 64
// float4 values of its chunk in FP32, the warp and the CTA combine in FP64 in
// a fixed order, and one warp per sum adds the matrix's chunk partials in
// index order.
#include <cuda_bf16.h>

#include <cmath>

#include "internal.h"
#include "ptx.cuh"

namespace puro {
namespace {

constexpr int kMuonhThreads = 256;
constexpr int kMuonhUnroll = 4;
constexpr int64_t kMinChunk4 = 1024;   // float4 values per CTA (4096 elements) ...
constexpr int64_t kMaxChunk4 = 16384;  // ... up to 65536 elements: <= 64 per thread
constexpr int kMaxGroup = 128;         // matrices per launch (the table is a kernel parameter)

// float4 values per CTA for a matrix of n4 float4 values (about 1024 CTAs
// for mid-sized matrices; a function of n alone).
int64_t chunk4_of(int64_t n4) {
    const int64_t c = (n4 + 1023) / 1024;
    return c < kMinChunk4 ? kMinChunk4 : (c > kMaxChunk4 ? kMaxChunk4 : c);
}
int64_t chunks_of(int64_t n4) { return n4 <= 0 ? 0 : (n4 + chunk4_of(n4) - 1) / chunk4_of(n4); }

// The matrices of one launch, passed by value.
struct MuonhGroup {
    int count;
    int total_blocks;
    int block_start[kMaxGroup + 1];  // CTAs of matrix m: [block_start[m], block_start[m+1])
    float4 *w[kMaxGroup];
    const float4 *u[kMaxGroup];
    uint2 *wb[kMaxGroup];            // bf16 copy (4 values per uint2), or null
    int64_t n4[kMaxGroup];
    int64_t chunk4[kMaxGroup];
    double radius[kMaxGroup];
    double eta;
    double *partials;                // [3][total_blocks]
    double *sums;                    // [count][3]
};

__device__ __forceinline__ double warp_sum_f64(double v) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, off);
    return v;  // identical in every lane (each step adds the same two values)
}

// The matrix a CTA works on (binary search of the block prefix).
__device__ __forceinline__ int matrix_of(const MuonhGroup &g, int b) {
    int lo = 0, hi = g.count - 1;
    while (lo < hi) {
        const int mid = (lo + hi + 1) >> 1;
        if (g.block_start[mid] <= b) lo = mid; else hi = mid - 1;
    }
    return lo;
}

// Per-CTA partial sums {S_ww, S_wu, S_uu} of one chunk.
__global__ void __launch_bounds__(kMuonhThreads) muonh_reduce_kernel(const __grid_constant__ MuonhGroup g) {
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    const int m = matrix_of(g, b);
    const int64_t c4 = g.chunk4[m];
    const int64_t lo = static_cast<int64_t>(b - g.block_start[m]) * c4;
    const int64_t hi = lo + c4 < g.n4[m] ? lo + c4 : g.n4[m];
    const float4 *__restrict__ w = g.w[m];
    const float4 *__restrict__ u = g.u[m];
    float sww = 0.0f, swu = 0.0f, suu = 0.0f;
    int64_t i = lo + threadIdx.x;
    constexpr int64_t kStep = kMuonhThreads;
    for (; i + (kMuonhUnroll - 1) * kStep < hi; i += kMuonhUnroll * kStep) {  // loads in flight, then math
        float4 a[kMuonhUnroll], v[kMuonhUnroll];
#pragma unroll
        for (int j = 0; j < kMuonhUnroll; ++j) {
            a[j] = __ldg(w + i + j * kStep);
            v[j] = __ldg(u + i + j * kStep);
        }
#pragma unroll
        for (int j = 0; j < kMuonhUnroll; ++j) {
            sww += fmaf(a[j].x, a[j].x, a[j].y * a[j].y) + fmaf(a[j].z, a[j].z, a[j].w * a[j].w);
            swu += fmaf(a[j].x, v[j].x, a[j].y * v[j].y) + fmaf(a[j].z, v[j].z, a[j].w * v[j].w);
            suu += fmaf(v[j].x, v[j].x, v[j].y * v[j].y) + fmaf(v[j].z, v[j].z, v[j].w * v[j].w);
        }
    }
    for (; i < hi; i += kStep) {
        const float4 a = __ldg(w + i), v = __ldg(u + i);
        sww += fmaf(a.x, a.x, a.y * a.y) + fmaf(a.z, a.z, a.w * a.w);
        swu += fmaf(a.x, v.x, a.y * v.y) + fmaf(a.z, v.z, a.w * v.w);
        suu += fmaf(v.x, v.x, v.y * v.y) + fmaf(v.z, v.z, v.w * v.w);
    }
    __shared__ double red[3][kMuonhThreads / 32];
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const double d0 = warp_sum_f64(sww), d1 = warp_sum_f64(swu), d2 = warp_sum_f64(suu);
    if (lane == 0) {
        red[0][warp] = d0;
        red[1][warp] = d1;
        red[2][warp] = d2;
    }
    __syncthreads();
    if (threadIdx.x < 3) {
        double s = 0.0;
#pragma unroll
        for (int k = 0; k < kMuonhThreads / 32; ++k) s += red[threadIdx.x][k];
        g.partials[threadIdx.x * g.total_blocks + b] = s;
    }
}

// sums[m][k] = the matrix's chunk partials of sum k, in index order (CTA m,
// warp k: lane-strided fp64 sums, then the butterfly).
__global__ void __launch_bounds__(96) muonh_finalize_kernel(const __grid_constant__ MuonhGroup g) {
    pdl_wait();
    pdl_launch_dependents();
    const int m = blockIdx.x, k = threadIdx.x >> 5, lane = threadIdx.x & 31;
    double s = 0.0;
    for (int b = g.block_start[m] + lane; b < g.block_start[m + 1]; b += 32) s += g.partials[k * g.total_blocks + b];
    s = warp_sum_f64(s);
    if (lane == 0) g.sums[3 * m + k] = s;
}

// W <- s (W - c u) on one chunk, c and s from the matrix's sums (fp64, once
// per CTA).
__global__ void __launch_bounds__(kMuonhThreads) muonh_apply_kernel(const __grid_constant__ MuonhGroup g) {
    pdl_wait();
    pdl_launch_dependents();
    const int b = blockIdx.x;
    const int m = matrix_of(g, b);
    __shared__ float cs[2];
    if (threadIdx.x == 0) {
        const double sww = g.sums[3 * m], swu = g.sums[3 * m + 1], suu = g.sums[3 * m + 2];
        const double r = g.radius[m];
        // a zero Muon direction takes no step (the equation divides by ||u||)
        const double c = suu > 0.0 ? g.eta * r / sqrt(suu) : 0.0;
        const double tn2 = sww - 2.0 * c * swu + c * c * suu;  // ||W~||_F^2
        cs[0] = static_cast<float>(c);
        cs[1] = static_cast<float>(r / sqrt(tn2));
    }
    __syncthreads();
    const float c = cs[0], s = cs[1];
    const int64_t c4 = g.chunk4[m];
    const int64_t lo = static_cast<int64_t>(b - g.block_start[m]) * c4;
    const int64_t hi = lo + c4 < g.n4[m] ? lo + c4 : g.n4[m];
    float4 *__restrict__ w = g.w[m];
    const float4 *__restrict__ u = g.u[m];
    uint2 *__restrict__ wb = g.wb[m];
    for (int64_t i = lo + threadIdx.x; i < hi; i += kMuonhThreads) {
        const float4 a = w[i], v = __ldg(u + i);
        float4 r;
        r.x = __fmul_rn(s, fmaf(-c, v.x, a.x));
        r.y = __fmul_rn(s, fmaf(-c, v.y, a.y));
        r.z = __fmul_rn(s, fmaf(-c, v.z, a.z));
        r.w = __fmul_rn(s, fmaf(-c, v.w, a.w));
        w[i] = r;
        if (wb) {
            __nv_bfloat162 l2 = __floats2bfloat162_rn(r.x, r.y), h2 = __floats2bfloat162_rn(r.z, r.w);
            wb[i] = make_uint2(*reinterpret_cast<uint32_t *>(&l2), *reinterpret_cast<uint32_t *>(&h2));
        }
    }
}

bool aligned(const void *p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }
bool valid_scalars(double eta, double radius) {
    return eta >= 0.0 && radius > 0.0 && std::isfinite(eta) && std::isfinite(radius);
}

// Checks one matrix and adds it to the group (n > 0 only).
puro_status_t add_matrix(MuonhGroup &g, float *w, const float *u, void *wb, int64_t n, double radius) {
    if (n < 0 || n % 4) return PURO_ERR_INVALID_ARG;
    if (!w || !u || !aligned(w, 16) || !aligned(u, 16) || !aligned(wb, 8)) return PURO_ERR_INVALID_ARG;
    const int64_t n4 = n / 4;
    const int64_t blocks = static_cast<int64_t>(g.total_blocks) + chunks_of(n4);
    if (blocks > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    const int m = g.count++;
    g.w[m] = reinterpret_cast<float4 *>(w);
    g.u[m] = reinterpret_cast<const float4 *>(u);
    g.wb[m] = static_cast<uint2 *>(wb);
    g.n4[m] = n4;
    g.chunk4[m] = chunk4_of(n4);
    g.radius[m] = radius;
    g.block_start[m] = g.total_blocks;
    g.total_blocks = static_cast<int>(blocks);
    g.block_start[m + 1] = g.total_blocks;
    return PURO_OK;
}

enum MuonhPass { kReduce = 1, kApply = 2 };

cudaError_t run_group(const MuonhGroup &g, int passes, cudaStream_t s) {
    if (g.count == 0) return cudaSuccess;
    if (passes & kReduce) {
        cudaError_t e = launch_pdl(muonh_reduce_kernel, dim3(g.total_blocks), dim3(kMuonhThreads), 0, s, g);
        if (e != cudaSuccess) return e;
        e = launch_pdl(muonh_finalize_kernel, dim3(g.count), dim3(96), 0, s, g);
        if (e != cudaSuccess) return e;
    }
    if (passes & kApply) return launch_pdl(muonh_apply_kernel, dim3(g.total_blocks), dim3(kMuonhThreads), 0, s, g);
    return cudaSuccess;
}

puro_status_t status_of(cudaError_t e) { return e == cudaSuccess ? PURO_OK : PURO_ERR_CUDA; }

}  // namespace
}  // namespace puro

using namespace puro;

#define PURO_MUONH_API extern "C" __attribute__((visibility("default")))

PURO_MUONH_API size_t puro_muonh_workspace_size(int64_t n) {
    return n <= 0 ? 0 : 3 * sizeof(double) * static_cast<size_t>(chunks_of(n / 4));
}

PURO_MUONH_API puro_status_t puro_muonh_reduce(const float *w, const float *u, int64_t n, double *sums,
                                               void *workspace, size_t workspace_bytes, void *stream) {
    if (n < 0 || n % 4) return PURO_ERR_INVALID_ARG;
    if (!sums || !aligned(sums, 8)) return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (n == 0) return status_of(cudaMemsetAsync(sums, 0, 3 * sizeof(double), s));
    if (!workspace || !aligned(workspace, 8) || workspace_bytes < puro_muonh_workspace_size(n))
        return PURO_ERR_INVALID_ARG;
    MuonhGroup g{};
    puro_status_t st = add_matrix(g, const_cast<float *>(w), u, nullptr, n, 1.0);
    if (st != PURO_OK) return st;
    g.partials = static_cast<double *>(workspace);
    g.sums = sums;
    return status_of(run_group(g, kReduce, s));
}

PURO_MUONH_API puro_status_t puro_muonh_apply(float *w, const float *u, int64_t n, const double *sums, double eta,
                                              double radius, void *w_bf16, void *stream) {
    if (n < 0 || n % 4 || !valid_scalars(eta, radius)) return PURO_ERR_INVALID_ARG;
    if (n == 0) return PURO_OK;
    if (!sums || !aligned(sums, 8)) return PURO_ERR_INVALID_ARG;
    MuonhGroup g{};
    puro_status_t st = add_matrix(g, w, u, w_bf16, n, radius);
    if (st != PURO_OK) return st;
    g.eta = eta;
    g.sums = const_cast<double *>(sums);
    return status_of(run_group(g, kApply, static_cast<cudaStream_t>(stream)));
}

PURO_MUONH_API puro_status_t puro_muonh_step(float *w, const float *u, int64_t n, double eta, double radius,
                                             double *sums, void *workspace, size_t workspace_bytes, void *w_bf16,
                                             void *stream) {
    puro_muonh_matrix_t m{w, u, w_bf16, n, radius};
    if (n == 0) return (n % 4 == 0 && valid_scalars(eta, radius)) ? PURO_OK : PURO_ERR_INVALID_ARG;
    return puro_muonh_step_grouped(&m, 1, eta, sums, workspace, workspace_bytes, stream);
}

PURO_MUONH_API size_t puro_muonh_grouped_workspace_size(const puro_muonh_matrix_t *mats, int32_t count) {
    if (!mats || count <= 0) return 0;
    size_t total = 0, batch = 0;
    for (int32_t i = 0; i < count; ++i) {
        batch += static_cast<size_t>(chunks_of(mats[i].n / 4));
        if ((i + 1) % kMaxGroup == 0 || i + 1 == count) {  // launches of kMaxGroup matrices reuse the scratch
            total = batch > total ? batch : total;
            batch = 0;
        }
    }
    return 3 * sizeof(double) * total;
}

PURO_MUONH_API puro_status_t puro_muonh_step_grouped(const puro_muonh_matrix_t *mats, int32_t count, double eta,
                                                     double *sums, void *workspace, size_t workspace_bytes,
                                                     void *stream) {
    if (count < 0 || (count > 0 && !mats)) return PURO_ERR_INVALID_ARG;
    if (!std::isfinite(eta) || !(eta >= 0.0)) return PURO_ERR_INVALID_ARG;
    if (count == 0) return PURO_OK;
    if (!sums || !aligned(sums, 8)) return PURO_ERR_INVALID_ARG;
    for (int32_t i = 0; i < count; ++i)  // every matrix is checked before anything is enqueued
        if (mats[i].n < 0 || mats[i].n % 4 || !valid_scalars(eta, mats[i].radius) ||
            (mats[i].n > 0 && (!mats[i].w || !mats[i].u || !aligned(mats[i].w, 16) || !aligned(mats[i].u, 16) ||
                               !aligned(mats[i].w_bf16, 8))))
            return PURO_ERR_INVALID_ARG;
    if (!workspace || !aligned(workspace, 8) || workspace_bytes < puro_muonh_grouped_workspace_size(mats, count))
        return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    for (int32_t first = 0; first < count; first += kMaxGroup) {
        const int32_t last = first + kMaxGroup < count ? first + kMaxGroup : count;
        MuonhGroup g{};
        g.eta = eta;
        g.partials = static_cast<double *>(workspace);
        int32_t i = first;
        while (i < last) {  // runs of non-empty matrices share a launch; empty ones get zero sums
            if (mats[i].n == 0) {
                cudaError_t e = cudaMemsetAsync(sums + 3 * i, 0, 3 * sizeof(double), s);
                if (e != cudaSuccess) return PURO_ERR_CUDA;
                ++i;
                continue;
            }
            g = MuonhGroup{};
            g.eta = eta;
            g.partials = static_cast<double *>(workspace);
            g.sums = sums + 3 * i;
            while (i < last && mats[i].n > 0) {
                puro_status_t st = add_matrix(g, mats[i].w, mats[i].u, mats[i].w_bf16, mats[i].n, mats[i].radius);
                if (st != PURO_OK) return st;
                ++i;
            }
            cudaError_t e = run_group(g, kReduce | kApply, s);
            if (e != cudaSuccess) return PURO_ERR_CUDA;
        }
    }
    return PURO_OK;
}
