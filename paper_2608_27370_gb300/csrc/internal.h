// internal.h -- declarations shared by the CUDA translation units of the
// FP8 linear-path library (not part of the public C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>

#include "puro_fp8.h"

namespace puro {

// How a quantiser groups values (section "FP8 Mixed-Precision Training").
enum QuantKind : int {
    kQuantBlockAct = 0,     // 1x128 groups along cols (q) and along rows (q_t)
    kQuantBlockWeight = 1,  // 128x128 blocks; q_t = transposed codes
    kQuantTensor = 2,       // one scale for the whole tensor
};

struct QuantArgs {
    const uint16_t *x;        // bf16 [rows, cols]
    int64_t rows, cols;
    int fmt;                  // 0 = E4M3, 1 = E5M2
    QuantKind kind;
    const uint32_t *amax;     // kQuantTensor only
    uint8_t *scale_u8;        // block scale vectors of q (tensor-core layout)
    uint8_t *scale_t_u8;      // block scale vectors of q_t (tensor-core layout)
    float *scale_f;           // tensor scale_inv for q
    float *scale_t_f;         // tensor scale_inv for q_t (may be null)
    bool has_t;
};

cudaError_t launch_amax(const uint16_t *x, int64_t n, uint32_t *amax, cudaStream_t s);

// tm_x: bf16 [rows, cols], box {128, 128}, no swizzle.
// tm_q: u8 [rows, cols], box {128, 128}, no swizzle.
// tm_qt: u8 [cols, rows], box {128, 128}, 128-byte swizzle (only if has_t).
cudaError_t launch_quantize(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                            const CUtensorMap &tm_qt, cudaStream_t s);

// Writes only the per-tensor scale_inv (used for empty tensors).
cudaError_t launch_tensor_scale_only(const QuantArgs &a, cudaStream_t s);

// Operand kinds of the tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T.
enum GemmKind : int {
    kGemmBF16 = 0,       // kind::f16, bf16 operands
    kGemmFP8Tensor = 1,  // kind::f8f6f4, per-tensor scale_inv product in the epilogue
    kGemmFP8Block = 2,   // kind::mxf8f6f4 with E8M0 group scales
};

struct GemmArgs {
    GemmKind kind;
    int a_fmt, b_fmt;            // FP8 formats (0 = E4M3, 1 = E5M2)
    int64_t M, N, K;
    // kGemmFP8Block: scale vectors of A and B in the tensor-core layout,
    // [rows/128][ceil(K/512)][512] bytes each.
    const uint8_t *sfa;
    const uint8_t *sfb;
    // kGemmFP8Tensor: dequantisation factors of A and B.
    const float *sia, *sib;
    int32_t *status;             // optional device status word
    uint64_t wait_timeout_ns;
    int num_sms;
    // split reduction (FP8 kinds only): splits > 1 needs `workspace` of
    // splitk_workspace_bytes(M, N, K) bytes; `out` is D (bf16)
    int splits;
    void *workspace;
    void *out;
};

// tm_a: A [M, K], tm_b: B [N, K] (128-byte swizzle, box {128 bytes, rows}),
// tm_d: D [M, N] bf16 (128-byte swizzle, box {64, 32}),
// tm_ws: workspace [splits * M, N] fp32 (128-byte swizzle, box {32, 32});
// only read when g.splits > 1.
cudaError_t launch_gemm(const GemmArgs &g, const CUtensorMap &tm_a, const CUtensorMap &tm_b,
                        const CUtensorMap &tm_d, const CUtensorMap &tm_ws, cudaStream_t s);

// The FP8 GEMM entry behind puro_fp8_linear_{fprop,dgrad,wgrad}: validates,
// encodes the tensor maps and launches (D = A * B^T).
puro_status_t fp8_gemm_entry(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, void *d, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, void *stream);

// Split count the GEMM uses for a shape (1: no split), and the workspace it
// then needs.  Host-only, shape-only (plans for 152 SMs).
int choose_splits(int64_t M, int64_t N, int64_t K, bool bf16);
size_t splitk_workspace_bytes(int64_t M, int64_t N, int64_t K, bool bf16);

// Tile shape of the GEMM kernel (rows of A per CTA tile, rows of B) and the
// bytes of K per pipeline stage (128: 4 stages, 128-byte swizzle; 64: 8
// stages, 64-byte swizzle).
constexpr int kGemmBM = 128;
constexpr int kGemmBN = 256;
constexpr int kGemmBKBytes = 128;

}  // namespace puro
