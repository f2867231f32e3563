// internal.h -- declarations shared by the CUDA translation units of the
// FP8 linear-path library (not part of the public C ABI).
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <cstddef>
#include <cstdint>

#include "puro_fp8.h"

namespace puro {

// Launch `kern` on `s` with programmatic stream serialisation (the kernel
// calls pdl_wait() before touching global memory; see ptx.cuh).
template <typename... KArgs, typename... Args>
inline cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, size_t smem, cudaStream_t s,
                              Args &&...args) {
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = grid;
    cfg.blockDim = block;
    cfg.dynamicSmemBytes = smem;
    cfg.stream = s;
    cudaLaunchAttribute attr;
    attr.id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr.val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = &attr;
    cfg.numAttrs = 1;
    return cudaLaunchKernelEx(&cfg, kern, static_cast<Args &&>(args)...);
}


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
    int32_t *status;          // optional device status word (PURO_ERR_TIMEOUT when a tile load is given up)
    uint64_t wait_ns;         // bound on each tile-load wait
};

cudaError_t launch_amax(const uint16_t *x, int64_t n, uint32_t *amax, cudaStream_t s);

// Many weights quantised in one launch (128x128 blocks, optional transposed
// copies): each weight's three tensor maps (as puro_fp8_quantize builds them)
// and scale-vector pointers travel in the kernel's parameter block, so one
// launch takes at most kWeightGroupMax weights.
constexpr int kWeightGroupMax = 64;
struct WeightGroup {
    CUtensorMap x[kWeightGroupMax], q[kWeightGroupMax], qt[kWeightGroupMax];
    uint8_t *scale[kWeightGroupMax], *scale_t[kWeightGroupMax];
    int tile_start[kWeightGroupMax + 1];  // first 128x128 tile of each weight; [count] = all tiles
    int tiles_n[kWeightGroupMax];         // column tiles of each weight (cols / 128)
    int kb_rows[kWeightGroupMax];         // rows / 128 (k-blocks of the transposed copy)
    int count;
    int32_t *status;                      // optional device status word
    uint64_t wait_ns;                     // bound on each tile-load wait
};
cudaError_t launch_quantize_weights(const WeightGroup &g, int fmt, bool has_t, cudaStream_t s);

// Producers fused ahead of the activation quantiser.
enum QuantProd : int {
    kProdNone = 0,
    kProdRmsNorm = 1,  // y = bf16((h * rstd[row]) * gamma[col])
    kProdSwiGlu = 2,   // y = bf16(silu(gate) * up)
};
struct ProdArgs {
    const float *rstd;      // kProdRmsNorm: [rows]
    const uint16_t *gamma;  // kProdRmsNorm: bf16 [cols], or null (no gain)
    bool write_y;           // also store y (through tm_y)
    const uint16_t *up;     // kProdSwiGlu: bf16 [rows, cols], rows ld elements apart
    int64_t ld;             // kProdSwiGlu: row stride of up (and of the gate tm_x maps)
};

// rstd[r] = 1 / sqrt(mean(h[r,:]^2) + eps) (cols a multiple of 8).
cudaError_t launch_rmsnorm_rstd(const uint16_t *h, int64_t rows, int64_t cols, float eps, float *rstd, cudaStream_t s);
// y = bf16((h * rstd) * gamma), the unfused application.
cudaError_t launch_rmsnorm_apply(const uint16_t *h, int64_t rows, int64_t cols, const float *rstd,
                                 const uint16_t *gamma, uint16_t *y, cudaStream_t s);

// tm_x: bf16 [rows, cols], box {128, 128}, no swizzle.
// tm_q: u8 [rows, cols], box {128, 128}, no swizzle.
// tm_qt: u8 [cols, rows], box {128, 128}, 128-byte swizzle (only if has_t).
cudaError_t launch_quantize(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                            const CUtensorMap &tm_qt, cudaStream_t s);

// The activation quantiser fed by RMSNorm (a.kind must be kQuantBlockAct):
// tm_x maps h; tm_y (bf16 [rows, cols], box {128, 128}, no swizzle) is
// written only when prod.write_y.
cudaError_t launch_quantize_rmsnorm(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                    const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                    cudaStream_t s);

// The activation quantiser fed by SwiGLU (a.kind must be kQuantBlockAct, rows
// and cols multiples of 128): tm_x maps the gate (bf16 [rows, cols], row
// stride prod.ld elements), prod.up the up projection with the same stride.
cudaError_t launch_quantize_swiglu(const QuantArgs &a, const CUtensorMap &tm_x, const CUtensorMap &tm_q,
                                   const CUtensorMap &tm_qt, const CUtensorMap &tm_y, const ProdArgs &prod,
                                   cudaStream_t s);
// y = bf16(silu(gate) * up), the unfused application (cols a multiple of 8;
// gate and up rows ld elements apart, y contiguous).
cudaError_t launch_swiglu_apply(const uint16_t *gate, const uint16_t *up, int64_t rows, int64_t cols, int64_t ld,
                                uint16_t *y, cudaStream_t s);

// Writes only the per-tensor scale_inv (used for empty tensors).
cudaError_t launch_tensor_scale_only(const QuantArgs &a, cudaStream_t s);

// Operand kinds of the tensor-core GEMM D[M,N] = A[M,K] * B[N,K]^T.
enum GemmKind : int {
    kGemmBF16 = 0,       // kind::f16, bf16 operands
    kGemmFP8Tensor = 1,  // kind::f8f6f4, per-tensor scale_inv product in the epilogue
    kGemmFP8Block = 2,   // kind::mxf8f6f4 with E8M0 group scales
};

// Output forms of the GEMM kernel.
enum GemmOut : int {
    kGemmOutBF16 = 0,        // D in BF16
    kGemmOutF32Partial = 1,  // FP32 partial tiles of a split reduction (workspace)
    kGemmOutF32Add = 2,      // D (FP32) += the product (main-grad accumulation)
    kGemmOutQuant = 3,       // D rounded to BF16, then its blockwise FP8 copies (block kind, 256-wide, unsplit)
};

struct GemmArgs {
    GemmKind kind;
    int a_fmt, b_fmt;            // FP8 formats (0 = E4M3, 1 = E5M2)
    int64_t M, N, K;
    int tile_n;                  // 256, or 224 (block kind, unsplit; see choose_tile_n)
    // kGemmFP8Block: scale vectors of B (the 224-wide form gathers them
    // itself; the 256-wide form loads them through GemmMaps::sfb).
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
    // out is an FP32 main-grad [M, N] that receives out += A * B^T (block
    // or per-tensor kinds; 256-wide tiles)
    bool accumulate_f32;
    // kGemmOutQuant (block kind): the epilogue quantises bf16(D) into the
    // rowwise copy q [M, N] (scales q_scale) and, when qt is set, the
    // transposed copy qt [N, M] (scales qt_scale), in format q_fmt; D itself
    // is stored in BF16 only when d_bf16 is set.
    bool quant_out;
    int q_fmt;
    uint8_t *q, *q_scale, *qt, *qt_scale;
    void *d_bf16;
};

// Tensor maps of one GEMM launch.
//   a:   A [M, K] (128-byte swizzle, box {128 bytes, 128 rows})
//   b:   B [N, K] (box {128 bytes, tile_n / 2 rows}: half of a tile per CTA)
//   d:   D [M, N] bf16 (tile_n 256: 128-byte swizzle, box {64, 32};
//        tile_n 224: 64-byte swizzle, box {32, 32}); with accumulate_f32, the
//        FP32 main-grad [M, N] (128-byte swizzle, box {32, 32})
//   ws:  workspace [splits * splitk_rows_per_chunk(M), N] fp32 (128-byte
//        swizzle, box {32, 32}); only read when g.splits > 1
//   sfa, sfb (kGemmFP8Block only): the scale vectors of A / B,
//        [rows/128][ceil(K/512)][512] bytes viewed as uint32
//        [rows/128 * ceil(K/512), 128], box {128, 1}
struct GemmMaps {
    CUtensorMap a, b, d, ws, sfa, sfb;
};

cudaError_t launch_gemm(const GemmArgs &g, const GemmMaps &m, cudaStream_t s);
// Two block-scaled GEMMs with BF16 output in one launch (the Dgrad and Wgrad
// of one linear): 256-wide tiles, neither reduction split.
cudaError_t launch_gemm_grouped(const GemmArgs &g0, const GemmMaps &m0, const GemmArgs &g1, const GemmMaps &m1,
                                cudaStream_t s);

// The FP8 GEMM entry behind puro_fp8_linear_{fprop,dgrad,wgrad}: validates,
// encodes the tensor maps and launches (D = A * B^T).
puro_status_t fp8_gemm_entry(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, void *d, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, void *stream);

// The host-side argument checks of fp8_gemm_entry alone (no CUDA call).
puro_status_t fp8_gemm_validate(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, const void *d);

// Split count the GEMM uses for a shape (1: no split), and the workspace it
// then needs.  Host-only, shape-only (plans for 152 SMs).
int choose_splits(int64_t M, int64_t N, int64_t K, bool bf16);
size_t splitk_workspace_bytes(int64_t M, int64_t N, int64_t K, bool bf16);
int64_t splitk_rows_per_chunk(int64_t M);  // M rounded up to a whole 256-row pair tile
// Whether a linear's Dgrad (dX [M, K], reduction N) and Wgrad (dW [N, K],
// reduction M) are modelled faster as one grouped launch (balanced
// schedule, Wgrad unsplit) than as two launches with the Wgrad split into
// w_splits chunks.  Host-only, shape-only.
bool grouped_backward_faster(int64_t M, int64_t N, int64_t K, int w_splits);
// Tile width (256 or 224) of an unsplit block-scaled GEMM: modelled waves x
// per-tile time of the two forms.  Host-only, shape-only.
int choose_tile_n(int64_t M, int64_t N, int64_t K);

// Tile shape of the GEMM kernel: rows of A per CTA (a CTA pair computes
// 2 * kGemmBM rows), columns of a tile (rows of B per pair), and the bytes
// of K per pipeline stage (one 128-byte swizzle row).
constexpr int kGemmBM = 128;
constexpr int kGemmBN = 256;
constexpr int kGemmBKBytes = 128;

}  // namespace puro
