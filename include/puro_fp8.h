/*
 * puro_fp8.h -- C ABI of the GB300 (sm_103a) FP8 linear-layer training path.
 *
 * The method (Puro-2B, section "FP8 Mixed-Precision Training"; appendix
 * "Production Training Details", paragraph "FP8 implementation pipeline"
 * and its precision-flow figure):
 *   - every Transformer linear layer runs its three GEMMs -- Fprop
 *     Y = X W^T, Dgrad dX = dY W, Wgrad dW = dY^T X -- from FP8 operands,
 *     accumulates in FP32 and writes a BF16 output;
 *   - operands are E4M3; inputs and weights are quantised from BF16
 *     just ahead of the GEMM, with scales computed online per local
 *     group: 1x128 groups along the GEMM reduction dimension for activations
 *     and activation gradients, 128x128 blocks for weights;
 *   - each group scale is a power of two (E8M0 expressiveness);
 *   - the quantised input is kept for Wgrad.
 * A per-tensor (a single scale per tensor, the contrast drawn in the
 * same section) mode and the E5M2 format are provided as well.
 *
 * Conventions for every entry point
 *   - Ownership: the caller allocates and owns every buffer.  The library
 *     allocates no memory, never synchronises the stream (except
 *     puro_fp8_get_status, which says so) and keeps no state between calls.
 *   - Ordering: all work is enqueued on `stream` (a cudaStream_t passed as
 *     void*; NULL is the legacy default stream) in call order.
 *   - Pointers: device pointers unless marked "host".  Every tensor pointer
 *     must be 16-byte aligned.
 *   - Errors: argument violations are detected on the host before anything
 *     is enqueued and return PURO_ERR_INVALID_ARG or PURO_ERR_UNSUPPORTED;
 *     a failed launch returns PURO_ERR_CUDA.  No entry point traps or
 *     asserts on the device.  Non-finite data is carried in-band (NaN codes,
 *     E8M0 0xFF, NaN scale_inv).  A GEMM or quantiser kernel whose wait on
 *     the device exceeds its bound (puro_set_wait_timeout_ns) stops working
 *     on its tiles, lets its own copies in flight land, exits cleanly and
 *     stores PURO_ERR_TIMEOUT in *dev_status when dev_status is non-NULL;
 *     the outputs of such a call are then incomplete.
 *   - Layout: every tensor is row-major and dense.  A quantised GEMM operand
 *     is stored [rows, red] with the reduction dimension `red` contiguous;
 *     all three GEMMs read both operands this way ("TN"), which is why the
 *     quantiser can emit a transposed copy.
 *
 * Scale layouts
 *   PURO_SCALE_TENSOR : `scale` is one float, the dequantisation factor
 *                       scale_inv = fp32(1 / fp32(fmt_max / amax)).
 *   PURO_SCALE_BLOCK  : uint8 E8M0 exponents g (scale 2^(g-127)) stored as
 *                       the tensor cores read them ("scale vectors"): for an
 *                       operand [rows, red], KB = red/128 k-blocks in
 *                       KG = ceil(KB/4) groups, the buffer is
 *                       [rows/128][KG][512] bytes and byte
 *                           16*l + 4*j + b   of chunk (rb, kg)
 *                       holds g of row 128*rb + 32*j + l, k-block 4*kg + b
 *                       (l < 32, j < 4, b < 4); bytes of k-blocks >= KB are
 *                       127.  One 512-byte chunk is exactly the 32-line x
 *                       16-byte image tcgen05.cp loads for 128 rows, and b is
 *                       the MMA scale id.
 *                       role ACT: g of the 1x128 group (row, k-block).
 *                       role WEIGHT: g of the 128x128 block (row/128,
 *                       k-block), i.e. repeated over the block's rows.
 *                       Size: rows * KG * 4 bytes (puro_fp8_scale_bytes).
 *   g = 0xFF marks a group that held Inf or NaN; its codes are NaN.
 */
#ifndef PURO_FP8_H
#define PURO_FP8_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum {
    PURO_OK = 0,
    PURO_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad shape, bad enum */
    PURO_ERR_UNSUPPORTED = 2,  /* valid request this build does not implement */
    PURO_ERR_CUDA = 3,         /* a CUDA runtime/driver call failed */
    PURO_ERR_TIMEOUT = 4       /* device-side bounded wait expired (see dev_status) */
} puro_status_t;

typedef enum { PURO_E4M3 = 0, PURO_E5M2 = 1 } puro_fp8_format_t;
typedef enum { PURO_SCALE_TENSOR = 0, PURO_SCALE_BLOCK = 1 } puro_scaling_t;
typedef enum { PURO_ROLE_ACT = 0, PURO_ROLE_WEIGHT = 1 } puro_role_t;

/* One quantised GEMM operand, as produced by puro_fp8_quantize. */
typedef struct {
    const uint8_t *data;  /* device, [rows, red] FP8 codes, row-major        */
    const void *scale;    /* device, layout per `scaling` and `role` above   */
    int64_t rows;         /* non-reduction extent                            */
    int64_t red;          /* reduction extent (contiguous)                   */
    int32_t fmt;          /* puro_fp8_format_t                               */
    int32_t scaling;      /* puro_scaling_t                                  */
    int32_t role;         /* puro_role_t (BLOCK only; ignored for TENSOR)    */
    int32_t reserved;     /* must be 0                                       */
} puro_fp8_tensor_t;

/*
 * amax: max |x| over a BF16 tensor -- the online scale statistic of the
 * section "FP8 Mixed-Precision Training" ("compute scales online").
 *   x         : device, [rows, cols] bf16, 16-byte aligned.
 *   amax_bits : device, one uint32.  The call zeroes it (stream-ordered)
 *               and then writes the bf16 bit pattern of max |x| (sign
 *               cleared) into its low 16 bits.  Computed as an integer max
 *               of (bits & 0x7FFF): exact, order independent, and NaN
 *               propagating (any NaN gives a value > 0x7F80).
 * rows == 0 or cols == 0 is valid and yields 0.
 */
puro_status_t puro_fp8_amax(const void *x, int64_t rows, int64_t cols,
                            uint32_t *amax_bits, void *stream);

/*
 * quantize: BF16 -> FP8 with online scales (section "FP8 Mixed-Precision
 * Training"), optionally emitting the transposed copy that Wgrad consumes
 * (same section: the quantised input is kept for Wgrad).
 *   x        : device [rows, cols] bf16.
 *   fmt      : PURO_E4M3 or PURO_E5M2.
 *   scaling  : PURO_SCALE_BLOCK (the paper's recipe) or PURO_SCALE_TENSOR.
 *   role     : BLOCK only.  ACT: 1x128 groups along cols for q and along
 *              rows for q_t.  WEIGHT: 128x128 blocks; q_t holds exactly the
 *              transposed codes and scale_t the transposed grid.
 *   amax_bits: TENSOR only: device uint32 written by puro_fp8_amax on this
 *              same x; NULL in BLOCK mode.
 *   q, scale : rowwise copy [rows, cols] and its scales (layouts above).
 *   q_t, scale_t : optional transposed copy [cols, rows] and its scales.
 *              BLOCK: both NULL or both non-NULL.  TENSOR: scale_t may be
 *              NULL; when given it receives the same scale_inv.
 * Codes: code = RNE_satfinite(x * 2^(127-g)) in BLOCK mode, where g is the
 * smallest exponent with amax <= fmt_max * 2^(g-127) (clamped to [0,254]);
 * code = RNE_satfinite(fp32(x * scale)) in TENSOR mode, scale =
 * fp32(fmt_max / amax) (1 if amax == 0, FLT_MAX if the quotient overflows).
 * Negative values that round to zero give -0 (0x80).
 * Shapes: BLOCK needs rows % 128 == 0 and cols % 128 == 0.  TENSOR needs
 * cols % 16 == 0, and rows % 16 == 0 when q_t is requested.  An empty
 * tensor (rows or cols 0) writes no codes, so x, q and q_t may be NULL;
 * in TENSOR mode it still writes scale_inv = 1 (amax of nothing is 0).
 * dev_status: optional device int32, written only when a tile-load wait on
 *   the device runs out (PURO_ERR_TIMEOUT); the caller zeroes it.
 */
puro_status_t puro_fp8_quantize(const void *x, int64_t rows, int64_t cols,
                                int32_t fmt, int32_t scaling, int32_t role,
                                const uint32_t *amax_bits,
                                uint8_t *q, void *scale,
                                uint8_t *q_t, void *scale_t,
                                int32_t *dev_status, void *stream);

/*
 * Many weights quantised in one call.
 *
 * The weights are quantised once per optimizer step (section "FP8
 * Mixed-Precision Training": 128x128 blocks, the transposed copy sharing
 * the block scales), so a caller can quantise all of a model's weights at
 * once.  Each entry is quantised exactly as
 *     puro_fp8_quantize(w, rows, cols, fmt, PURO_SCALE_BLOCK,
 *                       PURO_ROLE_WEIGHT, NULL, q, scale, q_t, scale_t)
 * would, with the same codes and scales bit for bit, but the tiles of up to
 * 64 weights share one launch (more weights: one launch per 64).
 *   w: bf16 [rows, cols] row-major, 16-byte aligned; rows and cols
 *     multiples of 128 (an entry with rows or cols 0 is skipped).
 *   q, scale: the rowwise copy [rows, cols] and its scale vectors
 *     (puro_fp8_scale_bytes(rows, cols) bytes).
 *   q_t, scale_t: the transposed copy [cols, rows] and its scale vectors,
 *     or both NULL; either every non-empty entry has a transposed copy or
 *     none does.
 * fmt: PURO_E4M3 or PURO_E5M2 for all entries.  The table is read on the
 * host during the call (it may be freed on return); every entry is checked
 * before anything is enqueued.  dev_status: as in puro_fp8_quantize.
 */
typedef struct {
    const void *w;
    int64_t rows, cols;
    uint8_t *q;
    void *scale;
    uint8_t *q_t;
    void *scale_t;
} puro_fp8_weight_t;

puro_status_t puro_fp8_quantize_weights(const puro_fp8_weight_t *weights, int32_t count, int32_t fmt,
                                        int32_t *dev_status, void *stream);

/*
 * RMSNorm fused ahead of the blockwise activation quantiser.
 *
 * The model normalises the hidden states with RMSNorm before the attention
 * and MLP projections (section "Model architecture and pretraining system":
 * the Qwen3 architecture); this entry point takes the pre-norm rows h and
 * emits the FP8 operands of the projection directly:
 *     rstd[r] = 1 / sqrt(mean_k h[r,k]^2 + eps)     (fp32, written)
 *     y[r,k]  = bf16((h[r,k] * rstd[r]) * gamma[k])  (fp32 products)
 * and then quantises y exactly as puro_fp8_quantize does with
 * PURO_SCALE_BLOCK / PURO_ROLE_ACT (1x128 groups, optional transposed copy).
 *   h: bf16 [rows, cols]; rows and cols multiples of 128; 16-byte aligned.
 *   gamma: bf16 [cols] gain, or NULL for none.
 *   eps >= 0.
 *   rstd: fp32 [rows], written (kept for the RMSNorm backward).
 *   y: bf16 [rows, cols], or NULL: y itself is written only when asked.
 *   q, scale, q_t, scale_t, dev_status: as in puro_fp8_quantize.
 * rstd is an fp32 sum of squares in a fixed order, so it agrees with an
 * exact computation to within a few fp32 ulps; y and every code and scale
 * are then exactly determined by rstd.  Two kernels on `stream`; h is read
 * twice (the second time largely from L2).
 */
puro_status_t puro_fp8_quantize_rmsnorm(const void *h, int64_t rows, int64_t cols, const void *gamma, float eps,
                                        int32_t fmt, float *rstd, void *y, uint8_t *q, void *scale, uint8_t *q_t,
                                        void *scale_t, int32_t *dev_status, void *stream);

/*
 * The same RMSNorm without the quantiser: rstd and y (bf16) as above, cols
 * a multiple of 8.  The unfused comparison for the fused entry point.
 */
puro_status_t puro_rmsnorm_bf16(const void *h, int64_t rows, int64_t cols, const void *gamma, float eps,
                                float *rstd, void *y, void *stream);

/*
 * SwiGLU fused ahead of the blockwise activation quantiser.
 *
 * The model's MLP is gated (section "Model architecture and pretraining
 * system": the Qwen3 architecture): the down projection receives
 *     y[r,k] = bf16(silu(gate[r,k]) * up[r,k]),   silu(g) = g / (1 + e^-g),
 * evaluated in fp32 (sigmoid from e^-|g|, so nothing overflows; the
 * exponential and the reciprocal are single special-function instructions,
 * with subnormal values of e^-|g| kept by an exact power-of-two scaling).
 * This entry
 * point quantises y exactly as puro_fp8_quantize does with PURO_SCALE_BLOCK /
 * PURO_ROLE_ACT (1x128 groups, optional transposed copy) without writing y,
 * which the MLP's backward does not need (it keeps gate and up).
 *   gate, up: bf16 [rows, cols] with rows ld elements apart (ld >= cols, a
 *     multiple of 8): the two halves of one [rows, 2*cols] gate/up output are
 *     passed as gate = out, up = out + cols, ld = 2*cols.  16-byte aligned.
 *   rows and cols multiples of 128.
 *   y: bf16 [rows, cols] contiguous, or NULL: written only when asked.
 *   q, scale, q_t, scale_t, dev_status: as in puro_fp8_quantize.
 * Every code and scale is an exact function of y.  y itself agrees with the
 * exactly rounded silu(gate) * up to within one bf16 ulp, and equals it for
 * all but about 1e-5 of typical inputs.  One kernel on `stream`; gate and up
 * are each read once.
 */
puro_status_t puro_fp8_quantize_swiglu(const void *gate, const void *up, int64_t rows, int64_t cols, int64_t ld,
                                       int32_t fmt, void *y, uint8_t *q, void *scale, uint8_t *q_t, void *scale_t,
                                       int32_t *dev_status, void *stream);

/*
 * The same SwiGLU without the quantiser: y (bf16, contiguous [rows, cols]) as
 * above, cols a multiple of 8.  The unfused comparison for the fused entry
 * point.
 */
puro_status_t puro_swiglu_bf16(const void *gate, const void *up, int64_t rows, int64_t cols, int64_t ld, void *y,
                               void *stream);

/*
 * The three FP8 GEMMs of a linear layer with weight W [N, K], input X [M, K]
 * and output gradient dY [M, N] (appendix "FP8 implementation pipeline":
 * Fprop, Dgrad and Wgrad all use blockwise E4M3 operands).  Each computes
 *     D[i, j] = sum_r sA(i, r) sB(j, r) qA[i, r] qB[j, r]
 * with FP32 accumulation on the tensor cores and BF16 (RNE) output, where
 * the scales are the E8M0 group scales (BLOCK) or the two scale_inv values
 * (TENSOR, applied in the epilogue).
 *   fprop: A = x   (Xq   [M, K], ACT)    B = w   (Wq   [N, K], WEIGHT)  -> y  [M, N]
 *   dgrad: A = dy  (dYq  [M, N], ACT)    B = w_t (Wq^T [K, N], WEIGHT)  -> dx [M, K]
 *   wgrad: A = dy_t(dYq^T[N, M], ACT)    B = x_t (Xq^T [K, M], ACT)     -> dw [N, K]
 * (the GEMM itself does not depend on the roles: every BLOCK operand carries
 * per-row scale vectors).
 * Both operands must use the same `scaling`.  BLOCK: all extents multiples
 * of 128.  TENSOR: extents multiples of 16.  A zero reduction extent writes
 * zeros; a zero output extent is a no-op.
 *   workspace, workspace_bytes: optional scratch (may be NULL/0), 16-byte
 *     aligned.  When the output has fewer 128x256 tiles than the GPU has
 *     SMs and at least puro_fp8_workspace_size(...) bytes are given, the
 *     reduction is split into chunks whose FP32 partial tiles go to the
 *     workspace and are summed (in fixed chunk order, then rounded once to
 *     BF16) by a second kernel on the same stream.  Results are within the
 *     output tolerance either way, and deterministic for a given split.
 *     The workspace is only written, never read before being written.
 *   dev_status: optional device int32, written only on a device-side
 *     timeout (PURO_ERR_TIMEOUT).  The caller zeroes it.
 */
puro_status_t puro_fp8_linear_fprop(const puro_fp8_tensor_t *x, const puro_fp8_tensor_t *w,
                                    void *y, void *workspace, size_t workspace_bytes,
                                    int32_t *dev_status, void *stream);
puro_status_t puro_fp8_linear_dgrad(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t,
                                    void *dx, void *workspace, size_t workspace_bytes,
                                    int32_t *dev_status, void *stream);
puro_status_t puro_fp8_linear_wgrad(const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t,
                                    void *dw, void *workspace, size_t workspace_bytes,
                                    int32_t *dev_status, void *stream);

/*
 * Dgrad and Wgrad of one linear in one call.
 *
 *   dx = dy * w_t^T     (as puro_fp8_linear_dgrad)
 *   dw = dy_t * x_t^T   (as puro_fp8_linear_wgrad)
 * The two are independent (both need only the quantised output gradient),
 * so when both run as unsplit 256-wide block-scaled GEMMs they share one
 * persistent launch: the tiles of the GEMM with the longer reduction first,
 * then the other's.  Where the long tiles do not divide evenly over the CTA
 * pairs, the pairs with one long tile fewer first take about a long tile's
 * worth of short ones, so the pairs finish together.  A Wgrad that would
 * split its reduction with the given workspace joins the Dgrad unsplit in
 * such a launch when that is modelled faster (it is for every linear of the
 * Qwen2-1.5B and Qwen3-1.7B shapes at their token counts).  Each output of a
 * grouped launch is bit-identical to the separate call's without a
 * workspace.  Otherwise (per-tensor scaling, a split reduction, the
 * 224-wide tile form, an empty extent) the two GEMMs are launched one after
 * the other, exactly as the separate entry points would.  Arguments as for
 * those entry points; one workspace serves both (its bytes: the larger of
 * the two puro_fp8_workspace_size values).  Both are validated before
 * anything is enqueued.
 */
puro_status_t puro_fp8_linear_backward(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t, void *dx,
                                       const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw,
                                       void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                       void *stream);

/*
 * Dgrad with the next quantisation fused into its epilogue.
 *
 * The backward pass carries the output gradient of one linear, through the
 * elementwise steps between layers, to the output gradient dY of the linear
 * before it, and the FP8 pipeline quantises that dY twice: rowwise for the
 * layer's Dgrad and transposed for its Wgrad (appendix "FP8 implementation
 * pipeline"; section "FP8 Mixed-Precision Training": activation gradients
 * in E4M3 with 1x128 groups along the reduction dimension).  Where the Dgrad
 * output is that next dY, this entry point computes
 *     dx = dy * w_t^T        (as puro_fp8_linear_dgrad; BLOCK scaling only)
 * and quantises bf16(dx) in the GEMM's epilogue, writing exactly what
 * puro_fp8_quantize(dx, M, K, fmt, PURO_SCALE_BLOCK, PURO_ROLE_ACT, ...)
 * writes from the same BF16 values:
 *   dxq [M, K] u8, dxq_scale: 1x128 groups along K (the scale layout of a
 *     BLOCK operand [M, K], puro_fp8_scale_bytes(M, K) bytes);
 *   dxq_t [K, M] u8, dxq_t_scale: groups of 128 rows of dx, stored
 *     transposed (operand [K, M], puro_fp8_scale_bytes(K, M) bytes), or both
 *     NULL for no transposed copy;
 *   dx: bf16 [M, K], or NULL: then the BF16 product is not written;
 *   fmt: PURO_E4M3 or PURO_E5M2, the format of both copies.
 * dy, w_t: as in puro_fp8_linear_dgrad (both BLOCK; M, N, K multiples of
 * 128).  The reduction is never split (no workspace).  All pointers 16-byte
 * aligned.  dx, when written, equals puro_fp8_linear_dgrad's output for an
 * unsplit reduction, bit for bit, and every code and scale is an exact
 * function of those BF16 values.  One kernel on `stream`; K == 0 gives zero
 * codes with exponent 127 (memsets).  dev_status as for the GEMMs.
 */
puro_status_t puro_fp8_linear_dgrad_quantize(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t,
                                             int32_t fmt, void *dx, uint8_t *dxq, void *dxq_scale,
                                             uint8_t *dxq_t, void *dxq_t_scale, int32_t *dev_status,
                                             void *stream);

/*
 * Wgrad accumulated into an FP32 main-grad:
 *     main_grad[n, k] += sum_m sA(n, m) sB(k, m) qA[n, m] qB[k, m]
 * (appendix "FP8 implementation pipeline": the weight gradient is
 * accumulated in FP32 across micro-batches, the main-grad of the optimizer).
 * Same operands, scaling rules and workspace as puro_fp8_linear_wgrad;
 * main_grad is FP32 [N, K], row-major, 16-byte aligned, read and written.
 * Each element receives exactly one FP32 addition per call (of the FP32
 * product, or of the fixed-order sum of the split partials), so results are
 * deterministic.  A zero reduction extent leaves main_grad unchanged.
 */
puro_status_t puro_fp8_linear_wgrad_main_grad(const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t,
                                              float *main_grad, void *workspace, size_t workspace_bytes,
                                              int32_t *dev_status, void *stream);

/*
 * Wgrad without allocation and without caller-supplied scratch.
 *
 * The paper has no counterpart to this entry point; it serves callers that
 * cannot allocate device memory while they run the backward pass -- plugin
 * hosts that own every device buffer and forbid allocations in their
 * execution callbacks, latency-critical code that cannot afford
 * cudaMalloc's device-wide synchronisation, or callers with a fixed memory
 * budget -- and so cannot provide the scratch puro_fp8_linear_wgrad's
 * split-reduction schedule wants.
 *
 * Same operands, output and results as puro_fp8_linear_wgrad with a large
 * enough workspace.  The scratch is a fixed PURO_NOALLOC_SCRATCH_BYTES
 * (40 MiB) array inside the library's device image, held by every GPU that
 * loads the library until the process exits; no cudaMalloc, cudaFree or
 * allocating library call is made.
 *   - Arguments are checked exactly as puro_fp8_linear_wgrad checks them
 *     (PURO_ERR_INVALID_ARG for a malformed call); then a shape whose split
 *     schedule needs more than PURO_NOALLOC_SCRATCH_BYTES (see
 *     puro_fp8_workspace_size) returns PURO_ERR_UNSUPPORTED.  Both before
 *     any work is enqueued.
 *   - The first call on each device looks up the array's device address
 *     (cudaGetSymbolAddress) with that device current and caches it for the
 *     life of the process; make that first call before any stream capture
 *     begins.  The cached address belongs to the device's current context:
 *     after cudaDeviceReset (or any other teardown of that context) it is
 *     stale, and this entry point must not be called again in the process.
 *   - All calls share the one array, which keeps the last call's contents.
 *     Nothing in it needs to start at zero: each call writes every scratch
 *     byte before reading it.  Calls whose executions overlap on the GPU
 *     (different streams without ordering) race on the array: order them.
 */
#define PURO_NOALLOC_SCRATCH_BYTES (40u * 1024u * 1024u)
puro_status_t puro_fp8_linear_wgrad_noalloc(const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw,
                                            int32_t *dev_status, void *stream);

/*
 * Kernel launches puro_fp8_linear_backward makes for block-scaled operands
 * of a linear with M tokens, N output and K input features, given
 * workspace_bytes of (16-byte aligned) workspace: 1 for a grouped launch,
 * else one per GEMM plus one per split reduction.  0 for an empty extent.
 * Host-only, no CUDA call.
 */
int32_t puro_fp8_linear_backward_launches(int64_t M, int64_t N, int64_t K, size_t workspace_bytes);

/*
 * Bytes of a PURO_SCALE_BLOCK scale buffer for an operand [rows, red]
 * (rows * ceil(red/512) * 4).  Host-only, no CUDA call.
 */
size_t puro_fp8_scale_bytes(int64_t rows, int64_t red);

/*
 * Scratch bytes that let a GEMM with output [rows_out, cols_out] and
 * reduction extent `red` use its split-reduction schedule (0 if it never
 * would): splits * ceil(rows_out/128)*128 * cols_out * 4.  Host-only, no
 * CUDA call.
 */
size_t puro_fp8_workspace_size(int64_t rows_out, int64_t cols_out, int64_t red);

/*
 * Copy *dev_status to *host_out (host pointer).  Synchronises `stream`.
 */
puro_status_t puro_fp8_get_status(const int32_t *dev_status, int32_t *host_out, void *stream);

/*
 * BF16 build of the same three GEMMs on the same tensor cores, for the
 * FP8-versus-BF16 comparison the paper reports (appendix "MuonH
 * Scaling-Ladder Analysis", "Precision and throughput decomposition").
 * Operands are BF16, row-major, reduction dimension contiguous (the same
 * TN forms as above; the caller supplies W^T, dY^T, X^T for dgrad/wgrad).
 *   fprop: x [M,K], w [N,K]      -> y  [M,N]
 *   dgrad: dy [M,N], w_t [K,N]   -> dx [M,K]
 *   wgrad: dy_t [N,M], x_t [K,M] -> dw [N,K]
 * Extents must be multiples of 8.
 */
puro_status_t puro_bf16_linear_fprop(const void *x, const void *w, void *y,
                                     int64_t M, int64_t N, int64_t K,
                                     int32_t *dev_status, void *stream);
puro_status_t puro_bf16_linear_dgrad(const void *dy, const void *w_t, void *dx,
                                     int64_t M, int64_t N, int64_t K,
                                     int32_t *dev_status, void *stream);
puro_status_t puro_bf16_linear_wgrad(const void *dy_t, const void *x_t, void *dw,
                                     int64_t M, int64_t N, int64_t K,
                                     int32_t *dev_status, void *stream);

/*
 * Wall-time bound (nanoseconds, process-wide, default 2e9) of every
 * device-side pipeline wait in the GEMM kernels.  Fault-detection tests
 * lower it to force the PURO_ERR_TIMEOUT path without hanging the GPU.
 */
void puro_set_wait_timeout_ns(uint64_t ns);

/*
 * Tile width of unsplit block-scaled GEMMs (process-wide): 0 (default) lets
 * a per-shape cost model choose; 256 or 224 forces that form.  The 256-wide
 * form shares half of its tensor-memory accumulator between consecutive
 * tiles; the 224-wide form double-buffers it.  Both compute the same
 * products (summation order differs only by tile boundaries, which do not
 * cross the reduction).  Any other value returns PURO_ERR_INVALID_ARG.
 * For tests and tuning; the paper has no counterpart.
 */
puro_status_t puro_set_gemm_tile_n(int32_t tile_n);

/*
 * MuonH hyperball step (section "Hyperball Optimization", Eq.
 * hyperball-update), for one wrapped matrix W (FP32 master weight) and its
 * Muon update direction u:
 *     u_hat = u / ||u||_F,   W~ = W - eta R u_hat,   W <- R W~ / ||W~||_F,
 * R = ||W_0||_F being the matrix's fixed radius (puro_muonh_reduce of W_0
 * with itself gives R^2 as sums[0]).  The Muon orthogonalisation that
 * produces u is not part of this step (the paper does not specify it).
 *
 * The step is two passes over memory: a reduction of the three sums
 *     sums = {S_ww, S_wu, S_uu} = {sum W^2, sum W u, sum u^2}   (fp64)
 * and an update W <- s (W - c u), c = eta R / sqrt(S_uu),
 * s = R / sqrt(S_ww - 2 c S_wu + c^2 S_uu), with c and s rounded to fp32.
 * The sums are additive over any partition of the matrix: a caller that
 * shards W across devices runs puro_muonh_reduce on each shard, all-reduces
 * the three doubles, then runs puro_muonh_apply on each shard.
 *   w, u: fp32, n values (any shape; the Frobenius norm is that of the
 *     flattened matrix), n a multiple of 4, 16-byte aligned; w updated in place.
 *   sums: device double[3], 8-byte aligned (written by reduce, read by apply).
 *   workspace: device scratch of puro_muonh_workspace_size(n) bytes, 8-byte
 *     aligned (per-block partial sums).
 *   eta >= 0 (the Hyperball learning rate), radius > 0, both finite.
 *   w_bf16: optional bf16 [n] copy of the updated W (8-byte aligned), or NULL.
 * A zero direction (S_uu = 0) takes no step: W is only projected (the
 * equation is undefined there).  If W~ = 0 the result is NaN.  The
 * reduction order is fixed by n alone, so results are deterministic and the
 * same on every device.  n = 0 does nothing (reduce writes zero sums).
 * Three kernels for the step: the chunk sums, their fixed-order total, and
 * the update.
 */
size_t puro_muonh_workspace_size(int64_t n);
puro_status_t puro_muonh_reduce(const float *w, const float *u, int64_t n, double *sums, void *workspace,
                                size_t workspace_bytes, void *stream);
puro_status_t puro_muonh_apply(float *w, const float *u, int64_t n, const double *sums, double eta, double radius,
                               void *w_bf16, void *stream);
/* reduce then apply, on one device (three kernels on `stream`). */
puro_status_t puro_muonh_step(float *w, const float *u, int64_t n, double eta, double radius, double *sums,
                              void *workspace, size_t workspace_bytes, void *w_bf16, void *stream);

/*
 * The same step for many matrices at once (every wrapped matrix of a model):
 * three kernel launches per 128 matrices instead of three per matrix.  Each
 * matrix is cut into chunks by its own size alone, so its result is bit for
 * bit the one puro_muonh_step gives.
 *   mats: host array of `count` descriptors (read during the call only).
 *   sums: device double[count][3], written (the three sums of each matrix).
 *   workspace: puro_muonh_grouped_workspace_size(mats, count) bytes.
 * Every descriptor is checked before anything is enqueued.
 */
typedef struct {
    float *w;           /* fp32 master weight [n], updated in place (16-byte aligned) */
    const float *u;     /* fp32 Muon direction [n] (16-byte aligned) */
    void *w_bf16;       /* bf16 copy [n] written after the update (8-byte aligned), or NULL */
    int64_t n;          /* number of values, a multiple of 4 */
    double radius;      /* R = ||W_0||_F > 0 */
} puro_muonh_matrix_t;

size_t puro_muonh_grouped_workspace_size(const puro_muonh_matrix_t *mats, int32_t count);
puro_status_t puro_muonh_step_grouped(const puro_muonh_matrix_t *mats, int32_t count, double eta, double *sums,
                                      void *workspace, size_t workspace_bytes, void *stream);

/* Human-readable name of a status code (static string). */
const char *puro_status_string(puro_status_t s);

#ifdef __cplusplus
}
#endif

#endif /* PURO_FP8_H */
