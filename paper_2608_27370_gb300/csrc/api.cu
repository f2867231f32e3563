// api.cu -- the C ABI declared in include/puro_fp8.h: argument validation
// (entirely on the host, before anything is enqueued), TMA descriptor
// encoding and kernel launch.  See the header for the contract of every
// entry point.
#include <atomic>
#include <mutex>

#include "internal.h"
#include "puro_fp8.h"

#define PURO_API extern "C" __attribute__((visibility("default")))

namespace puro {
namespace {

std::atomic<uint64_t> g_wait_timeout_ns{2000000000ull};  // 2 s
std::atomic<int> g_tile_n{0};                             // 0: cost model; 224 / 256: forced

using EncodeTiledFn = CUresult (*)(CUtensorMap *, CUtensorMapDataType, cuuint32_t, void *, const cuuint64_t *,
                                   const cuuint64_t *, const cuuint32_t *, const cuuint32_t *,
                                   CUtensorMapInterleave, CUtensorMapSwizzle, CUtensorMapL2promotion,
                                   CUtensorMapFloatOOBfill);

EncodeTiledFn encode_fn() {
    static EncodeTiledFn fn = nullptr;
    static std::once_flag once;
    std::call_once(once, [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q{};
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            fn = reinterpret_cast<EncodeTiledFn>(p);
    });
    return fn;
}

// 2-D tensor map over a row-major [outer, inner] matrix.
bool make_map(CUtensorMap *m, CUtensorMapDataType dt, const void *base, uint64_t inner, uint64_t outer,
              uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, CUtensorMapSwizzle sw) {
    EncodeTiledFn fn = encode_fn();
    if (!fn) return false;
    const cuuint64_t dims[2] = {inner, outer};
    const cuuint64_t strides[1] = {row_bytes};
    const cuuint32_t box[2] = {box_inner, box_outer};
    const cuuint32_t estr[2] = {1, 1};
    return fn(m, dt, 2, const_cast<void *>(base), dims, strides, box, estr, CU_TENSOR_MAP_INTERLEAVE_NONE, sw,
              CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE) == CUDA_SUCCESS;
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

// Scale vectors of a BLOCK operand [rows, red] as uint32 [rows/128 *
// ceil(red/512), 128]: one 512-byte chunk (128 rows x four k-blocks) per row
// of the map, loaded whole (box {128, 1}); rows past the end read as zero.
bool make_scale_map(CUtensorMap *m, const void *scale, int64_t rows, int64_t red) {
    const uint64_t chunks = static_cast<uint64_t>((rows + 127) / 128) * static_cast<uint64_t>((red / 128 + 3) / 4);
    return make_map(m, CU_TENSOR_MAP_DATA_TYPE_UINT32, scale, 128, chunks, 512, 128, 1, CU_TENSOR_MAP_SWIZZLE_NONE);
}

int sm_count() {
    static int cache[64] = {0};
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (dev >= 0 && dev < 64 && cache[dev]) return cache[dev];
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess) return 0;
    if (dev >= 0 && dev < 64) cache[dev] = n;
    return n;
}

puro_status_t cuda_status(cudaError_t e) { return e == cudaSuccess ? PURO_OK : PURO_ERR_CUDA; }

bool valid_fmt(int32_t f) { return f == PURO_E4M3 || f == PURO_E5M2; }

// Shape/pointer checks shared by the FP8 GEMM entry points.
puro_status_t check_operand(const puro_fp8_tensor_t *t) {
    if (!t || !t->data || !t->scale) return PURO_ERR_INVALID_ARG;
    if (!aligned16(t->data) || !aligned16(t->scale)) return PURO_ERR_INVALID_ARG;
    if (t->rows < 0 || t->red < 0 || !valid_fmt(t->fmt) || t->reserved != 0) return PURO_ERR_INVALID_ARG;
    if (t->rows > INT32_MAX || t->red > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    if (t->scaling == PURO_SCALE_BLOCK) {
        if (t->role != PURO_ROLE_ACT && t->role != PURO_ROLE_WEIGHT) return PURO_ERR_INVALID_ARG;
        if (t->rows % 128 || t->red % 128) return PURO_ERR_INVALID_ARG;
    } else if (t->scaling == PURO_SCALE_TENSOR) {
        if (t->rows % 16 || t->red % 16) return PURO_ERR_INVALID_ARG;
    } else {
        return PURO_ERR_INVALID_ARG;
    }
    return PURO_OK;
}

// What a validated GEMM call needs enqueued.
enum GemmAction { kGemmNothing, kGemmZeroFill, kGemmLaunch };

// The argument checks of D = A * B^T (host only, no CUDA call).
puro_status_t validate_fp8_gemm(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, const void *d) {
    puro_status_t st = check_operand(a);
    if (st != PURO_OK) return st;
    st = check_operand(b);
    if (st != PURO_OK) return st;
    if (a->red != b->red || a->scaling != b->scaling) return PURO_ERR_INVALID_ARG;
    if (!d || !aligned16(d)) return PURO_ERR_INVALID_ARG;
    return PURO_OK;
}

// Validates D = A * B^T and prepares its launch (nothing is enqueued here).
puro_status_t prepare_fp8_gemm(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, void *d, void *workspace,
                               size_t workspace_bytes, int32_t *dev_status, bool accumulate_f32, GemmArgs *gout,
                               GemmMaps *mout, GemmAction *action) {
    const puro_status_t st = validate_fp8_gemm(a, b, d);
    if (st != PURO_OK) return st;
    const int64_t M = a->rows, N = b->rows, K = a->red;
    *action = kGemmNothing;
    gout->M = M;
    gout->N = N;
    gout->out = d;
    if (M == 0 || N == 0) return PURO_OK;
    if (K == 0) {  // an empty reduction: the product is zero (a main-grad is left as it is)
        if (!accumulate_f32) *action = kGemmZeroFill;
        return PURO_OK;
    }
    const bool block = a->scaling == PURO_SCALE_BLOCK;

    // Split the reduction across CTA pairs when the output has too few tiles
    // to fill the GPU and the caller supplied enough aligned scratch;
    // otherwise the block-scaled kind picks its tile width.
    const int sp = choose_splits(M, N, K, false);
    const bool split = sp > 1 && workspace && aligned16(workspace) &&
                       workspace_bytes >= splitk_workspace_bytes(M, N, K, false);
    const int forced = g_tile_n.load();
    const int tile_n = (block && !split && !accumulate_f32) ? (forced ? forced : choose_tile_n(M, N, K)) : 256;

    GemmMaps m{};
    if (!make_map(&m.a, CU_TENSOR_MAP_DATA_TYPE_UINT8, a->data, K, M, K, kGemmBKBytes, kGemmBM,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, b->data, K, N, K, kGemmBKBytes,
                  static_cast<uint32_t>(tile_n / 2), CU_TENSOR_MAP_SWIZZLE_128B) ||
        !(accumulate_f32
              ? make_map(&m.d, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, d, N, M, N * 4, 32, 32, CU_TENSOR_MAP_SWIZZLE_128B)
              : make_map(&m.d, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, d, N, M, N * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B)))
        return PURO_ERR_CUDA;
    m.ws = m.d;
    m.sfa = m.d;
    m.sfb = m.d;
    GemmArgs g{};
    g.kind = block ? kGemmFP8Block : kGemmFP8Tensor;
    g.a_fmt = a->fmt;
    g.b_fmt = b->fmt;
    g.M = M;
    g.N = N;
    g.K = K;
    g.tile_n = tile_n;
    if (block) {
        if (!make_scale_map(&m.sfa, a->scale, M, K) || !make_scale_map(&m.sfb, b->scale, N, K)) return PURO_ERR_CUDA;
        g.sfb = static_cast<const uint8_t *>(b->scale);
    } else {
        g.sia = static_cast<const float *>(a->scale);
        g.sib = static_cast<const float *>(b->scale);
    }
    g.status = dev_status;
    g.wait_timeout_ns = g_wait_timeout_ns.load();
    g.num_sms = sm_count();
    if (g.num_sms <= 0) return PURO_ERR_CUDA;
    g.out = d;
    g.splits = 1;
    g.accumulate_f32 = accumulate_f32;
    if (split) {
        const uint64_t rows = static_cast<uint64_t>(sp) * static_cast<uint64_t>(splitk_rows_per_chunk(M));
        if (!make_map(&m.ws, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, workspace, N, rows, N * 4, 32, 32,
                      CU_TENSOR_MAP_SWIZZLE_128B))
            return PURO_ERR_CUDA;
        g.splits = sp;
        g.workspace = workspace;
    }
    *gout = g;
    *mout = m;
    *action = kGemmLaunch;
    return PURO_OK;
}

puro_status_t run_fp8_gemm(GemmAction action, const GemmArgs &g, const GemmMaps &m, cudaStream_t s) {
    if (action == kGemmZeroFill) return cuda_status(cudaMemsetAsync(g.out, 0, static_cast<size_t>(g.M * g.N) * 2, s));
    if (action == kGemmLaunch) return cuda_status(launch_gemm(g, m, s));
    return PURO_OK;
}

// D[M,N] = A[M,K] * B[N,K]^T over quantised operands.
// accumulate_f32: d is an FP32 [M, N] main-grad that receives d += A * B^T.
puro_status_t fp8_gemm(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, void *d, void *workspace,
                       size_t workspace_bytes, int32_t *dev_status, void *stream, bool accumulate_f32 = false) {
    GemmArgs g{};
    GemmMaps m{};
    GemmAction action;
    const puro_status_t st =
        prepare_fp8_gemm(a, b, d, workspace, workspace_bytes, dev_status, accumulate_f32, &g, &m, &action);
    if (st != PURO_OK) return st;
    return run_fp8_gemm(action, g, m, static_cast<cudaStream_t>(stream));
}

// How a linear's backward (Dgrad dX [M, K] over N, Wgrad dW [N, K] over M,
// block-scaled) runs, given `ws` usable workspace bytes: one grouped launch
// when both GEMMs are 256-wide and unsplit -- or when the Wgrad would split
// its reduction but one grouped launch with it unsplit is modelled faster --
// else each GEMM on its own (a split Wgrad adds its reduction kernel).
struct BackwardPlan {
    bool grouped;        // one launch for both
    bool wgrad_unsplit;  // the Wgrad gives up the split it would take, to join the Dgrad
    int launches;        // kernel launches
};

BackwardPlan plan_backward(int64_t M, int64_t N, int64_t K, size_t ws) {
    auto split_of = [&](int64_t r, int64_t c, int64_t red) {
        const int sp = choose_splits(r, c, red, false);
        return (sp > 1 && ws >= splitk_workspace_bytes(r, c, red, false)) ? sp : 1;
    };
    auto tile_of = [&](int64_t r, int64_t c, int64_t red) {
        const int forced = g_tile_n.load();
        return forced ? forced : choose_tile_n(r, c, red);
    };
    BackwardPlan b{};
    const int sd = split_of(M, K, N), sw = split_of(N, K, M);
    if (sd == 1 && tile_of(M, K, N) == 256 && tile_of(N, K, M) == 256) {
        if (sw == 1)
            b.grouped = true;
        else
            b.grouped = b.wgrad_unsplit = grouped_backward_faster(M, N, K, sw);
    }
    b.launches = b.grouped ? 1 : (sd > 1 ? 2 : 1) + (sw > 1 ? 2 : 1);
    return b;
}

// Dgrad and Wgrad of one linear: one grouped launch when plan_backward says
// so (the problem with the longer reduction first; the balanced schedule
// lets the pairs with fewer of its tiles take more of the other's), else two.
puro_status_t fp8_backward(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t, void *dx,
                           const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw, void *workspace,
                           size_t workspace_bytes, int32_t *dev_status, void *stream) {
    puro_status_t st = validate_fp8_gemm(dy, w_t, dx);  // both calls' arguments first
    if (st != PURO_OK) return st;
    st = validate_fp8_gemm(dy_t, x_t, dw);
    if (st != PURO_OK) return st;
    GemmArgs gd{}, gw{};
    GemmMaps md{}, mw{};
    GemmAction ad, aw;
    st = prepare_fp8_gemm(dy, w_t, dx, workspace, workspace_bytes, dev_status, false, &gd, &md, &ad);
    if (st != PURO_OK) return st;
    const size_t ws_usable = (workspace && aligned16(workspace)) ? workspace_bytes : 0;
    const bool both_block = dy->scaling == PURO_SCALE_BLOCK && dy_t->scaling == PURO_SCALE_BLOCK;
    const bool unsplit_w = both_block && dy->rows > 0 && dy->red > 0 && w_t->rows > 0 &&
                           plan_backward(dy->rows, dy->red, w_t->rows, ws_usable).wgrad_unsplit;
    st = prepare_fp8_gemm(dy_t, x_t, dw, unsplit_w ? nullptr : workspace, unsplit_w ? 0 : workspace_bytes, dev_status,
                          false, &gw, &mw, &aw);
    if (st != PURO_OK) return st;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    const bool grouped = ad == kGemmLaunch && aw == kGemmLaunch && gd.kind == kGemmFP8Block &&
                         gw.kind == kGemmFP8Block && gd.splits == 1 && gw.splits == 1 && gd.tile_n == 256 &&
                         gw.tile_n == 256;
    if (grouped)
        return cuda_status(gw.K >= gd.K ? launch_gemm_grouped(gw, mw, gd, md, s) : launch_gemm_grouped(gd, md, gw, mw, s));
    st = run_fp8_gemm(ad, gd, md, s);
    if (st != PURO_OK) return st;
    return run_fp8_gemm(aw, gw, mw, s);
}

puro_status_t bf16_gemm(const void *a, const void *b, void *d, int64_t M, int64_t N, int64_t K,
                        int32_t *dev_status, void *stream) {
    if (!a || !b || !d || !aligned16(a) || !aligned16(b) || !aligned16(d)) return PURO_ERR_INVALID_ARG;
    if (M < 0 || N < 0 || K < 0 || M % 8 || N % 8 || K % 8) return PURO_ERR_INVALID_ARG;
    if (M > INT32_MAX || N > INT32_MAX || K > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (M == 0 || N == 0) return PURO_OK;
    if (K == 0) return cuda_status(cudaMemsetAsync(d, 0, static_cast<size_t>(M * N) * 2, s));
    GemmMaps m{};
    if (!make_map(&m.a, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, a, K, M, K * 2, kGemmBKBytes / 2, kGemmBM,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m.b, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, b, K, N, K * 2, kGemmBKBytes / 2, kGemmBN / 2,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m.d, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, d, N, M, N * 2, 32, 32, CU_TENSOR_MAP_SWIZZLE_64B))
        return PURO_ERR_CUDA;
    m.ws = m.d;
    m.sfa = m.d;
    m.sfb = m.d;
    GemmArgs g{};
    g.kind = kGemmBF16;
    g.M = M;
    g.N = N;
    g.K = K;
    g.tile_n = 256;
    g.status = dev_status;
    g.wait_timeout_ns = g_wait_timeout_ns.load();
    g.num_sms = sm_count();
    if (g.num_sms <= 0) return PURO_ERR_CUDA;
    g.splits = 1;
    g.out = d;
    return cuda_status(launch_gemm(g, m, s));
}

// D[M,N] = A[M,K] * B[N,K]^T (block-scaled operands), rounded to BF16 and
// quantised in the epilogue into the blockwise activation copies of D: Dq
// [M, N] with 1x128 groups along N and, when q_t is given, Dq^T [N, M] with
// groups of 128 rows; D itself in BF16 only when d is given.
puro_status_t fp8_gemm_quant(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, int32_t fmt, void *d,
                             uint8_t *q, void *q_scale, uint8_t *q_t, void *q_t_scale, int32_t *dev_status,
                             void *stream) {
    puro_status_t st = check_operand(a);
    if (st != PURO_OK) return st;
    st = check_operand(b);
    if (st != PURO_OK) return st;
    if (a->red != b->red || a->scaling != PURO_SCALE_BLOCK || b->scaling != PURO_SCALE_BLOCK)
        return PURO_ERR_INVALID_ARG;
    if (!valid_fmt(fmt)) return PURO_ERR_INVALID_ARG;
    if (!q || !q_scale || !aligned16(q) || !aligned16(q_scale)) return PURO_ERR_INVALID_ARG;
    if ((q_t == nullptr) != (q_t_scale == nullptr)) return PURO_ERR_INVALID_ARG;
    if (q_t && (!aligned16(q_t) || !aligned16(q_t_scale))) return PURO_ERR_INVALID_ARG;
    if (d && !aligned16(d)) return PURO_ERR_INVALID_ARG;
    const int64_t M = a->rows, N = b->rows, K = a->red;  // multiples of 128 (check_operand)
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    if (M == 0 || N == 0) return PURO_OK;
    if (K == 0) {  // a zero product: zero codes, scale exponent 127 (as the quantiser gives an all-zero tensor)
        cudaError_t e = cudaMemsetAsync(q, 0, static_cast<size_t>(M * N), s);
        if (e == cudaSuccess) e = cudaMemsetAsync(q_scale, 127, static_cast<size_t>(M * ((N / 128 + 3) / 4) * 4), s);
        if (e == cudaSuccess && q_t) e = cudaMemsetAsync(q_t, 0, static_cast<size_t>(M * N), s);
        if (e == cudaSuccess && q_t)
            e = cudaMemsetAsync(q_t_scale, 127, static_cast<size_t>(N * ((M / 128 + 3) / 4) * 4), s);
        if (e == cudaSuccess && d) e = cudaMemsetAsync(d, 0, static_cast<size_t>(M * N) * 2, s);
        return cuda_status(e);
    }
    GemmMaps m{};
    if (!make_map(&m.a, CU_TENSOR_MAP_DATA_TYPE_UINT8, a->data, K, M, K, kGemmBKBytes, kGemmBM,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_map(&m.b, CU_TENSOR_MAP_DATA_TYPE_UINT8, b->data, K, N, K, kGemmBKBytes, kGemmBN / 2,
                  CU_TENSOR_MAP_SWIZZLE_128B) ||
        !make_scale_map(&m.sfa, a->scale, M, K) || !make_scale_map(&m.sfb, b->scale, N, K))
        return PURO_ERR_CUDA;
    m.d = m.a;  // the quantising epilogue stores from registers: no output map (the kernel prefetches tm_d)
    m.ws = m.a;
    GemmArgs g{};
    g.kind = kGemmFP8Block;
    g.a_fmt = a->fmt;
    g.b_fmt = b->fmt;
    g.M = M;
    g.N = N;
    g.K = K;
    g.tile_n = 256;
    g.sfb = static_cast<const uint8_t *>(b->scale);
    g.status = dev_status;
    g.wait_timeout_ns = g_wait_timeout_ns.load();
    g.num_sms = sm_count();
    if (g.num_sms <= 0) return PURO_ERR_CUDA;
    g.out = d;
    g.splits = 1;
    g.quant_out = true;
    g.q_fmt = fmt;
    g.q = q;
    g.q_scale = static_cast<uint8_t *>(q_scale);
    g.qt = q_t;
    g.qt_scale = static_cast<uint8_t *>(q_t_scale);
    g.d_bf16 = d;
    return cuda_status(launch_gemm(g, m, s));
}

}  // namespace

puro_status_t fp8_gemm_entry(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, void *d, void *workspace,
                             size_t workspace_bytes, int32_t *dev_status, void *stream) {
    return fp8_gemm(a, b, d, workspace, workspace_bytes, dev_status, stream);
}

puro_status_t fp8_gemm_validate(const puro_fp8_tensor_t *a, const puro_fp8_tensor_t *b, const void *d) {
    return validate_fp8_gemm(a, b, d);
}

}  // namespace puro

using namespace puro;

PURO_API puro_status_t puro_fp8_quantize_weights(const puro_fp8_weight_t *weights, int32_t count, int32_t fmt,
                                                 int32_t *dev_status, void *stream) {
    if (count < 0 || (count > 0 && !weights) || !valid_fmt(fmt)) return PURO_ERR_INVALID_ARG;
    if (count == 0) return PURO_OK;
    bool has_t = false;  // from the first non-empty entry; empty entries are skipped unchecked
    for (int32_t i = 0; i < count; ++i)
        if (weights[i].rows > 0 && weights[i].cols > 0) {
            has_t = weights[i].q_t != nullptr;
            break;
        }
    for (int32_t i = 0; i < count; ++i) {  // every argument checked before anything is enqueued
        const puro_fp8_weight_t &w = weights[i];
        if (w.rows < 0 || w.cols < 0 || w.rows % 128 || w.cols % 128) return PURO_ERR_INVALID_ARG;
        if (w.rows > INT32_MAX || w.cols > INT32_MAX) return PURO_ERR_UNSUPPORTED;
        if (w.rows == 0 || w.cols == 0) continue;
        if ((w.q_t != nullptr) != has_t || (w.scale_t != nullptr) != has_t) return PURO_ERR_INVALID_ARG;
        if (!w.w || !w.q || !w.scale || !aligned16(w.w) || !aligned16(w.q) || !aligned16(w.scale) ||
            !aligned16(w.q_t) || !aligned16(w.scale_t))
            return PURO_ERR_INVALID_ARG;
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    static thread_local WeightGroup g;  // 26 KB: kept off the stack
    g.status = dev_status;
    g.wait_ns = g_wait_timeout_ns.load();
    int32_t i = 0;
    while (i < count) {
        g.count = 0;
        g.tile_start[0] = 0;
        int64_t tiles = 0;
        for (; i < count && g.count < kWeightGroupMax; ++i) {
            const puro_fp8_weight_t &w = weights[i];
            if (w.rows == 0 || w.cols == 0) continue;
            const int64_t wt = (w.rows / 128) * (w.cols / 128);
            if (tiles + wt > INT32_MAX) break;
            const int k = g.count;
            if (!make_map(&g.x[k], CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, w.w, w.cols, w.rows, w.cols * 2, 128, 128,
                          CU_TENSOR_MAP_SWIZZLE_NONE) ||
                !make_map(&g.q[k], CU_TENSOR_MAP_DATA_TYPE_UINT8, w.q, w.cols, w.rows, w.cols, 128, 128,
                          CU_TENSOR_MAP_SWIZZLE_NONE))
                return PURO_ERR_CUDA;
            if (has_t) {
                if (!make_map(&g.qt[k], CU_TENSOR_MAP_DATA_TYPE_UINT8, w.q_t, w.rows, w.cols, w.rows, 128, 128,
                              CU_TENSOR_MAP_SWIZZLE_128B))
                    return PURO_ERR_CUDA;
            } else {
                g.qt[k] = g.q[k];
            }
            g.scale[k] = static_cast<uint8_t *>(w.scale);
            g.scale_t[k] = static_cast<uint8_t *>(w.scale_t);
            g.tiles_n[k] = static_cast<int>(w.cols / 128);
            g.kb_rows[k] = static_cast<int>(w.rows / 128);
            tiles += wt;
            g.tile_start[k + 1] = static_cast<int>(tiles);
            ++g.count;
        }
        if (g.count == 0 && i < count) return PURO_ERR_UNSUPPORTED;  // one weight beyond the tile index range
        const puro_status_t st = cuda_status(launch_quantize_weights(g, fmt, has_t, s));
        if (st != PURO_OK) return st;
    }
    return PURO_OK;
}

PURO_API puro_status_t puro_fp8_amax(const void *x, int64_t rows, int64_t cols, uint32_t *amax_bits, void *stream) {
    if (!amax_bits || rows < 0 || cols < 0) return PURO_ERR_INVALID_ARG;
    if ((reinterpret_cast<uintptr_t>(amax_bits) & 3u) != 0) return PURO_ERR_INVALID_ARG;
    const int64_t n = rows * cols;
    if (n > 0 && (!x || !aligned16(x))) return PURO_ERR_INVALID_ARG;
    return cuda_status(launch_amax(static_cast<const uint16_t *>(x), n, amax_bits, static_cast<cudaStream_t>(stream)));
}

PURO_API puro_status_t puro_fp8_quantize(const void *x, int64_t rows, int64_t cols, int32_t fmt, int32_t scaling,
                                         int32_t role, const uint32_t *amax_bits, uint8_t *q, void *scale,
                                         uint8_t *q_t, void *scale_t, int32_t *dev_status, void *stream) {
    if (!valid_fmt(fmt) || rows < 0 || cols < 0) return PURO_ERR_INVALID_ARG;
    if ((q_t == nullptr) != (scale_t == nullptr) && scaling == PURO_SCALE_BLOCK) return PURO_ERR_INVALID_ARG;
    const bool has_t = q_t != nullptr;
    QuantArgs a{};
    a.fmt = fmt;
    a.rows = rows;
    a.cols = cols;
    a.has_t = has_t;
    a.status = dev_status;
    a.wait_ns = g_wait_timeout_ns.load();
    if (scaling == PURO_SCALE_BLOCK) {
        if (role != PURO_ROLE_ACT && role != PURO_ROLE_WEIGHT) return PURO_ERR_INVALID_ARG;
        if (amax_bits != nullptr) return PURO_ERR_INVALID_ARG;
        if (rows % 128 || cols % 128) return PURO_ERR_INVALID_ARG;
        a.kind = role == PURO_ROLE_ACT ? kQuantBlockAct : kQuantBlockWeight;
        a.scale_u8 = static_cast<uint8_t *>(scale);
        a.scale_t_u8 = static_cast<uint8_t *>(scale_t);
    } else if (scaling == PURO_SCALE_TENSOR) {
        if (!amax_bits || (reinterpret_cast<uintptr_t>(amax_bits) & 3u)) return PURO_ERR_INVALID_ARG;
        if (cols % 16 || (has_t && rows % 16)) return PURO_ERR_INVALID_ARG;
        a.kind = kQuantTensor;
        a.scale_f = static_cast<float *>(scale);
        a.scale_t_f = static_cast<float *>(scale_t);
        if ((reinterpret_cast<uintptr_t>(scale) & 3u) || (reinterpret_cast<uintptr_t>(scale_t) & 3u))
            return PURO_ERR_INVALID_ARG;
    } else {
        return PURO_ERR_INVALID_ARG;
    }
    const bool empty = rows == 0 || cols == 0;
    // Empty tensors write no codes (their buffers may be NULL); per-tensor
    // mode still writes scale_inv.
    if (!aligned16(q) || !aligned16(scale) || !aligned16(q_t) || !aligned16(scale_t)) return PURO_ERR_INVALID_ARG;
    if (!empty && (!q || !scale)) return PURO_ERR_INVALID_ARG;
    if (empty && scaling == PURO_SCALE_TENSOR && !scale) return PURO_ERR_INVALID_ARG;
    if (rows > INT32_MAX || cols > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    if (!empty && (!x || !aligned16(x))) return PURO_ERR_INVALID_ARG;
    a.amax = amax_bits;
    if (empty) {
        if (scaling == PURO_SCALE_TENSOR)  // empty tensor: amax is 0, scale_inv is 1
            return cuda_status(launch_tensor_scale_only(a, static_cast<cudaStream_t>(stream)));
        return PURO_OK;
    }
    a.x = static_cast<const uint16_t *>(x);
    CUtensorMap tm_x, tm_q, tm_qt;
    if (!make_map(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, x, cols, rows, cols * 2, 128, 128,
                  CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !make_map(&tm_q, CU_TENSOR_MAP_DATA_TYPE_UINT8, q, cols, rows, cols, 128, 128, CU_TENSOR_MAP_SWIZZLE_NONE))
        return PURO_ERR_CUDA;
    if (has_t) {
        if (!make_map(&tm_qt, CU_TENSOR_MAP_DATA_TYPE_UINT8, q_t, rows, cols, rows, 128, 128,
                      CU_TENSOR_MAP_SWIZZLE_128B))
            return PURO_ERR_CUDA;
    } else {
        tm_qt = tm_q;
    }
    return cuda_status(launch_quantize(a, tm_x, tm_q, tm_qt, static_cast<cudaStream_t>(stream)));
}

// RMSNorm (rows of h, optional bf16 gain) fused ahead of the blockwise
// activation quantiser; see the header.
PURO_API puro_status_t puro_fp8_quantize_rmsnorm(const void *h, int64_t rows, int64_t cols, const void *gamma,
                                                 float eps, int32_t fmt, float *rstd, void *y, uint8_t *q, void *scale,
                                                 uint8_t *q_t, void *scale_t, int32_t *dev_status, void *stream) {
    if (!valid_fmt(fmt) || rows < 0 || cols < 0 || !(eps >= 0.0f)) return PURO_ERR_INVALID_ARG;
    if (rows % 128 || cols % 128) return PURO_ERR_INVALID_ARG;
    if ((q_t == nullptr) != (scale_t == nullptr)) return PURO_ERR_INVALID_ARG;
    if (rows > INT32_MAX || cols > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    if (rows == 0 || cols == 0) return PURO_OK;
    if (!h || !rstd || !q || !scale) return PURO_ERR_INVALID_ARG;
    if (!aligned16(h) || !aligned16(gamma) || !aligned16(y) || !aligned16(q) || !aligned16(scale) ||
        !aligned16(q_t) || !aligned16(scale_t) || (reinterpret_cast<uintptr_t>(rstd) & 3u))
        return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    QuantArgs a{};
    a.fmt = fmt;
    a.rows = rows;
    a.cols = cols;
    a.has_t = q_t != nullptr;
    a.kind = kQuantBlockAct;
    a.scale_u8 = static_cast<uint8_t *>(scale);
    a.scale_t_u8 = static_cast<uint8_t *>(scale_t);
    a.status = dev_status;
    a.wait_ns = g_wait_timeout_ns.load();
    a.x = static_cast<const uint16_t *>(h);
    CUtensorMap tm_x, tm_q, tm_qt, tm_y;
    if (!make_map(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, h, cols, rows, cols * 2, 128, 128,
                  CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !make_map(&tm_q, CU_TENSOR_MAP_DATA_TYPE_UINT8, q, cols, rows, cols, 128, 128, CU_TENSOR_MAP_SWIZZLE_NONE))
        return PURO_ERR_CUDA;
    tm_qt = tm_q;
    if (a.has_t && !make_map(&tm_qt, CU_TENSOR_MAP_DATA_TYPE_UINT8, q_t, rows, cols, rows, 128, 128,
                             CU_TENSOR_MAP_SWIZZLE_128B))
        return PURO_ERR_CUDA;
    tm_y = tm_x;
    if (y && !make_map(&tm_y, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, y, cols, rows, cols * 2, 128, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE))
        return PURO_ERR_CUDA;
    cudaError_t e = launch_rmsnorm_rstd(static_cast<const uint16_t *>(h), rows, cols, eps, rstd, s);
    if (e != cudaSuccess) return cuda_status(e);
    ProdArgs prod{rstd, static_cast<const uint16_t *>(gamma), y != nullptr};
    return cuda_status(launch_quantize_rmsnorm(a, tm_x, tm_q, tm_qt, tm_y, prod, s));
}

// SwiGLU fused ahead of the activation quantiser.
PURO_API puro_status_t puro_fp8_quantize_swiglu(const void *gate, const void *up, int64_t rows, int64_t cols,
                                                int64_t ld, int32_t fmt, void *y, uint8_t *q, void *scale,
                                                uint8_t *q_t, void *scale_t, int32_t *dev_status, void *stream) {
    if (!valid_fmt(fmt) || rows < 0 || cols < 0 || ld < cols || ld % 8) return PURO_ERR_INVALID_ARG;
    if (rows % 128 || cols % 128) return PURO_ERR_INVALID_ARG;
    if ((q_t == nullptr) != (scale_t == nullptr)) return PURO_ERR_INVALID_ARG;
    if (rows > INT32_MAX || cols > INT32_MAX || ld > INT32_MAX) return PURO_ERR_UNSUPPORTED;
    if (rows == 0 || cols == 0) return PURO_OK;
    if (!gate || !up || !q || !scale) return PURO_ERR_INVALID_ARG;
    if (!aligned16(gate) || !aligned16(up) || !aligned16(y) || !aligned16(q) || !aligned16(scale) ||
        !aligned16(q_t) || !aligned16(scale_t))
        return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    QuantArgs a{};
    a.fmt = fmt;
    a.rows = rows;
    a.cols = cols;
    a.has_t = q_t != nullptr;
    a.kind = kQuantBlockAct;
    a.scale_u8 = static_cast<uint8_t *>(scale);
    a.scale_t_u8 = static_cast<uint8_t *>(scale_t);
    a.status = dev_status;
    a.wait_ns = g_wait_timeout_ns.load();
    a.x = static_cast<const uint16_t *>(gate);
    CUtensorMap tm_x, tm_q, tm_qt, tm_y;
    if (!make_map(&tm_x, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, gate, cols, rows, ld * 2, 128, 128,
                  CU_TENSOR_MAP_SWIZZLE_NONE) ||
        !make_map(&tm_q, CU_TENSOR_MAP_DATA_TYPE_UINT8, q, cols, rows, cols, 128, 128, CU_TENSOR_MAP_SWIZZLE_NONE))
        return PURO_ERR_CUDA;
    tm_qt = tm_q;
    if (a.has_t && !make_map(&tm_qt, CU_TENSOR_MAP_DATA_TYPE_UINT8, q_t, rows, cols, rows, 128, 128,
                             CU_TENSOR_MAP_SWIZZLE_128B))
        return PURO_ERR_CUDA;
    tm_y = tm_x;
    if (y && !make_map(&tm_y, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, y, cols, rows, cols * 2, 128, 128,
                       CU_TENSOR_MAP_SWIZZLE_NONE))
        return PURO_ERR_CUDA;
    ProdArgs prod{};
    prod.write_y = y != nullptr;
    prod.up = static_cast<const uint16_t *>(up);
    prod.ld = ld;
    return cuda_status(launch_quantize_swiglu(a, tm_x, tm_q, tm_qt, tm_y, prod, s));
}

// The same SwiGLU without the quantiser (the unfused comparison).
PURO_API puro_status_t puro_swiglu_bf16(const void *gate, const void *up, int64_t rows, int64_t cols, int64_t ld,
                                        void *y, void *stream) {
    if (rows < 0 || cols < 0 || cols % 8 || ld < cols || ld % 8) return PURO_ERR_INVALID_ARG;
    if (rows == 0 || cols == 0) return PURO_OK;
    if (!gate || !up || !y || !aligned16(gate) || !aligned16(up) || !aligned16(y)) return PURO_ERR_INVALID_ARG;
    return cuda_status(launch_swiglu_apply(static_cast<const uint16_t *>(gate), static_cast<const uint16_t *>(up),
                                           rows, cols, ld, static_cast<uint16_t *>(y),
                                           static_cast<cudaStream_t>(stream)));
}

// The same RMSNorm without the quantiser (the unfused comparison).
PURO_API puro_status_t puro_rmsnorm_bf16(const void *h, int64_t rows, int64_t cols, const void *gamma, float eps,
                                         float *rstd, void *y, void *stream) {
    if (rows < 0 || cols < 0 || cols % 8 || !(eps >= 0.0f)) return PURO_ERR_INVALID_ARG;
    if (rows == 0 || cols == 0) return PURO_OK;
    if (!h || !rstd || !y || !aligned16(h) || !aligned16(gamma) || !aligned16(y) ||
        (reinterpret_cast<uintptr_t>(rstd) & 3u))
        return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = launch_rmsnorm_rstd(static_cast<const uint16_t *>(h), rows, cols, eps, rstd, s);
    if (e != cudaSuccess) return cuda_status(e);
    return cuda_status(launch_rmsnorm_apply(static_cast<const uint16_t *>(h), rows, cols, rstd,
                                            static_cast<const uint16_t *>(gamma), static_cast<uint16_t *>(y), s));
}

PURO_API puro_status_t puro_fp8_linear_fprop(const puro_fp8_tensor_t *x, const puro_fp8_tensor_t *w, void *y,
                                             void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                             void *stream) {
    return fp8_gemm(x, w, y, workspace, workspace_bytes, dev_status, stream);
}

PURO_API puro_status_t puro_fp8_linear_dgrad(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t, void *dx,
                                             void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                             void *stream) {
    return fp8_gemm(dy, w_t, dx, workspace, workspace_bytes, dev_status, stream);
}

PURO_API puro_status_t puro_fp8_linear_backward(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t, void *dx,
                                                const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw,
                                                void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                                void *stream) {
    return fp8_backward(dy, w_t, dx, dy_t, x_t, dw, workspace, workspace_bytes, dev_status, stream);
}

PURO_API puro_status_t puro_fp8_linear_dgrad_quantize(const puro_fp8_tensor_t *dy, const puro_fp8_tensor_t *w_t,
                                                      int32_t fmt, void *dx, uint8_t *dxq, void *dxq_scale,
                                                      uint8_t *dxq_t, void *dxq_t_scale, int32_t *dev_status,
                                                      void *stream) {
    return fp8_gemm_quant(dy, w_t, fmt, dx, dxq, dxq_scale, dxq_t, dxq_t_scale, dev_status, stream);
}

PURO_API puro_status_t puro_fp8_linear_wgrad(const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t, void *dw,
                                             void *workspace, size_t workspace_bytes, int32_t *dev_status,
                                             void *stream) {
    return fp8_gemm(dy_t, x_t, dw, workspace, workspace_bytes, dev_status, stream);
}

PURO_API puro_status_t puro_fp8_linear_wgrad_main_grad(const puro_fp8_tensor_t *dy_t, const puro_fp8_tensor_t *x_t,
                                                       float *main_grad, void *workspace, size_t workspace_bytes,
                                                       int32_t *dev_status, void *stream) {
    return fp8_gemm(dy_t, x_t, main_grad, workspace, workspace_bytes, dev_status, stream, true);
}

PURO_API int32_t puro_fp8_linear_backward_launches(int64_t M, int64_t N, int64_t K, size_t workspace_bytes) {
    if (M <= 0 || N <= 0 || K <= 0) return 0;
    return plan_backward(M, N, K, workspace_bytes).launches;
}

PURO_API size_t puro_fp8_workspace_size(int64_t rows_out, int64_t cols_out, int64_t red) {
    if (rows_out <= 0 || cols_out <= 0 || red <= 0) return 0;
    return splitk_workspace_bytes(rows_out, cols_out, red, false);
}

PURO_API size_t puro_fp8_scale_bytes(int64_t rows, int64_t red) {
    if (rows <= 0 || red <= 0) return 0;
    return static_cast<size_t>(rows) * static_cast<size_t>((red / 128 + 3) / 4) * 4;
}

PURO_API puro_status_t puro_fp8_get_status(const int32_t *dev_status, int32_t *host_out, void *stream) {
    if (!dev_status || !host_out || (reinterpret_cast<uintptr_t>(dev_status) & 3u)) return PURO_ERR_INVALID_ARG;
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    cudaError_t e = cudaMemcpyAsync(host_out, dev_status, sizeof(int32_t), cudaMemcpyDeviceToHost, s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    return cuda_status(e);
}

PURO_API puro_status_t puro_bf16_linear_fprop(const void *x, const void *w, void *y, int64_t M, int64_t N,
                                              int64_t K, int32_t *dev_status, void *stream) {
    return bf16_gemm(x, w, y, M, N, K, dev_status, stream);
}

PURO_API puro_status_t puro_bf16_linear_dgrad(const void *dy, const void *w_t, void *dx, int64_t M, int64_t N,
                                              int64_t K, int32_t *dev_status, void *stream) {
    // dX [M, K] = dY [M, N] * (W^T [K, N])^T
    return bf16_gemm(dy, w_t, dx, M, K, N, dev_status, stream);
}

PURO_API puro_status_t puro_bf16_linear_wgrad(const void *dy_t, const void *x_t, void *dw, int64_t M, int64_t N,
                                              int64_t K, int32_t *dev_status, void *stream) {
    // dW [N, K] = dY^T [N, M] * (X^T [K, M])^T
    return bf16_gemm(dy_t, x_t, dw, N, K, M, dev_status, stream);
}

PURO_API void puro_set_wait_timeout_ns(uint64_t ns) { g_wait_timeout_ns.store(ns); }

PURO_API puro_status_t puro_set_gemm_tile_n(int32_t tile_n) {
    if (tile_n != 0 && tile_n != 224 && tile_n != 256) return PURO_ERR_INVALID_ARG;
    g_tile_n.store(tile_n);
    return PURO_OK;
}

PURO_API const char *puro_status_string(puro_status_t s) {
    switch (s) {
        case PURO_OK: return "PURO_OK";
        case PURO_ERR_INVALID_ARG: return "PURO_ERR_INVALID_ARG";
        case PURO_ERR_UNSUPPORTED: return "PURO_ERR_UNSUPPORTED";
        case PURO_ERR_CUDA: return "PURO_ERR_CUDA";
        case PURO_ERR_TIMEOUT: return "PURO_ERR_TIMEOUT";
        default: return "PURO_ERR_UNKNOWN";
    }
}
