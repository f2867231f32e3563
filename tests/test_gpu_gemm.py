"""GPU parity of the three GEMMs of a linear layer (Fprop, Dgrad, Wgrad)
against the oracle's fp64 products, element by element, within
|gpu - ref| <= 2^-7 |ref| + 1e-3 rms(ref).

Shapes span several output tiles (256 x 256 or 256 x 224 pair tiles) with
ragged last tiles; the per-tensor and BF16 cases also have ragged reduction
tails.  The block-scaled cases run with each tile form forced and with the
per-shape choice.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import (assert_close, bits, check_gemm_every_tile, host, oracle_linear, par_quantize_blocks_128x128,
                     par_quantize_cols_128x1, par_quantize_rows_1x128, run_linear)

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


def _inputs(M, N, K, seed, t3=False):
    x = (W.student_t3_f32((M, K), DEV, seed) if t3 else W.normal_f32((M, K), 1.0, DEV, seed)).to(torch.bfloat16)
    w = W.normal_bf16((N, K), 0.02, DEV, seed + 1)
    dy = W.normal_bf16((M, N), 1e-3, DEV, seed + 2)
    return x, w, dy


@pytest.fixture(params=[0, 224, 256], ids=["tile_auto", "tile224", "tile256"])
def tile_n(request):
    P.puro_set_gemm_tile_n(request.param)
    yield request.param
    P.puro_set_gemm_tile_n(0)


@pytest.mark.parametrize("M,N,K", [(128, 128, 128), (384, 640, 384), (256, 1536, 1536), (512, 256, 1024),
                                   (640, 1152, 2560)])
def test_block_linear(M, N, K, tile_n):
    x, w, dy = _inputs(M, N, K, 1000 + M + N + K, t3=True)
    out = run_linear(x, w, dy, P.SCALE_BLOCK)
    ref = oracle_linear(x, w, dy, P.SCALE_BLOCK)
    assert_close(out["y"], ref["y"], "fprop")
    assert_close(out["dx"], ref["dx"], "dgrad")
    assert_close(out["dw"], ref["dw"], "wgrad")


@pytest.mark.parametrize("fmts", [(P.E4M3, P.E4M3, P.E5M2), (P.E5M2, P.E5M2, P.E5M2)])
def test_block_linear_e5m2(fmts, tile_n):
    M, N, K = 256, 384, 256
    x, w, dy = _inputs(M, N, K, 77)
    out = run_linear(x, w, dy, P.SCALE_BLOCK, *fmts)
    ref = oracle_linear(x, w, dy, P.SCALE_BLOCK, *fmts)
    for k in ("y", "dx", "dw"):
        assert_close(out[k], ref[k], k)


@pytest.mark.parametrize("M,N,K", [(256, 1536, 1536), (272, 400, 208), (16, 16, 16), (144, 528, 272)])
def test_tensor_linear(M, N, K):
    x, w, dy = _inputs(M, N, K, 2000 + M + N + K)
    out = run_linear(x, w, dy, P.SCALE_TENSOR)
    ref = oracle_linear(x, w, dy, P.SCALE_TENSOR)
    assert_close(out["y"], ref["y"], "fprop")
    assert_close(out["dx"], ref["dx"], "dgrad")
    assert_close(out["dw"], ref["dw"], "wgrad")


@pytest.mark.parametrize("M,N,K", [(256, 1536, 1536), (272, 400, 208)])
def test_tensor_linear_e5m2_gradients(M, N, K):
    # the hybrid recipe the FP8 section contrasts with its own: per-tensor
    # scales, X and W in E4M3, the output gradient in E5M2 (Dgrad and Wgrad
    # multiply an E5M2 operand by an E4M3 one)
    x, w, dy = _inputs(M, N, K, 2100 + M + N + K)
    out = run_linear(x, w, dy, P.SCALE_TENSOR, P.E4M3, P.E4M3, P.E5M2, step_calls=True)
    ref = oracle_linear(x, w, dy, P.SCALE_TENSOR, P.E4M3, P.E4M3, P.E5M2)
    for k in ("y", "dx", "dw"):
        assert_close(out[k], ref[k], k)


@pytest.mark.parametrize("M,N,K", [(128, 256, 64), (264, 392, 200), (512, 1536, 1536)])
def test_bf16_linear(M, N, K):
    x, w, dy = _inputs(M, N, K, 3000 + M)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=DEV)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    dw = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    P.puro_bf16_linear_fprop(x, w, y, M, N, K)
    P.puro_bf16_linear_dgrad(dy, w.t().contiguous(), dx, M, N, K)
    P.puro_bf16_linear_wgrad(dy.t().contiguous(), x.t().contiguous(), dw, M, N, K)
    torch.cuda.synchronize()
    X, Wd, dY = (O.bf16_to_double(bits(t)) for t in (x, w, dy))
    assert_close(y, O.gemm_tn(X, Wd, 8), "bf16 fprop")
    assert_close(dx, O.gemm_tn(dY, np.ascontiguousarray(Wd.T), 8), "bf16 dgrad")
    assert_close(dw, O.gemm_tn(np.ascontiguousarray(dY.T), np.ascontiguousarray(X.T), 8), "bf16 wgrad")


def test_fprop_of_transposed_weight_equals_dgrad_bitwise():
    """Dgrad is Fprop of the linear whose weight is W^T: same kernel, same
    operand bytes, so the outputs are identical bit for bit."""
    M, N, K = 256, 512, 384
    x, w, dy = _inputs(M, N, K, 55)
    out = run_linear(x, w, dy, P.SCALE_BLOCK)
    y2 = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    P.puro_fp8_linear_fprop(out["dyq"].rowwise, out["wq"].colwise, y2)
    torch.cuda.synchronize()
    assert torch.equal(y2.view(torch.int16), out["dx"].view(torch.int16))


def test_zero_reduction_writes_zeros_and_empty_output_is_noop():
    import ctypes
    lib = P.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    buf = torch.zeros(4096, dtype=torch.uint8, device=DEV)
    p = buf.data_ptr()
    a = P.puro_fp8_tensor_t(p, p, 256, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b = P.puro_fp8_tensor_t(p, p, 128, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, 0)
    y = torch.full((256, 128), 7.0, dtype=torch.bfloat16, device=DEV)
    assert lib.puro_fp8_linear_fprop(ctypes.byref(a), ctypes.byref(b), y.data_ptr(), None, 0, None, stream) == 0
    torch.cuda.synchronize()
    assert torch.all(y == 0)
    a0 = P.puro_fp8_tensor_t(p, p, 0, 128, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b1 = P.puro_fp8_tensor_t(p, p, 128, 128, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, 0)
    y.fill_(3.0)
    assert lib.puro_fp8_linear_fprop(ctypes.byref(a0), ctypes.byref(b1), y.data_ptr(), None, 0, None, stream) == 0
    torch.cuda.synchronize()
    assert torch.all(y == 3.0)


def test_gemm_status_word_stays_clear_on_success():
    M, N, K = 256, 256, 256
    x, w, dy = _inputs(M, N, K, 91)
    out = run_linear(x, w, dy, P.SCALE_BLOCK)  # asserts the status word is 0
    assert torch.isfinite(out["y"].float()).all()


@pytest.mark.parametrize("scaling,M,N,K", [(P.SCALE_BLOCK, 8192, 256, 256), (P.SCALE_BLOCK, 4096, 384, 1536),
                                           (P.SCALE_TENSOR, 4112, 400, 208)])
def test_wgrad_split_reduction(scaling, M, N, K):
    """Small-output Wgrad with a long reduction (tokens): with a workspace
    the reduction is split across CTAs (FP32 partials + a fixed-order sum);
    both schedules must meet the tolerance against the oracle."""
    x, w, dy = _inputs(M, N, K, 4000 + M + N, t3=True)
    xq = P.quantize(x, P.E4M3, scaling, P.ROLE_ACT)
    dyq = P.quantize(dy, P.E4M3, scaling, P.ROLE_ACT)
    ws_bytes = P.puro_fp8_workspace_size(N, K, M)
    assert ws_bytes > 0, "this shape should take the split schedule"
    ws = torch.full((ws_bytes,), 0xFF, dtype=torch.uint8, device=DEV)  # NaN garbage: must be overwritten
    dw_split = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    dw_plain = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw_split, workspace=ws)
    P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw_plain)
    torch.cuda.synchronize()
    ref = oracle_linear(x, w, dy, scaling)["dw"]
    assert_close(dw_split, ref, "wgrad (split reduction)")
    assert_close(dw_plain, ref, "wgrad (single pass)")
    # too small a workspace silently falls back to the single-pass schedule
    dw_small = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw_small, workspace=ws[: ws_bytes // 2])
    torch.cuda.synchronize()
    assert torch.equal(dw_small.view(torch.int16), dw_plain.view(torch.int16))


@pytest.mark.parametrize("M,N,K,split", [(512, 384, 640, False), (640, 1152, 2560, False), (8192, 256, 256, True),
                                         (4096, 384, 1536, True)])
def test_wgrad_main_grad_accumulates_in_fp32(M, N, K, split):
    """main_grad += dY^T X, twice from the same FP32 start: the result is the
    start plus twice the oracle's product (within the GEMM tolerance), it is
    deterministic, and the split schedule (with a workspace) agrees."""
    x, w, dy = _inputs(M, N, K, 5000 + M + N + K, t3=True)
    xq = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    ws = None
    if split:
        ws_bytes = P.puro_fp8_workspace_size(N, K, M)
        assert ws_bytes > 0, "this shape should take the split schedule"
        ws = torch.full((ws_bytes,), 0xFF, dtype=torch.uint8, device=DEV)
    main0 = W.normal_f32((N, K), 0.05, DEV, 6000 + M)
    runs = []
    for _ in range(2):
        main = main0.clone()
        P.puro_fp8_linear_wgrad_main_grad(dyq.colwise, xq.colwise, main, workspace=ws)
        P.puro_fp8_linear_wgrad_main_grad(dyq.colwise, xq.colwise, main, workspace=ws)
        runs.append(main)
    torch.cuda.synchronize()
    assert torch.equal(runs[0], runs[1]), "main-grad accumulation is not deterministic"
    dw_ref = oracle_linear(x, w, dy, P.SCALE_BLOCK)["dw"]
    start = main0.double().cpu().numpy()
    got = runs[0].double().cpu().numpy()
    ok, ratio = O.within_tolerance(got - start, 2.0 * dw_ref)
    assert ok, f"main-grad increment outside tolerance (worst ratio {ratio:.3g})"
    # and the FP32 sum keeps far more than BF16's precision: typical error
    # well below a BF16 ulp of the increment
    rel = np.abs((got - start) - 2.0 * dw_ref) / np.maximum(np.abs(2.0 * dw_ref), 1e-30)
    assert float(np.median(rel)) < 2.0 ** -12, f"median relative error {float(np.median(rel)):.3g}"


def test_wgrad_main_grad_zero_reduction_leaves_it_unchanged():
    import ctypes
    lib = P.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    buf = torch.zeros(4096, dtype=torch.uint8, device=DEV)
    p = buf.data_ptr()
    a = P.puro_fp8_tensor_t(p, p, 256, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b = P.puro_fp8_tensor_t(p, p, 384, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    main = W.normal_f32((256, 384), 1.0, DEV, 77)
    before = main.clone()
    assert lib.puro_fp8_linear_wgrad_main_grad(ctypes.byref(a), ctypes.byref(b), main.data_ptr(), None, 0, None,
                                               stream) == 0
    torch.cuda.synchronize()
    assert torch.equal(main, before)


def test_backward_groups_a_wgrad_that_would_split():
    """qkv shape at 8192 tokens with a workspace: the Wgrad ([2048, 1536]
    output, 48 tiles) would split its reduction, but one grouped launch with
    it unsplit is modelled faster, so both outputs are bit-identical to the
    separate calls without a workspace, and within tolerance of the oracle."""
    M, N, K = 8192, 2048, 1536
    assert P.puro_fp8_workspace_size(N, K, M) > 0, "the Wgrad alone would split"
    ws_bytes = max(P.puro_fp8_workspace_size(M, K, N), P.puro_fp8_workspace_size(N, K, M))
    assert P.puro_fp8_linear_backward_launches(M, N, K, ws_bytes) == 1
    x, w, dy = _inputs(M, N, K, 6500, t3=True)
    xq = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    wq = P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    dx, dw = torch.empty((M, K), dtype=torch.bfloat16, device=DEV), torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    dx1, dw1 = torch.empty_like(dx), torch.empty_like(dw)
    ws = torch.full((ws_bytes,), 0xFF, dtype=torch.uint8, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_fp8_linear_backward(dyq.rowwise, wq.colwise, dx, dyq.colwise, xq.colwise, dw, ws, dev_status=status)
    P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, dx1)
    P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw1)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    assert torch.equal(dx.view(torch.int16), dx1.view(torch.int16))
    assert torch.equal(dw.view(torch.int16), dw1.view(torch.int16)), "dW is not the unsplit Wgrad's"
    rng = np.random.default_rng(6501)
    dYt = O.dequant_rows_1x128(*par_quantize_cols_128x1(bits(dy), P.E4M3), P.E4M3)
    Xt = O.dequant_rows_1x128(*par_quantize_cols_128x1(bits(x), P.E4M3), P.E4M3)
    check_gemm_every_tile(dw, dYt, Xt, rng, "grouped wgrad")


@pytest.mark.parametrize("M,N,K", [(8192, 4096, 2048),     # both unsplit: one grouped launch
                                   (4096, 2304, 1536),     # ragged last rounds in both
                                   (2048, 1536, 1536)])    # Wgrad small enough to split: two launches
def test_grouped_backward_equals_separate_calls(M, N, K):
    """puro_fp8_linear_backward gives the same dX and dW as the separate
    Dgrad and Wgrad calls, bit for bit (without a workspace both run
    unsplit, as the grouped launch does), and within tolerance of the
    oracle."""
    x, w, dy = _inputs(M, N, K, 6000 + M + N + K)
    xq = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    wq = P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    dx, dw = torch.empty((M, K), dtype=torch.bfloat16, device=DEV), torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    dx1, dw1 = torch.empty_like(dx), torch.empty_like(dw)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_fp8_linear_backward(dyq.rowwise, wq.colwise, dx, dyq.colwise, xq.colwise, dw, dev_status=status)
    P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, dx1)
    P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw1)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    assert torch.equal(dx.view(torch.int16), dx1.view(torch.int16)), "dX differs from the separate Dgrad"
    assert torch.equal(dw.view(torch.int16), dw1.view(torch.int16)), "dW differs from the separate Wgrad"
    if M * N * K <= 4096 * 2304 * 1536:
        ref = oracle_linear(x, w, dy, P.SCALE_BLOCK)
        assert_close(dx, ref["dx"], "grouped dgrad")
        assert_close(dw, ref["dw"], "grouped wgrad")
    # with a workspace (the Wgrad may split): still within tolerance of the separate calls' results
    ws = torch.empty(max(16, P.puro_fp8_workspace_size(M, K, N), P.puro_fp8_workspace_size(N, K, M)),
                     dtype=torch.uint8, device=DEV)
    P.puro_fp8_linear_backward(dyq.rowwise, wq.colwise, dx, dyq.colwise, xq.colwise, dw, ws, status)
    torch.cuda.synchronize()
    assert torch.equal(dx.view(torch.int16), dx1.view(torch.int16))
    assert P.puro_fp8_get_status(status) == 0


# --------------------------------------------------------------------------
# Several tiles per CTA pair.  The persistent grid holds at most 76 pairs on
# GB300 (152 SMs), so outputs of 256 or more 256-wide pair tiles make every
# pair loop over 3-4 tiles: the persistent schedule, the alternation of the
# accumulator buffers in tensor memory (two whole 256-column buffers for the
# dense kinds, the shifted pair for the block-scaled kind) and the reuse of
# the epilogue's staging.  Each output is checked on the cross product of one
# sampled row and column in every 32 (every 32 x 32 piece of every tile).
# Shapes: Y [4112, 4224] 17 x 17 pair tiles (ragged last row and column
# tiles), dX [4112, 3968] 17 x 16, dW [4224, 3968] 17 x 16; the Wgrad
# reduction (M = 4112 tokens) ends in a partial K stage.
# --------------------------------------------------------------------------
MANY_M, MANY_N, MANY_K = 4112, 4224, 3968


def _f64(a):
    return np.ascontiguousarray(a, dtype=np.float64)


@pytest.mark.parametrize("fmt_g", [P.E4M3, P.E5M2], ids=["e4m3", "e5m2_gradients"])
def test_tensor_linear_many_tiles_per_pair(fmt_g):
    """Per-tensor scaling (workload C1's recipe), E4M3 throughout or with
    E5M2 output gradients (the hybrid recipe), as the training step calls it."""
    M, N, K = MANY_M, MANY_N, MANY_K
    x, w, dy = _inputs(M, N, K, 7100 + fmt_g)
    out = run_linear(x, w, dy, P.SCALE_TENSOR, P.E4M3, P.E4M3, fmt_g, step_calls=True)
    ops = []
    for t, q, fmt in ((x, out["xq"], P.E4M3), (w, out["wq"], P.E4M3), (dy, out["dyq"], fmt_g)):
        amax, codes, si = O.quantize_tensor(bits(t), fmt)
        assert int(host(q.amax)[0]) & 0xFFFF == amax
        assert np.array_equal(host(q.rowwise.data), codes), "per-tensor codes (several tiles per CTA)"
        assert np.array_equal(host(q.colwise.data), np.ascontiguousarray(codes.T)), "transposed per-tensor codes"
        ops.append(O.dequant_tensor(codes, si, fmt))
    X, Wd, dY = ops
    rng = np.random.default_rng(7200 + fmt_g)
    check_gemm_every_tile(out["y"], X, Wd, rng, "per-tensor fprop")
    check_gemm_every_tile(out["dx"], dY, _f64(Wd.T), rng, "per-tensor dgrad")
    check_gemm_every_tile(out["dw"], _f64(dY.T), _f64(X.T), rng, "per-tensor wgrad")


def test_bf16_linear_many_tiles_per_pair():
    """The BF16 comparison build (kind::f16) on the same multi-tile shapes."""
    M, N, K = MANY_M, MANY_N, MANY_K
    x, w, dy = _inputs(M, N, K, 7300)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=DEV)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    dw = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_bf16_linear_fprop(x, w, y, M, N, K, dev_status=status)
    P.puro_bf16_linear_dgrad(dy, w.t().contiguous(), dx, M, N, K, dev_status=status)
    P.puro_bf16_linear_wgrad(dy.t().contiguous(), x.t().contiguous(), dw, M, N, K, dev_status=status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    X, Wd, dY = (O.bf16_to_double(bits(t)) for t in (x, w, dy))
    rng = np.random.default_rng(7301)
    check_gemm_every_tile(y, X, Wd, rng, "bf16 fprop")
    check_gemm_every_tile(dx, dY, _f64(Wd.T), rng, "bf16 dgrad")
    check_gemm_every_tile(dw, _f64(dY.T), _f64(X.T), rng, "bf16 wgrad")


def test_block_linear_many_tiles_per_pair(tile_n):
    """The paper's blockwise recipe on the same multi-tile shapes (M a
    multiple of 128 here), both tile forms, separate (unsplit) calls."""
    M, N, K = 4096, MANY_N, MANY_K
    x, w, dy = _inputs(M, N, K, 7400, t3=True)
    out = run_linear(x, w, dy, P.SCALE_BLOCK)
    xb, wb, dyb = bits(x), bits(w), bits(dy)
    X = O.dequant_rows_1x128(*par_quantize_rows_1x128(xb, P.E4M3), P.E4M3)
    Xt = O.dequant_rows_1x128(*par_quantize_cols_128x1(xb, P.E4M3), P.E4M3)
    Wd = O.dequant_blocks_128x128(*par_quantize_blocks_128x128(wb, P.E4M3), P.E4M3)
    dY = O.dequant_rows_1x128(*par_quantize_rows_1x128(dyb, P.E4M3), P.E4M3)
    dYt = O.dequant_rows_1x128(*par_quantize_cols_128x1(dyb, P.E4M3), P.E4M3)
    rng = np.random.default_rng(7401 + tile_n)
    check_gemm_every_tile(out["y"], X, Wd, rng, "block fprop")
    check_gemm_every_tile(out["dx"], dY, _f64(Wd.T), rng, "block dgrad")
    check_gemm_every_tile(out["dw"], dYt, Xt, rng, "block wgrad")


def test_wgrad_main_grad_unsplit_gate_up_shape():
    """main_grad += dY^T X into the FP32 [17920, 1536] main-grad of the
    gate_up projection, unsplit (70 x 6 = 420 pair tiles, 5-6 per pair):
    the increment against the oracle on every 32 x 32 piece of every tile."""
    M, N, K = 1024, 17920, 1536
    x, w, dy = _inputs(M, N, K, 7500, t3=True)
    xq = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    assert P.puro_fp8_workspace_size(N, K, M) == 0, "this output is large enough not to split"
    main0 = W.normal_f32((N, K), 0.05, DEV, 7501)
    main = main0.clone()
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_fp8_linear_wgrad_main_grad(dyq.colwise, xq.colwise, main, dev_status=status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    rng = np.random.default_rng(7502)
    from _parity import sample_every
    rows, cols = sample_every(N, rng), sample_every(K, rng)
    r_t, c_t = (torch.from_numpy(v).to(DEV) for v in (rows, cols))
    dYt = O.dequant_rows_1x128(*par_quantize_cols_128x1(bits(dy[:, r_t]), P.E4M3), P.E4M3)
    Xt = O.dequant_rows_1x128(*par_quantize_cols_128x1(bits(x[:, c_t]), P.E4M3), P.E4M3)
    ref = O.gemm_tn(dYt, Xt, 8)
    inc = (main[r_t][:, c_t].double() - main0[r_t][:, c_t].double()).cpu().numpy()
    ok, ratio = O.within_tolerance(inc, ref)
    assert ok, f"main-grad increment outside tolerance (worst ratio {ratio:.3g})"
