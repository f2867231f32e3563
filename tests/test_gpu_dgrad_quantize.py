"""The Dgrad whose epilogue quantises its own output (the next layer's dY):
puro_fp8_linear_dgrad_quantize against puro_fp8_linear_dgrad, the oracle's
fp64 product and the oracle's blockwise quantiser.

The product comes from the same kernel arithmetic as the plain (unsplit)
Dgrad, so its BF16 output must equal puro_fp8_linear_dgrad's bit for bit
and lie within |gpu - ref| <= 2^-7 |ref| + 1e-3 rms(ref) of the oracle.
Every code and scale must equal, bit for bit, the oracle's 1x128 (rowwise)
and 128x1 (transposed) quantisation of those BF16 values: both sides take
each scale decision from the same BF16 bits.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import assert_close, bits, check_block_act_quant, sample_index

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


def _operands(M, N, K, seed, zero_rows=True):
    """dY [M, N] ~ N(0, 1e-3) times per-row powers of two (row scales up to
    2^12 apart) with a few zero rows, quantised rowwise; the layer's weight
    W [N, K] ~ 0.02 t3, quantised in 128x128 blocks with its transposed copy
    W^T [K, N] (the Dgrad's B operand)."""
    gen = torch.Generator(device=DEV)
    gen.manual_seed(seed)
    dy = W.normal_f32((M, N), 1e-3, DEV, seed) * torch.exp2(torch.randint(-6, 7, (M, 1), generator=gen,
                                                                          device=DEV).float())
    if zero_rows and M >= 8:
        dy[torch.randint(0, M, (4,), generator=gen, device=DEV)] = 0.0
    dy = dy.to(torch.bfloat16)
    w = W.student_t3_f32((N, K), DEV, seed + 1).mul_(0.02).to(torch.bfloat16)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, transpose=False)
    wq = P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
    return dy, w, dyq, wq


def _empty_q(rows, cols, with_t=True):
    row = P.FP8Operand(torch.empty((rows, cols), dtype=torch.uint8, device=DEV),
                       P.empty_scales(rows, cols, P.SCALE_BLOCK, P.ROLE_ACT, DEV))
    col = P.FP8Operand(torch.empty((cols, rows), dtype=torch.uint8, device=DEV),
                       P.empty_scales(cols, rows, P.SCALE_BLOCK, P.ROLE_ACT, DEV)) if with_t else None
    return P.Quantized(row, col)


def _fused(dyq, wq, fmt, dx, q, status=None):
    P.puro_fp8_linear_dgrad_quantize(dyq.rowwise, wq.colwise, fmt, dx, q.rowwise.data, q.rowwise.scale,
                                     q.colwise.data if q.colwise is not None else None,
                                     q.colwise.scale if q.colwise is not None else None, dev_status=status)


@pytest.mark.parametrize("M,N,K,fmt", [(128, 128, 128, P.E4M3), (384, 640, 384, P.E4M3), (512, 1536, 1024, P.E4M3),
                                       (640, 256, 2560, P.E5M2), (1024, 2048, 1536, P.E5M2)])
def test_matches_the_plain_dgrad_and_the_quantiser(M, N, K, fmt):
    dy, w, dyq, wq = _operands(M, N, K, 100 + M + N + K)
    dx_ref = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, dx_ref)  # no workspace: unsplit
    dx = torch.full((M, K), float("nan"), dtype=torch.bfloat16, device=DEV)
    q = _empty_q(M, K)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    _fused(dyq, wq, fmt, dx, q, status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    assert torch.equal(dx.view(torch.int16), dx_ref.view(torch.int16)), "BF16 product differs from the plain Dgrad"
    check_block_act_quant(dx, q, fmt)
    # the product itself, against the oracle's fp64 Dgrad of the same BF16 inputs
    dyq_o, dys_o = O.quantize_rows_1x128(bits(dy), P.E4M3)
    wq_o, ws_o = O.quantize_blocks_128x128(bits(w), P.E4M3)
    wd = O.dequant_blocks_128x128(wq_o, ws_o, P.E4M3)
    ref = O.gemm_tn(O.dequant_rows_1x128(dyq_o, dys_o, P.E4M3), np.ascontiguousarray(wd.T), 8)
    assert_close(dx, ref, "dgrad")


def test_optional_outputs_do_not_change_the_codes():
    M, N, K = 512, 768, 640
    _, _, dyq, wq = _operands(M, N, K, 41)
    q_all = _empty_q(M, K)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    _fused(dyq, wq, P.E4M3, dx, q_all)
    q_nodx = _empty_q(M, K)
    _fused(dyq, wq, P.E4M3, None, q_nodx)
    q_rows = _empty_q(M, K, with_t=False)
    _fused(dyq, wq, P.E4M3, None, q_rows)
    torch.cuda.synchronize()
    for a, b in ((q_all.rowwise.data, q_nodx.rowwise.data), (q_all.rowwise.scale, q_nodx.rowwise.scale),
                 (q_all.colwise.data, q_nodx.colwise.data), (q_all.colwise.scale, q_nodx.colwise.scale),
                 (q_all.rowwise.data, q_rows.rowwise.data), (q_all.rowwise.scale, q_rows.rowwise.scale)):
        assert torch.equal(a, b)
    check_block_act_quant(dx, q_all, P.E4M3)


def test_non_finite_groups():
    # a NaN in one row of dY makes that row of dX NaN: its row groups and
    # every column group it belongs to take the non-finite scale and NaN codes
    M, N, K = 256, 256, 384
    dy, w, _, wq = _operands(M, N, K, 57, zero_rows=False)
    dy[37, 5] = float("nan")
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, transpose=False)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    q = _empty_q(M, K)
    _fused(dyq, wq, P.E4M3, dx, q)
    torch.cuda.synchronize()
    assert torch.isnan(dx[37].float()).all()
    check_block_act_quant(dx, q, P.E4M3)


def test_empty_reduction_gives_zero_codes_and_empty_output_is_a_no_op():
    import ctypes
    lib = P.load_library()
    stream = torch.cuda.current_stream().cuda_stream
    M, K = 256, 384
    buf = torch.zeros(4096, dtype=torch.uint8, device=DEV)
    p = buf.data_ptr()
    a = P.puro_fp8_tensor_t(p, p, M, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b = P.puro_fp8_tensor_t(p, p, K, 0, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, 0)
    q = _empty_q(M, K)
    for t in (q.rowwise.data, q.rowwise.scale, q.colwise.data, q.colwise.scale):
        t.fill_(0x55)
    dx = torch.full((M, K), 1.0, dtype=torch.bfloat16, device=DEV)
    ptrs = [t.data_ptr() for t in (dx, q.rowwise.data, q.rowwise.scale, q.colwise.data, q.colwise.scale)]
    assert lib.puro_fp8_linear_dgrad_quantize(ctypes.byref(a), ctypes.byref(b), P.E4M3, *ptrs, None, stream) == 0
    torch.cuda.synchronize()
    assert not dx.any()
    check_block_act_quant(dx, q, P.E4M3)
    # no rows: nothing written
    a0 = P.puro_fp8_tensor_t(p, p, 0, 128, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b1 = P.puro_fp8_tensor_t(p, p, K, 128, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, 0)
    q.rowwise.data.fill_(0x55)
    assert lib.puro_fp8_linear_dgrad_quantize(ctypes.byref(a0), ctypes.byref(b1), P.E4M3, *ptrs, None, stream) == 0
    torch.cuda.synchronize()
    assert bool((q.rowwise.data == 0x55).all())


@pytest.mark.slow
@pytest.mark.parametrize("name,N,K", [("down", 1536, 8960), ("gate_up", 17920, 1536)])
def test_c5_full_size_sampled(name, N, K):
    """The C5 Dgrad of `down` (dX [32768, 8960]) and of `gate_up` (dX
    [32768, 1536]) at full size: dX equal to the plain Dgrad everywhere,
    codes and scales bit-exact on sampled rows and columns."""
    M = 32768
    _, _, dyq, wq = _operands(M, N, K, 7000 + N)
    dx_ref = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, dx_ref)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    q = _empty_q(M, K)
    _fused(dyq, wq, P.E4M3, dx, q)
    torch.cuda.synchronize()
    assert torch.equal(dx.view(torch.int16), dx_ref.view(torch.int16)), name
    rng = np.random.default_rng(7001 + N)
    rows = torch.from_numpy(sample_index(M, 256, rng)).to(DEV)
    cols = torch.from_numpy(sample_index(K, 64, rng)).to(DEV)
    check_block_act_quant(dx, q, P.E4M3, rows=rows, cols=cols)
