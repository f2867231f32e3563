"""Failure detection without a GPU fault.

Every wait on the device is bounded in wall time: the pipeline waits of the
GEMM kernels and the tile-load waits of the quantiser kernels.  Here the
bound is dropped to zero, so any wait that is not already satisfied gives
up: the kernel must record PURO_ERR_TIMEOUT in the caller's status word,
let its own copies (and MMAs) in flight finish, free tensor memory and
return -- no trap, no hang -- and the context must stay usable (the next
call, with the normal bound, is correct).  The multi-tile cases give up in
the middle of a persistent schedule, with tiles of the same CTA already
done.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import (assert_close, bits, check_block_act_quant, check_block_weight_quant, check_gemm_every_tile,
                     check_tensor_quant, oracle_linear, par_quantize_blocks_128x128, par_quantize_rows_1x128)

pytestmark = pytest.mark.gpu
DEV = "cuda"
DEFAULT_WAIT_NS = 2_000_000_000


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


@pytest.mark.parametrize("kind", ["block", "tensor", "bf16"])
def test_wait_timeout_sets_status_and_context_survives(kind):
    M, N, K = 512, 512, 8192  # 64 k-blocks through a 4-stage ring: the pipeline must wait
    x = W.normal_bf16((M, K), 1.0, DEV, 1)
    w = W.normal_bf16((N, K), 0.02, DEV, 2)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    if kind == "bf16":
        run = lambda st: P.puro_bf16_linear_fprop(x, w, y, M, N, K, dev_status=st)  # noqa: E731
    else:
        sc = P.SCALE_BLOCK if kind == "block" else P.SCALE_TENSOR
        xq = P.quantize(x, P.E4M3, sc, P.ROLE_ACT, transpose=False)
        wq = P.quantize(w, P.E4M3, sc, P.ROLE_WEIGHT, transpose=False)
        run = lambda st: P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, y, dev_status=st)  # noqa: E731
    torch.cuda.synchronize()

    P.puro_set_wait_timeout_ns(0)
    try:
        run(status)
        torch.cuda.synchronize()
    finally:
        P.puro_set_wait_timeout_ns(DEFAULT_WAIT_NS)
    assert P.puro_fp8_get_status(status) == P.PURO_ERR_TIMEOUT

    # the context is intact: the same call with the normal bound is correct
    status.zero_()
    run(status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == P.PURO_OK
    if kind == "bf16":
        import oracle as O
        ref = O.gemm_tn(O.bf16_to_double(bits(x)), O.bf16_to_double(bits(w)), 8)
    else:
        sc = P.SCALE_BLOCK if kind == "block" else P.SCALE_TENSOR
        ref = oracle_linear(x, w, torch.zeros((M, N), dtype=torch.bfloat16, device=DEV), sc)["y"]
    assert_close(y, ref, f"{kind} fprop after a timed-out launch")


def _timed_out_then_correct(run, status):
    """run(status) with a zero wait bound must report PURO_ERR_TIMEOUT; the
    same call with the normal bound must then succeed."""
    torch.cuda.synchronize()
    P.puro_set_wait_timeout_ns(0)
    try:
        run(status)
        torch.cuda.synchronize()
    finally:
        P.puro_set_wait_timeout_ns(DEFAULT_WAIT_NS)
    assert P.puro_fp8_get_status(status) == P.PURO_ERR_TIMEOUT
    status.zero_()
    run(status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == P.PURO_OK


@pytest.mark.parametrize("kind", ["block", "tensor", "bf16"])
def test_wait_timeout_mid_schedule_many_tiles_per_pair(kind):
    """4096 x 4096 x 8192: 256 pair tiles, three to four per CTA pair, each
    with 32-64 K stages through the 3-deep ring."""
    M, N, K = 4096, 4096, 8192
    x = W.normal_bf16((M, K), 1.0, DEV, 3)
    w = W.normal_bf16((N, K), 0.02, DEV, 4)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=DEV)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    rng = np.random.default_rng(5 + len(kind))
    if kind == "bf16":
        _timed_out_then_correct(lambda st: P.puro_bf16_linear_fprop(x, w, y, M, N, K, dev_status=st), status)
        check_gemm_every_tile(y, O.bf16_to_double(bits(x)), O.bf16_to_double(bits(w)), rng, "bf16 fprop")
        return
    sc = P.SCALE_BLOCK if kind == "block" else P.SCALE_TENSOR
    xq = P.quantize(x, P.E4M3, sc, P.ROLE_ACT, transpose=False)
    wq = P.quantize(w, P.E4M3, sc, P.ROLE_WEIGHT, transpose=False)
    _timed_out_then_correct(lambda st: P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, y, dev_status=st), status)
    if kind == "block":
        X = O.dequant_rows_1x128(*par_quantize_rows_1x128(bits(x), P.E4M3), P.E4M3)
        Wd = O.dequant_blocks_128x128(*par_quantize_blocks_128x128(bits(w), P.E4M3), P.E4M3)
    else:
        _, xc, xsi = O.quantize_tensor(bits(x), P.E4M3)
        _, wc, wsi = O.quantize_tensor(bits(w), P.E4M3)
        X, Wd = O.dequant_tensor(xc, xsi, P.E4M3), O.dequant_tensor(wc, wsi, P.E4M3)
    check_gemm_every_tile(y, X, Wd, rng, f"{kind} fprop after a timed-out launch")


QSHAPE = (4096, 4096)  # 1024 tiles of 128 x 128: three to four per persistent CTA


@pytest.mark.parametrize("kind", ["act", "weight", "tensor", "weights_grouped", "rmsnorm", "swiglu"])
def test_quantiser_wait_timeout_sets_status_and_context_survives(kind):
    """Each quantiser kernel gives up on a tile load that has not landed: the
    status word reads PURO_ERR_TIMEOUT, and the same call with the normal
    bound then gives every byte the oracle gives."""
    R, C = QSHAPE
    x = (W.student_t3_f32((R, C), DEV, 21) * 2.0).to(torch.bfloat16)
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    if kind in ("act", "weight", "tensor"):
        sc = P.SCALE_TENSOR if kind == "tensor" else P.SCALE_BLOCK
        role = P.ROLE_WEIGHT if kind == "weight" else P.ROLE_ACT
        q = P.quantize(x, P.E4M3, sc, role)
        _timed_out_then_correct(lambda st: P.quantize(x, P.E4M3, sc, role, out=q, dev_status=st), status)
        if kind == "tensor":
            check_tensor_quant(x, q, P.E4M3)
        elif kind == "weight":
            check_block_weight_quant(x, q, P.E4M3)
        else:
            check_block_act_quant(x, q, P.E4M3)
    elif kind == "weights_grouped":
        q = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
        table = P.weight_table([(x, q)])
        _timed_out_then_correct(lambda st: P.puro_fp8_quantize_weights(table, P.E4M3, dev_status=st), status)
        check_block_weight_quant(x, q, P.E4M3)
    elif kind == "rmsnorm":
        rstd = torch.empty(R, dtype=torch.float32, device=DEV)
        y = torch.empty_like(x)
        q = P.quantize(torch.empty_like(x))
        _timed_out_then_correct(lambda st: P.puro_fp8_quantize_rmsnorm(
            x, None, 1e-6, P.E4M3, rstd, y, q.rowwise.data, q.rowwise.scale, q.colwise.data, q.colwise.scale,
            dev_status=st), status)
        check_block_act_quant(y, q, P.E4M3)
        ref = O.rmsnorm_apply_f32(bits(x), rstd.cpu().numpy())
        assert np.array_equal(bits(y), ref), "normalised y after a timed-out launch"
    else:
        up = W.normal_bf16((R, C), 1.0, DEV, 22)
        h = torch.empty_like(x)
        q = P.quantize(torch.empty_like(x))
        _timed_out_then_correct(lambda st: P.puro_fp8_quantize_swiglu(
            x, up, P.E4M3, h, q.rowwise.data, q.rowwise.scale, q.colwise.data, q.colwise.scale, dev_status=st),
            status)
        check_block_act_quant(h, q, P.E4M3)
