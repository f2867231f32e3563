"""SwiGLU fused ahead of the blockwise activation quantiser.

y = bf16(silu(gate) * up) is evaluated in fp32 on the GPU and in fp64 by the
oracle, so y may differ from the oracle's correctly rounded value by one
bf16 ulp where the exact value lies within the fp32 error of a rounding
boundary (rare: the test bounds how often).  Every FP8 code and scale is an
exact function of y, so given the kernel's own y they must equal the
oracle's bit for bit; a call that does not store y must produce the same
bytes as one that does.
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import bits, check_block_act_quant

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


def _gate_up(rows, cols, seed, fused_layout):
    """gate ~ 3 t3 (both tails of the sigmoid, a few gates at +-40..120, where
    e^g is subnormal in fp32, and exact zeros), up ~ N(0,1) times per-row
    powers of two; as the two halves
    of one [rows, 2 cols] output when fused_layout, else two tensors."""
    g = W.student_t3_f32((rows, cols), DEV, seed) * 3.0
    gen = torch.Generator(device=DEV)
    gen.manual_seed(seed + 1)
    idx = torch.randint(0, rows * cols, (96,), generator=gen, device=DEV)
    special = torch.tensor([0.0, 40.0, -40.0, 80.0, -80.0, 55.5, -61.0, 0.0, -79.5, -90.0, -100.0, 120.0],
                           device=DEV).repeat(8)
    g.view(-1)[idx] = special
    k = torch.randint(-6, 7, (rows, 1), generator=gen, device=DEV).float()
    u = W.normal_f32((rows, cols), 1.0, DEV, seed + 2) * torch.exp2(k)
    if fused_layout:
        gu = torch.cat([g, u], dim=1).to(torch.bfloat16)
        return gu[:, :cols], gu[:, cols:]
    return g.to(torch.bfloat16), u.to(torch.bfloat16)


def _empty_q(rows, cols, with_t=True):
    row = P.FP8Operand(torch.empty((rows, cols), dtype=torch.uint8, device=DEV),
                       P.empty_scales(rows, cols, P.SCALE_BLOCK, P.ROLE_ACT, DEV))
    col = P.FP8Operand(torch.empty((cols, rows), dtype=torch.uint8, device=DEV),
                       P.empty_scales(cols, rows, P.SCALE_BLOCK, P.ROLE_ACT, DEV)) if with_t else None
    return P.Quantized(row, col)


def _check_y(y: torch.Tensor, gate, up):
    ref = O.swiglu(bits(gate), bits(up))
    got = bits(y)
    rv = torch.from_numpy(ref.view(np.int16)).view(torch.bfloat16).double().numpy()
    gv = torch.from_numpy(got.view(np.int16)).view(torch.bfloat16).double().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(rv), 2.0 ** -126))) - 7)
    err = np.abs(gv - rv)
    assert float((err / ulp).max()) <= 1.0, "y differs from the oracle by more than one bf16 ulp"
    frac = np.count_nonzero(got != ref) / got.size
    assert frac <= 1e-3, f"{frac:.2e} of y values differ from the correctly rounded result"


@pytest.mark.parametrize("rows,cols,fused_layout,fmt", [(256, 640, False, P.E4M3), (384, 1536, True, P.E4M3),
                                                        (128, 8960, True, P.E4M3), (1024, 2048, True, P.E5M2),
                                                        (640, 384, False, P.E5M2)])
def test_fused_swiglu_quantize(rows, cols, fused_layout, fmt):
    gate, up = _gate_up(rows, cols, 900 + rows + cols, fused_layout)
    y = torch.full((rows, cols), float("nan"), dtype=torch.bfloat16, device=DEV)
    q = _empty_q(rows, cols)
    P.puro_fp8_quantize_swiglu(gate, up, fmt, y, q.rowwise.data, q.rowwise.scale, q.colwise.data, q.colwise.scale)
    # the same call without y: identical bytes
    q2 = _empty_q(rows, cols)
    P.puro_fp8_quantize_swiglu(gate, up, fmt, None, q2.rowwise.data, q2.rowwise.scale, q2.colwise.data,
                               q2.colwise.scale)
    torch.cuda.synchronize()
    _check_y(y, gate, up)
    check_block_act_quant(y, q, fmt)
    for a, b in ((q.rowwise.data, q2.rowwise.data), (q.rowwise.scale, q2.rowwise.scale),
                 (q.colwise.data, q2.colwise.data), (q.colwise.scale, q2.colwise.scale)):
        assert torch.equal(a, b), "storing y changed the codes"


def test_rowwise_only_and_unfused_agree():
    rows, cols = 256, 1536
    gate, up = _gate_up(rows, cols, 77, True)
    y1 = torch.empty((rows, cols), dtype=torch.bfloat16, device=DEV)
    y2 = torch.empty_like(y1)
    q = _empty_q(rows, cols, with_t=False)
    P.puro_fp8_quantize_swiglu(gate, up, P.E4M3, y1, q.rowwise.data, q.rowwise.scale)
    P.puro_swiglu_bf16(gate, up, y2)
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
    check_block_act_quant(y1, q, P.E4M3)
    # the unfused output fed to the plain quantiser gives the same codes
    qu = P.quantize(y2, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    torch.cuda.synchronize()
    assert torch.equal(qu.rowwise.data, q.rowwise.data)
    assert torch.equal(qu.rowwise.scale, q.rowwise.scale)


def test_unfused_handles_a_ragged_width():
    rows, cols = 3, 40  # any multiple of 8
    gate, up = _gate_up(rows, cols, 31, True)
    y = torch.empty((rows, cols), dtype=torch.bfloat16, device=DEV)
    P.puro_swiglu_bf16(gate, up, y)
    torch.cuda.synchronize()
    _check_y(y, gate, up)


def test_fused_rejects_a_ragged_shape_on_the_host():
    gate = torch.zeros((200, 256), dtype=torch.bfloat16, device=DEV)
    q = _empty_q(200, 256, with_t=False)
    with pytest.raises(P.PuroError):
        P.puro_fp8_quantize_swiglu(gate, gate, P.E4M3, None, q.rowwise.data, q.rowwise.scale)
