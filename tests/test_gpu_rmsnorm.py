"""RMSNorm fused ahead of the blockwise activation quantiser.

The one floating-point decision with a free summation order is rstd (an
fp32 sum of squares): it is compared with the oracle's fp64 value within a
bound derived from the fp32 accumulation.  Everything downstream is exactly
determined by rstd, so given the kernel's own rstd the normalised values y
(bf16) and every FP8 code and scale must equal the oracle's bit for bit.
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


def _bf16_from_bits(b: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(np.ascontiguousarray(b).view(np.int16)).view(torch.bfloat16)


def _h(rows, cols, seed):
    """Student-t(3) rows with per-row scales 2^-6 .. 2^6 (a spread of rstd)."""
    h = W.student_t3_f32((rows, cols), DEV, seed)
    g = torch.Generator(device=DEV)
    g.manual_seed(seed + 1)
    k = torch.randint(-6, 7, (rows, 1), generator=g, device=DEV).float()
    return (h * torch.exp2(k)).to(torch.bfloat16)


def _empty_q(rows, cols):
    return P.Quantized(
        P.FP8Operand(torch.empty((rows, cols), dtype=torch.uint8, device=DEV),
                     P.empty_scales(rows, cols, P.SCALE_BLOCK, P.ROLE_ACT, DEV)),
        P.FP8Operand(torch.empty((cols, rows), dtype=torch.uint8, device=DEV),
                     P.empty_scales(cols, rows, P.SCALE_BLOCK, P.ROLE_ACT, DEV)))


@pytest.mark.parametrize("rows,cols,gain,write_y", [(256, 640, True, True), (384, 1536, False, True),
                                                    (1024, 2048, True, False), (128, 8960, True, True)])
def test_fused_rmsnorm_quantize(rows, cols, gain, write_y):
    eps = 1e-6
    h = _h(rows, cols, 700 + rows + cols)
    gamma = W.normal_f32((cols,), 0.1, DEV, 800 + cols).add_(1.0).to(torch.bfloat16) if gain else None
    rstd = torch.empty(rows, dtype=torch.float32, device=DEV)
    y = torch.full((rows, cols), float("nan"), dtype=torch.bfloat16, device=DEV) if write_y else None
    q = _empty_q(rows, cols)
    P.puro_fp8_quantize_rmsnorm(h, gamma, eps, P.E4M3, rstd, y, q.rowwise.data, q.rowwise.scale, q.colwise.data,
                                q.colwise.scale)
    torch.cuda.synchronize()

    # rstd: fp32 sum of cols/64 squares per accumulator, then a 32-way tree
    ref = O.rmsnorm_rstd(bits(h), eps)
    got = rstd.double().cpu().numpy()
    bound = (cols / 64 + 8) * 2.0 ** -24
    rel = np.abs(got - ref) / ref
    assert float(rel.max()) <= bound, f"rstd relative error {float(rel.max()):.3g} > {bound:.3g}"

    # y and the codes, exactly, given the kernel's rstd
    y_ref = O.rmsnorm_apply_f32(bits(h), rstd.cpu().numpy(), None if gamma is None else bits(gamma))
    if write_y:
        yb = bits(y)
        bad = np.argwhere(yb != y_ref)
        assert bad.size == 0, f"normalised y: {len(bad)} values differ; first at {tuple(bad[0])}"
    check_block_act_quant(_bf16_from_bits(y_ref).to(DEV), q, P.E4M3)


def test_unfused_rmsnorm_matches_the_fused_one():
    rows, cols = 256, 1536
    h = _h(rows, cols, 901)
    gamma = W.normal_f32((cols,), 0.1, DEV, 902).add_(1.0).to(torch.bfloat16)
    r1 = torch.empty(rows, dtype=torch.float32, device=DEV)
    r2 = torch.empty_like(r1)
    y1 = torch.empty((rows, cols), dtype=torch.bfloat16, device=DEV)
    y2 = torch.empty_like(y1)
    q = _empty_q(rows, cols)
    P.puro_fp8_quantize_rmsnorm(h, gamma, 1e-6, P.E4M3, r1, y1, q.rowwise.data, q.rowwise.scale)
    P.puro_rmsnorm_bf16(h, gamma, 1e-6, r2, y2)
    torch.cuda.synchronize()
    assert torch.equal(r1, r2)
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
