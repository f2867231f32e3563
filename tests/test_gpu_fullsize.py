"""GPU parity at the full sizes of the benchmark workloads, in the launch
configuration the benchmark times: weights through the grouped weight
quantiser, Dgrad and Wgrad through puro_fp8_linear_backward with a
workspace (one grouped launch where both are unsplit, a split reduction for
small-output Wgrads), as in the training step.

C1 (one linear, M=256) is compared element by element in both scaling
modes.  C2-C6 (C6: the paper's own Qwen3-1.7B-shaped model) use the
paper's blockwise recipe:
  - quantised bytes: every FP8 byte and scale of X, W and dY (both copies)
    on C2, C3, C4 and on layers 0, 13 and 27 of C5; W in full and X, dY on
    the first/last 128 and 96 random rows and columns on the other 25 C5
    layers and on C6;
  - GEMM outputs (every layer of C5): the cross product of the first 128,
    the last 128 and 96 random row and column indices of each output, i.e.
    the four complete corner 128x128 tiles plus 9216 seeded random entries,
    against the oracle's fp64 products.
"""
import numpy as np
import pytest
import torch

import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import (assert_close, check_block_act_quant, check_block_weight_quant, check_linear_sampled,
                     check_tensor_quant, oracle_linear, run_linear)

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


@pytest.mark.parametrize("scaling", [P.SCALE_TENSOR, P.SCALE_BLOCK])
def test_c1_full(scaling):
    wl = W.WORKLOADS["C1"]
    li = W.make_linear(wl, 0, 0, DEV)
    out = run_linear(li.x, li.w, li.dy, scaling, step_calls=True)
    if scaling == P.SCALE_TENSOR:
        check_tensor_quant(li.x, out["xq"], P.E4M3)
        check_tensor_quant(li.w, out["wq"], P.E4M3)
        check_tensor_quant(li.dy, out["dyq"], P.E4M3)
    else:
        check_block_act_quant(li.x, out["xq"], P.E4M3)
        check_block_weight_quant(li.w, out["wq"], P.E4M3)
        check_block_act_quant(li.dy, out["dyq"], P.E4M3)
    ref = oracle_linear(li.x, li.w, li.dy, scaling)
    assert_close(out["y"], ref["y"], "fprop")
    assert_close(out["dx"], ref["dx"], "dgrad")
    assert_close(out["dw"], ref["dw"], "wgrad")


def _sampled(key, layer, idx, seed, full_bytes=False):
    wl = W.WORKLOADS[key]
    li = W.make_linear(wl, layer, idx, DEV)
    out = run_linear(li.x, li.w, li.dy, P.SCALE_BLOCK, step_calls=True)
    check_linear_sampled(li.x, li.w, li.dy, out, np.random.default_rng(seed), full_bytes=full_bytes)
    del out, li
    torch.cuda.empty_cache()


@pytest.mark.parametrize("idx", [0, 1])
def test_c2_attention_projections(idx):
    _sampled("C2", 0, idx, 20 + idx, full_bytes=True)


@pytest.mark.parametrize("idx", [0, 1])
def test_c3_mlp_with_outliers(idx):
    _sampled("C3", 0, idx, 30 + idx, full_bytes=True)


@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_c4_decoder_layer(idx):
    _sampled("C4", 0, idx, 40 + idx, full_bytes=True)


C5_FULL_LAYERS = (0, 13, 27)


@pytest.mark.parametrize("layer", range(28))
def test_c5_layer(layer):
    """All four linears of one C5 layer: every byte on layers 0, 13 and 27,
    sampled rows and columns on the others; sampled GEMM outputs on all."""
    for idx in range(4):
        _sampled("C5", layer, idx, 500 + 4 * layer + idx, full_bytes=layer in C5_FULL_LAYERS)


@pytest.mark.parametrize("layer", [0, 27])
@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_c6_paper_model_layers(layer, idx):
    """The paper's own model shape (Qwen3-1.7B linears, M = 8192)."""
    _sampled("C6", layer, idx, 600 + 4 * layer + idx)


def test_c5_rmsnorm_quantize_full_size():
    """The fused RMSNorm -> quantise on the C5 qkv/gate_up input [32768, 1536]
    (with a gain), sampled: rstd of sampled rows within its bound, y and the
    codes bit-exact given the kernel's rstd on sampled rows and columns."""
    import oracle as O
    from _parity import bits, sample_index

    M, K = 32768, 1536
    h = (W.student_t3_f32((M, K), DEV, 5100) * 4.0).to(torch.bfloat16)
    gamma = W.normal_f32((K,), 0.1, DEV, 5101).add_(1.0).to(torch.bfloat16)
    rstd = torch.empty(M, dtype=torch.float32, device=DEV)
    y = torch.empty((M, K), dtype=torch.bfloat16, device=DEV)
    q = P.quantize(torch.empty((M, K), dtype=torch.bfloat16, device=DEV))
    P.puro_fp8_quantize_rmsnorm(h, gamma, 1e-6, P.E4M3, rstd, y, q.rowwise.data, q.rowwise.scale, q.colwise.data,
                                q.colwise.scale)
    torch.cuda.synchronize()
    rng = np.random.default_rng(5102)
    rows = torch.from_numpy(sample_index(M, 256, rng)).to(DEV)
    cols = torch.from_numpy(sample_index(K, 64, rng)).to(DEV)
    ref = O.rmsnorm_rstd(bits(h[rows]), 1e-6)
    rel = np.abs(rstd[rows].double().cpu().numpy() - ref) / ref
    assert float(rel.max()) <= (K / 64 + 8) * 2.0 ** -24
    y_ref = O.rmsnorm_apply_f32(bits(h[rows]), rstd[rows].cpu().numpy(), bits(gamma))
    assert np.array_equal(bits(y[rows]), y_ref), "normalised y differs on sampled rows"
    check_block_act_quant(y, q, P.E4M3, rows=rows, cols=cols)


def test_c5_swiglu_quantize_full_size():
    """The fused SwiGLU -> quantise on the C5 down input [32768, 8960] from the
    gate/up output [32768, 17920], sampled: h within one bf16 ulp of the
    oracle on sampled rows, the codes bit-exact given the kernel's h."""
    import oracle as O
    from _parity import bits, sample_index

    M, F = 32768, 8960
    gu = (W.student_t3_f32((M, 2 * F), DEV, 5200) * 3.0).to(torch.bfloat16)
    h = torch.empty((M, F), dtype=torch.bfloat16, device=DEV)
    q = P.quantize(torch.empty((M, F), dtype=torch.bfloat16, device=DEV))
    P.puro_fp8_quantize_swiglu(gu[:, :F], gu[:, F:], P.E4M3, h, q.rowwise.data, q.rowwise.scale, q.colwise.data,
                               q.colwise.scale)
    torch.cuda.synchronize()
    rng = np.random.default_rng(5201)
    rows = torch.from_numpy(sample_index(M, 256, rng)).to(DEV)
    cols = torch.from_numpy(sample_index(F, 64, rng)).to(DEV)
    g_rows = gu[rows]
    ref = O.swiglu(bits(g_rows[:, :F]), bits(g_rows[:, F:]))
    got = bits(h[rows])
    rv = torch.from_numpy(ref.view(np.int16)).view(torch.bfloat16).double().numpy()
    gv = torch.from_numpy(got.view(np.int16)).view(torch.bfloat16).double().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(rv), 2.0 ** -126))) - 7)
    assert float((np.abs(gv - rv) / ulp).max()) <= 1.0
    assert np.count_nonzero(got != ref) / got.size <= 1e-3
    check_block_act_quant(h, q, P.E4M3, rows=rows, cols=cols)
