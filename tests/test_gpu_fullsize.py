"""GPU parity at the full sizes of the benchmark workloads, in the launch
configuration the benchmark times.

C1 (one linear, M=256) is compared element by element in both scaling
modes.  C2-C6 (C6: the paper's own Qwen3-1.7B-shaped model) use the
paper's blockwise recipe and are compared on sampled
outputs the oracle computes one by one: every quantised byte and scale on
sampled rows and columns, and every GEMM output on the cross product of
sampled rows and columns (which contains the four corner 128x128 tiles).
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
    out = run_linear(li.x, li.w, li.dy, scaling)
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


def _sampled(key, layer, idx, seed):
    wl = W.WORKLOADS[key]
    li = W.make_linear(wl, layer, idx, DEV)
    out = run_linear(li.x, li.w, li.dy, P.SCALE_BLOCK)
    check_linear_sampled(li.x, li.w, li.dy, out, np.random.default_rng(seed))
    del out, li
    torch.cuda.empty_cache()


@pytest.mark.parametrize("idx", [0, 1])
def test_c2_attention_projections(idx):
    _sampled("C2", 0, idx, 20 + idx)


@pytest.mark.parametrize("idx", [0, 1])
def test_c3_mlp_with_outliers(idx):
    _sampled("C3", 0, idx, 30 + idx)


@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_c4_decoder_layer(idx):
    _sampled("C4", 0, idx, 40 + idx)


@pytest.mark.parametrize("layer", [0, 13, 27])
@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_c5_layers(layer, idx):
    _sampled("C5", layer, idx, 500 + 4 * layer + idx)


@pytest.mark.parametrize("layer", [0, 27])
@pytest.mark.parametrize("idx", [0, 1, 2, 3])
def test_c6_paper_model_layers(layer, idx):
    """The paper's own model shape (Qwen3-1.7B linears, M = 8192)."""
    _sampled("C6", layer, idx, 600 + 4 * layer + idx)
