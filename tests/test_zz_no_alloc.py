"""The allocation-free Wgrad entry point (puro_fp8_linear_wgrad_noalloc).

It exists for callers that cannot obtain device memory while they run the
backward pass (engine plugins that own every device buffer, latency-critical
code that cannot pay for cudaMalloc's device-wide synchronisation, fixed
memory budgets): instead of caller-supplied scratch, its split-reduction
schedule uses a fixed array inside the library.  This test calls it through
the C ABI on two calls in a row with different inputs.  Both calls take the
same split schedule as the regular puro_fp8_linear_wgrad given a workspace,
and sum the same FP32 partials in the same fixed order, so each output must
equal the regular one bit for bit: a wrong offset into the shared array, or
bytes the previous call left in it, would show.  Each output is also checked
against the oracle's fp64 dW within the GEMM tolerance.  An oversize request
must be refused.  The file is named so that pytest collects it last.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import bits

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module")
def lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    return P.load_library()


def _operands(M, N, K, seed):
    """Quantised Wgrad operands dY^T [N, M] and X^T [K, M] (blockwise E4M3),
    and the oracle's fp64 dW of the same BF16 inputs."""
    x = W.student_t3_f32((M, K), DEV, seed).to(torch.bfloat16)
    dy = W.normal_bf16((M, N), 1e-3, DEV, seed + 1)
    xq = P.quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    dyq = P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT)
    xb, dyb = bits(x), bits(dy)
    dYt = O.dequant_rows_1x128(*O.quantize_cols_128x1(dyb, P.E4M3), P.E4M3)
    Xt = O.dequant_rows_1x128(*O.quantize_cols_128x1(xb, P.E4M3), P.E4M3)
    return dyq.colwise, xq.colwise, O.gemm_tn(dYt, Xt, 8)


def _as_f64(t):
    return t.float().cpu().numpy().astype(np.float64)


def test_noalloc_wgrad_matches_regular_entry_point_twice(lib):
    M, N, K = 8192, 256, 384  # 4 output tiles, long reduction: the split schedule is taken
    ws_bytes = P.puro_fp8_workspace_size(N, K, M)
    assert 0 < ws_bytes <= 40 * 1024 * 1024
    stream = torch.cuda.current_stream().cuda_stream
    status = torch.zeros(1, dtype=torch.int32, device=DEV)
    for call, seed in enumerate((71, 93)):
        dyt, xt, dw_ref = _operands(M, N, K, seed)
        ref = torch.empty((N, K), dtype=torch.bfloat16, device=DEV)
        ws = torch.empty(ws_bytes, dtype=torch.uint8, device=DEV)
        P.puro_fp8_linear_wgrad(dyt, xt, ref, workspace=ws)
        out = torch.full((N, K), float("nan"), dtype=torch.bfloat16, device=DEV)
        a, b = dyt.as_c(), xt.as_c()
        st = lib.puro_fp8_linear_wgrad_noalloc(ctypes.byref(a), ctypes.byref(b), out.data_ptr(), status.data_ptr(),
                                               stream)
        assert st == P.PURO_OK, f"call {call}: status {st}"
        torch.cuda.synchronize()
        assert P.puro_fp8_get_status(status) == 0
        assert torch.equal(out.view(torch.int16), ref.view(torch.int16)), \
            f"call {call}: differs from the regular entry point given a workspace"
        ok, ratio = O.within_tolerance(_as_f64(out), dw_ref)
        assert ok, f"call {call}: outside tolerance of the oracle (worst ratio {ratio:.3g})"


def test_noalloc_wgrad_refuses_oversize_requests(lib):
    # output [2048, 1792] over 32768 tokens would need 4 x 2048 x 1792 x 4 B
    # = 58.7 MB of split scratch, more than the fixed 40 MiB
    assert P.puro_fp8_workspace_size(2048, 1792, 32768) > 40 * 1024 * 1024
    fake = 0x100000  # never dereferenced: the request is refused on the host
    a = P.puro_fp8_tensor_t(fake, fake, 2048, 32768, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    b = P.puro_fp8_tensor_t(fake, fake, 1792, 32768, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, 0)
    st = lib.puro_fp8_linear_wgrad_noalloc(ctypes.byref(a), ctypes.byref(b), fake, None, None)
    assert st == P.PURO_ERR_UNSUPPORTED
