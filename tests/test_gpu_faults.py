"""Failure detection without a GPU fault.

Every pipeline wait in the GEMM kernels is bounded in wall time.  Here the
bound is dropped to zero, so any wait that is not already satisfied gives
up: the kernel must record PURO_ERR_TIMEOUT in the caller's status word,
drain its own copies and MMAs, free tensor memory and return -- no trap, no
hang -- and the context must stay usable (the next call, with the normal
bound, is correct).
"""
import pytest
import torch

import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import assert_close, bits, oracle_linear

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
