"""Launch one of the library's fused or optimizer kernels a few times on a
fixed synthetic input, for profiling with ncu (one kernel per run, small
enough that a full capture ends in seconds).  Not part of the library.

    python -m paper_2608_27370_gb300.microbench.kernels swiglu   # [8192, 6144] from gate/up [8192, 12288]
    python -m paper_2608_27370_gb300.microbench.kernels rmsnorm  # [32768, 1536] with a gain
    python -m paper_2608_27370_gb300.microbench.kernels muonh    # gate_up [17920, 1536] + down [1536, 8960]
    python -m paper_2608_27370_gb300.microbench.kernels gemm     # down Fprop, M = 8192, N = 1536, K = 8960
    python -m paper_2608_27370_gb300.microbench.kernels gemm_k1536  # gate_up Fprop, M = 8192, N = 17920, K = 1536
    python -m paper_2608_27370_gb300.microbench.kernels dgrad_quant  # down Dgrad + both FP8 copies of dX, M = 8192
    python -m paper_2608_27370_gb300.microbench.kernels quant    # gate_up output gradient [8192, 17920], both copies

Each input is larger than L2.  Every call is made twice: the second is the
one to capture (ncu -s skips the first).
"""
import math
import sys

import torch

import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W


def main(which: str) -> None:
    dev = "cuda"
    P.load_library()
    if which == "swiglu":
        M, F = 8192, 6144
        gu = W.student_t3_f32((M, 2 * F), dev, 41).to(torch.bfloat16)
        q = P.quantize(torch.empty((M, F), dtype=torch.bfloat16, device=dev))
        for _ in range(2):
            P.puro_fp8_quantize_swiglu(gu[:, :F], gu[:, F:], P.E4M3, None, q.rowwise.data, q.rowwise.scale,
                                       q.colwise.data, q.colwise.scale)
    elif which == "rmsnorm":
        M, K = 32768, 1536
        h = W.normal_bf16((M, K), 1.0, dev, 31)
        g = W.normal_bf16((K,), 0.1, dev, 33).add_(1.0)
        rstd = torch.empty(M, dtype=torch.float32, device=dev)
        q = P.quantize(h)
        for _ in range(2):
            P.puro_fp8_quantize_rmsnorm(h, g, 1e-6, P.E4M3, rstd, None, q.rowwise.data, q.rowwise.scale,
                                        q.colwise.data, q.colwise.scale)
    elif which == "muonh":
        mats = []
        for j, (N, K) in enumerate(((17920, 1536), (1536, 8960))):
            w = W.normal_f32((N, K), 0.02, dev, 70 + j)
            u = W.normal_f32((N, K), 1.0 / math.sqrt(K), dev, 90 + j)
            mats.append((w, u, torch.empty((N, K), dtype=torch.bfloat16, device=dev),
                         float(torch.linalg.vector_norm(w.double()))))
        sums = torch.empty((len(mats), 3), dtype=torch.float64, device=dev)
        ws = torch.empty(P.puro_muonh_grouped_workspace_size(mats), dtype=torch.uint8, device=dev)
        for _ in range(2):
            P.puro_muonh_step_grouped(mats, 4.08e-4, sums, ws)
    elif which in ("gemm", "gemm_k1536"):
        M, N, K = (8192, 1536, 8960) if which == "gemm" else (8192, 17920, 1536)
        a = P.quantize(W.normal_bf16((M, K), 1.0, dev, 1), transpose=False)
        b = P.quantize(W.normal_bf16((N, K), 0.02, dev, 2), P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, transpose=False)
        d = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
        for _ in range(2):
            P.puro_fp8_linear_fprop(a.rowwise, b.rowwise, d)
    elif which == "dgrad_quant":
        # down Dgrad at M = 8192: dY [8192, 1536] x W [1536, 8960] -> dX [8192, 8960] quantised in the epilogue
        M, N, K = 8192, 1536, 8960
        dyq = P.quantize(W.normal_bf16((M, N), 1e-3, dev, 4), transpose=False)
        wt = P.quantize(W.normal_bf16((N, K), 0.02, dev, 5), P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT).colwise
        q = P.quantize(torch.empty((M, K), dtype=torch.bfloat16, device=dev))
        for _ in range(2):
            P.puro_fp8_linear_dgrad_quantize(dyq.rowwise, wt, P.E4M3, None, q.rowwise.data, q.rowwise.scale,
                                             q.colwise.data, q.colwise.scale)
    elif which == "quant":
        dy = W.normal_bf16((8192, 17920), 1e-3, dev, 3)
        q = P.quantize(dy)
        for _ in range(2):
            P.quantize(dy, out=q)
    else:
        raise SystemExit(f"unknown kernel {which!r}: swiglu, rmsnorm, muonh, gemm, gemm_k1536, dgrad_quant or quant")
    torch.cuda.synchronize()
    print("ok", which)


if __name__ == "__main__":
    main(sys.argv[1] if len(sys.argv) > 1 else "swiglu")
