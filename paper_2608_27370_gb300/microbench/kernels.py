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
    python -m paper_2608_27370_gb300.microbench.kernels quant_small  # qkv / o_proj / gate_up input [32768, 1536], both copies
    python -m paper_2608_27370_gb300.microbench.kernels gemm_oproj   # o_proj Fprop, M = 32768, N = 1536, K = 1536
    python -m paper_2608_27370_gb300.microbench.kernels tensor   # per-tensor scaling: amax, quantise, down Fprop, M = 8192
    python -m paper_2608_27370_gb300.microbench.kernels bf16     # down Fprop on BF16 operands (kind::f16), M = 8192
    python -m paper_2608_27370_gb300.microbench.kernels weight   # one weight's 128x128-block cast: gate_up W [17920, 1536]
    python -m paper_2608_27370_gb300.microbench.kernels weights  # one grouped launch: the four weights of eight C5 layers
    python -m paper_2608_27370_gb300.microbench.kernels splitk   # qkv Wgrad at M = 32768: split reduction, BF16 and FP32 main-grad
    python -m paper_2608_27370_gb300.microbench.kernels unfused  # the unfused producers: RMSNorm [32768, 1536], SwiGLU [8192, 6144]

Most inputs are larger than L2 (ncu flushes the caches before each pass in
any case).  Every call is made twice: the second is the one to capture
(ncu -s skips the first call's launches).
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
    elif which in ("gemm", "gemm_k1536", "gemm_oproj"):
        M, N, K = {"gemm": (8192, 1536, 8960), "gemm_k1536": (8192, 17920, 1536),
                   "gemm_oproj": (32768, 1536, 1536)}[which]
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
    elif which in ("quant", "quant_small"):
        dy = W.normal_bf16((8192, 17920) if which == "quant" else (32768, 1536), 1e-3, dev, 3)
        q = P.quantize(dy)
        for _ in range(2):
            P.quantize(dy, out=q)
    elif which == "tensor":
        # per-tensor current scaling of the down Fprop at M = 8192: amax and the
        # per-tensor cast (both copies) of X and W, then the GEMM with the
        # scale_inv product in its epilogue (five kernel launches per call)
        M, N, K = 8192, 1536, 8960
        x = W.normal_bf16((M, K), 1.0, dev, 6)
        w = W.normal_bf16((N, K), 0.02, dev, 7)
        d = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
        xq = wq = None
        for _ in range(2):
            xq = P.quantize(x, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT, out=xq)
            wq = P.quantize(w, P.E4M3, P.SCALE_TENSOR, P.ROLE_WEIGHT, out=wq)
            P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, d)
    elif which == "bf16":
        M, N, K = 8192, 1536, 8960
        x = W.normal_bf16((M, K), 1.0, dev, 8)
        w = W.normal_bf16((N, K), 0.02, dev, 9)
        d = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
        for _ in range(2):
            P.puro_bf16_linear_fprop(x, w, d, M, N, K)
    elif which == "weight":
        w = W.normal_bf16((17920, 1536), 0.02, dev, 10)
        q = P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
        for _ in range(2):
            P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, out=q)
    elif which == "weights":
        # the step's grouped weight cast: 32 weights (eight C5 layers' qkv,
        # o_proj, gate_up, down; 1.5 GB of BF16) in one launch, both copies
        entries = []
        for layer in range(8):
            for j, (_, N, K) in enumerate(W.QWEN2_1P5B_LINEARS):
                w = W.normal_bf16((N, K), 0.02, dev, 100 + 4 * layer + j)
                entries.append((w, P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)))
        table = P.weight_table(entries)
        for _ in range(2):
            P.puro_fp8_quantize_weights(table, P.E4M3)
    elif which == "splitk":
        # the qkv Wgrad of C5 (dW [2048, 1536], reduction over M = 32768): a
        # 2048 x 1536 output has too few tiles for the SMs, so the reduction
        # is split through FP32 partials; once into BF16 dW, once added to an
        # FP32 main-grad (two kernel launches each)
        M, N, K = 32768, 2048, 1536
        dyt = P.quantize(W.normal_bf16((N, M), 1e-3, dev, 11), transpose=False).rowwise
        xt = P.quantize(W.normal_bf16((K, M), 1.0, dev, 12), transpose=False).rowwise
        dw = torch.empty((N, K), dtype=torch.bfloat16, device=dev)
        main = torch.zeros((N, K), dtype=torch.float32, device=dev)
        ws = torch.empty(max(16, P.puro_fp8_workspace_size(N, K, M)), dtype=torch.uint8, device=dev)
        for _ in range(2):
            P.puro_fp8_linear_wgrad(dyt, xt, dw, ws)
            P.puro_fp8_linear_wgrad_main_grad(dyt, xt, main, ws)
    elif which == "unfused":
        # the comparison kernels of the fused producers (three launches per call)
        h = W.normal_bf16((32768, 1536), 1.0, dev, 13)
        g = W.normal_bf16((1536,), 0.1, dev, 14).add_(1.0)
        rstd = torch.empty(32768, dtype=torch.float32, device=dev)
        y = torch.empty_like(h)
        gu = W.student_t3_f32((8192, 12288), dev, 15).to(torch.bfloat16)
        hs = torch.empty((8192, 6144), dtype=torch.bfloat16, device=dev)
        for _ in range(2):
            P.puro_rmsnorm_bf16(h, g, 1e-6, rstd, y)
            P.puro_swiglu_bf16(gu[:, :6144], gu[:, 6144:], hs)
    else:
        raise SystemExit(f"unknown kernel {which!r}: swiglu, rmsnorm, muonh, gemm, gemm_k1536, gemm_oproj, "
                         "dgrad_quant, quant, quant_small, tensor, bf16, weight, weights, splitk or unfused")
    torch.cuda.synchronize()
    print("ok", which)


if __name__ == "__main__":
    main(sys.argv[1] if len(sys.argv) > 1 else "swiglu")
