#!/usr/bin/env python3
"""Benchmark of the FP8 linear training path on GB300.

One step = one forward + backward pass of every linear layer of the
workload through the library's C ABI, in the paper's recipe (section "FP8
Mixed-Precision Training"; appendix "FP8 implementation pipeline"):

  first every weight W (128x128 blocks, with the transposed copy), 64 weights
      per launch
  forward, layer 0 .. L-1, each linear: quantise X (1x128 groups, rowwise for
      Fprop and the transposed copy kept for Wgrad), Fprop Y = X W^T
  backward, layer L-1 .. 0, each linear in reverse: quantise dY (rowwise and
      transposed), Dgrad dX = dY W and Wgrad dW = dY^T X (one grouped launch
      when neither splits its reduction)

Default workload: the 28-layer Qwen2-1.5B linear stack at M = 32768 tokens
(qkv, o_proj, gate_up, down per layer), distinct seeded inputs per layer,
all resident in HBM before timing; per-layer inputs (2.4 GB) exceed L2.

Prints one JSON line (rank 0).  `value` is whole-step FP8 fwd+bwd TFLOP/s
(3 GEMMs x 2MNK per linear, divided by the step time including all
quantisation).  `roofline` is measured live with CUDA events around every
launch of the dominant kernel inside the timed steps.
"""
from __future__ import annotations

import argparse
import json
import os
import statistics
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "FP8 linear fwd+bwd TFLOP/s and % of FP8 peak; quantise HBM GB/s"
FALLBACK_PEAKS = {"hbm_gbs": 6800.0, "bf16_tflops": 1900.0, "bf16_tflops_sustained": 1700.0}
# GB300's nominal figures, reported beside the measured denominators as
# context: dense FP8 tensor rate and HBM3e bandwidth.
NOMINAL_FP8_DENSE_TFLOPS = 4500.0
NOMINAL_HBM_GBS = 7900.0
FP8_PER_BF16 = 2.0  # nominal dense ratio (4.5 / 2.25 PFLOP/s)
FP8_FLOP_PER_CLK_SM = 16384  # dense FP8 tensor-pipe rate per SM (a 256x256x32 pair MMA per 128 cycles)

# DRAM bytes (dram__bytes_read.sum + dram__bytes_write.sum) per algorithmic
# byte over the 8 GEMM launches and the 9 quantise launches of one layer
# of the C5 workload (block scaling, M = 32768), from per-kernel ncu
# captures of at most four launches each of a one-layer run (about 4 GB on
# the device).  All 28 layers have the same
# shapes, so one layer's calls stand for the step.  Each figure holds only
# for the kernel sources it was captured on (sha1 prefix over the listed
# files) and is reported as null once they change or for another workload.
CAPTURED_TRAFFIC = {
    "gemm": {"files": ["gemm.cu", "ptx.cuh", "internal.h", "api.cu", "quant_math.cuh"], "sha1": "17ee2a9d639da521",
             "bytes_per_algorithmic_byte": 5599.3e6 / 5004.2036e6},
    "quantize": {"files": ["quantize.cu", "ptx.cuh", "quant_math.cuh"], "sha1": "8b99029e4df2986b",
                 "bytes_per_algorithmic_byte": 4533.1e6 / 5004.2036e6},
}
CAPTURED_TRAFFIC_WORKLOAD = ("C5", 32768, "block")


def captured_traffic(kind: str, workload, algorithmic_bytes_per_launch: float) -> "int | None":
    """DRAM bytes per launch of `kind` if the capture applies, else None: the
    captured layer's DRAM bytes per algorithmic byte times the algorithmic
    bytes of the step's average launch (the GEMM launches of a layer are the
    same in every layer; the quantiser's grouped weight launch covers 56
    weights (14 layers) in the step and four in the captured layer, so its
    average launch differs and the ratio carries over)."""
    import hashlib

    if tuple(workload) != CAPTURED_TRAFFIC_WORKLOAD:
        return None
    rec = CAPTURED_TRAFFIC[kind]
    h = hashlib.sha1()
    for f in rec["files"]:
        with open(os.path.join(ROOT, "paper_2608_27370_gb300", "csrc", f), "rb") as fh:
            h.update(fh.read())
    if not h.hexdigest().startswith(rec["sha1"]):
        return None
    return int(round(rec["bytes_per_algorithmic_byte"] * algorithmic_bytes_per_launch))


def load_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return d, "measured"
    return dict(FALLBACK_PEAKS), "fallback"


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=10)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--config", default="C5")
    ap.add_argument("--scaling", choices=["block", "tensor"], default="block")
    ap.add_argument("--layers", type=int, default=None, help="override layer count (profiling runs only)")
    ap.add_argument("--tokens", type=int, default=None, help="override M (profiling runs only)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-bf16", action="store_true")
    ap.add_argument("--no-clocks", action="store_true")
    ap.add_argument("--no-paper-model", action="store_true", help="skip the C6 (paper model shape), E5M2-gradient, per-tensor, producer/epilogue-fusion and MuonH lines")
    return ap.parse_args()


# ----------------------------------------------------------------------------
# multi-rank timing: one process per GPU, each a full replica of the step
# (the linears of different replicas share nothing, so no collective runs on
# the data path); the job's time is the slowest rank's
# ----------------------------------------------------------------------------
def max_over_ranks(seconds: float, world: int, device) -> float:
    """The maximum of a per-rank duration over all ranks, then a barrier."""
    if world <= 1:
        return seconds
    import torch
    import torch.distributed as dist

    t = torch.tensor([seconds], device=device, dtype=torch.float64)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    dist.barrier()
    return float(t.item())


def job_value(world: int, units_per_rank: float, step_seconds: float) -> float:
    """Whole-job throughput: the units every rank processed over the job's step time."""
    return world * units_per_rank / step_seconds


# ----------------------------------------------------------------------------
# clocks during the timed region
# ----------------------------------------------------------------------------
class ClockSampler:
    QUERY = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
             "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
             "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_index: int, enabled: bool = True):
        self.proc = None
        self.path = None
        self.gpu = gpu_index
        if not enabled:
            return
        try:
            fd, self.path = tempfile.mkstemp(prefix="clocks_", suffix=".csv")
            os.close(fd)
            self.f = open(self.path, "w")
            self.proc = subprocess.Popen(["nvidia-smi", f"--id={gpu_index}", f"--query-gpu={self.QUERY}",
                                          "--format=csv,noheader,nounits", "-lms", "200"],
                                         stdout=self.f, stderr=subprocess.DEVNULL)
        except (OSError, FileNotFoundError):
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.f.close()
        sm, mx, reasons = [], [], set()
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) < 9:
                continue
            try:
                sm.append(float(parts[1]))
                mx.append(float(parts[2]))
            except ValueError:
                continue
            for n, v in zip(names, parts[5:9]):
                if v.lower() == "active":
                    reasons.add(n)
        os.unlink(self.path)
        if not sm:
            return None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(mx), "samples": len(sm),
                "reasons": sorted(reasons)}


# ----------------------------------------------------------------------------
# the stack of linears and one step through the C ABI
# ----------------------------------------------------------------------------
class LaunchTimer:
    """CUDA events around launches, grouped by kernel category."""

    def __init__(self, torch):
        self.torch = torch
        self.pending = []  # (category, label, units, start, end)
        self.enabled = False
        self.label = None  # what the next run() call is (a shape), for the per-call breakdown

    def run(self, cat: str, units: float, fn, *args, **kw):
        label, self.label = self.label, None
        if not self.enabled:
            return fn(*args, **kw)
        s = self.torch.cuda.Event(enable_timing=True)
        e = self.torch.cuda.Event(enable_timing=True)
        s.record()
        fn(*args, **kw)
        e.record()
        self.pending.append((cat, label or cat, units, s, e))

    def totals(self):
        out = {}
        for cat, _, units, s, e in self.pending:
            t = s.elapsed_time(e) * 1e-3
            c = out.setdefault(cat, {"time_s": 0.0, "units": 0.0, "launches": 0})
            c["time_s"] += t
            c["units"] += units
            c["launches"] += 1
        return out

    def by_label(self, cat: str, unit_scale: float):
        """Per labelled call of category `cat`: launches, mean microseconds
        and units per second (times unit_scale), slowest rate first."""
        agg = {}
        for c, label, units, s, e in self.pending:
            if c != cat:
                continue
            a = agg.setdefault(label, [0, 0.0, 0.0])
            a[0] += 1
            a[1] += s.elapsed_time(e) * 1e-3
            a[2] += units
        rows = [{"call": k, "launches": n, "mean_us": t / n * 1e6, "rate": u / t * unit_scale}
                for k, (n, t, u) in agg.items()]
        return sorted(rows, key=lambda r: r["rate"])


class LinearStack:
    def __init__(self, P, W, torch, wl, device, scaling, layers, M):
        self.P, self.torch = P, torch
        self.scaling = P.SCALE_BLOCK if scaling == "block" else P.SCALE_TENSOR
        self.wl = wl
        self.L = layers
        self.M = M
        self.device = device
        self.timer = LaunchTimer(torch)
        self.launches_per_step = 0
        wl_eff = W.Workload(wl.key, wl.description, M, layers, wl.linears, wl.recipe, wl.scaling)
        self.inputs = [[W.make_linear(wl_eff, l, j, device) for j in range(len(wl.linears))] for l in range(layers)]
        u8, bf = torch.uint8, torch.bfloat16
        sc = self.scaling
        # persistent per layer: quantised weights (both copies) and the transposed X copy for Wgrad
        self.wq, self.xqt = [], []
        for l in range(layers):
            wrow, xrow = [], []
            for j, (_, N, K) in enumerate(wl.linears):
                wrow.append(P.Quantized(
                    P.FP8Operand(torch.empty((N, K), dtype=u8, device=device),
                                 P.empty_scales(N, K, sc, P.ROLE_WEIGHT, device), scaling=sc, role=P.ROLE_WEIGHT),
                    P.FP8Operand(torch.empty((K, N), dtype=u8, device=device),
                                 P.empty_scales(K, N, sc, P.ROLE_WEIGHT, device), scaling=sc, role=P.ROLE_WEIGHT),
                    torch.zeros(1, dtype=torch.int32, device=device) if sc == P.SCALE_TENSOR else None))
                xrow.append(P.FP8Operand(torch.empty((K, M), dtype=u8, device=device),
                                         P.empty_scales(K, M, sc, P.ROLE_ACT, device), scaling=sc))
            self.wq.append(wrow)
            self.xqt.append(xrow)
        # shared across layers (consumed right after they are produced)
        self.xq, self.dyq, self.y, self.dx, self.dw = [], [], [], [], []
        for j, (_, N, K) in enumerate(wl.linears):
            amax = torch.zeros(1, dtype=torch.int32, device=device) if sc == P.SCALE_TENSOR else None
            self.xq.append(P.FP8Operand(torch.empty((M, K), dtype=u8, device=device),
                                        P.empty_scales(M, K, sc, P.ROLE_ACT, device), scaling=sc))
            self.dyq.append(P.Quantized(
                P.FP8Operand(torch.empty((M, N), dtype=u8, device=device), P.empty_scales(M, N, sc, P.ROLE_ACT, device),
                             scaling=sc),
                P.FP8Operand(torch.empty((N, M), dtype=u8, device=device), P.empty_scales(N, M, sc, P.ROLE_ACT, device),
                             scaling=sc), amax))
            self.y.append(torch.empty((M, N), dtype=bf, device=device))
            self.dx.append(torch.empty((M, K), dtype=bf, device=device))
            self.dw.append(torch.empty((N, K), dtype=bf, device=device))
        self.xamax = [torch.zeros(1, dtype=torch.int32, device=device) for _ in wl.linears]
        # block scaling: every weight of the step quantised by one grouped call
        # (one launch per 64 weights) at the start of the step
        self.wtable = None
        if self.scaling == P.SCALE_BLOCK:
            self.wtable = P.weight_table([(self.inputs[l][j].w, self.wq[l][j]) for l in range(layers)
                                          for j in range(len(wl.linears))])
            self.wbytes = sum(self._qbytes(N, K, P.ROLE_WEIGHT) for _, N, K in wl.linears) * layers
        self.grad_fmt = P.E4M3
        # scratch for split reductions of small-output GEMMs (Wgrad of qkv / o_proj)
        ws = max([P.puro_fp8_workspace_size(N, K, M) for _, N, K in wl.linears] +
                 [P.puro_fp8_workspace_size(M, N, K) for _, N, K in wl.linears] +
                 [P.puro_fp8_workspace_size(M, K, N) for _, N, K in wl.linears] + [16])
        self.workspace = torch.empty(ws, dtype=torch.uint8, device=device)

    # bytes each quantise launch moves by definition (read bf16, write both
    # FP8 copies and their scales)
    def _qbytes(self, rows, cols, role):
        n = rows * cols
        if self.scaling == self.P.SCALE_TENSOR:
            return 4 * n + 8
        if role == self.P.ROLE_WEIGHT:
            return 4 * n + 2 * (rows // 128) * (cols // 128)
        return 4 * n + 2 * n // 128

    def set_grad_format(self, fmt):
        """FP8 format of the output-gradient operands (E4M3 by default; E5M2
        is the wider-range variant the FP8 section contrasts it with)."""
        self.grad_fmt = fmt
        for q in self.dyq:
            q.rowwise.fmt = fmt
            q.colwise.fmt = fmt

    def _quant(self, x, role, q: "object", fmt=None):
        P, T = self.P, self.timer
        rows, cols = x.shape
        if self.scaling == P.SCALE_TENSOR:
            T.run("amax", 2 * rows * cols, P.puro_fp8_amax, x, q.amax)
            self.launches_per_step += 1
        fmt = P.E4M3 if fmt is None else fmt
        T.label = f"{'weight' if role == P.ROLE_WEIGHT else 'act'} [{rows}, {cols}]"
        T.run("quantize", self._qbytes(rows, cols, role), P.puro_fp8_quantize, x, fmt, self.scaling, role,
              q.amax if self.scaling == P.SCALE_TENSOR else None, q.rowwise.data, q.rowwise.scale,
              q.colwise.data, q.colwise.scale)
        self.launches_per_step += 1

    def _backward_launches(self, N, K):
        # the library's own plan for puro_fp8_linear_backward with this workspace
        if self.scaling == self.P.SCALE_BLOCK:
            return self.P.puro_fp8_linear_backward_launches(self.M, N, K, self.workspace.numel())
        return self._gemm_launches(self.M, K, N) + self._gemm_launches(N, K, self.M)

    def _gemm_launches(self, rows_out, cols_out, red):
        # one GEMM kernel, plus the reduction kernel when the split schedule is taken
        ws = self.P.puro_fp8_workspace_size(rows_out, cols_out, red)
        return 2 if 0 < ws <= self.workspace.numel() else 1

    def step(self, hooks=None):
        """One step.  `hooks` (the end-to-end measurement) is told when a
        layer's forward or backward starts, picks each Wgrad's output buffer
        and is handed each finished dW; the calls made are the same."""
        P, T = self.P, self.timer
        self.launches_per_step = 0
        if self.wtable is not None:
            T.label = f"all {self.wtable.count} weights, grouped"
            T.run("quantize", self.wbytes, P.puro_fp8_quantize_weights, self.wtable, P.E4M3)
            self.launches_per_step += -(-self.wtable.count // 64)
        for l in range(self.L):
            if hooks is not None:
                hooks.before_forward(l)
            for j, (name, N, K) in enumerate(self.wl.linears):
                li = self.inputs[l][j]
                if self.wtable is None:
                    self._quant(li.w, P.ROLE_WEIGHT, self.wq[l][j])
                xq = P.Quantized(self.xq[j], self.xqt[l][j], self.xamax[j])
                self._quant(li.x, P.ROLE_ACT, xq)
                T.label = f"fprop {name}"
                T.run("gemm", 2.0 * self.M * N * K, P.puro_fp8_linear_fprop, self.xq[j], self.wq[l][j].rowwise,
                      self.y[j], self.workspace)
                self.launches_per_step += self._gemm_launches(self.M, N, K)
        for l in reversed(range(self.L)):
            if hooks is not None:
                hooks.before_backward(l)
            for j in reversed(range(len(self.wl.linears))):
                name, N, K = self.wl.linears[j]
                li = self.inputs[l][j]
                dw = self.dw[j] if hooks is None else hooks.dw(l, j)
                self._quant(li.dy, P.ROLE_ACT, self.dyq[j], self.grad_fmt)
                # Dgrad and Wgrad of the linear: one grouped launch when both run unsplit
                T.label = f"dgrad+wgrad {name}"
                T.run("gemm", 4.0 * self.M * N * K, P.puro_fp8_linear_backward, self.dyq[j].rowwise,
                      self.wq[l][j].colwise, self.dx[j], self.dyq[j].colwise, self.xqt[l][j], dw,
                      self.workspace)
                self.launches_per_step += self._backward_launches(N, K)
                if hooks is not None:
                    hooks.after_backward(l, j, dw)

    def flops_per_step(self):
        return self.L * sum(6.0 * self.M * N * K for _, N, K in self.wl.linears)

    def gemm_algorithmic_bytes_per_call(self):
        """Algorithmic bytes per GEMM kernel launch of the step (a grouped
        backward launch of a linear's Dgrad and Wgrad counts once; a split
        reduction's summing kernel is part of its GEMM): both FP8 operands and
        their scales read once and the BF16 output written once, per GEMM
        (every layer has the same shapes)."""
        M, tot, calls = self.M, 0, 0
        for _, N, K in self.wl.linears:
            tot += M * K + N * K + 2 * M * N + M * K // 128 + N * K // 16384   # fprop
            tot += M * N + K * N + 2 * M * K + M * N // 128 + K * N // 16384   # dgrad
            tot += N * M + K * M + 2 * N * K + N * M // 128 + K * M // 128     # wgrad
            calls += 1 + (1 if self._backward_launches(N, K) == 1 else 2)
        return tot / calls

    def quantize_kernel_launches_per_step(self):
        """Quantiser kernel launches of one step: the grouped weight call is
        one launch per 64 weights."""
        acts = 2 * self.L * len(self.wl.linears)
        if self.wtable is not None:
            return acts + -(-self.wtable.count // 64)
        return acts + self.L * len(self.wl.linears)


def bf16_layer_speedup(P, torch, stack):
    """Same three GEMMs of layer 0's linears in BF16 (tcgen05 kind::f16) vs
    FP8 (blockwise, kind::mxf8f6f4), GEMM time only, operands already in
    the layout each GEMM reads."""
    dev = stack.device
    M = stack.M
    li0 = stack.inputs[0]
    bufs = []
    for j, (_, N, K) in enumerate(stack.wl.linears):
        li = li0[j]
        bufs.append((li.x, li.w, li.dy, li.w.t().contiguous(), li.dy.t().contiguous(), li.x.t().contiguous(), N, K))

    def run_bf16():
        for j, (x, w, dy, wt, dyt, xt, N, K) in enumerate(bufs):
            P.puro_bf16_linear_fprop(x, w, stack.y[j], M, N, K)
        for j, (x, w, dy, wt, dyt, xt, N, K) in enumerate(bufs):
            P.puro_bf16_linear_dgrad(dy, wt, stack.dx[j], M, N, K)
            P.puro_bf16_linear_wgrad(dyt, xt, stack.dw[j], M, N, K)

    def run_fp8():
        for j, (_, N, K) in enumerate(stack.wl.linears):
            P.puro_fp8_linear_fprop(stack.xq[j], stack.wq[0][j].rowwise, stack.y[j])
        for j, (_, N, K) in enumerate(stack.wl.linears):
            P.puro_fp8_linear_dgrad(stack.dyq[j].rowwise, stack.wq[0][j].colwise, stack.dx[j], stack.workspace)
            P.puro_fp8_linear_wgrad(stack.dyq[j].colwise, stack.xqt[0][j], stack.dw[j], stack.workspace)

    def timeit(fn, reps=5):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) * 1e-3 / reps

    # fill the FP8 operands of layer 0 (quantise once, outside the timing)
    for j, (_, N, K) in enumerate(stack.wl.linears):
        li = li0[j]
        P.quantize(li.w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT, out=stack.wq[0][j])
        P.quantize(li.x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, out=P.Quantized(stack.xq[j], stack.xqt[0][j]))
        P.quantize(li.dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, out=stack.dyq[j])
    t_bf16 = timeit(run_bf16)
    t_fp8 = timeit(run_fp8)
    flops = sum(6.0 * M * N * K for _, N, K in stack.wl.linears)
    del bufs

    # Wgrad into an FP32 main-grad (the paper's FP32 gradient accumulation)
    # against the BF16-output Wgrad, same operands
    mains = [torch.zeros((N, K), dtype=torch.float32, device=dev) for _, N, K in stack.wl.linears]

    def run_wgrad_bf16():
        for j in range(len(stack.wl.linears)):
            P.puro_fp8_linear_wgrad(stack.dyq[j].colwise, stack.xqt[0][j], stack.dw[j], stack.workspace)

    def run_wgrad_main():
        for j in range(len(stack.wl.linears)):
            P.puro_fp8_linear_wgrad_main_grad(stack.dyq[j].colwise, stack.xqt[0][j], mains[j], stack.workspace)

    t_wb = timeit(run_wgrad_bf16)
    t_wm = timeit(run_wgrad_main)
    wflops = sum(2.0 * M * N * K for _, N, K in stack.wl.linears)
    del mains
    torch.cuda.empty_cache()
    return {"layer": 0, "bf16_gemm_tflops": flops / t_bf16 / 1e12, "fp8_gemm_tflops": flops / t_fp8 / 1e12,
            "fp8_over_bf16": t_bf16 / t_fp8, "paper_fp8_over_bf16_whole_model_rtx5090": 1.36,
            "wgrad_bf16_out_tflops": wflops / t_wb / 1e12, "wgrad_fp32_main_grad_tflops": wflops / t_wm / 1e12}


def rmsnorm_fusion_measure(P, W, torch, device):
    """RMSNorm fused ahead of the activation quantiser against RMSNorm (bf16
    y written and read back) followed by the quantiser, on the inputs of the
    qkv / gate_up projections of C5 ([32768, 1536]) and C6 ([8192, 2048])."""

    def timeit(fn, reps=20):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) * 1e-3 / reps

    out = []
    for key, (M, K) in (("C5", (32768, 1536)), ("C6", (8192, 2048))):
        # rotate over inputs totalling more than twice L2: no reuse across calls
        nbuf = max(2, -(-300_000_000 // (M * K * 2)))
        hs = [W.normal_bf16((M, K), 1.0, device, 31 + i) for i in range(nbuf)]
        gamma = W.normal_bf16((K,), 0.1, device, 33).add_(1.0)
        rstd = torch.empty(M, dtype=torch.float32, device=device)
        y = torch.empty((M, K), dtype=torch.bfloat16, device=device)
        q = P.quantize(hs[0])
        it = [0]

        def fused():
            it[0] = (it[0] + 1) % nbuf
            P.puro_fp8_quantize_rmsnorm(hs[it[0]], gamma, 1e-6, P.E4M3, rstd, None, q.rowwise.data, q.rowwise.scale,
                                        q.colwise.data, q.colwise.scale)

        def unfused():
            it[0] = (it[0] + 1) % nbuf
            P.puro_rmsnorm_bf16(hs[it[0]], gamma, 1e-6, rstd, y)
            P.quantize(y, out=q)

        tf, tu = timeit(fused), timeit(unfused)
        n = M * K
        # algorithmic bytes of the fused op: read h, write both FP8 copies,
        # their scales and rstd
        fused_bytes = 2 * n + 2 * n + 2 * n // 128 + 4 * M
        out.append({"input": f"{key} qkv/gate_up input [{M}, {K}]", "fused_us": tf * 1e6, "unfused_us": tu * 1e6,
                    "fused_over_unfused_time": tf / tu, "fused_algorithmic_gbs": fused_bytes / tf / 1e9})
        del hs, y, q
        torch.cuda.empty_cache()
    return out


def swiglu_fusion_measure(P, W, torch, device):
    """SwiGLU fused ahead of the activation quantiser against SwiGLU (bf16 h
    written and read back) followed by the quantiser, on the down-projection
    inputs of C5 (F = 8960) and C6 (F = 6144): gate and up are the two halves
    of one [M, 2F] gate/up output."""

    def timeit(fn, reps=20):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) * 1e-3 / reps

    out = []
    for key, (M, F) in (("C5", (32768, 8960)), ("C6", (8192, 6144))):
        # rotate over inputs totalling more than twice L2: no reuse across calls
        nbuf = max(2, -(-300_000_000 // (M * 2 * F * 2)))
        gus = [W.student_t3_f32((M, 2 * F), device, 41 + i).to(torch.bfloat16) for i in range(nbuf)]
        h = torch.empty((M, F), dtype=torch.bfloat16, device=device)
        q = P.quantize(h)
        it = [0]

        def fused():
            it[0] = (it[0] + 1) % nbuf
            gu = gus[it[0]]
            P.puro_fp8_quantize_swiglu(gu[:, :F], gu[:, F:], P.E4M3, None, q.rowwise.data, q.rowwise.scale,
                                       q.colwise.data, q.colwise.scale)

        def unfused():
            it[0] = (it[0] + 1) % nbuf
            gu = gus[it[0]]
            P.puro_swiglu_bf16(gu[:, :F], gu[:, F:], h)
            P.quantize(h, out=q)

        tf, tu = timeit(fused), timeit(unfused)
        n = M * F
        # algorithmic bytes of the fused op: read gate and up, write both FP8
        # copies and their scales
        fused_bytes = 4 * n + 2 * n + 2 * n // 128
        out.append({"input": f"{key} down-projection input [{M}, {F}] from gate/up [{M}, {2 * F}]",
                    "fused_us": tf * 1e6, "unfused_us": tu * 1e6, "fused_over_unfused_time": tf / tu,
                    "fused_algorithmic_gbs": fused_bytes / tf / 1e9})
        del gus, h, q
        torch.cuda.empty_cache()
    return out


def dgrad_quantize_fusion_measure(P, W, torch, device):
    """The Dgrad that quantises its own output in the epilogue
    (puro_fp8_linear_dgrad_quantize: both blockwise copies of dX, no BF16
    dX) against the BF16 Dgrad followed by the activation quantiser, and
    against the BF16 Dgrad alone, on the four Dgrad shapes of C5 (M =
    32768).  E4M3 operands and outputs."""

    def timeit(fn, reps=20):
        for _ in range(3):
            fn()
        torch.cuda.synchronize()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) * 1e-3 / reps

    wl = W.WORKLOADS["C5"]
    M = wl.M
    out = []
    for j, (name, N, K) in enumerate(wl.linears):
        # rotate over output gradients totalling more than twice L2
        nbuf = max(2, -(-300_000_000 // (M * N)))
        dyqs = []
        for i in range(nbuf):
            dy = W.normal_bf16((M, N), 1e-3, device, 8100 + 16 * j + i)
            dyqs.append(P.quantize(dy, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, transpose=False))
            del dy
        wt = P.quantize(W.normal_bf16((N, K), 0.02, device, 8200 + j), P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT).colwise
        dx = torch.empty((M, K), dtype=torch.bfloat16, device=device)
        q = P.quantize(dx)
        it = [0]

        def nxt():
            it[0] = (it[0] + 1) % nbuf
            return dyqs[it[0]].rowwise

        def fused():
            P.puro_fp8_linear_dgrad_quantize(nxt(), wt, P.E4M3, None, q.rowwise.data, q.rowwise.scale,
                                             q.colwise.data, q.colwise.scale)

        def unfused():
            P.puro_fp8_linear_dgrad(nxt(), wt, dx)
            P.quantize(dx, out=q)

        def dgrad_only():
            P.puro_fp8_linear_dgrad(nxt(), wt, dx)

        tf, tu, td = timeit(fused), timeit(unfused), timeit(dgrad_only)
        flop = 2.0 * M * N * K
        out.append({"linear": f"C5 {name} Dgrad: dY [{M}, {N}] x W -> dX [{M}, {K}]",
                    "fused_us": tf * 1e6, "unfused_us": tu * 1e6, "dgrad_bf16_us": td * 1e6,
                    "fused_over_unfused_time": tf / tu, "fused_tflops": flop / tf / 1e12,
                    "dgrad_bf16_tflops": flop / td / 1e12})
        del dyqs, wt, dx, q
        torch.cuda.empty_cache()
    return out


def muonh_measure(P, W, torch, device, peaks, steps=3, warmup=2):
    """The MuonH hyperball step over every wrapped matrix of C5 (the 112
    linear weights of the 28 layers, 1.30 G parameters): fp32 master weights
    and Muon directions resident in HBM, the bf16 weight copy written."""
    import math

    wl = W.WORKLOADS["C5"]
    mats = []
    for l in range(wl.layers):
        for j, (_, N, K) in enumerate(wl.linears):
            w = W.normal_f32((N, K), 0.02, device, 7000 + 16 * l + j)
            u = W.normal_f32((N, K), 1.0 / math.sqrt(K), device, 9000 + 16 * l + j)
            mats.append((w, u, torch.empty((N, K), dtype=torch.bfloat16, device=device),
                         float(torch.linalg.vector_norm(w.double()))))
    sums = torch.empty((len(mats), 3), dtype=torch.float64, device=device)
    ws = torch.empty(P.puro_muonh_grouped_workspace_size(mats), dtype=torch.uint8, device=device)

    def step():  # every matrix in one grouped step: three launches
        P.puro_muonh_step_grouped(mats, 4.08e-4, sums, ws)

    for _ in range(warmup):
        step()
    torch.cuda.synchronize()
    s = torch.cuda.Event(enable_timing=True)
    e = torch.cuda.Event(enable_timing=True)
    s.record()
    for _ in range(steps):
        step()
    e.record()
    torch.cuda.synchronize()
    t = s.elapsed_time(e) * 1e-3 / steps
    n = sum(w.numel() for w, _, _, _ in mats)
    # algorithmic bytes per element: read W and u (reduce), read W and u,
    # write W and the bf16 copy (apply)
    gbs = 22.0 * n / t / 1e9
    out = {"workload": f"MuonH hyperball step over C5's {len(mats)} linear weights ({n / 1e9:.2f} G fp32 parameters)",
           "ms_per_step": t * 1e3, "params_per_s": n / t, "algorithmic_gbs": gbs,
           "hbm_frac": gbs / peaks["hbm_gbs"], "launches_per_step": 3 * (-(-len(mats) // 128)), "steps": steps,
           "warmup": warmup}
    del mats, sums, ws
    torch.cuda.empty_cache()
    return out


def timed_steps(torch, stack, steps, warmup):
    """Step time of `stack` (CUDA events around `steps` steps after `warmup`)
    and the per-category launch totals of the last timed step (per-launch
    events only there, as in the main measurement)."""
    for _ in range(warmup):
        stack.step()
    torch.cuda.synchronize()
    stack.timer.pending.clear()
    s = torch.cuda.Event(enable_timing=True)
    e = torch.cuda.Event(enable_timing=True)
    s.record()
    for i in range(steps):
        stack.timer.enabled = i == steps - 1
        stack.step()
    e.record()
    torch.cuda.synchronize()
    stack.timer.enabled = False
    return s.elapsed_time(e) * 1e-3 / steps, stack.timer.totals()


def grad_format_measure(P, torch, stack, steps=3, warmup=2):
    """The same step with E5M2 output-gradient operands (weights and
    activations stay E4M3): the quantiser writes E5M2 codes for dY and its
    transposed copy, and Dgrad / Wgrad take one E5M2 operand."""
    stack.set_grad_format(P.E5M2)
    try:
        step_s, per = timed_steps(torch, stack, steps, warmup)
    finally:
        stack.set_grad_format(P.E4M3)
    g, q = per["gemm"], per["quantize"]
    return {"variant": "dY and dY^T in E5M2, X and W in E4M3 (block scaling)",
            "value": stack.flops_per_step() / step_s / 1e12, "unit": "TFLOP/s", "ms_per_step": step_s * 1e3,
            "steps": steps, "warmup": warmup, "gemm_only_tflops": g["units"] / g["time_s"] / 1e12,
            "quantize_gbs": q["units"] / q["time_s"] / 1e9}


def tensor_scaling_measure(P, W, torch, device, layers=4, steps=3, warmup=2, grad_fmt=None):
    """The C5 step with per-tensor current scaling (the contrast the FP8
    section draws: one scale per tensor, from an amax pass) on `layers` of
    its 28 layers: amax, per-tensor quantise (both copies), and the three
    FP8 GEMMs with the scale_inv product applied in the epilogue.  With
    grad_fmt = E5M2 the output gradients are cast to E5M2 (the hybrid
    recipe: E4M3 forward, E5M2 backward)."""
    wl = W.WORKLOADS["C5"]
    stack = LinearStack(P, W, torch, wl, device, "tensor", layers, wl.M)
    if grad_fmt is not None:
        stack.set_grad_format(grad_fmt)
    step_s, per = timed_steps(torch, stack, steps, warmup)
    g, q = per["gemm"], per["quantize"]
    grads = "E5M2" if grad_fmt == P.E5M2 else "E4M3"
    out = {"workload": f"C5 with per-tensor scaling, {grads} output gradients, {layers} of its 28 layers, M={wl.M}",
           "value": stack.flops_per_step() / step_s / 1e12, "unit": "TFLOP/s", "ms_per_step": step_s * 1e3,
           "steps": steps, "warmup": warmup, "gemm_only_tflops": g["units"] / g["time_s"] / 1e12,
           "quantize_gbs": q["units"] / q["time_s"] / 1e9,
           "amax_gbs": per["amax"]["units"] / per["amax"]["time_s"] / 1e9 if "amax" in per else None}
    del stack
    torch.cuda.empty_cache()
    return out


def paper_model_measure(P, W, torch, device, scaling, steps=5, warmup=3):
    """The same step on the paper's own production model shape: C6, the
    28-layer Qwen3-1.7B linear stack at its training micro-batch (2 x 4096
    tokens).  Device-resident inputs, CUDA events around the timed steps."""
    wl = W.WORKLOADS["C6"]
    stack = LinearStack(P, W, torch, wl, device, scaling, wl.layers, wl.M)
    torch.cuda.synchronize()
    step_s, per = timed_steps(torch, stack, steps, warmup)
    g, q = per["gemm"], per["quantize"]
    out = {"workload": f"{wl.key}: " + wl.description, "value": stack.flops_per_step() / step_s / 1e12,
           "unit": "TFLOP/s", "ms_per_step": step_s * 1e3, "tokens_per_s": wl.M / step_s, "steps": steps,
           "warmup": warmup, "gemm_only_tflops": g["units"] / g["time_s"] / 1e12,
           "quantize_gbs": q["units"] / q["time_s"] / 1e9}
    del stack
    torch.cuda.empty_cache()
    return out


def library_context(torch, stack):
    """Library context, not part of the path: the same twelve GEMMs as
    bf16_layer_speedup (Fprop, Dgrad and Wgrad of layer 0's four linears,
    operands already in the layout each GEMM reads, GEMM time only) through
    torch's wrappers of NVIDIA's libraries, and ours with per-tensor scales
    beside them (bf16_layer_speedup has ours blockwise): cuBLASLt FP8 (torch._scaled_mm)
    with E4M3 operands and per-tensor fp32 scales, cuBLASLt MXFP8 with one
    E8M0 scale per 32 elements of K (the blockwise recipe's arithmetic, each
    1x128 scale repeated four times) where this torch build accepts it, and
    cuBLAS BF16 (torch.matmul).  The operand values are the workload's, cast
    to FP8 by torch; every scale is 1."""
    f8 = torch.float8_e4m3fn
    dev = stack.device
    M = stack.M
    li0 = stack.inputs[0]
    ops = []
    for j, (_, N, K) in enumerate(stack.wl.linears):
        li = li0[j]
        x8, w8, dy8 = li.x.to(f8), (li.w * 50.0).to(f8), (li.dy * 1000.0).to(f8)
        # row-major A [rows, red] and column-major B [red, cols] of each GEMM
        ops.append(("fprop", x8, w8.t(), li.x, li.w.t(), N, K))
        ops.append(("dgrad", dy8, w8.t().contiguous().t(), li.dy, li.w, N, K))
        ops.append(("wgrad", dy8.t().contiguous(), x8.t().contiguous().t(), li.dy.t(), li.x, N, K))
    one = torch.ones((), dtype=torch.float32, device=dev)

    def mx_scales(rows, red):
        def up(a, b):
            return (a + b - 1) // b * b
        # E8M0 1.0 (byte 127) in the library's blocked layout: its size is
        # the padded [rows, red / 32] grid (128-row by 4-column blocks)
        return torch.full((up(rows, 128), up((red + 31) // 32, 4)), 127, dtype=torch.uint8,
                          device=dev).view(torch.float8_e8m0fnu)

    def timeit(fn, reps=5):
        for _ in range(2):
            fn()
        torch.cuda.synchronize()
        s = torch.cuda.Event(enable_timing=True)
        e = torch.cuda.Event(enable_timing=True)
        s.record()
        for _ in range(reps):
            fn()
        e.record()
        torch.cuda.synchronize()
        return s.elapsed_time(e) * 1e-3 / reps

    flops = sum(6.0 * M * N * K for _, N, K in stack.wl.linears)
    out = {"layer": 0, "note": "NVIDIA libraries through torch, for context; not on the path"}

    def per_tensor():
        for _, a, b, _, _, _, _ in ops:
            torch._scaled_mm(a, b, one, one, out_dtype=torch.bfloat16)

    def bf16():
        for _, _, _, a, b, _, _ in ops:
            torch.matmul(a, b)

    # ours, the same twelve GEMMs with per-tensor scales (E4M3, scale_inv product in the epilogue)
    import paper_2608_27370_gb300 as P
    ours_t = []
    for j, (_, N, K) in enumerate(stack.wl.linears):
        li = li0[j]
        ours_t.append((P.quantize(li.x, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT),
                       P.quantize(li.w, P.E4M3, P.SCALE_TENSOR, P.ROLE_WEIGHT),
                       P.quantize(li.dy, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT)))

    def ours_per_tensor():
        for j, (xq, wq, dyq) in enumerate(ours_t):
            P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, stack.y[j])
        for j, (xq, wq, dyq) in enumerate(ours_t):
            P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, stack.dx[j], stack.workspace)
            P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, stack.dw[j], stack.workspace)

    out["ours_fp8_per_tensor_tflops"] = flops / timeit(ours_per_tensor) / 1e12
    del ours_t
    try:
        out["cublaslt_fp8_per_tensor_tflops"] = flops / timeit(per_tensor) / 1e12
    except (RuntimeError, TypeError) as exc:
        out["cublaslt_fp8_per_tensor_tflops"] = None
        out["cublaslt_fp8_per_tensor_unavailable"] = str(exc).splitlines()[0][:200]
    try:
        mx = [(a, b, mx_scales(a.shape[0], a.shape[1]), mx_scales(b.shape[1], b.shape[0])) for _, a, b, *_ in ops]

        def mxfp8():
            for a, b, sa, sb in mx:
                torch._scaled_mm(a, b, sa, sb, out_dtype=torch.bfloat16)

        out["cublaslt_mxfp8_tflops"] = flops / timeit(mxfp8) / 1e12
        del mx
    except (RuntimeError, TypeError, AttributeError) as exc:
        out["cublaslt_mxfp8_tflops"] = None
        out["cublaslt_mxfp8_unavailable"] = str(exc).splitlines()[0][:200]
    out["cublas_bf16_tflops"] = flops / timeit(bf16) / 1e12
    del ops
    torch.cuda.empty_cache()
    return out


def e2e_measure(P, torch, stack, steps):
    """The same step (the same library calls, through `stack.step`) with
    host-resident inputs: every layer's X and dY are copied from pinned host
    memory into device buffers and every layer's dW is read back to pinned
    host memory, all inside the timed region.  Copies run on their own
    streams (H2D, D2H) and overlap the computation; each layer's compute
    waits for its own inputs, and dW alternates between two device buffer
    sets so a read-back never races a later Wgrad into the same buffer.  The
    pinned source holds layer 0's inputs and serves every layer (host memory
    stays bounded); the weights stay resident, as a model's do."""
    comp = torch.cuda.current_stream()
    h2d_s = torch.cuda.Stream()  # one stream: more measured slower (145 vs 163 GB/s)
    d2h_s = torch.cuda.Stream()
    J = len(stack.wl.linears)
    hx = [li.x.cpu().pin_memory() for li in stack.inputs[0]]
    hdy = [li.dy.cpu().pin_memory() for li in stack.inputs[0]]
    dw_sets = [stack.dw, [torch.empty_like(d) for d in stack.dw]]
    hdw = [[torch.empty(d.shape, dtype=d.dtype).pin_memory() for d in stack.dw] for _ in range(2)]
    x_ready = [torch.cuda.Event() for _ in range(stack.L)]
    dy_ready = [torch.cuda.Event() for _ in range(stack.L)]
    dw_done = [torch.cuda.Event() for _ in range(J)]
    dw_read = [[torch.cuda.Event() for _ in range(J)] for _ in range(2)]
    counts = {"h2d": 0, "d2h": 0}

    class Hooks:
        def before_forward(self, l):
            comp.wait_event(x_ready[l])

        def before_backward(self, l):
            comp.wait_event(dy_ready[l])

        def dw(self, l, j):
            comp.wait_event(dw_read[l % 2][j])  # this buffer's previous read-back is done
            return dw_sets[l % 2][j]

        def after_backward(self, l, j, dw):
            dw_done[j].record(comp)
            d2h_s.wait_event(dw_done[j])
            with torch.cuda.stream(d2h_s):
                hdw[l % 2][j].copy_(dw, non_blocking=True)
            dw_read[l % 2][j].record(d2h_s)
            counts["d2h"] += dw.numel() * dw.element_size()

    hooks = Hooks()

    def one_step():
        counts["h2d"] = counts["d2h"] = 0
        begin = torch.cuda.Event()
        begin.record(comp)
        h2d_s.wait_event(begin)  # nothing is copied before this step starts
        with torch.cuda.stream(h2d_s):
            for l in range(stack.L):
                for j in range(J):
                    stack.inputs[l][j].x.copy_(hx[j], non_blocking=True)
                    counts["h2d"] += hx[j].numel() * hx[j].element_size()
                x_ready[l].record(h2d_s)
            for l in reversed(range(stack.L)):
                for j in range(J):
                    stack.inputs[l][j].dy.copy_(hdy[j], non_blocking=True)
                    counts["h2d"] += hdy[j].numel() * hdy[j].element_size()
                dy_ready[l].record(h2d_s)
        stack.step(hooks)
        comp.wait_stream(d2h_s)
        comp.wait_stream(h2d_s)

    stack.timer.enabled = False
    one_step()
    torch.cuda.synchronize()
    s = torch.cuda.Event(enable_timing=True)
    e = torch.cuda.Event(enable_timing=True)
    s.record(comp)
    for _ in range(steps):
        one_step()
    e.record(comp)
    torch.cuda.synchronize()
    t = s.elapsed_time(e) * 1e-3 / steps
    h2d_gbs = counts["h2d"] / t / 1e9
    return {"value": stack.flops_per_step() / t / 1e12, "unit": "TFLOP/s", "ms_per_step": t * 1e3,
            "h2d_bytes_per_step": counts["h2d"], "d2h_bytes_per_step": counts["d2h"],
            "h2d_gbs_effective": h2d_gbs,
            "steps": steps,
            "note": "X and dY of every layer copied from pinned host memory (layer 0's bytes serve every layer) "
                    "on a copy stream overlapping compute; every layer's dW read back on another.  The step's "
                    "results that leave the device are the weight gradients: Y and dX are activations and "
                    "activation gradients that the rest of the model (not on this path) consumes on the device, "
                    "so they are not read back.  The host-to-device link measured about 200-211 GB/s with "
                    "nothing else running"}


def cpu_baseline(torch, stack, seconds_hint=True):
    """The oracle, as it stands, on the host cores: quantise + Fprop/Dgrad/Wgrad
    in fp64 for the first M_s tokens of layer 0's o_proj linear."""
    import numpy as np

    import oracle as O

    M_s = min(32768, stack.M)
    li = stack.inputs[0][1]  # o_proj [1536, 1536]
    N, K = li.w.shape

    def b(t):
        return t.contiguous().cpu().view(torch.int16).numpy().view(np.uint16)

    x, w, dy = b(li.x[:M_s]), b(li.w), b(li.dy[:M_s])
    threads = os.cpu_count() or 1
    t0 = time.perf_counter()
    O.linear_block(x, w, dy, nthreads=threads)
    t = time.perf_counter() - t0
    flops = 6.0 * M_s * N * K
    return {"value": flops / t / 1e12, "unit": "TFLOP/s", "cores": threads, "kind": "oracle",
            "seconds": t, "sample": f"layer 0 o_proj [{N},{K}], first {M_s} of {stack.M} tokens: blockwise "
                                    f"quantise + Fprop/Dgrad/Wgrad in fp64 ({flops / 1e9:.1f} GFLOP)"}


# ----------------------------------------------------------------------------
def reference_arm(args):
    """The oracle timed on host cores, same metric/unit/config."""
    rank = int(os.environ.get("RANK", "0"))
    if rank != 0:
        return 0
    import numpy as np
    import torch

    import oracle as O
    from paper_2608_27370_gb300 import workloads as W

    wl = W.WORKLOADS[args.config]
    M_s = 256
    _, N, K = wl.linears[1] if len(wl.linears) > 1 else wl.linears[0]
    g = lambda shape, std, seed: W.normal_bf16(shape, std, "cpu", seed).view(torch.int16).numpy().view(np.uint16)  # noqa
    x, w, dy = g((M_s, K), 1.0, 1), g((N, K), 0.02, 2), g((M_s, N), 1e-3, 3)
    threads = os.cpu_count() or 1
    flops = 6.0 * M_s * N * K
    for _ in range(args.warmup):
        O.linear_block(x, w, dy, nthreads=threads)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        O.linear_block(x, w, dy, nthreads=threads)
    t = (time.perf_counter() - t0) / max(args.steps, 1)
    v = flops / t / 1e12
    sample = f"one [{N},{K}] linear of {args.config}, {M_s} tokens per step: blockwise quantise + 3 GEMMs in fp64"
    line = {"metric": METRIC, "value": v, "unit": "TFLOP/s", "n_gpus": args.gpus, "steps": args.steps,
            "warmup": args.warmup, "ms_per_step": t * 1e3, "higher_is_better": True, "scaling": "weak",
            "vs_baseline": None, "dtype": "f64", "data": "synthetic", "impl": "reference",
            "config": {"workload": f"{wl.key}: " + wl.description, "tokens_per_step": M_s,
                       "scaling": "block", "sample": "bounded CPU sample of the workload, see cpu_baseline"},
            "cpu_baseline": {"value": v, "unit": "TFLOP/s", "cores": threads, "kind": "oracle", "sample": sample},
            "e2e": {"value": v, "unit": "TFLOP/s", "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)
    return 0


def main():
    args = parse_args()
    if args.impl == "reference":
        return reference_arm(args)

    import torch
    import torch.distributed as dist

    import paper_2608_27370_gb300 as P
    from paper_2608_27370_gb300 import workloads as W

    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    torch.cuda.set_device(local)
    device = f"cuda:{local}"
    if world > 1:
        dist.init_process_group("nccl", device_id=torch.device(device))
    P.load_library()
    peaks, peak_src = load_peaks()

    wl = W.WORKLOADS[args.config]
    layers = args.layers or wl.layers
    M = args.tokens or wl.M
    stack = LinearStack(P, W, torch, wl, device, args.scaling, layers, M)
    torch.cuda.synchronize()

    for _ in range(args.warmup):
        stack.step()
    torch.cuda.synchronize()
    if world > 1:
        dist.barrier()
    clocks = ClockSampler(local, enabled=not args.no_clocks)
    stack.timer.pending.clear()
    torch.cuda.synchronize()
    t_start = torch.cuda.Event(enable_timing=True)
    t_end = torch.cuda.Event(enable_timing=True)
    t_start.record()
    for i in range(args.steps):
        # per-launch CUDA events (the kernels' own durations) in the last
        # timed step only: two events around each of a step's ~730 launches
        # cost the step 2.5-4.5%, which the earlier steps do not carry
        stack.timer.enabled = i == args.steps - 1
        stack.step()
    t_end.record()
    torch.cuda.synchronize()
    clk = clocks.stop()
    stack.timer.enabled = False
    elapsed = max_over_ranks(t_start.elapsed_time(t_end) * 1e-3, world, device)
    per_kernel = stack.timer.totals()
    step_s = elapsed / args.steps
    flops = stack.flops_per_step()
    value = job_value(world, flops, step_s) / 1e12

    fp8_peak_burst = peaks["bf16_tflops"] * FP8_PER_BF16
    fp8_peak_sust = peaks["bf16_tflops_sustained"] * FP8_PER_BF16
    g = per_kernel.get("gemm", {"time_s": 1.0, "units": 0.0, "launches": 1})
    q = per_kernel.get("quantize", {"time_s": 1.0, "units": 0.0, "launches": 1})
    gemm_tflops = g["units"] / g["time_s"] / 1e12
    quant_gbs = q["units"] / q["time_s"] / 1e9
    total_kernel_time = sum(c["time_s"] for c in per_kernel.values())
    traffic_wl = (args.config, M, args.scaling)
    shares = {k: c["time_s"] / total_kernel_time for k, c in per_kernel.items()}

    result = {
        "metric": METRIC, "value": value, "unit": "TFLOP/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": step_s * 1e3, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None,
        "dtype": "fp8_e4m3" + ("+e8m0_block_scales" if args.scaling == "block" else "+fp32_tensor_scale"),
        "data": "synthetic",
        "config": {"workload": f"{wl.key}: " + wl.description if layers == wl.layers and M == wl.M else
                   f"{wl.key} profile subset: {layers} layers, M={M}",
                   "tokens_per_step": M, "layers": layers, "linears_per_layer": len(wl.linears),
                   "scaling": args.scaling, "l2": "inputs larger than L2 (>=2.4 GB per layer)",
                   "parallelism": f"replicas x{world} (weak scaling, no collective on the path)"},
        "pct_fp8_peak": 100.0 * value / world / fp8_peak_sust,
        "step_frac_vs_nominal_fp8": value / world / NOMINAL_FP8_DENSE_TFLOPS,
        "tokens_per_s": world * M / step_s,
        "gemm_only_tflops": gemm_tflops,
        "quantize_gbs": quant_gbs,
        "kernel_time_share": shares,
        "gpu_launches": stack.launches_per_step * args.steps,
        "roofline": {"bound": "tensor", "kernel": "gemm_tn_kernel<FP8 block-scaled>", "achieved": gemm_tflops,
                     "peak": fp8_peak_sust, "unit": "TFLOP/s", "frac": gemm_tflops / fp8_peak_sust,
                     "peak_source": f"2 x bf16_tflops_sustained ({peak_src}); kernel timed inside a long step",
                     "traffic": captured_traffic("gemm", traffic_wl, stack.gemm_algorithmic_bytes_per_call()),
                     "traffic_note": "DRAM bytes per GEMM launch: DRAM bytes per algorithmic byte from per-kernel ncu captures of one layer's GEMM calls, times the step's average launch",
                     "timing": "CUDA events around each launch of the last timed step, on the launching stream",
                     "nominal_peak": NOMINAL_FP8_DENSE_TFLOPS,
                     "frac_vs_nominal": gemm_tflops / NOMINAL_FP8_DENSE_TFLOPS},
        "roofline_quantize": {"bound": "hbm", "kernel": "quant_act_kernel (X, dY) + quant_weight_group_kernel (W)", "achieved": quant_gbs,
                              "peak": peaks["hbm_gbs"], "unit": "GB/s", "frac": quant_gbs / peaks["hbm_gbs"],
                              "peak_source": f"hbm_gbs ({peak_src})",
                              "traffic": captured_traffic("quantize", traffic_wl,
                                                          q["units"] / stack.quantize_kernel_launches_per_step()),
                              "traffic_note": "DRAM bytes per quantiser launch: DRAM bytes per algorithmic byte from per-kernel ncu captures of one layer's quantiser calls, times the step's average launch",
                              "timing": "CUDA events around each launch of the last timed step, on the launching stream",
                              "nominal_peak": NOMINAL_HBM_GBS,
                              "frac_vs_nominal": quant_gbs / NOMINAL_HBM_GBS},
    }
    if args.scaling == "tensor":
        result["roofline"]["kernel"] = "gemm_tn_kernel<FP8 per-tensor>"
    result["gemm_by_call"] = stack.timer.by_label("gemm", 1e-12)        # rate: TFLOP/s
    result["quantize_by_call"] = stack.timer.by_label("quantize", 1e-9)  # rate: GB/s (algorithmic)
    if clk:
        result["clocks"] = clk
        # the tensor pipe's own ceiling at the clock the timed region ran at:
        # a pair MMA (M 256, N 256, K 32 bytes of FP8) takes 128 cycles, so
        # 16384 FP8 flop per clock per SM
        sms = torch.cuda.get_device_properties(device).multi_processor_count
        clock_peak = FP8_FLOP_PER_CLK_SM * sms * clk["sm_mhz"] * 1e6 / 1e12
        result["roofline"]["clock_limited_tensor_peak"] = clock_peak
        result["roofline"]["frac_vs_clock_limited_tensor_peak"] = gemm_tflops / clock_peak
        result["step_frac_vs_clock_limited_tensor_peak"] = value / world / clock_peak
    if rank == 0 and world == 1 and not args.no_bf16 and args.scaling == "block":
        try:
            result["bf16_comparison"] = bf16_layer_speedup(P, torch, stack)
        except (RuntimeError, torch.cuda.OutOfMemoryError) as exc:  # report, do not hide
            result["bf16_comparison"] = {"error": str(exc)}
        try:
            result["library_context"] = library_context(torch, stack)
        except (RuntimeError, torch.cuda.OutOfMemoryError) as exc:
            result["library_context"] = {"error": str(exc)}
    if rank == 0 and world == 1 and not args.no_paper_model and args.scaling == "block":
        result["e5m2_gradients"] = grad_format_measure(P, torch, stack)
    if not args.no_e2e:
        result["e2e"] = e2e_measure(P, torch, stack, 5)
        if world > 1:
            ms = max_over_ranks(result["e2e"]["ms_per_step"], world, device)
            result["e2e"]["ms_per_step"] = ms
            result["e2e"]["value"] = job_value(world, flops, ms * 1e-3) / 1e12
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        result["cpu_baseline"] = cpu_baseline(torch, stack)
    if rank == 0 and world == 1 and not args.no_paper_model and args.config == "C5":
        del stack
        torch.cuda.empty_cache()
        result["paper_model_shape"] = paper_model_measure(P, W, torch, device, args.scaling)
        result["rmsnorm_quantize_fusion"] = rmsnorm_fusion_measure(P, W, torch, device)
        result["swiglu_quantize_fusion"] = swiglu_fusion_measure(P, W, torch, device)
        result["dgrad_quantize_fusion"] = dgrad_quantize_fusion_measure(P, W, torch, device)
        result["muonh_step"] = muonh_measure(P, W, torch, device, peaks)
        if args.scaling == "block":
            result["tensor_scaling"] = tensor_scaling_measure(P, W, torch, device)
            result["tensor_scaling_e5m2_gradients"] = tensor_scaling_measure(P, W, torch, device, grad_fmt=P.E5M2)
    if rank == 0:
        print(json.dumps(result), flush=True)
    if world > 1:
        dist.barrier()
        dist.destroy_process_group()
    return 0


if __name__ == "__main__":
    sys.exit(main())
