"""GB300 (sm_103a) FP8 linear-layer training path of Puro-2B.

Python binding of ``libpuro_fp8.so`` (C ABI in ``include/puro_fp8.h``).
Every function here is argument marshalling only: it checks that the torch
tensors it is handed are CUDA, contiguous and of the right dtype, and passes
their device pointers, the sizes and the current CUDA stream to the library
entry point of the same name.  All arithmetic runs in the library's CUDA
kernels.  There is no fallback: if the library is missing, every call raises
:class:`PuroError`.

The method (paper section "FP8 Mixed-Precision Training"; appendix
"Production Training Details", paragraph "FP8 implementation pipeline"):
E4M3 operands for all three GEMMs of every linear layer, power-of-two scales
computed online for 1x128 groups along the reduction dimension (activations
and activation gradients) or 128x128 blocks (weights), FP32 accumulation and
BF16 output.
"""
from __future__ import annotations

import ctypes
import os
from dataclasses import dataclass
from typing import Optional

import torch

from . import _build

E4M3, E5M2 = 0, 1
SCALE_TENSOR, SCALE_BLOCK = 0, 1
ROLE_ACT, ROLE_WEIGHT = 0, 1

PURO_OK = 0
PURO_ERR_INVALID_ARG = 1
PURO_ERR_UNSUPPORTED = 2
PURO_ERR_CUDA = 3
PURO_ERR_TIMEOUT = 4

LIB_PATH = _build.LIB
HEADER_PATH = os.path.join(_build.INCLUDE, "puro_fp8.h")


class PuroError(RuntimeError):
    def __init__(self, fn: str, status: int):
        self.status = status
        names = {1: "PURO_ERR_INVALID_ARG", 2: "PURO_ERR_UNSUPPORTED", 3: "PURO_ERR_CUDA", 4: "PURO_ERR_TIMEOUT"}
        super().__init__(f"{fn} returned {names.get(status, status)}")


class puro_fp8_tensor_t(ctypes.Structure):
    """Mirror of the C struct puro_fp8_tensor_t."""
    _fields_ = [
        ("data", ctypes.c_void_p),
        ("scale", ctypes.c_void_p),
        ("rows", ctypes.c_int64),
        ("red", ctypes.c_int64),
        ("fmt", ctypes.c_int32),
        ("scaling", ctypes.c_int32),
        ("role", ctypes.c_int32),
        ("reserved", ctypes.c_int32),
    ]


_P = ctypes.c_void_p
_I64 = ctypes.c_int64
_I32 = ctypes.c_int32
_SIGNATURES = {
    "puro_fp8_amax": (_I32, [_P, _I64, _I64, _P, _P]),
    "puro_fp8_quantize": (_I32, [_P, _I64, _I64, _I32, _I32, _I32, _P, _P, _P, _P, _P, _P, _P]),
    "puro_fp8_quantize_rmsnorm": (_I32, [_P, _I64, _I64, _P, ctypes.c_float, _I32, _P, _P, _P, _P, _P, _P, _P, _P]),
    "puro_rmsnorm_bf16": (_I32, [_P, _I64, _I64, _P, ctypes.c_float, _P, _P, _P]),
    "puro_fp8_quantize_swiglu": (_I32, [_P, _P, _I64, _I64, _I64, _I32, _P, _P, _P, _P, _P, _P, _P]),
    "puro_muonh_workspace_size": (ctypes.c_size_t, [_I64]),
    "puro_muonh_reduce": (_I32, [_P, _P, _I64, _P, _P, ctypes.c_size_t, _P]),
    "puro_muonh_apply": (_I32, [_P, _P, _I64, _P, ctypes.c_double, ctypes.c_double, _P, _P]),
    "puro_muonh_step": (_I32, [_P, _P, _I64, ctypes.c_double, ctypes.c_double, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_muonh_grouped_workspace_size": (ctypes.c_size_t, [_P, _I32]),
    "puro_muonh_step_grouped": (_I32, [_P, _I32, ctypes.c_double, _P, _P, ctypes.c_size_t, _P]),
    "puro_swiglu_bf16": (_I32, [_P, _P, _I64, _I64, _I64, _P, _P]),
    "puro_fp8_linear_fprop": (_I32, [_P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_fp8_linear_dgrad": (_I32, [_P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_fp8_linear_wgrad": (_I32, [_P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_fp8_linear_dgrad_quantize": (_I32, [_P, _P, _I32, _P, _P, _P, _P, _P, _P, _P]),
    "puro_fp8_linear_backward": (_I32, [_P, _P, _P, _P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_fp8_quantize_weights": (_I32, [_P, _I32, _I32, _P, _P]),
    "puro_fp8_linear_wgrad_main_grad": (_I32, [_P, _P, _P, _P, ctypes.c_size_t, _P, _P]),
    "puro_fp8_linear_wgrad_noalloc": (_I32, [_P, _P, _P, _P, _P]),
    "puro_fp8_workspace_size": (ctypes.c_size_t, [_I64, _I64, _I64]),
    "puro_fp8_linear_backward_launches": (_I32, [_I64, _I64, _I64, ctypes.c_size_t]),
    "puro_fp8_scale_bytes": (ctypes.c_size_t, [_I64, _I64]),
    "puro_fp8_get_status": (_I32, [_P, _P, _P]),
    "puro_bf16_linear_fprop": (_I32, [_P, _P, _P, _I64, _I64, _I64, _P, _P]),
    "puro_bf16_linear_dgrad": (_I32, [_P, _P, _P, _I64, _I64, _I64, _P, _P]),
    "puro_bf16_linear_wgrad": (_I32, [_P, _P, _P, _I64, _I64, _I64, _P, _P]),
    "puro_set_wait_timeout_ns": (None, [ctypes.c_uint64]),
    "puro_set_gemm_tile_n": (ctypes.c_int, [ctypes.c_int32]),
    "puro_status_string": (ctypes.c_char_p, [_I32]),
}

_lib = None


def load_library(path: Optional[str] = None):
    """Load libpuro_fp8.so (built by ``__graft_entry__.build()``); raises if absent."""
    global _lib
    if _lib is not None and path is None:
        return _lib
    p = path or LIB_PATH
    if not os.path.exists(p):
        raise RuntimeError(
            f"libpuro_fp8.so not found at {p}: build it with `python -c 'import __graft_entry__ as g; g.build()'`")
    lib = ctypes.CDLL(p)
    for name, (res, args) in _SIGNATURES.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    if path is None:
        _lib = lib
    return lib


def _check(fn: str, status: int) -> None:
    if status != PURO_OK:
        raise PuroError(fn, status)


def _stream(stream) -> int:
    if stream is None:
        return torch.cuda.current_stream().cuda_stream
    if isinstance(stream, torch.cuda.Stream):
        return stream.cuda_stream
    return int(stream)


def _ptr(t: Optional[torch.Tensor], dtype=None, name: str = "tensor") -> Optional[int]:
    if t is None:
        return None
    if t.numel() == 0:
        return t.data_ptr() or None
    if not t.is_cuda:
        raise ValueError(f"{name} must be a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if dtype is not None and t.dtype not in (dtype if isinstance(dtype, tuple) else (dtype,)):
        raise ValueError(f"{name} has dtype {t.dtype}, expected {dtype}")
    return t.data_ptr()


# --------------------------------------------------------------------------
# Entry points (same names as the C ABI)
# --------------------------------------------------------------------------
def puro_fp8_amax(x: torch.Tensor, amax_bits: torch.Tensor, stream=None) -> None:
    rows, cols = (x.shape[0], x.shape[1]) if x.dim() == 2 else (1, x.numel())
    st = load_library().puro_fp8_amax(_ptr(x, torch.bfloat16, "x"), rows, cols,
                                      _ptr(amax_bits, (torch.int32, torch.uint32), "amax_bits"), _stream(stream))
    _check("puro_fp8_amax", st)


def puro_fp8_quantize(x: torch.Tensor, fmt: int, scaling: int, role: int, amax_bits: Optional[torch.Tensor],
                      q: torch.Tensor, scale: torch.Tensor, q_t: Optional[torch.Tensor] = None,
                      scale_t: Optional[torch.Tensor] = None, dev_status: Optional[torch.Tensor] = None,
                      stream=None) -> None:
    rows, cols = x.shape
    u8 = torch.uint8
    sdt = u8 if scaling == SCALE_BLOCK else torch.float32
    st = load_library().puro_fp8_quantize(
        _ptr(x, torch.bfloat16, "x"), rows, cols, fmt, scaling, role,
        _ptr(amax_bits, (torch.int32, torch.uint32), "amax_bits"), _ptr(q, u8, "q"), _ptr(scale, sdt, "scale"),
        _ptr(q_t, u8, "q_t"), _ptr(scale_t, sdt, "scale_t"), _ptr(dev_status, torch.int32, "dev_status"),
        _stream(stream))
    _check("puro_fp8_quantize", st)


def puro_fp8_quantize_rmsnorm(h: torch.Tensor, gamma: Optional[torch.Tensor], eps: float, fmt: int,
                              rstd: torch.Tensor, y: Optional[torch.Tensor], q: torch.Tensor, scale: torch.Tensor,
                              q_t: Optional[torch.Tensor] = None, scale_t: Optional[torch.Tensor] = None,
                              dev_status: Optional[torch.Tensor] = None, stream=None) -> None:
    """RMSNorm of the rows of h (bf16, optional bf16 gain) fused ahead of the
    blockwise activation quantiser: writes rstd (fp32 [rows]), optionally y
    (bf16), and the codes and scales as puro_fp8_quantize does."""
    rows, cols = h.shape
    u8 = torch.uint8
    st = load_library().puro_fp8_quantize_rmsnorm(
        _ptr(h, torch.bfloat16, "h"), rows, cols, _ptr(gamma, torch.bfloat16, "gamma"), float(eps), fmt,
        _ptr(rstd, torch.float32, "rstd"), _ptr(y, torch.bfloat16, "y"), _ptr(q, u8, "q"), _ptr(scale, u8, "scale"),
        _ptr(q_t, u8, "q_t"), _ptr(scale_t, u8, "scale_t"), _ptr(dev_status, torch.int32, "dev_status"),
        _stream(stream))
    _check("puro_fp8_quantize_rmsnorm", st)


def _gate_up(gate: torch.Tensor, up: torch.Tensor):
    """Pointers and the shared row stride of gate / up (bf16 [rows, cols]
    CUDA tensors with unit column stride, e.g. the halves of one output)."""
    for name, t in (("gate", gate), ("up", up)):
        if not t.is_cuda or t.dtype != torch.bfloat16 or t.dim() != 2:
            raise ValueError(f"{name} must be a 2-D bf16 CUDA tensor")
        if t.numel() and t.stride(1) != 1:
            raise ValueError(f"{name} must have unit column stride")
    if gate.shape != up.shape:
        raise ValueError("gate and up differ in shape")
    rows, cols = gate.shape
    ld = gate.stride(0) if rows > 1 else cols
    if rows > 1 and up.stride(0) != ld:
        raise ValueError("gate and up must share one row stride")
    return gate.data_ptr() or None, up.data_ptr() or None, rows, cols, ld


class puro_fp8_weight_t(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("rows", ctypes.c_int64), ("cols", ctypes.c_int64),
                ("q", ctypes.c_void_p), ("scale", ctypes.c_void_p), ("q_t", ctypes.c_void_p),
                ("scale_t", ctypes.c_void_p)]


def weight_table(entries):
    """The host table of puro_fp8_quantize_weights for a fixed list of
    (w bf16 [rows, cols], Quantized with rowwise [rows, cols] and optional
    colwise [cols, rows] operands): build it once and pass it to every call
    (the tensors must stay alive and in place)."""
    table = (puro_fp8_weight_t * max(1, len(entries)))()
    u8 = torch.uint8
    for i, (w, q) in enumerate(entries):
        col = q.colwise
        table[i] = puro_fp8_weight_t(_ptr(w, torch.bfloat16, "w"), w.shape[0], w.shape[1],
                                     _ptr(q.rowwise.data, u8, "q"), _ptr(q.rowwise.scale, u8, "scale"),
                                     _ptr(col.data, u8, "q_t") if col is not None else None,
                                     _ptr(col.scale, u8, "scale_t") if col is not None else None)
    table.count = len(entries)
    return table


def puro_fp8_quantize_weights(entries, fmt: int = E4M3, dev_status: Optional[torch.Tensor] = None,
                              stream=None) -> None:
    """Quantise many weights in 128x128 blocks in one call: entries is a list
    of (w, Quantized) pairs or a table from weight_table().  Same bytes as
    quantize(w, fmt, SCALE_BLOCK, ROLE_WEIGHT, out=q) for each."""
    table = entries if isinstance(entries, ctypes.Array) else weight_table(entries)
    st = load_library().puro_fp8_quantize_weights(table, table.count, fmt,
                                                  _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check("puro_fp8_quantize_weights", st)


def puro_fp8_quantize_swiglu(gate: torch.Tensor, up: torch.Tensor, fmt: int, y: Optional[torch.Tensor],
                             q: torch.Tensor, scale: torch.Tensor, q_t: Optional[torch.Tensor] = None,
                             scale_t: Optional[torch.Tensor] = None, dev_status: Optional[torch.Tensor] = None,
                             stream=None) -> None:
    """SwiGLU (silu(gate) * up, bf16) fused ahead of the blockwise activation
    quantiser: writes the codes and scales as puro_fp8_quantize does, and y
    (bf16) only when given.  gate and up may be row-strided views."""
    g, u, rows, cols, ld = _gate_up(gate, up)
    u8 = torch.uint8
    st = load_library().puro_fp8_quantize_swiglu(
        g, u, rows, cols, ld, fmt, _ptr(y, torch.bfloat16, "y"), _ptr(q, u8, "q"), _ptr(scale, u8, "scale"),
        _ptr(q_t, u8, "q_t"), _ptr(scale_t, u8, "scale_t"), _ptr(dev_status, torch.int32, "dev_status"),
        _stream(stream))
    _check("puro_fp8_quantize_swiglu", st)


def puro_swiglu_bf16(gate: torch.Tensor, up: torch.Tensor, y: torch.Tensor, stream=None) -> None:
    g, u, rows, cols, ld = _gate_up(gate, up)
    st = load_library().puro_swiglu_bf16(g, u, rows, cols, ld, _ptr(y, torch.bfloat16, "y"), _stream(stream))
    _check("puro_swiglu_bf16", st)


def puro_muonh_workspace_size(n: int) -> int:
    return int(load_library().puro_muonh_workspace_size(n))


def puro_muonh_reduce(w: torch.Tensor, u: torch.Tensor, sums: torch.Tensor, workspace: torch.Tensor,
                      stream=None) -> None:
    """sums (fp64 [3], device) = {sum W^2, sum W u, sum u^2} of fp32 W and u."""
    if w.numel() != u.numel():
        raise ValueError("w and u differ in size")
    st = load_library().puro_muonh_reduce(_ptr(w, torch.float32, "w"), _ptr(u, torch.float32, "u"), w.numel(),
                                          _ptr(sums, torch.float64, "sums"), _ptr(workspace, None, "workspace"),
                                          workspace.numel() * workspace.element_size(), _stream(stream))
    _check("puro_muonh_reduce", st)


def puro_muonh_apply(w: torch.Tensor, u: torch.Tensor, sums: torch.Tensor, eta: float, radius: float,
                     w_bf16: Optional[torch.Tensor] = None, stream=None) -> None:
    if w.numel() != u.numel() or (w_bf16 is not None and w_bf16.numel() != w.numel()):
        raise ValueError("w, u and w_bf16 differ in size")
    st = load_library().puro_muonh_apply(_ptr(w, torch.float32, "w"), _ptr(u, torch.float32, "u"), w.numel(),
                                         _ptr(sums, torch.float64, "sums"), float(eta), float(radius),
                                         _ptr(w_bf16, torch.bfloat16, "w_bf16"), _stream(stream))
    _check("puro_muonh_apply", st)


def puro_muonh_step(w: torch.Tensor, u: torch.Tensor, eta: float, radius: float, sums: torch.Tensor,
                    workspace: torch.Tensor, w_bf16: Optional[torch.Tensor] = None, stream=None) -> None:
    """One MuonH hyperball update of the fp32 master weight w (in place)
    along the Muon direction u; optionally writes the bf16 copy."""
    if w.numel() != u.numel() or (w_bf16 is not None and w_bf16.numel() != w.numel()):
        raise ValueError("w, u and w_bf16 differ in size")
    st = load_library().puro_muonh_step(_ptr(w, torch.float32, "w"), _ptr(u, torch.float32, "u"), w.numel(),
                                        float(eta), float(radius), _ptr(sums, torch.float64, "sums"),
                                        _ptr(workspace, None, "workspace"),
                                        workspace.numel() * workspace.element_size(),
                                        _ptr(w_bf16, torch.bfloat16, "w_bf16"), _stream(stream))
    _check("puro_muonh_step", st)


class puro_muonh_matrix_t(ctypes.Structure):
    _fields_ = [("w", ctypes.c_void_p), ("u", ctypes.c_void_p), ("w_bf16", ctypes.c_void_p),
                ("n", ctypes.c_int64), ("radius", ctypes.c_double)]


def _muonh_table(mats):
    """ctypes array of descriptors from (w, u, w_bf16 or None, radius) tuples."""
    arr = (puro_muonh_matrix_t * max(1, len(mats)))()
    for i, (w, u, wb, r) in enumerate(mats):
        if w.numel() != u.numel() or (wb is not None and wb.numel() != w.numel()):
            raise ValueError(f"matrix {i}: w, u and w_bf16 differ in size")
        arr[i] = puro_muonh_matrix_t(_ptr(w, torch.float32, "w"), _ptr(u, torch.float32, "u"),
                                     _ptr(wb, torch.bfloat16, "w_bf16"), w.numel(), float(r))
    return arr


def puro_muonh_grouped_workspace_size(mats) -> int:
    return int(load_library().puro_muonh_grouped_workspace_size(_muonh_table(mats), len(mats)))


def puro_muonh_step_grouped(mats, eta: float, sums: torch.Tensor, workspace: torch.Tensor, stream=None) -> None:
    """The hyperball step for every (w, u, w_bf16 or None, radius) in mats;
    sums: fp64 [len(mats), 3] on the device."""
    table = _muonh_table(mats)
    st = load_library().puro_muonh_step_grouped(table, len(mats), float(eta), _ptr(sums, torch.float64, "sums"),
                                                _ptr(workspace, None, "workspace"),
                                                workspace.numel() * workspace.element_size(), _stream(stream))
    _check("puro_muonh_step_grouped", st)


def muonh_radius(w0: torch.Tensor) -> float:
    """R = ||W_0||_F (fp64, through puro_muonh_reduce; synchronises)."""
    sums = torch.empty(3, dtype=torch.float64, device=w0.device)
    ws = torch.empty(max(8, puro_muonh_workspace_size(w0.numel())), dtype=torch.uint8, device=w0.device)
    puro_muonh_reduce(w0, w0, sums, ws)
    return float(sums[0].sqrt().item())


def puro_rmsnorm_bf16(h: torch.Tensor, gamma: Optional[torch.Tensor], eps: float, rstd: torch.Tensor,
                      y: torch.Tensor, stream=None) -> None:
    """The same RMSNorm without the quantiser (rstd fp32, y bf16)."""
    rows, cols = h.shape
    st = load_library().puro_rmsnorm_bf16(_ptr(h, torch.bfloat16, "h"), rows, cols,
                                          _ptr(gamma, torch.bfloat16, "gamma"), float(eps),
                                          _ptr(rstd, torch.float32, "rstd"), _ptr(y, torch.bfloat16, "y"),
                                          _stream(stream))
    _check("puro_rmsnorm_bf16", st)


@dataclass
class FP8Operand:
    """A quantised GEMM operand: codes [rows, red] plus scales (torch tensors kept alive here)."""
    data: torch.Tensor
    scale: torch.Tensor
    fmt: int = E4M3
    scaling: int = SCALE_BLOCK
    role: int = ROLE_ACT

    @property
    def rows(self) -> int:
        return self.data.shape[0]

    @property
    def red(self) -> int:
        return self.data.shape[1]

    def as_c(self) -> puro_fp8_tensor_t:
        return puro_fp8_tensor_t(_ptr(self.data, torch.uint8, "data"), _ptr(self.scale, None, "scale"),
                                 self.data.shape[0], self.data.shape[1], self.fmt, self.scaling, self.role, 0)


def _gemm(name: str, a: FP8Operand, b: FP8Operand, out: torch.Tensor, workspace, dev_status, stream,
          out_dtype=torch.bfloat16) -> None:
    ca, cb = a.as_c(), b.as_c()
    ws_ptr = _ptr(workspace, None, "workspace")
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    fn = getattr(load_library(), name)
    st = fn(ctypes.byref(ca), ctypes.byref(cb), _ptr(out, out_dtype, "out"), ws_ptr, ws_bytes,
            _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check(name, st)


def puro_fp8_linear_fprop(x: FP8Operand, w: FP8Operand, y: torch.Tensor, workspace=None, dev_status=None,
                          stream=None) -> None:
    """Y [M,N] = X [M,K] . W [N,K]^T."""
    _gemm("puro_fp8_linear_fprop", x, w, y, workspace, dev_status, stream)


def puro_fp8_linear_dgrad(dy: FP8Operand, w_t: FP8Operand, dx: torch.Tensor, workspace=None, dev_status=None,
                          stream=None) -> None:
    """dX [M,K] = dY [M,N] . W [N,K] (B operand = W^T [K,N])."""
    _gemm("puro_fp8_linear_dgrad", dy, w_t, dx, workspace, dev_status, stream)


def puro_fp8_linear_backward(dy: FP8Operand, w_t: FP8Operand, dx: torch.Tensor, dy_t: FP8Operand,
                             x_t: FP8Operand, dw: torch.Tensor, workspace=None, dev_status=None, stream=None) -> None:
    """dX [M,K] = dY . W and dW [N,K] = dY^T . X in one call (one grouped
    launch when both are unsplit block-scaled GEMMs)."""
    c = [op.as_c() for op in (dy, w_t, dy_t, x_t)]
    ws_bytes = workspace.numel() * workspace.element_size() if workspace is not None else 0
    st = load_library().puro_fp8_linear_backward(
        ctypes.byref(c[0]), ctypes.byref(c[1]), _ptr(dx, torch.bfloat16, "dx"), ctypes.byref(c[2]),
        ctypes.byref(c[3]), _ptr(dw, torch.bfloat16, "dw"), _ptr(workspace, None, "workspace"), ws_bytes,
        _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check("puro_fp8_linear_backward", st)


def puro_fp8_linear_dgrad_quantize(dy: FP8Operand, w_t: FP8Operand, fmt: int, dx: Optional[torch.Tensor],
                                   dxq: torch.Tensor, dxq_scale: torch.Tensor, dxq_t: Optional[torch.Tensor] = None,
                                   dxq_t_scale: Optional[torch.Tensor] = None, dev_status=None, stream=None) -> None:
    """dX [M,K] = dY [M,N] . W [N,K], rounded to BF16 and quantised in the
    GEMM's epilogue into the blockwise activation copies (dxq [M,K] with
    1x128 groups; dxq_t [K,M] with 128-row groups, optional); dx (bf16) is
    written only when given."""
    ca, cb = dy.as_c(), w_t.as_c()
    u8 = torch.uint8
    st = load_library().puro_fp8_linear_dgrad_quantize(
        ctypes.byref(ca), ctypes.byref(cb), fmt, _ptr(dx, torch.bfloat16, "dx"), _ptr(dxq, u8, "dxq"),
        _ptr(dxq_scale, u8, "dxq_scale"), _ptr(dxq_t, u8, "dxq_t"), _ptr(dxq_t_scale, u8, "dxq_t_scale"),
        _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check("puro_fp8_linear_dgrad_quantize", st)


def puro_fp8_linear_wgrad(dy_t: FP8Operand, x_t: FP8Operand, dw: torch.Tensor, workspace=None, dev_status=None,
                          stream=None) -> None:
    """dW [N,K] = dY^T [N,M] . X [M,K] (operands dY^T [N,M], X^T [K,M])."""
    _gemm("puro_fp8_linear_wgrad", dy_t, x_t, dw, workspace, dev_status, stream)


def puro_fp8_linear_wgrad_main_grad(dy_t: FP8Operand, x_t: FP8Operand, main_grad: torch.Tensor, workspace=None,
                                    dev_status=None, stream=None) -> None:
    """main_grad [N,K] (FP32) += dY^T [N,M] . X [M,K]: the weight gradient
    accumulated in FP32 (operands dY^T [N,M], X^T [K,M])."""
    _gemm("puro_fp8_linear_wgrad_main_grad", dy_t, x_t, main_grad, workspace, dev_status, stream,
          out_dtype=torch.float32)


def puro_fp8_linear_wgrad_noalloc(dy_t: FP8Operand, x_t: FP8Operand, dw: torch.Tensor, dev_status=None,
                                  stream=None) -> None:
    """dW [N,K] = dY^T X without allocating and without caller scratch: for
    callers that cannot obtain device memory while running the backward
    pass.  The split-reduction scratch is a fixed 40 MiB array inside the
    library (see the header for the limits and ordering rules)."""
    ca, cb = dy_t.as_c(), x_t.as_c()
    st = load_library().puro_fp8_linear_wgrad_noalloc(ctypes.byref(ca), ctypes.byref(cb),
                                                      _ptr(dw, torch.bfloat16, "dw"),
                                                      _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check("puro_fp8_linear_wgrad_noalloc", st)


def puro_fp8_linear_backward_launches(M: int, N: int, K: int, workspace_bytes: int) -> int:
    """Kernel launches of puro_fp8_linear_backward for block-scaled operands
    (M tokens, N out, K in features) given a workspace of that many bytes."""
    return int(load_library().puro_fp8_linear_backward_launches(M, N, K, workspace_bytes))


def puro_fp8_workspace_size(rows_out: int, cols_out: int, red: int) -> int:
    return int(load_library().puro_fp8_workspace_size(rows_out, cols_out, red))


def puro_fp8_get_status(dev_status: torch.Tensor, stream=None) -> int:
    out = ctypes.c_int32(0)
    st = load_library().puro_fp8_get_status(_ptr(dev_status, torch.int32, "dev_status"), ctypes.byref(out),
                                            _stream(stream))
    _check("puro_fp8_get_status", st)
    return out.value


def _bf16(name, a, b, out, M, N, K, dev_status, stream):
    fn = getattr(load_library(), name)
    st = fn(_ptr(a, torch.bfloat16, "a"), _ptr(b, torch.bfloat16, "b"), _ptr(out, torch.bfloat16, "out"), M, N, K,
            _ptr(dev_status, torch.int32, "dev_status"), _stream(stream))
    _check(name, st)


def puro_bf16_linear_fprop(x, w, y, M, N, K, dev_status=None, stream=None) -> None:
    _bf16("puro_bf16_linear_fprop", x, w, y, M, N, K, dev_status, stream)


def puro_bf16_linear_dgrad(dy, w_t, dx, M, N, K, dev_status=None, stream=None) -> None:
    _bf16("puro_bf16_linear_dgrad", dy, w_t, dx, M, N, K, dev_status, stream)


def puro_bf16_linear_wgrad(dy_t, x_t, dw, M, N, K, dev_status=None, stream=None) -> None:
    _bf16("puro_bf16_linear_wgrad", dy_t, x_t, dw, M, N, K, dev_status, stream)


def puro_set_wait_timeout_ns(ns: int) -> None:
    load_library().puro_set_wait_timeout_ns(int(ns))


def puro_set_gemm_tile_n(tile_n: int) -> None:
    """0: per-shape choice; 224 or 256: force that block-scaled GEMM form."""
    _check("puro_set_gemm_tile_n", load_library().puro_set_gemm_tile_n(int(tile_n)))


# --------------------------------------------------------------------------
# Allocation helpers (torch allocates; the library computes)
# --------------------------------------------------------------------------
@dataclass
class Quantized:
    """Both copies produced by one quantise call."""
    rowwise: FP8Operand
    colwise: Optional[FP8Operand]
    amax: Optional[torch.Tensor] = None


def scale_vec_shape(rows: int, red: int):
    """Shape of a blockwise scale buffer for an operand [rows, red]: 512-byte
    tensor-core scale-vector chunks per 128 rows and 4 k-blocks."""
    return (rows // 128, (red // 128 + 3) // 4, 512)


def empty_scales(rows: int, red: int, scaling: int, role: int, device) -> torch.Tensor:
    if scaling == SCALE_TENSOR:
        return torch.empty(1, dtype=torch.float32, device=device)
    return torch.empty(scale_vec_shape(rows, red), dtype=torch.uint8, device=device)


def puro_fp8_scale_bytes(rows: int, red: int) -> int:
    return int(load_library().puro_fp8_scale_bytes(rows, red))


def quantize(x: torch.Tensor, fmt: int = E4M3, scaling: int = SCALE_BLOCK, role: int = ROLE_ACT,
             transpose: bool = True, out: Optional[Quantized] = None, dev_status: Optional[torch.Tensor] = None,
             stream=None) -> Quantized:
    """Quantise x [rows, cols] (bf16) into a rowwise operand [rows, cols] and,
    if ``transpose``, a columnwise operand [cols, rows]; per-tensor mode runs
    the amax kernel first."""
    rows, cols = x.shape
    dev = x.device
    if out is None:
        q = torch.empty((rows, cols), dtype=torch.uint8, device=dev)
        s = empty_scales(rows, cols, scaling, role, dev)
        colwise = None
        if transpose:
            colwise = FP8Operand(torch.empty((cols, rows), dtype=torch.uint8, device=dev),
                                 empty_scales(cols, rows, scaling, role, dev), fmt, scaling, role)
        amax = torch.zeros(1, dtype=torch.int32, device=dev) if scaling == SCALE_TENSOR else None
        out = Quantized(FP8Operand(q, s, fmt, scaling, role), colwise, amax)
    if scaling == SCALE_TENSOR:
        puro_fp8_amax(x, out.amax, stream)
    puro_fp8_quantize(x, fmt, scaling, role, out.amax if scaling == SCALE_TENSOR else None, out.rowwise.data,
                      out.rowwise.scale, out.colwise.data if out.colwise else None,
                      out.colwise.scale if out.colwise else None, dev_status=dev_status, stream=stream)
    return out


__all__ = [n for n in dir() if n.startswith("puro_")] + [
    "E4M3", "E5M2", "SCALE_TENSOR", "SCALE_BLOCK", "ROLE_ACT", "ROLE_WEIGHT", "PuroError", "FP8Operand",
    "Quantized", "quantize", "load_library", "empty_scales", "scale_vec_shape", "LIB_PATH", "HEADER_PATH",
]
