"""CPU oracle for the FP8 linear training path (Puro-2B).

TEST INFRASTRUCTURE ONLY.  This package is imported by the test suite, by
``__graft_entry__.smoke()`` and by the CPU-baseline leg of ``bench.py``;
the product library never loads it and shares no code with it.

The arithmetic lives in ``puro_oracle.c`` (plain C, fp64, IEEE round to
nearest even).  This module only builds it with gcc, loads it with ctypes
and moves numpy arrays in and out.  The definitions it follows are those of
the paper's section "FP8 Mixed-Precision Training" (E4M3 operands, 1x128
groups along the reduction dimension for activations and activation
gradients, 128x128 blocks for weights, power-of-two scales) and of the
appendix paragraph "FP8 implementation pipeline" (Fprop, Dgrad and Wgrad all
from FP8 operands, BF16 output).  Layouts here are the natural ones:
row-major tensors, row-major scale grids.

Parity pins: every function here is pinned by ``tests/test_oracle_*.py``
against closed forms, exhaustive enumerations, brute force and library
routines; none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess

import numpy as np

E4M3 = 0
E5M2 = 1
FMT_MAX = {E4M3: 448.0, E5M2: 57344.0}

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "puro_oracle.c")
_SO = os.path.join(_HERE, "libpuro_oracle.so")
_lib = None


def build(force: bool = False) -> str:
    """Compile the oracle into ``oracle/libpuro_oracle.so`` (gcc, no fast-math)."""
    if force or not os.path.exists(_SO) or os.path.getmtime(_SO) < os.path.getmtime(_SRC):
        tmp = _SO + ".tmp.%d" % os.getpid()
        cmd = ["gcc", "-std=c11", "-O2", "-ffp-contract=off", "-fno-fast-math", "-fPIC",
               "-shared", "-pthread", _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _SO)
    return _SO


def _load():
    global _lib
    if _lib is not None:
        return _lib
    build()
    lib = ctypes.CDLL(_SO)
    P = ctypes.c_void_p
    I64 = ctypes.c_int64
    I = ctypes.c_int
    sig = {
        "oracle_fmt_max": (ctypes.c_double, [I]),
        "oracle_fp8_decode": (ctypes.c_double, [ctypes.c_uint8, I]),
        "oracle_fp8_encode": (ctypes.c_uint8, [ctypes.c_double, I]),
        "oracle_bf16_from_double": (ctypes.c_uint16, [ctypes.c_double]),
        "oracle_amax_bf16": (ctypes.c_uint16, [P, I64]),
        "oracle_e8m0_from_amax": (ctypes.c_uint8, [ctypes.c_uint16, I]),
        "oracle_quantize_rows_1x128": (None, [P, I64, I64, I, P, P]),
        "oracle_quantize_blocks_128x128": (None, [P, I64, I64, I, P, P]),
        "oracle_quantize_tensor": (None, [P, I64, I, ctypes.c_uint16, P, P]),
        "oracle_dequant_rows_1x128": (None, [P, P, I64, I64, I, P]),
        "oracle_dequant_blocks_128x128": (None, [P, P, I64, I64, I, P]),
        "oracle_dequant_tensor": (None, [P, I64, I, ctypes.c_float, P]),
        "oracle_bf16_to_double": (None, [P, I64, P]),
        "oracle_gemm_tn": (I, [P, P, I64, I64, I64, P, I]),
        "oracle_dot_pairs": (None, [P, P, I64, P, P, I64, P]),
        "oracle_fp8_decode_array": (None, [P, I64, I, P]),
        "oracle_fp8_encode_array": (None, [P, I64, I, P]),
        "oracle_bf16_from_double_array": (None, [P, I64, P]),
        "oracle_e8m0_from_amax_array": (None, [P, I64, I, P]),
        "oracle_rmsnorm_rstd": (None, [P, I64, I64, ctypes.c_double, P]),
        "oracle_rmsnorm_apply_f32": (None, [P, I64, I64, P, P, P]),
        "oracle_swiglu": (None, [P, P, I64, I64, I64, P]),
        "oracle_frobenius_norm": (ctypes.c_double, [P, I64]),
        "oracle_muonh_step": (None, [P, P, I64, ctypes.c_double, ctypes.c_double, P]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def _p(a: np.ndarray):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.c_void_p)


def _bits(x) -> np.ndarray:
    """bf16 bit patterns as a contiguous uint16 array (accepts uint16/int16 arrays)."""
    a = np.ascontiguousarray(x)
    if a.dtype == np.int16:
        a = a.view(np.uint16)
    assert a.dtype == np.uint16, a.dtype
    return a


# --------------------------------------------------------------------------
# codec
# --------------------------------------------------------------------------
def decode(codes, fmt: int) -> np.ndarray:
    c = np.ascontiguousarray(codes, dtype=np.uint8)
    out = np.empty(c.shape, np.float64)
    _load().oracle_fp8_decode_array(_p(c), c.size, fmt, _p(out))
    return out


def encode(values, fmt: int) -> np.ndarray:
    v = np.ascontiguousarray(values, dtype=np.float64)
    out = np.empty(v.shape, np.uint8)
    _load().oracle_fp8_encode_array(_p(v), v.size, fmt, _p(out))
    return out


def bf16_from_double(values) -> np.ndarray:
    v = np.ascontiguousarray(values, dtype=np.float64)
    out = np.empty(v.shape, np.uint16)
    _load().oracle_bf16_from_double_array(_p(v), v.size, _p(out))
    return out


def bf16_to_double(bits) -> np.ndarray:
    b = _bits(bits)
    out = np.empty(b.shape, np.float64)
    _load().oracle_bf16_to_double(_p(b), b.size, _p(out))
    return out


def fmt_max(fmt: int) -> float:
    return _load().oracle_fmt_max(fmt)


# --------------------------------------------------------------------------
# amax and group scales
# --------------------------------------------------------------------------
def amax_bf16(x) -> int:
    b = _bits(x)
    return int(_load().oracle_amax_bf16(_p(b), b.size))


def e8m0_from_amax(amax_bits, fmt: int):
    if np.isscalar(amax_bits):
        return int(_load().oracle_e8m0_from_amax(int(amax_bits), fmt))
    a = np.ascontiguousarray(amax_bits, dtype=np.uint16)
    out = np.empty(a.shape, np.uint8)
    _load().oracle_e8m0_from_amax_array(_p(a), a.size, fmt, _p(out))
    return out


# --------------------------------------------------------------------------
# quantisation (natural layouts)
# --------------------------------------------------------------------------
def quantize_rows_1x128(x, fmt: int):
    """1x128 groups along each row. Returns (q [R,C] u8, s [R, C/128] u8)."""
    b = _bits(x)
    R, C = b.shape
    assert C % 128 == 0
    q = np.empty((R, C), np.uint8)
    s = np.empty((R, C // 128), np.uint8)
    _load().oracle_quantize_rows_1x128(_p(b), R, C, fmt, _p(q), _p(s))
    return q, s


def quantize_cols_128x1(x, fmt: int):
    """128x1 groups down each column, stored transposed: the rowwise rule
    applied to x^T.  Returns (q_t [C,R] u8, s_t [C, R/128] u8)."""
    return quantize_rows_1x128(np.ascontiguousarray(_bits(x).T), fmt)


def quantize_blocks_128x128(x, fmt: int):
    """128x128 blocks. Returns (q [R,C] u8, s [R/128, C/128] u8)."""
    b = _bits(x)
    R, C = b.shape
    assert R % 128 == 0 and C % 128 == 0
    q = np.empty((R, C), np.uint8)
    s = np.empty((R // 128, C // 128), np.uint8)
    _load().oracle_quantize_blocks_128x128(_p(b), R, C, fmt, _p(q), _p(s))
    return q, s


def quantize_tensor(x, fmt: int, amax_bits: int | None = None):
    """Per-tensor current scaling. Returns (amax_bits, q u8 same shape, scale_inv fp32)."""
    b = _bits(x)
    if amax_bits is None:
        amax_bits = amax_bf16(b)
    q = np.empty(b.shape, np.uint8)
    si = np.zeros(1, np.float32)
    _load().oracle_quantize_tensor(_p(b), b.size, fmt, int(amax_bits), _p(q), _p(si))
    return int(amax_bits), q, float(si[0])


def dequant_rows_1x128(q, s, fmt: int) -> np.ndarray:
    q = np.ascontiguousarray(q, np.uint8)
    s = np.ascontiguousarray(s, np.uint8)
    R, C = q.shape
    out = np.empty((R, C), np.float64)
    _load().oracle_dequant_rows_1x128(_p(q), _p(s), R, C, fmt, _p(out))
    return out


def dequant_blocks_128x128(q, s, fmt: int) -> np.ndarray:
    q = np.ascontiguousarray(q, np.uint8)
    s = np.ascontiguousarray(s, np.uint8)
    R, C = q.shape
    out = np.empty((R, C), np.float64)
    _load().oracle_dequant_blocks_128x128(_p(q), _p(s), R, C, fmt, _p(out))
    return out


def dequant_tensor(q, scale_inv: float, fmt: int) -> np.ndarray:
    q = np.ascontiguousarray(q, np.uint8)
    out = np.empty(q.shape, np.float64)
    _load().oracle_dequant_tensor(_p(q), q.size, fmt, ctypes.c_float(scale_inv), _p(out))
    return out


# --------------------------------------------------------------------------
# GEMM
# --------------------------------------------------------------------------
def gemm_tn(a, b, nthreads: int = 1) -> np.ndarray:
    """out[m, n] = sum_k a[m, k] * b[n, k] in fp64 (plain k order)."""
    a = np.ascontiguousarray(a, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    M, K = a.shape
    N, K2 = b.shape
    assert K == K2
    out = np.empty((M, N), np.float64)
    rc = _load().oracle_gemm_tn(_p(a), _p(b), M, N, K, _p(out), int(nthreads))
    if rc != 0:
        raise MemoryError("oracle_gemm_tn failed")
    return out


def dot_pairs(a, b, ai, bi) -> np.ndarray:
    """out[i] = sum_k a[ai[i], k] * b[bi[i], k] in fp64."""
    a = np.ascontiguousarray(a, np.float64)
    b = np.ascontiguousarray(b, np.float64)
    ai = np.ascontiguousarray(ai, np.int64)
    bi = np.ascontiguousarray(bi, np.int64)
    assert a.shape[1] == b.shape[1] and ai.shape == bi.shape
    out = np.empty(ai.shape, np.float64)
    _load().oracle_dot_pairs(_p(a), _p(b), a.shape[1], _p(ai), _p(bi), ai.size, _p(out))
    return out


# --------------------------------------------------------------------------
# One linear layer, fully, in the paper's recipe (small sizes)
# --------------------------------------------------------------------------
def linear_block(x, w, dy, fmt_x: int = E4M3, fmt_w: int = E4M3, fmt_g: int = E4M3,
                 nthreads: int = 1):
    """Blockwise recipe for one linear: X [M,K], W [N,K], dY [M,N] (bf16 bits).

    Quantise X rowwise (groups along K, for Fprop) and columnwise (groups
    along M, for Wgrad); W in 128x128 blocks (W^T shares the block scales);
    dY rowwise (groups along N, for Dgrad) and columnwise (groups along M,
    for Wgrad).  Returns the quantised tensors and the fp64 GEMM results.
    """
    xq, xs = quantize_rows_1x128(x, fmt_x)
    xqt, xst = quantize_cols_128x1(x, fmt_x)
    wq, ws = quantize_blocks_128x128(w, fmt_w)
    dyq, dys = quantize_rows_1x128(dy, fmt_g)
    dyqt, dyst = quantize_cols_128x1(dy, fmt_g)
    X = dequant_rows_1x128(xq, xs, fmt_x)
    Xt = dequant_rows_1x128(xqt, xst, fmt_x)
    W = dequant_blocks_128x128(wq, ws, fmt_w)
    Wt = np.ascontiguousarray(W.T)
    dY = dequant_rows_1x128(dyq, dys, fmt_g)
    dYt = dequant_rows_1x128(dyqt, dyst, fmt_g)
    return dict(
        xq=xq, xs=xs, xqt=xqt, xst=xst, wq=wq, ws=ws, dyq=dyq, dys=dys, dyqt=dyqt, dyst=dyst,
        y=gemm_tn(X, W, nthreads), dx=gemm_tn(dY, Wt, nthreads), dw=gemm_tn(dYt, Xt, nthreads),
    )


def linear_tensor(x, w, dy, fmt_x: int = E4M3, fmt_w: int = E4M3, fmt_g: int = E4M3,
                  nthreads: int = 1):
    """Per-tensor recipe for one linear (one scale per tensor; the transposed
    copy of each operand carries the same codes, transposed)."""
    ax, xq, xsi = quantize_tensor(x, fmt_x)
    aw, wq, wsi = quantize_tensor(w, fmt_w)
    ag, dyq, dysi = quantize_tensor(dy, fmt_g)
    X = dequant_tensor(xq, xsi, fmt_x)
    W = dequant_tensor(wq, wsi, fmt_w)
    dY = dequant_tensor(dyq, dysi, fmt_g)
    return dict(
        amax_x=ax, amax_w=aw, amax_dy=ag, xq=xq, wq=wq, dyq=dyq, x_si=xsi, w_si=wsi, dy_si=dysi,
        y=gemm_tn(X, W, nthreads), dx=gemm_tn(dY, np.ascontiguousarray(W.T), nthreads),
        dw=gemm_tn(np.ascontiguousarray(dY.T), np.ascontiguousarray(X.T), nthreads),
    )


def rmsnorm_rstd(h, eps: float) -> np.ndarray:
    """Per-row 1/sqrt(mean(h^2) + eps) of a bf16 [rows, cols] matrix, fp64."""
    hb = np.ascontiguousarray(_bits(h))
    rows, cols = hb.shape
    out = np.empty(rows, np.float64)
    _load().oracle_rmsnorm_rstd(_p(hb), rows, cols, ctypes.c_double(eps), _p(out))
    return out


def rmsnorm_apply_f32(h, rstd_f32, gamma=None) -> np.ndarray:
    """bf16 bits of (h * rstd) * gamma in fp32 (gamma None: no gain)."""
    hb = np.ascontiguousarray(_bits(h))
    rows, cols = hb.shape
    r = np.ascontiguousarray(np.asarray(rstd_f32, np.float32))
    assert r.shape == (rows,)
    g = None if gamma is None else np.ascontiguousarray(_bits(gamma))
    out = np.empty((rows, cols), np.uint16)
    _load().oracle_rmsnorm_apply_f32(_p(hb), rows, cols, _p(r), None if g is None else _p(g), _p(out))
    return out


def swiglu(g, u) -> np.ndarray:
    """bf16 bits of silu(g) * u (fp64, one rounding) for bf16 [rows, cols]
    matrices g and u.  Row-strided views (e.g. the two halves of one
    [rows, 2 cols] array) are passed with their row stride, not copied."""
    gb, ub = _bits(g), _bits(u)
    assert gb.shape == ub.shape and gb.ndim == 2
    rows, cols = gb.shape

    def strided(a):
        if a.strides[1] == 2 and a.strides[0] % 2 == 0 and a.strides[0] >= 2 * cols:
            return a, a.strides[0] // 2
        a = np.ascontiguousarray(a)
        return a, cols

    gb, ldg = strided(gb)
    ub, ldu = strided(ub)
    if ldg != ldu:
        gb, ub, ldg = np.ascontiguousarray(gb), np.ascontiguousarray(ub), cols
    out = np.empty((rows, cols), np.uint16)
    if rows and cols:
        _load().oracle_swiglu(ctypes.c_void_p(gb.ctypes.data), ctypes.c_void_p(ub.ctypes.data), rows, cols, ldg,
                              _p(out))
    return out


def frobenius_norm(x) -> float:
    """||x||_F of an fp32 array (any shape), accumulated in fp64."""
    a = np.ascontiguousarray(np.asarray(x, np.float32))
    return float(_load().oracle_frobenius_norm(_p(a), a.size))


def muonh_step(w, u, eta: float, radius: float) -> np.ndarray:
    """The hyperball update of fp32 W along the Muon direction u (same
    shape): R W~ / ||W~||_F with W~ = W - eta R u / ||u||_F, in fp64."""
    wa = np.ascontiguousarray(np.asarray(w, np.float32))
    ua = np.ascontiguousarray(np.asarray(u, np.float32))
    assert wa.shape == ua.shape
    out = np.empty(wa.shape, np.float64)
    _load().oracle_muonh_step(_p(wa), _p(ua), wa.size, ctypes.c_double(eta), ctypes.c_double(radius), _p(out))
    return out


def within_tolerance(gpu, ref):
    """The acceptance rule for BF16 GEMM outputs against the fp64 result:
    |gpu - ref| <= 2^-7 |ref| + 1e-3 rms(ref).  Returns (ok, worst ratio)."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    rms = float(np.sqrt(np.mean(ref * ref))) if ref.size else 0.0
    bound = 2.0 ** -7 * np.abs(ref) + 1e-3 * rms
    err = np.abs(gpu - ref)
    ratio = float(np.max(err / np.maximum(bound, 1e-300))) if ref.size else 0.0
    return bool(np.all(err <= bound)), ratio
