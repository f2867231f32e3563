"""Helpers shared by the GPU parity tests: run one linear layer through the
C ABI, rebuild the oracle's view of the same bytes, compare.

The oracle never sees a byte produced by the CUDA path: it quantises the
same BF16 inputs itself and forms its own fp64 products.  Layout
conversions between the oracle's natural scale grids and the library's
tensor-core scale vectors are plain index permutations.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np
import torch

import oracle as O
import paper_2608_27370_gb300 as P


# Host threads for the oracle at full size.  The oracle's ctypes calls
# release the GIL, so bands of a tensor are quantised in parallel threads;
# every quantisation group lies inside one band (bands are cut along the
# other axis, or at multiples of 128), so the result is exactly the single
# call's.
NTHREADS = max(1, min(32, os.cpu_count() or 1))


def _bands(n: int, align: int) -> list:
    """Split range(n) into about NTHREADS bands whose starts are multiples of align."""
    units = max(1, -(-n // align))
    per = max(1, -(-units // NTHREADS))
    return [(a * align, min(n, (a + per) * align)) for a in range(0, units, per)]


def par_quantize_rows_1x128(xb: np.ndarray, fmt: int):
    """O.quantize_rows_1x128 on bands of rows (each row's groups stay whole)."""
    bands = _bands(xb.shape[0], 1)
    with ThreadPoolExecutor(len(bands)) as ex:
        parts = list(ex.map(lambda b: O.quantize_rows_1x128(xb[b[0]:b[1]], fmt), bands))
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def par_quantize_cols_128x1(xb: np.ndarray, fmt: int):
    """O.quantize_cols_128x1 on bands of columns (each column's groups stay whole)."""
    bands = _bands(xb.shape[1], 1)
    with ThreadPoolExecutor(len(bands)) as ex:
        parts = list(ex.map(lambda b: O.quantize_cols_128x1(np.ascontiguousarray(xb[:, b[0]:b[1]]), fmt), bands))
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def par_quantize_blocks_128x128(wb: np.ndarray, fmt: int):
    """O.quantize_blocks_128x128 on bands of whole 128-row blocks."""
    bands = _bands(wb.shape[0], 128)
    with ThreadPoolExecutor(len(bands)) as ex:
        parts = list(ex.map(lambda b: O.quantize_blocks_128x128(wb[b[0]:b[1]], fmt), bands))
    return np.concatenate([p[0] for p in parts]), np.concatenate([p[1] for p in parts])


def par_gemm_tn(a: np.ndarray, b: np.ndarray) -> np.ndarray:
    return O.gemm_tn(a, b, NTHREADS)


def bits(t: torch.Tensor) -> np.ndarray:
    """bf16 tensor -> uint16 numpy array of its bit patterns (host copy)."""
    return t.detach().contiguous().cpu().view(torch.int16).numpy().view(np.uint16)


def host(t: torch.Tensor) -> np.ndarray:
    return t.detach().cpu().numpy()


def bf16_values(t: torch.Tensor) -> np.ndarray:
    return t.detach().float().cpu().numpy().astype(np.float64)


# --------------------------------------------------------------------------
# Running the path
# --------------------------------------------------------------------------
def run_linear(x, w, dy, scaling=P.SCALE_BLOCK, fmt_x=P.E4M3, fmt_w=P.E4M3, fmt_g=P.E4M3, step_calls=False):
    """Quantise X, W, dY (rowwise + transposed copies) and run the three GEMMs.

    With ``step_calls`` the calls are the training step's: a blockwise weight
    goes through the grouped weight quantiser (puro_fp8_quantize_weights),
    and Dgrad and Wgrad through puro_fp8_linear_backward with a workspace
    large enough for any split, so a small-output Wgrad splits its reduction
    and two unsplit block-scaled GEMMs share one launch.  Otherwise each
    operand has its own quantise call and each GEMM its own unsplit call."""
    M, K = x.shape
    N = w.shape[0]
    dev = x.device
    xq = P.quantize(x, fmt_x, scaling, P.ROLE_ACT)
    if step_calls and scaling == P.SCALE_BLOCK:
        u8 = torch.uint8
        wq = P.Quantized(
            P.FP8Operand(torch.empty((N, K), dtype=u8, device=dev), P.empty_scales(N, K, scaling, P.ROLE_WEIGHT, dev),
                         fmt_w, scaling, P.ROLE_WEIGHT),
            P.FP8Operand(torch.empty((K, N), dtype=u8, device=dev), P.empty_scales(K, N, scaling, P.ROLE_WEIGHT, dev),
                         fmt_w, scaling, P.ROLE_WEIGHT))
        P.puro_fp8_quantize_weights([(w, wq)], fmt_w)
    else:
        wq = P.quantize(w, fmt_w, scaling, P.ROLE_WEIGHT)
    dyq = P.quantize(dy, fmt_g, scaling, P.ROLE_ACT)
    y = torch.empty((M, N), dtype=torch.bfloat16, device=dev)
    dx = torch.empty((M, K), dtype=torch.bfloat16, device=dev)
    dw = torch.empty((N, K), dtype=torch.bfloat16, device=dev)
    status = torch.zeros(1, dtype=torch.int32, device=dev)
    if step_calls:
        ws = torch.empty(max(16, P.puro_fp8_workspace_size(M, N, K), P.puro_fp8_workspace_size(M, K, N),
                             P.puro_fp8_workspace_size(N, K, M)), dtype=torch.uint8, device=dev)
        P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, y, ws, dev_status=status)
        P.puro_fp8_linear_backward(dyq.rowwise, wq.colwise, dx, dyq.colwise, xq.colwise, dw, ws, dev_status=status)
    else:
        P.puro_fp8_linear_fprop(xq.rowwise, wq.rowwise, y, dev_status=status)
        P.puro_fp8_linear_dgrad(dyq.rowwise, wq.colwise, dx, dev_status=status)
        P.puro_fp8_linear_wgrad(dyq.colwise, xq.colwise, dw, dev_status=status)
    torch.cuda.synchronize()
    assert P.puro_fp8_get_status(status) == 0
    return dict(xq=xq, wq=wq, dyq=dyq, y=y, dx=dx, dw=dw)


# --------------------------------------------------------------------------
# Scale layouts: the oracle's natural per-row grid [rows, KB] <-> the
# library's tensor-core scale vectors [rows/128, ceil(KB/4), 512]
# (byte 16*l + 4*j + b of chunk (rb, kg) = row 128*rb + 32*j + l,
# k-block 4*kg + b; padding k-blocks hold 127).  Pure index permutations.
# --------------------------------------------------------------------------
def to_scale_vec(g_rows: np.ndarray) -> np.ndarray:
    rows, kb = g_rows.shape
    kg = (kb + 3) // 4
    pad = np.full((rows, kg * 4), 127, np.uint8)
    pad[:, :kb] = g_rows
    a = pad.reshape(rows // 128, 4, 32, kg, 4)           # [rb, j, l, kg, b]
    return np.ascontiguousarray(a.transpose(0, 3, 2, 1, 4).reshape(rows // 128, kg, 512))


def from_scale_vec(v: np.ndarray, kb: int) -> np.ndarray:
    rb, kg, _ = v.shape
    a = v.reshape(rb, kg, 32, 4, 4).transpose(0, 3, 2, 1, 4)  # [rb, j, l, kg, b]
    return np.ascontiguousarray(a.reshape(rb * 128, kg * 4)[:, :kb])


def scales_of(op: "P.FP8Operand") -> np.ndarray:
    """The exponents of an operand's scale vectors as a [rows, KB] grid."""
    return from_scale_vec(host(op.scale), op.red // 128)


# --------------------------------------------------------------------------
# Comparisons
# --------------------------------------------------------------------------
def assert_close(gpu: torch.Tensor, ref: np.ndarray, what: str):
    g = bf16_values(gpu)
    ok, ratio = O.within_tolerance(g, ref)
    if not ok:
        rms = float(np.sqrt(np.mean(ref * ref)))
        bound = 2.0 ** -7 * np.abs(ref) + 1e-3 * rms
        bad = np.argwhere(np.abs(g - ref) > bound)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {ref.size} outside tolerance (worst ratio {ratio:.3g}); "
                             f"first at {i}: gpu {g[i]!r} ref {ref[i]!r}")


def assert_bytes(gpu: torch.Tensor, ref: np.ndarray, what: str):
    g = host(gpu)
    assert g.shape == ref.shape, (what, g.shape, ref.shape)
    if not np.array_equal(g, ref):
        bad = np.argwhere(g != ref)
        i = tuple(bad[0])
        raise AssertionError(f"{what}: {len(bad)} of {ref.size} bytes differ; first at {i}: "
                             f"gpu {g[i]:#04x} ref {ref[i]:#04x}")


def check_block_act_quant(x: torch.Tensor, q: P.Quantized, fmt: int, rows=None, cols=None):
    """Bit-exact check of a 1x128 quantisation (rowwise + transposed copy).
    rows/cols: optional index subsets (full-size sampling)."""
    xb = bits(x if rows is None else x[rows])
    q_ref, s_ref = par_quantize_rows_1x128(xb, fmt)
    qr = q.rowwise.data if rows is None else q.rowwise.data[rows]
    assert_bytes(qr, q_ref, "rowwise codes")
    if rows is None:  # the whole buffer, padding bytes included
        assert_bytes(q.rowwise.scale, to_scale_vec(s_ref), "rowwise scale vectors")
    else:
        assert np.array_equal(scales_of(q.rowwise)[host(rows)], s_ref), "rowwise scales (sampled rows)"
    if q.colwise is None:
        return
    xc = xb if (rows is None and cols is None) else bits(x if cols is None else x[:, cols])
    qt_ref, st_ref = par_quantize_cols_128x1(xc, fmt)
    qc = q.colwise.data if cols is None else q.colwise.data[cols]
    assert_bytes(qc, qt_ref, "transposed codes")
    if cols is None:
        assert_bytes(q.colwise.scale, to_scale_vec(st_ref), "transposed scale vectors")
    else:
        assert np.array_equal(scales_of(q.colwise)[host(cols)], st_ref), "transposed scales (sampled columns)"


def check_block_weight_quant(w: torch.Tensor, q: P.Quantized, fmt: int):
    q_ref, s_ref = par_quantize_blocks_128x128(bits(w), fmt)
    assert_bytes(q.rowwise.data, q_ref, "weight codes")
    assert_bytes(q.rowwise.scale, to_scale_vec(np.repeat(s_ref, 128, axis=0)), "weight scale vectors")
    if q.colwise is not None:
        assert_bytes(q.colwise.data, np.ascontiguousarray(q_ref.T), "transposed weight codes")
        assert_bytes(q.colwise.scale, to_scale_vec(np.repeat(np.ascontiguousarray(s_ref.T), 128, axis=0)),
                     "transposed weight scale vectors")


def check_tensor_quant(x: torch.Tensor, q: P.Quantized, fmt: int):
    amax, q_ref, si_ref = O.quantize_tensor(bits(x), fmt)
    got_amax = int(host(q.amax)[0]) & 0xFFFF
    assert got_amax == amax, f"amax {got_amax:#06x} != {amax:#06x}"
    assert_bytes(q.rowwise.data, q_ref, "tensor-scaled codes")
    got_si = host(q.rowwise.scale)[0]
    assert np.float32(got_si).tobytes() == np.float32(si_ref).tobytes(), (got_si, si_ref)
    if q.colwise is not None:
        assert_bytes(q.colwise.data, np.ascontiguousarray(q_ref.T), "transposed tensor-scaled codes")
        assert np.float32(host(q.colwise.scale)[0]).tobytes() == np.float32(si_ref).tobytes()


def oracle_linear(x, w, dy, scaling, fmt_x=P.E4M3, fmt_w=P.E4M3, fmt_g=P.E4M3, nthreads=8):
    xb, wb, dyb = bits(x), bits(w), bits(dy)
    if scaling == P.SCALE_BLOCK:
        return O.linear_block(xb, wb, dyb, fmt_x, fmt_w, fmt_g, nthreads)
    return O.linear_tensor(xb, wb, dyb, fmt_x, fmt_w, fmt_g, nthreads)


# --------------------------------------------------------------------------
# Full-size sampling (blockwise recipe)
# --------------------------------------------------------------------------
def sample_index(n: int, k_rand: int, rng: np.random.Generator) -> np.ndarray:
    """First 128, last 128 and k_rand random indices of range(n), sorted, unique."""
    edge = min(128, n)
    idx = np.concatenate([np.arange(edge), np.arange(n - edge, n), rng.choice(n, size=min(k_rand, n), replace=False)])
    return np.unique(idx)


def check_linear_sampled(x, w, dy, out, rng, k_rand=96, fmt=P.E4M3, full_bytes=False):
    """Blockwise recipe at full size.

    Quantised bytes: with ``full_bytes`` every FP8 byte and scale of X, W and
    dY (both copies) against the oracle; otherwise W in full and X, dY on
    sampled rows and columns (the first and last 128 and k_rand random ones).
    GEMM outputs: the cross product of sampled rows and columns of each
    output -- the first 128, the last 128 and k_rand random indices of each
    dimension -- which holds the four complete corner 128x128 tiles and
    k_rand^2 seeded random (m, n) entries (9216 at the default 96), against
    the oracle's fp64 products of the same operands."""
    M, K = x.shape
    N = w.shape[0]
    Ms = sample_index(M, k_rand, rng)
    Ns = sample_index(N, k_rand, rng)
    Ks = sample_index(K, k_rand, rng)
    Ms_t, Ns_t, Ks_t = (torch.from_numpy(a).to(x.device) for a in (Ms, Ns, Ks))

    # quantised operands
    if full_bytes:
        check_block_act_quant(x, out["xq"], fmt)
        check_block_act_quant(dy, out["dyq"], fmt)
    else:
        check_block_act_quant(x, out["xq"], fmt, rows=Ms_t, cols=Ks_t)
        check_block_act_quant(dy, out["dyq"], fmt, rows=Ms_t, cols=Ns_t)
    check_block_weight_quant(w, out["wq"], fmt)

    # oracle operands for the sampled products
    xr_q, xr_s = O.quantize_rows_1x128(bits(x[Ms_t]), fmt)            # X rows (groups along K)
    X_rows = O.dequant_rows_1x128(xr_q, xr_s, fmt)
    dyr_q, dyr_s = O.quantize_rows_1x128(bits(dy[Ms_t]), fmt)         # dY rows (groups along N)
    dY_rows = O.dequant_rows_1x128(dyr_q, dyr_s, fmt)
    wq, ws = par_quantize_blocks_128x128(bits(w), fmt)                # W blocks
    W = O.dequant_blocks_128x128(wq, ws, fmt)
    xc_q, xc_s = par_quantize_cols_128x1(bits(x[:, Ks_t]), fmt)       # X columns (groups along M)
    Xt_rows = O.dequant_rows_1x128(xc_q, xc_s, fmt)
    dyc_q, dyc_s = par_quantize_cols_128x1(bits(dy[:, Ns_t]), fmt)    # dY columns (groups along M)
    dYt_rows = O.dequant_rows_1x128(dyc_q, dyc_s, fmt)

    y_ref = par_gemm_tn(X_rows, W[Ns])                                 # Y[Ms, Ns]
    dx_ref = par_gemm_tn(dY_rows, np.ascontiguousarray(W.T[Ks]))       # dX[Ms, Ks]
    dw_ref = par_gemm_tn(dYt_rows, Xt_rows)                            # dW[Ns, Ks]
    assert_close(out["y"][Ms_t][:, Ns_t], y_ref, "fprop (sampled)")
    assert_close(out["dx"][Ms_t][:, Ks_t], dx_ref, "dgrad (sampled)")
    assert_close(out["dw"][Ns_t][:, Ks_t], dw_ref, "wgrad (sampled)")


# --------------------------------------------------------------------------
# Output coverage of a persistent GEMM: one sampled index in every 32
# consecutive rows / columns, so the cross product meets every 32 x 32 piece
# of every output tile (each epilogue warp's lane quarter and column chunk,
# both CTAs of a pair, both accumulator buffers).
# --------------------------------------------------------------------------
def sample_every(n: int, rng: np.random.Generator, group: int = 32) -> np.ndarray:
    """One random index in each run of `group` consecutive indices of range(n)
    (the last run may be short), plus the first and last index."""
    starts = np.arange(0, n, group)
    picks = starts + rng.integers(0, np.minimum(group, n - starts))
    return np.unique(np.concatenate([picks, [0, n - 1]]))


def check_gemm_every_tile(out: torch.Tensor, a: np.ndarray, b: np.ndarray, rng: np.random.Generator, what: str):
    """out [M, N] (bf16, device) against the fp64 product a[rows] . b[cols]^T
    on the cross product of sample_every rows and columns; a [M, K] and b
    [N, K] are the oracle's dequantised operands (fp64)."""
    rows = sample_every(out.shape[0], rng)
    cols = sample_every(out.shape[1], rng)
    ref = par_gemm_tn(np.ascontiguousarray(a[rows]), np.ascontiguousarray(b[cols]))
    r_t, c_t = (torch.from_numpy(v).to(out.device) for v in (rows, cols))
    assert_close(out[r_t][:, c_t], ref, what)
