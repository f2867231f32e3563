"""Pins for the oracle's three GEMMs (Fprop, Dgrad, Wgrad).

Pinned against: exact rational brute force in the block-factored form
sum_kb s_a s_b sum_k q_a q_b (Python Fractions, pure loops), the identity
Fprop(dY, W^T) == Dgrad(dY, W) bit for bit, Wgrad(A, B) == Wgrad(B, A)^T,
and an exact-integer special case compared with numpy's int64 matmul.
"""
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as O


def bf16_bits(a):
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _inputs(M, N, K, seed):
    g = np.random.default_rng(seed)
    x = bf16_bits(g.standard_normal((M, K)))
    w = bf16_bits(g.standard_normal((N, K)) * 0.02)
    dy = bf16_bits(g.standard_normal((M, N)) * 1e-3)
    return x, w, dy


def _frac_code(c, fmt):
    v = float(O.decode(np.array([c], np.uint8), fmt)[0])
    return None if not np.isfinite(v) else Fraction(v)


def test_fprop_exact_bruteforce_block_factored():
    M, N, K = 128, 256, 256
    x, w, dy = _inputs(M, N, K, 11)
    r = O.linear_block(x, w, dy)
    tbl = [_frac_code(c, O.E4M3) for c in range(256)]
    rng = np.random.default_rng(0)
    for _ in range(6):
        m, n = int(rng.integers(M)), int(rng.integers(N))
        total = Fraction(0)
        for kb in range(K // 128):
            sa = Fraction(2) ** (int(r["xs"][m, kb]) - 127)
            sb = Fraction(2) ** (int(r["ws"][n // 128, kb]) - 127)
            inner = Fraction(0)
            for k in range(kb * 128, kb * 128 + 128):
                inner += tbl[r["xq"][m, k]] * tbl[r["wq"][n, k]]
            total += sa * sb * inner
        exact = float(total)
        assert abs(r["y"][m, n] - exact) <= 1e-13 * max(abs(exact), 1e-30) + 1e-300


def test_wgrad_exact_bruteforce():
    M, N, K = 256, 128, 128
    x, w, dy = _inputs(M, N, K, 12)
    r = O.linear_block(x, w, dy)
    tbl = [_frac_code(c, O.E4M3) for c in range(256)]
    rng = np.random.default_rng(1)
    for _ in range(4):
        n, k = int(rng.integers(N)), int(rng.integers(K))
        total = Fraction(0)
        for mb in range(M // 128):
            sa = Fraction(2) ** (int(r["dyst"][n, mb]) - 127)
            sb = Fraction(2) ** (int(r["xst"][k, mb]) - 127)
            inner = sum((tbl[r["dyqt"][n, m]] * tbl[r["xqt"][k, m]] for m in range(mb * 128, mb * 128 + 128)), Fraction(0))
            total += sa * sb * inner
        assert abs(r["dw"][n, k] - float(total)) <= 1e-13 * abs(float(total)) + 1e-300


def test_dgrad_exact_bruteforce():
    M, N, K = 128, 256, 128
    x, w, dy = _inputs(M, N, K, 13)
    r = O.linear_block(x, w, dy)
    tbl = [_frac_code(c, O.E4M3) for c in range(256)]
    for m, k in [(0, 0), (127, 127), (64, 5)]:
        total = Fraction(0)
        for nb in range(N // 128):
            sa = Fraction(2) ** (int(r["dys"][m, nb]) - 127)
            sb = Fraction(2) ** (int(r["ws"][nb, k // 128]) - 127)
            inner = sum((tbl[r["dyq"][m, n]] * tbl[r["wq"][n, k]] for n in range(nb * 128, nb * 128 + 128)), Fraction(0))
            total += sa * sb * inner
        assert abs(r["dx"][m, k] - float(total)) <= 1e-13 * abs(float(total)) + 1e-300


def test_fprop_of_transposed_weight_is_dgrad():
    M, N, K = 256, 384, 256
    x, w, dy = _inputs(M, N, K, 21)
    r = O.linear_block(x, w, dy)
    wt = np.ascontiguousarray(w.T)          # [K, N] as a weight of a linear N -> K
    r2 = O.linear_block(dy, wt, np.zeros((M, K), np.uint16))
    assert np.array_equal(r2["y"], r["dx"])


def test_wgrad_swap_is_transpose():
    M, N, K = 256, 128, 256
    x, w, dy = _inputs(M, N, K, 22)
    r = O.linear_block(x, w, dy)
    # swap the roles of dY and X: the Wgrad of a linear with input dY and output-gradient X
    r2 = O.linear_block(dy, np.zeros((K, N), np.uint16), x)
    assert np.array_equal(r2["dw"], r["dw"].T)


def test_exact_integer_operands_against_numpy():
    """E4M3 values that are small integers, with group max 256 so every
    scale is 1: the fp64 sums are exact and equal an integer matmul."""
    rng = np.random.default_rng(7)
    M, N, K = 128, 256, 384
    xa = rng.integers(-16, 17, (M, K)).astype(np.int64)
    wa = rng.integers(-16, 17, (N, K)).astype(np.int64)
    xa[:, ::128] = 256
    wa[::128, ::128] = 256
    wa[::128, 1::128] = -256
    xq, xs = O.quantize_rows_1x128(bf16_bits(xa), O.E4M3)
    wq, ws = O.quantize_blocks_128x128(bf16_bits(wa), O.E4M3)
    assert np.all(xs == 127) and np.all(ws == 127)
    y = O.gemm_tn(O.dequant_rows_1x128(xq, xs, O.E4M3), O.dequant_blocks_128x128(wq, ws, O.E4M3))
    assert np.array_equal(y, (xa @ wa.T).astype(np.float64))


def test_tensor_mode_gemm_bruteforce():
    M, N, K = 64, 48, 80
    x, w, dy = _inputs(M, N, K, 31)
    r = O.linear_tensor(x, w, dy)
    tbl = [_frac_code(c, O.E4M3) for c in range(256)]
    sx, sw, sg = Fraction(r["x_si"]), Fraction(r["w_si"]), Fraction(r["dy_si"])
    for m, n in [(0, 0), (63, 47), (10, 20)]:
        exact = sx * sw * sum((tbl[r["xq"][m, k]] * tbl[r["wq"][n, k]] for k in range(K)), Fraction(0))
        assert abs(r["y"][m, n] - float(exact)) <= 1e-13 * abs(float(exact))
    for m, k in [(3, 5), (60, 79)]:
        exact = sg * sw * sum((tbl[r["dyq"][m, n]] * tbl[r["wq"][n, k]] for n in range(N)), Fraction(0))
        assert abs(r["dx"][m, k] - float(exact)) <= 1e-13 * abs(float(exact))
    for n, k in [(1, 2), (47, 79)]:
        exact = sg * sx * sum((tbl[r["dyq"][m, n]] * tbl[r["xq"][m, k]] for m in range(M)), Fraction(0))
        assert abs(r["dw"][n, k] - float(exact)) <= 1e-13 * abs(float(exact))


def test_dot_pairs_and_threads_agree_with_full_gemm():
    rng = np.random.default_rng(9)
    a = rng.standard_normal((37, 129))
    b = rng.standard_normal((23, 129))
    full1 = O.gemm_tn(a, b, 1)
    full4 = O.gemm_tn(a, b, 4)
    assert np.array_equal(full1, full4)
    ai = rng.integers(0, 37, 50)
    bi = rng.integers(0, 23, 50)
    assert np.array_equal(O.dot_pairs(a, b, ai, bi), full1[ai, bi])


def test_tolerance_rule():
    ref = np.array([1.0, -2.0, 0.0, 1e-6])
    ok, _ = O.within_tolerance(ref * (1 + 2 ** -8), ref)
    assert ok
    ok, _ = O.within_tolerance(ref * (1 + 2 ** -5), ref)
    assert not ok
