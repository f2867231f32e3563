"""Pins for the oracle's amax, power-of-two group scale and quantisers.

Pinned against: an independent closed form of the scale exponent taken from
the bf16 bit fields (all 32768 magnitudes, both formats), the invariant that
a group's largest code lies in (max/2, max], the quantise-dequantise error
bound, numpy's max on finite data, torch's float8 cast for the per-tensor
rule (library routine), transposition symmetry of 128x128 blocks, and
exact-value special cases.
"""
import numpy as np
import pytest
import torch

import oracle as O

FMTS = [O.E4M3, O.E5M2]
# exponent of fmt_max's binade: 448 = 1.75 * 2^8, 57344 = 1.75 * 2^15
MAX_EXP = {O.E4M3: 8, O.E5M2: 15}


def bf16_bits(a: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(a, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def closed_form_g(bits: int, fmt: int) -> int:
    """Integer rule from the bf16 fields: amax = 1.m * 2^e with e = E - 127
    (normal) -> smallest k with amax <= 1.75 * 2^(M+k) is k = e - M if
    1.m <= 1.75 (m <= 96/128) else e - M + 1; bf16 subnormals and tiny
    normals clamp at g = 0."""
    E = bits >> 7
    mant = bits & 0x7F
    if bits == 0:
        return 127
    if E == 0xFF:
        return 0xFF
    if E == 0:
        return 0
    g = E - MAX_EXP[fmt] + (1 if mant > 96 else 0)
    return min(max(g, 0), 254)


@pytest.mark.parametrize("fmt", FMTS)
def test_e8m0_closed_form_all_magnitudes(fmt):
    bits = np.arange(0, 0x8000, dtype=np.uint16)
    got = O.e8m0_from_amax(bits, fmt)
    want = np.array([closed_form_g(int(b), fmt) for b in bits], np.uint8)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("fmt", FMTS)
def test_e8m0_is_smallest_pow2_and_group_max_in_top_binade(fmt):
    bits = np.arange(1, 0x7F80, dtype=np.uint16)
    g = O.e8m0_from_amax(bits, fmt).astype(np.int64)
    a = O.bf16_to_double(bits)
    mx = O.fmt_max(fmt)
    s = 2.0 ** (g - 127)
    unclamped = g > 0
    assert np.all(a[unclamped] / s[unclamped] <= mx)
    assert np.all(a[unclamped] / s[unclamped] > mx / 2)     # one exponent smaller would saturate
    assert np.all(a[~unclamped] <= mx * 2.0 ** -127)          # clamped only when below the range
    # the encoded group maximum lands in [max/2, max]
    top = O.decode(O.encode(a[unclamped] / s[unclamped], fmt), fmt)
    assert np.all((top >= mx / 2) & (top <= mx))


def test_amax_matches_numpy_and_propagates_nonfinite():
    rng = np.random.default_rng(0)
    x = rng.standard_t(3, 100_000).astype(np.float32) * 3
    b = bf16_bits(x)
    ref = np.max(np.abs(O.bf16_to_double(b)))
    assert O.bf16_to_double(np.array([O.amax_bf16(b)], np.uint16))[0] == ref
    b2 = b.copy(); b2[777] = 0xFF80  # -inf
    assert O.amax_bf16(b2) == 0x7F80
    b3 = b2.copy(); b3[5] = 0x7FC1   # NaN beats inf
    assert O.amax_bf16(b3) > 0x7F80
    assert O.amax_bf16(np.zeros(10, np.uint16)) == 0
    assert O.amax_bf16(np.array([0x8000], np.uint16)) == 0  # -0


def _bound_check(x_bits, q, g_full, fmt):
    x = O.bf16_to_double(x_bits)
    s = 2.0 ** (g_full.astype(np.int64) - 127)
    v = O.decode(q, fmt) * s
    emin = 1 - (7 if fmt == O.E4M3 else 15)
    mb = 3 if fmt == O.E4M3 else 2
    y = np.abs(x) / s
    e = np.floor(np.log2(np.maximum(y, 2.0 ** emin)))
    half_ulp = 2.0 ** (e - mb - 1)  # half the spacing at |x|/s, subnormals included
    assert np.all(np.abs(x - v) <= s * half_ulp)


@pytest.mark.parametrize("fmt", FMTS)
def test_rows_1x128_error_bound_and_layout(fmt):
    rng = np.random.default_rng(3)
    x = rng.standard_t(3, (256, 512)).astype(np.float32)
    x[:, 7] *= 50.0  # outlier channel
    x[5, 128:256] = 0.0  # a zero group
    b = bf16_bits(x)
    q, s = O.quantize_rows_1x128(b, fmt)
    assert q.shape == (256, 512) and s.shape == (256, 4)
    assert s[5, 1] == 127 and np.all((q[5, 128:256] == 0) | (q[5, 128:256] == 0x80))
    g_full = np.repeat(s, 128, axis=1)
    _bound_check(b, q, g_full, fmt)
    # scale of each group is the closed form of that group's amax
    for r in (0, 5, 100):
        for gi in range(4):
            assert s[r, gi] == closed_form_g(O.amax_bf16(b[r, gi * 128:(gi + 1) * 128]), fmt)


@pytest.mark.parametrize("fmt", FMTS)
def test_blocks_128x128_error_bound_and_transpose_symmetry(fmt):
    rng = np.random.default_rng(4)
    w = (rng.standard_normal((256, 384)) * 0.02).astype(np.float32)
    w[130, 200] = 3.0
    b = bf16_bits(w)
    q, s = O.quantize_blocks_128x128(b, fmt)
    assert s.shape == (2, 3)
    g_full = np.repeat(np.repeat(s, 128, axis=0), 128, axis=1)
    _bound_check(b, q, g_full, fmt)
    qt, st = O.quantize_blocks_128x128(np.ascontiguousarray(b.T), fmt)
    assert np.array_equal(qt, q.T) and np.array_equal(st, s.T)
    # the 1x128 rule on a row equals the block rule when the row holds the block max
    assert s[1, 1] == closed_form_g(0x4040, fmt)  # 3.0


@pytest.mark.parametrize("fmt", FMTS)
def test_exact_values_quantise_to_themselves(fmt):
    """A group already made of FP8 values whose max is the format max has
    scale 1 and codes equal to the values' own codes."""
    rng = np.random.default_rng(5)
    top = 0x7E if fmt == O.E4M3 else 0x7B
    codes = rng.integers(0, top + 1, (128, 256)).astype(np.uint8)
    codes |= (rng.integers(0, 2, codes.shape) * 0x80).astype(np.uint8)
    codes[:, 0] = top
    codes[:, 128] = top | 0x80
    vals = O.decode(codes, fmt)
    b = bf16_bits(vals.astype(np.float32))  # FP8 values are exact in bf16 (<= 3 mantissa bits)
    assert np.array_equal(O.bf16_to_double(b), vals)
    q, s = O.quantize_rows_1x128(b, fmt)
    assert np.all(s == 127)
    assert np.array_equal(q, codes)


@pytest.mark.parametrize("fmt", FMTS)
def test_nonfinite_groups(fmt):
    x = np.ones((2, 256), np.float32)
    x[0, 3] = np.inf
    x[0, 4] = -2.0
    b = bf16_bits(x)
    b[1, 200] = 0x7FC0  # +NaN (torch's own float->bf16 cast yields 0xFFFF here)
    q, s = O.quantize_rows_1x128(b, fmt)
    assert s[0, 0] == 0xFF and s[1, 1] == 0xFF and s[0, 1] != 0xFF and s[1, 0] != 0xFF
    assert np.all(q[0, :128][x[0, :128] > 0] == 0x7F)
    assert q[0, 4] == 0xFF
    assert np.all(q[1, 128:] == 0x7F)


@pytest.mark.parametrize("fmt,tdtype", [(O.E4M3, torch.float8_e4m3fn), (O.E5M2, torch.float8_e5m2)])
def test_tensor_scaling_matches_torch_cast(fmt, tdtype):
    rng = np.random.default_rng(6)
    x = (rng.standard_normal((64, 256)) * 1e-3).astype(np.float32)
    x[3, 3] = -0.37
    b = bf16_bits(x)
    amax, q, si = O.quantize_tensor(b, fmt)
    assert amax == O.amax_bf16(b)
    xf = torch.from_numpy(O.bf16_to_double(b).astype(np.float32))
    a = torch.tensor(O.bf16_to_double(np.array([amax], np.uint16))[0], dtype=torch.float32)
    scale = torch.tensor(O.fmt_max(fmt), dtype=torch.float32) / a
    prod = xf * scale  # fp32 multiply, RN
    assert torch.all(prod.abs() <= O.fmt_max(fmt) * (1 + 2 ** -23))
    prod = prod.clamp(-O.fmt_max(fmt), O.fmt_max(fmt))
    ref = prod.to(tdtype).view(torch.uint8).numpy()
    assert np.array_equal(q, ref)
    assert np.float32(si) == (torch.tensor(1.0, dtype=torch.float32) / scale).item()
    # dequantised max recovers amax within half an FP8 ulp
    deq = O.dequant_tensor(q, si, fmt)
    amax_v = float(a)
    assert abs(np.max(np.abs(deq)) - amax_v) <= amax_v * 2.0 ** -(4 if fmt == O.E4M3 else 3)


def test_tensor_scaling_edge_cases():
    z = np.zeros(300, np.uint16)
    amax, q, si = O.quantize_tensor(z, O.E4M3)
    assert amax == 0 and si == 1.0 and np.all(q == 0)
    b = bf16_bits(np.array([1.0, -np.inf, 2.0], np.float32))
    _, q, si = O.quantize_tensor(b, O.E4M3)
    assert np.isnan(si) and list(q) == [0x7F, 0xFF, 0x7F]
    tiny = np.array([0x0001, 0x8001, 0x0000], np.uint16)  # smallest bf16 subnormals
    _, q, si = O.quantize_tensor(tiny, O.E4M3)
    # 448 / 2^-133 overflows fp32: the scale saturates at FLT_MAX
    assert si == np.float32(1.0) / np.float32(np.finfo(np.float32).max)
    assert q[0] == O.encode(np.array([float(np.float32(2.0 ** -133) * np.finfo(np.float32).max)]), O.E4M3)[0]
    assert q[1] == q[0] | 0x80
