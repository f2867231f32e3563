"""Pins of the oracle's SwiGLU producer (the down projection's input
silu(gate) * up, rounded once to bf16): the exact result at 60 significant
digits, the closed forms at g = 0 and for large |g|, torch's fp64 silu (a
library routine), and the row-strided layout of the fused gate/up output."""
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as O


def _bf16(values) -> np.ndarray:
    return torch.tensor(np.asarray(values, np.float32)).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def _val(bits: np.ndarray) -> np.ndarray:
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).view(torch.bfloat16).double().numpy()


def _rne_bf16_exact(x: Fraction) -> int:
    """bf16 bits of the exact rational x, rounded to nearest even (finite,
    normal or subnormal; the tests keep x inside the bf16 range)."""
    if x == 0:
        return 0
    sign = 0x8000 if x < 0 else 0
    a = abs(x)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    if Fraction(2) ** e > a:
        e -= 1
    e = max(e, -126)                       # subnormals share the minimum exponent
    q = a / Fraction(2) ** (e - 7)         # 8 significant bits: [128, 256) when normal
    n = q.numerator // q.denominator
    rem = q - n
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and n % 2 == 1):
        n += 1
    if n == 256:
        n, e = 128, e + 1
    if n < 128:                            # subnormal
        return sign | n
    return sign | ((e + 127) << 7) | (n - 128)


def _fraction(x) -> Fraction:
    """The exact value of an mpmath number (sign, mantissa, exponent)."""
    sign, man, exp, _ = x._mpf_
    v = Fraction(int(man)) * Fraction(2) ** int(exp)
    return -v if sign else v


def test_matches_the_exact_result_at_60_digits():
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 60
    rng = np.random.default_rng(11)
    # |g| <= 30 keeps 1 + e^-g away from 1 in fp64 (large |g|: the tests below)
    g = _bf16(np.concatenate([rng.standard_normal(1500) * 3.0, rng.uniform(-30.0, 30.0, 500)]))
    u = _bf16(rng.standard_normal(2000) * np.exp2(rng.integers(-8, 9, 2000)))
    got = O.swiglu(g.reshape(40, 50), u.reshape(40, 50)).ravel()
    gv, uv = _val(g), _val(u)
    for i in range(g.size):
        x = mpmath.mpf(float(gv[i])) / (1 + mpmath.exp(-mpmath.mpf(float(gv[i])))) * mpmath.mpf(float(uv[i]))
        want = _rne_bf16_exact(_fraction(x))
        assert int(got[i]) == want, (i, float(gv[i]), float(uv[i]), hex(int(got[i])), hex(want))


def test_zero_gate_gives_zero():
    u = _bf16([1.0, -3.0, 1e30, -1e-30, 0.0, 7.5])
    g = _bf16([0.0] * 6)
    h = O.swiglu(g.reshape(1, 6), u.reshape(1, 6))
    assert np.all(_val(h) == 0.0)


def test_large_positive_gate_is_the_plain_product():
    # for g >= 40, g / (1 + e^-g) differs from g by < 2^-57 relative, so the
    # result is the rounded product g * u (exact as a rational: two 8-bit
    # significands).  Where g * u is itself a bf16 tie the true value lies a
    # hair below it; an fp64 (or fp32) evaluation sees g * u and rounds to
    # even, the reading both the oracle and the kernels take.
    rng = np.random.default_rng(5)
    g = _bf16(rng.uniform(40.0, 3000.0, 4096))
    u = _bf16(rng.standard_normal(4096))
    h = O.swiglu(g.reshape(64, 64), u.reshape(64, 64)).ravel()
    prod = [_rne_bf16_exact(Fraction(float(a)) * Fraction(float(b))) for a, b in zip(_val(g), _val(u))]
    assert h.tolist() == prod


def test_large_negative_gate_vanishes_like_g_exp_g():
    # for g <= -40, silu(g) = g e^g (1 - e^g + ...): relative size of the
    # correction < 2^-57, so the result is the rounding of g e^g u
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 40
    gs = [-40.0, -45.5, -60.0, -64.0, -80.0]
    us = [1.0, -2.0, 1e10, 3e20, -5e25]
    h = O.swiglu(_bf16(gs).reshape(1, 5), _bf16(us).reshape(1, 5)).ravel()
    gv, uv = _val(_bf16(gs)), _val(_bf16(us))
    for i in range(5):
        x = mpmath.mpf(float(gv[i])) * mpmath.exp(mpmath.mpf(float(gv[i]))) * mpmath.mpf(float(uv[i]))
        assert int(h[i]) == _rne_bf16_exact(_fraction(x)), i


def test_torch_fp64_silu_agrees_almost_everywhere():
    # torch's double -> bfloat16 cast rounds through fp32 first (two
    # roundings), so a rare element may differ by one bf16 ulp
    rng = np.random.default_rng(8)
    g = _bf16(rng.standard_normal((256, 256)) * 4.0)
    u = _bf16(rng.standard_normal((256, 256)))
    h = O.swiglu(g, u)
    ref = torch.nn.functional.silu(torch.from_numpy(_val(g))) * torch.from_numpy(_val(u))
    ref_bits = ref.to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    diff = np.abs(h.astype(np.int32) - ref_bits.astype(np.int32))
    assert diff.max() <= 1
    assert np.count_nonzero(diff) <= 4


def test_row_strided_halves_of_a_fused_output():
    rng = np.random.default_rng(2)
    gu = _bf16(rng.standard_normal((96, 2 * 160)))
    g, u = gu[:, :160], gu[:, 160:]
    assert not g.flags["C_CONTIGUOUS"]
    a = O.swiglu(g, u)
    b = O.swiglu(np.ascontiguousarray(g), np.ascontiguousarray(u))
    assert np.array_equal(a, b)
    # and it is the gate half that goes through silu
    c = O.swiglu(np.ascontiguousarray(u), np.ascontiguousarray(g))
    assert not np.array_equal(a, c)
