"""Pins for the oracle's FP8 codec (E4M3 / E5M2, RNE with saturation).

Pinned against: the format table of the cited FP8 formats paper (golden
fixture), exhaustive enumeration of all 256 codes, exact midpoint
arithmetic, and torch's own float8 casts (a library routine) on every
bf16 bit pattern that does not need saturation.
"""
import os
from fractions import Fraction

import numpy as np
import pytest
import torch

import oracle as O

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "fp8_formats.txt")


def _golden_rows():
    rows = []
    for line in open(GOLDEN):
        line = line.strip()
        if not line or line.startswith("#"):
            continue
        fmt, field, pattern, value = line.split()
        rows.append((fmt, field, pattern, value))
    return rows


def _value(expr):
    if expr == "nan":
        return float("nan")
    if expr == "inf":
        return float("inf")
    return float(eval(expr, {"p2": lambda k: 2.0 ** k}))


@pytest.mark.parametrize("row", _golden_rows(), ids=lambda r: f"{r[0]}-{r[1]}-{r[2]}")
def test_golden_format_table(row):
    fmt_name, field, pattern, value = row
    fmt = O.E4M3 if fmt_name == "E4M3" else O.E5M2
    if field == "bias":
        # bias fixes the min normal: 2^(1 - bias)
        code = 0x08 if fmt == O.E4M3 else 0x04
        assert O.decode(np.array([code]), fmt)[0] == 2.0 ** (1 - int(value))
        return
    code = int(pattern.replace(".", ""), 2)
    v = _value(value)
    got = O.decode(np.array([code], np.uint8), fmt)[0]
    neg = O.decode(np.array([code | 0x80], np.uint8), fmt)[0]
    if np.isnan(v):
        assert np.isnan(got) and np.isnan(neg)
    else:
        assert got == v
        assert neg == -v and np.signbit(neg)
    if field == "max_normal":
        assert O.fmt_max(fmt) == v


@pytest.mark.parametrize("fmt", [O.E4M3, O.E5M2])
def test_exhaustive_round_trip(fmt):
    codes = np.arange(256, dtype=np.uint8)
    vals = O.decode(codes, fmt)
    back = O.encode(vals, fmt)
    for c in range(256):
        v = vals[c]
        if np.isnan(v):
            assert back[c] == 0x7F, hex(c)            # canonical NaN
        elif np.isinf(v):
            assert fmt == O.E5M2
            assert back[c] == (0xFB if v < 0 else 0x7B)  # satfinite: inf -> max
        else:
            assert back[c] == c, hex(c)


@pytest.mark.parametrize("fmt", [O.E4M3, O.E5M2])
def test_monotone_and_symmetric(fmt):
    top = 0x7E if fmt == O.E4M3 else 0x7B
    pos = O.decode(np.arange(0, top + 1, dtype=np.uint8), fmt)
    assert np.all(np.diff(pos) > 0)
    neg = O.decode(np.arange(0x80, 0x80 + top + 1, dtype=np.uint8), fmt)
    assert np.array_equal(neg, -pos)
    assert pos[-1] == O.fmt_max(fmt)


@pytest.mark.parametrize("fmt", [O.E4M3, O.E5M2])
def test_midpoints_round_to_even(fmt):
    top = 0x7E if fmt == O.E4M3 else 0x7B
    vals = O.decode(np.arange(0, top + 1, dtype=np.uint8), fmt)
    for c in range(top):
        lo, hi = vals[c], vals[c + 1]
        mid = (Fraction(lo) + Fraction(hi)) / 2
        m = float(mid)
        assert Fraction(m) == mid  # midpoints of FP8 values are exact doubles
        even = c if (c & 1) == 0 else c + 1  # mantissa LSB is the code LSB
        for sgn in (1.0, -1.0):
            sb = 0x80 if sgn < 0 else 0
            assert O.encode(np.array([sgn * m]), fmt)[0] == (even | sb)
            below = np.nextafter(m, 0.0)
            above = np.nextafter(m, np.inf)
            assert O.encode(np.array([sgn * below]), fmt)[0] == (c | sb)
            assert O.encode(np.array([sgn * above]), fmt)[0] == ((c + 1) | sb)


@pytest.mark.parametrize("fmt", [O.E4M3, O.E5M2])
def test_saturation_and_signed_zero(fmt):
    mx = O.fmt_max(fmt)
    maxc = 0x7E if fmt == O.E4M3 else 0x7B
    v = np.array([mx, mx * 1.01, mx * 4, np.inf, -mx * 1.5, -np.inf, 0.0, -0.0, -1e-30, 1e-30])
    got = O.encode(v, fmt)
    assert list(got) == [maxc, maxc, maxc, maxc, maxc | 0x80, maxc | 0x80, 0x00, 0x80, 0x80, 0x00]
    assert O.encode(np.array([np.nan]), fmt)[0] == 0x7F


def _all_bf16_values():
    bits = np.arange(65536, dtype=np.uint32).astype(np.uint16)
    return bits, O.bf16_to_double(bits)


@pytest.mark.parametrize("fmt,tdtype", [(O.E4M3, torch.float8_e4m3fn), (O.E5M2, torch.float8_e5m2)])
@pytest.mark.parametrize("scale_exp", [-12, -3, 0, 5, 13])
def test_matches_torch_cast_where_no_saturation(fmt, tdtype, scale_exp):
    """torch's float -> float8 cast rounds to nearest even but does not
    saturate, so only in-range values are compared."""
    _, vals = _all_bf16_values()
    v = vals * 2.0 ** scale_exp
    keep = np.isfinite(v) & (np.abs(v) <= O.fmt_max(fmt))
    v = v[keep]
    ours = O.encode(v, fmt)
    ref = torch.from_numpy(v).to(tdtype).view(torch.uint8).numpy()
    # torch keeps -0 for negative values that round to zero as well
    assert np.array_equal(ours, ref)


@pytest.mark.parametrize("fmt,tdtype", [(O.E4M3, torch.float8_e4m3fn), (O.E5M2, torch.float8_e5m2)])
def test_decode_matches_torch(fmt, tdtype):
    codes = np.arange(256, dtype=np.uint8)
    ours = O.decode(codes, fmt)
    ref = torch.from_numpy(codes).view(tdtype).to(torch.float64).numpy()
    both_nan = np.isnan(ours) & np.isnan(ref)
    assert np.array_equal(ours[~both_nan], ref[~both_nan])
    assert np.array_equal(np.isnan(ours), np.isnan(ref))


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(1)
    v = np.concatenate([rng.standard_normal(20000) * 10.0 ** rng.integers(-40, 38, 20000),
                        [0.0, -0.0, 1e-45, 3e38, 3.4e38, -3.4e38, 1.0 + 2 ** -8, 1.0 + 3 * 2 ** -9]])
    ours = O.bf16_from_double(v)
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    # torch goes through fp32 first (double rounding); compare where fp32 is exact
    exact = v.astype(np.float32).astype(np.float64) == v
    assert np.array_equal(ours[exact], ref[exact])
    back = O.bf16_to_double(ours)
    fin = np.isfinite(back)
    assert np.all(np.abs(back - v)[fin] <= np.abs(v[fin]) * 2.0 ** -8 + 2.0 ** -134)
    # overflow only beyond the largest finite bf16 plus half an ulp
    assert np.all(np.abs(v[~fin]) >= (2.0 - 2.0 ** -8) * 2.0 ** 127)
