"""Pins of the oracle's RMSNorm producer (the normalisation that the fused
RMSNorm -> quantise kernel applies before quantising): closed forms, exact
power-of-two scale invariance, exact rational arithmetic on small rows, and
torch's fp32 arithmetic for the fp32 application step."""
from fractions import Fraction
import math

import numpy as np
import torch

import oracle as O


def _bf16(values):
    return torch.tensor(values, dtype=torch.float32).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)


def test_constant_rows_closed_form():
    for c in (0.0, 1.0, -3.5, 0.0078125, 240.0):
        h = _bf16([[c] * 256])
        got = O.rmsnorm_rstd(h, 1e-6)[0]
        want = 1.0 / math.sqrt(c * c + 1e-6)
        assert abs(got - want) <= 1e-15 * want, (c, got, want)


def test_power_of_two_scaling_is_exact_without_eps():
    rng = np.random.default_rng(3)
    h = _bf16(rng.standard_normal((8, 384)).astype(np.float32))
    base = O.rmsnorm_rstd(h, 0.0)
    for k in (-20, -3, 1, 7, 40):
        hk = _bf16((torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).float() * 2.0 ** k).numpy())
        assert np.array_equal(O.rmsnorm_rstd(hk, 0.0), base * 2.0 ** -k), k


def test_exact_rational_mean_on_small_rows():
    rng = np.random.default_rng(5)
    h = _bf16(rng.standard_normal((6, 48)).astype(np.float32) * 3)
    vals = torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).double().numpy()
    got = O.rmsnorm_rstd(h, 1e-5)
    for r in range(h.shape[0]):
        mean = sum(Fraction(float(v)) ** 2 for v in vals[r]) / h.shape[1]
        want = 1.0 / math.sqrt(float(mean + Fraction(1e-5)))
        assert abs(got[r] - want) <= 4e-16 * want, (r, got[r], want)


def test_apply_matches_torch_fp32_then_bf16():
    rng = np.random.default_rng(7)
    h = _bf16(rng.standard_normal((16, 640)).astype(np.float32) * 5)
    gamma = _bf16(1.0 + 0.1 * rng.standard_normal(640).astype(np.float32))
    rstd = (1.0 / np.sqrt(np.mean(rng.standard_normal((16, 640)) ** 2, axis=1) + 1e-6)).astype(np.float32)
    ht = torch.from_numpy(h.view(np.int16)).view(torch.bfloat16).float()
    gt = torch.from_numpy(gamma.view(np.int16)).view(torch.bfloat16).float()
    rt = torch.from_numpy(rstd)[:, None]
    want_g = ((ht * rt) * gt).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    want_n = (ht * rt).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(O.rmsnorm_apply_f32(h, rstd, gamma), want_g)
    assert np.array_equal(O.rmsnorm_apply_f32(h, rstd, None), want_n)
    ones = _bf16(np.ones(640, np.float32))
    assert np.array_equal(O.rmsnorm_apply_f32(h, rstd, ones), want_n)
