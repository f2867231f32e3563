"""Pins of the oracle's MuonH hyperball step (section "Hyperball
Optimization", Eq. hyperball-update): a worked example with rational
norms, the sphere invariant, closed forms for eta = 0 and for an update
orthogonal to W, invariance to the scale of the Muon direction, and the
exact result at 50 digits on small inputs."""
import math

import numpy as np
import pytest

import oracle as O


def test_worked_example_with_rational_norms():
    # W = (5, 0) on the sphere R = 5, u along (0, 1): W~ = (5, -3.75) has
    # norm 6.25, so W_new = 5 * (5, -3.75) / 6.25 = (4, -3)
    w = np.array([5.0, 0.0], np.float32)
    for scale in (1.0, 7.0, 0.125):
        u = np.array([0.0, scale], np.float32)
        got = O.muonh_step(w, u, 0.75, 5.0)
        assert np.allclose(got, [4.0, -3.0], rtol=0, atol=1e-14), got
    # the same inside a larger matrix of zeros, and with the step reversed
    W = np.zeros((4, 8), np.float32)
    U = np.zeros((4, 8), np.float32)
    W[2, 3], U[1, 5] = 5.0, -2.0
    got = O.muonh_step(W, U, 0.75, 5.0)
    want = np.zeros((4, 8))
    want[2, 3], want[1, 5] = 4.0, 3.0
    assert np.allclose(got, want, rtol=0, atol=1e-14)


def test_result_lies_on_the_sphere():
    rng = np.random.default_rng(1)
    for n, eta in ((1000, 1e-3), (4096, 0.02), (77, 0.5)):
        w = rng.standard_normal(n).astype(np.float32)
        u = rng.standard_normal(n).astype(np.float32)
        r = float(rng.uniform(0.5, 40.0))
        got = O.muonh_step(w, u, eta, r)
        assert abs(math.sqrt(float(np.sum(got * got))) - r) <= 1e-13 * r


def test_zero_step_is_the_projection():
    rng = np.random.default_rng(2)
    w = rng.standard_normal((64, 48)).astype(np.float32)
    u = rng.standard_normal((64, 48)).astype(np.float32)
    r = 3.0
    got = O.muonh_step(w, u, 0.0, r)
    wd = w.astype(np.float64)
    want = r * wd / math.sqrt(float(np.sum(wd * wd)))  # numpy sums pairwise: rounding differs
    assert np.allclose(got, want, rtol=1e-13, atol=0)


def test_zero_direction_takes_no_step():
    # the equation divides by ||u|| = 0; the reading taken: no step
    rng = np.random.default_rng(6)
    w = rng.standard_normal(300).astype(np.float32)
    got = O.muonh_step(w, np.zeros(300, np.float32), 0.1, 2.0)
    assert np.array_equal(got, O.muonh_step(w, np.ones(300, np.float32), 0.0, 2.0))


def test_orthogonal_update_closed_form():
    # <W, u> = 0 and ||W|| = R:  ||W~||^2 = R^2 (1 + eta^2), so
    # W_new = (W - eta R u_hat) / sqrt(1 + eta^2)
    w = np.zeros(6, np.float32)
    u = np.zeros(6, np.float32)
    w[:3] = [2.0, -1.0, 2.0]      # norm 3
    u[3:] = [1.0, 2.0, 2.0]       # norm 3, orthogonal to w
    r, eta = 3.0, 0.3
    got = O.muonh_step(w, u, eta, r)
    want = (w.astype(np.float64) - eta * r * u.astype(np.float64) / 3.0) / math.sqrt(1.0 + eta * eta)
    assert np.allclose(got, want, rtol=1e-15, atol=1e-16)


def test_invariant_to_the_scale_of_the_muon_direction():
    rng = np.random.default_rng(3)
    w = rng.standard_normal(513).astype(np.float32)
    u = rng.standard_normal(513).astype(np.float32)
    base = O.muonh_step(w, u, 0.05, 7.0)
    for k in (-30, -3, 5, 40):
        scaled = (u * np.float32(2.0 ** k)).astype(np.float32)
        assert np.array_equal(O.muonh_step(w, scaled, 0.05, 7.0), base), k


def test_matches_the_exact_result_at_50_digits():
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 50
    rng = np.random.default_rng(4)
    w = rng.standard_normal(24).astype(np.float32)
    u = (rng.standard_normal(24) * 1e-3).astype(np.float32)
    eta, r = 0.125, 4.5
    got = O.muonh_step(w, u, eta, r)
    W = [mpmath.mpf(float(x)) for x in w]
    U = [mpmath.mpf(float(x)) for x in u]
    un = mpmath.sqrt(sum(x * x for x in U))
    T = [a - mpmath.mpf(eta) * r * b / un for a, b in zip(W, U)]
    tn = mpmath.sqrt(sum(x * x for x in T))
    for i in range(24):
        want = float(r * T[i] / tn)
        assert abs(got[i] - want) <= 4e-16 * abs(want) + 1e-300, (i, got[i], want)


def test_frobenius_norm_matches_numpy():
    rng = np.random.default_rng(5)
    x = rng.standard_normal((300, 200)).astype(np.float32)
    # index-order fp64 sum against numpy's pairwise one: 6e4 terms
    assert math.isclose(O.frobenius_norm(x), float(np.linalg.norm(x.astype(np.float64))), rel_tol=1e-12)
