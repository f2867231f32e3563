"""MuonH hyperball step on the GPU against the fp64 oracle.

The kernels reduce the three sums {sum W^2, sum W u, sum u^2} with FP32
per-thread chains of at most a few dozen chunk sums and FP64 above that,
round c = eta R / ||u|| and s = R / ||W~|| to fp32 and write
W <- s (W - c u) with one FMA and one multiply per element.  The sums'
relative error is then below about 64 * 2^-24 (4e-6) and each element's
below that plus three fp32 roundings, so the test accepts
|gpu - ref| <= 1e-5 |ref| + 1e-6 rms(ref) (the absolute term covers
elements where W - c u cancels).  The BF16 copy must be the fp32 result
rounded to nearest even, bit for bit.
"""
import math

import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W

pytestmark = pytest.mark.gpu
DEV = "cuda"


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


def _inputs(rows, cols, seed):
    """W ~ N(0, 0.02) (the initialisation) and a Muon-like direction u
    (rows of N(0, 1) / sqrt(cols), the scale of an orthogonalised update)."""
    w = W.normal_f32((rows, cols), 0.02, DEV, seed)
    u = W.normal_f32((rows, cols), 1.0 / math.sqrt(cols), DEV, seed + 1)
    return w, u


def _check(got: torch.Tensor, ref: np.ndarray):
    g = got.double().cpu().numpy()
    rms = float(np.sqrt(np.mean(ref * ref)))
    err = np.abs(g - ref)
    bound = 1e-5 * np.abs(ref) + 1e-6 * rms
    worst = float(np.max(err / bound))
    assert worst <= 1.0, f"MuonH result outside tolerance (worst ratio {worst:.3g})"


def _ws(n):
    return torch.empty(max(8, P.puro_muonh_workspace_size(n)), dtype=torch.uint8, device=DEV)


@pytest.mark.parametrize("rows,cols,eta", [(256, 640, 1e-3), (2048, 1536, 4.08e-4), (17920, 1536, 0.02),
                                           (12, 100, 0.3), (1536, 8960, 1e-3)])
def test_step_matches_the_oracle(rows, cols, eta):
    w0, u = _inputs(rows, cols, 1000 + rows + cols)
    n = w0.numel()
    radius = O.frobenius_norm(w0.cpu().numpy())
    # a weight already on the sphere, a step in, as in training
    w_start = w0 + 0.01 * W.normal_f32((rows, cols), 0.02, DEV, 7 + rows)
    w_start *= radius / float(torch.linalg.vector_norm(w_start.double()))
    w = w_start.clone()
    sums = torch.empty(3, dtype=torch.float64, device=DEV)
    wb = torch.empty((rows, cols), dtype=torch.bfloat16, device=DEV)
    P.puro_muonh_step(w, u, eta, radius, sums, _ws(n), wb)
    torch.cuda.synchronize()
    ws_h, u_h = w_start.cpu().numpy(), u.cpu().numpy()
    # the three sums
    s = sums.cpu().numpy()
    wd, ud = ws_h.astype(np.float64), u_h.astype(np.float64)
    for got, want in zip(s, (np.sum(wd * wd), np.sum(wd * ud), np.sum(ud * ud))):
        assert abs(got - want) <= 4e-6 * math.sqrt(np.sum(wd * wd) * np.sum(ud * ud)) + 4e-6 * abs(want)
    ref = O.muonh_step(ws_h, u_h, eta, radius)
    _check(w, ref)
    # on the sphere, and the bf16 copy is the fp32 result rounded
    assert abs(math.sqrt(float(torch.sum(w.double() ** 2))) - radius) <= 2e-5 * radius
    assert torch.equal(wb.view(torch.int16), w.to(torch.bfloat16).view(torch.int16))


def test_deterministic_and_shardable():
    rows, cols = 4096, 1536
    w0, u = _inputs(rows, cols, 5)
    n = w0.numel()
    radius = float(torch.linalg.vector_norm(w0.double()))
    sums = torch.empty(3, dtype=torch.float64, device=DEV)
    runs = []
    for _ in range(2):
        w = w0.clone()
        P.puro_muonh_step(w, u, 1e-3, radius, sums, _ws(n))
        runs.append(w)
    torch.cuda.synchronize()
    assert torch.equal(runs[0], runs[1]), "the step is not deterministic"
    # two shards: reduce each, add the sums (the all-reduce of a sharded
    # optimizer), apply each with the combined sums
    half = rows // 2
    parts = []
    for lo in (0, half):
        s = torch.empty(3, dtype=torch.float64, device=DEV)
        P.puro_muonh_reduce(w0[lo:lo + half], u[lo:lo + half], s, _ws(half * cols))
        parts.append(s)
    total = parts[0] + parts[1]
    w_sh = w0.clone()
    for lo in (0, half):
        P.puro_muonh_apply(w_sh[lo:lo + half], u[lo:lo + half], total, 1e-3, radius)
    torch.cuda.synchronize()
    ref = O.muonh_step(w0.cpu().numpy(), u.cpu().numpy(), 1e-3, radius)
    _check(w_sh, ref)
    # applying with the whole-matrix sums shard by shard is the same elementwise op, bit for bit
    P.puro_muonh_reduce(w0, u, sums, _ws(n))
    w_a, w_b = w0.clone(), w0.clone()
    P.puro_muonh_apply(w_a, u, sums, 1e-3, radius)
    for lo in (0, half):
        P.puro_muonh_apply(w_b[lo:lo + half], u[lo:lo + half], sums, 1e-3, radius)
    torch.cuda.synchronize()
    assert torch.equal(w_a, w_b)


def test_zero_direction_is_a_projection_and_empty_is_a_no_op():
    w0, _ = _inputs(128, 256, 9)
    w = w0.clone()
    sums = torch.empty(3, dtype=torch.float64, device=DEV)
    P.puro_muonh_step(w, torch.zeros_like(w0), 0.1, 2.0, sums, _ws(w.numel()))
    torch.cuda.synchronize()
    _check(w, O.muonh_step(w0.cpu().numpy(), np.zeros((128, 256), np.float32), 0.1, 2.0))
    e = torch.empty(0, dtype=torch.float32, device=DEV)
    P.puro_muonh_step(e, e, 0.1, 2.0, sums, _ws(8))
    P.puro_muonh_reduce(e, e, sums, _ws(8))
    torch.cuda.synchronize()
    assert torch.equal(sums, torch.zeros(3, dtype=torch.float64, device=DEV))


def test_radius_helper():
    w0, _ = _inputs(640, 384, 11)
    assert math.isclose(P.muonh_radius(w0), O.frobenius_norm(w0.cpu().numpy()), rel_tol=4e-6)


def test_grouped_step_equals_the_single_steps_bit_for_bit():
    # the model's four shapes (reduced M-independent sizes), a tiny matrix, an
    # empty one, and more than one launch's worth (130 > 128 matrices)
    shapes = [(2048, 1536), (1536, 1536), (8960, 1536), (1536, 8960), (4, 8), (0, 16)] + [(16, 64)] * 124
    mats, singles = [], []
    for i, (r, c) in enumerate(shapes):
        w, u = _inputs(r, c, 3000 + i)
        radius = 1.0 + 0.01 * i
        wb = torch.empty((r, c), dtype=torch.bfloat16, device=DEV) if i % 2 == 0 else None
        mats.append((w.clone(), u, wb, radius))
        singles.append((w.clone(), u, radius))
    sums = torch.empty((len(mats), 3), dtype=torch.float64, device=DEV)
    ws = torch.empty(max(8, P.puro_muonh_grouped_workspace_size(mats)), dtype=torch.uint8, device=DEV)
    P.puro_muonh_step_grouped(mats, 1e-3, sums, ws)
    s1 = torch.empty(3, dtype=torch.float64, device=DEV)
    for w, u, r in singles:
        P.puro_muonh_step(w, u, 1e-3, r, s1, _ws(max(4, w.numel())))
    torch.cuda.synchronize()
    for i, ((wg, u, wb, r), (w1, _, _)) in enumerate(zip(mats, singles)):
        assert torch.equal(wg, w1), f"matrix {i}: grouped and single steps differ"
        if wb is not None:
            assert torch.equal(wb.view(torch.int16), wg.to(torch.bfloat16).view(torch.int16))
    assert torch.equal(sums[5], torch.zeros(3, dtype=torch.float64, device=DEV))
    _check(mats[0][0], O.muonh_step(_inputs(2048, 1536, 3000)[0].cpu().numpy(),
                                    mats[0][1].cpu().numpy(), 1e-3, mats[0][3]))
