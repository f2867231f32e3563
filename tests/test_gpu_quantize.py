"""GPU parity of amax and the quantisers against the oracle: every amax,
every scale and every FP8 byte must match bit for bit.

Sizes span several 128x128 tiles; per-tensor cases include ragged tails
(extents that are multiples of 16 but not of 128).
"""
import numpy as np
import pytest
import torch

import oracle as O
import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import workloads as W
from _parity import bits, check_block_act_quant, check_block_weight_quant, check_tensor_quant, host, scales_of

pytestmark = pytest.mark.gpu
DEV = "cuda"
FMTS = [P.E4M3, P.E5M2]


@pytest.fixture(scope="module", autouse=True)
def _lib():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    P.load_library()


def _t3(shape, seed, scale=1.0):
    return (W.student_t3_f32(shape, DEV, seed) * scale).to(torch.bfloat16)


# ------------------------------------------------------------------ amax
# sizes past the eight-load unrolled loop of a full grid (152 SMs x 4 x 256
# threads x 8 vectors of 8 = 9.96M values) as well as below it
@pytest.mark.parametrize("n", [0, 1, 7, 8, 9, 1000, 4096 * 33 + 5, 3_000_001, 12_000_007, 41_943_043])
def test_amax_bit_exact(n):
    x = _t3((n,), 100 + n, 3.0)
    a = torch.full((1,), -1, dtype=torch.int32, device=DEV)
    P.puro_fp8_amax(x, a)
    torch.cuda.synchronize()
    want = O.amax_bf16(bits(x)) if n else 0
    assert int(host(a)[0]) == want


def test_amax_nonfinite_and_sign():
    x = torch.randn(50_000, device=DEV).to(torch.bfloat16)
    x[123] = -300.0
    a = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_fp8_amax(x, a)
    torch.cuda.synchronize()
    assert int(host(a)[0]) == O.amax_bf16(bits(x)) == 0x4396  # |-300| = 0x4396 in bf16
    x[40_000] = float("-inf")
    P.puro_fp8_amax(x, a)
    torch.cuda.synchronize()
    assert int(host(a)[0]) == 0x7F80
    x.view(torch.int16)[7] = 0x7FC1  # a NaN
    P.puro_fp8_amax(x, a)
    torch.cuda.synchronize()
    assert int(host(a)[0]) == O.amax_bf16(bits(x)) > 0x7F80


@pytest.mark.parametrize("pos", [0, 9_960_447, 19_999_999, 20_000_000, 20_000_004])
def test_amax_finds_a_single_maximum_anywhere(pos):
    # one value above all others at the first element, inside the unrolled
    # loop's range, in the last whole vector, and in the ragged tail
    n = 20_000_005
    x = (torch.rand(n, device=DEV) * 2 - 1).to(torch.bfloat16)
    x[pos] = -7.5
    a = torch.zeros(1, dtype=torch.int32, device=DEV)
    P.puro_fp8_amax(x, a)
    torch.cuda.synchronize()
    assert int(host(a)[0]) == 0x40F0  # |-7.5| in bf16


# ------------------------------------------------- 1x128 groups (activations)
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("shape", [(128, 128), (384, 640), (256, 1536), (1024, 256), (640, 384)])
def test_block_act_quantize(shape, fmt):
    x = _t3(shape, 7 + shape[0] + shape[1])
    x[:, 5] *= 50.0  # an outlier channel
    q = P.quantize(x, fmt, P.SCALE_BLOCK, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_block_act_quant(x, q, fmt)


@pytest.mark.parametrize("fmt", FMTS)
def test_block_act_quantize_rowwise_only(fmt):
    x = _t3((256, 384), 9)
    q = P.quantize(x, fmt, P.SCALE_BLOCK, P.ROLE_ACT, transpose=False)
    torch.cuda.synchronize()
    assert q.colwise is None
    check_block_act_quant(x, q, fmt)


@pytest.mark.parametrize("fmt", FMTS)
def test_block_act_special_values(fmt):
    """Zero groups, non-finite groups, bf16 subnormals, huge values, values
    that round to -0, and exact FP8 values."""
    x = _t3((256, 512), 11)
    xv = x.view(torch.int16)
    x[0:128, 0:128] = 0.0                                  # all-zero tile (row and column groups)
    x[3, 130] = float("inf")                               # one inf: its row group and column group
    xv[200, 300] = 0x7FC0                                  # +NaN
    xv[201, 301] = -1                                      # 0xFFFF: -NaN
    x[130, 384:512] = torch.tensor(1e-40).to(torch.bfloat16)   # bf16 subnormals (scale exponent clamps at 0)
    x[131, 384:512] = 3.0e38                                # near the bf16 max
    x[132, 384:400] = -1e-30                                # tiny negatives in a group with a large max
    x[132, 400] = 200.0
    q = P.quantize(x, fmt, P.SCALE_BLOCK, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_block_act_quant(x, q, fmt)
    s = scales_of(q.rowwise)  # [row, k-block]
    assert s[3, 1] == 0xFF and s[0, 0] == 127 and s[130, 3] == 0  # non-finite / zero / clamped


def test_block_act_canaries():
    """Guard bands around every output buffer stay untouched."""
    R, C, pad = 384, 256, 64
    x = _t3((R, C), 12)

    def guarded(n):
        buf = torch.full((n + 2 * pad,), 0xA5, dtype=torch.uint8, device=DEV)
        return buf, buf[pad:pad + n]

    ss, sst = P.scale_vec_shape(R, C), P.scale_vec_shape(C, R)
    bq, q = guarded(R * C)
    bs, s = guarded(int(np.prod(ss)))
    bqt, qt = guarded(R * C)
    bst, st = guarded(int(np.prod(sst)))
    P.puro_fp8_quantize(x, P.E4M3, P.SCALE_BLOCK, P.ROLE_ACT, None, q.view(R, C), s.view(*ss),
                        qt.view(C, R), st.view(*sst))
    torch.cuda.synchronize()
    for b in (bq, bs, bqt, bst):
        h = host(b)
        assert np.all(h[:pad] == 0xA5) and np.all(h[-pad:] == 0xA5)
    out = P.Quantized(P.FP8Operand(q.view(R, C), s.view(*ss)), P.FP8Operand(qt.view(C, R), st.view(*sst)))
    check_block_act_quant(x, out, P.E4M3)


# ----------------------------------------------- 128x128 blocks (weights)
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("shape", [(128, 128), (256, 384), (1536, 1536), (2048, 1536)])
def test_block_weight_quantize(shape, fmt):
    w = W.normal_bf16(shape, 0.02, DEV, 31 + shape[0])
    w[7, 9] = -1.5
    q = P.quantize(w, fmt, P.SCALE_BLOCK, P.ROLE_WEIGHT)
    torch.cuda.synchronize()
    check_block_weight_quant(w, q, fmt)


def test_block_weight_nonfinite_block():
    w = W.normal_bf16((256, 256), 0.02, DEV, 5)
    w[130, 3] = float("nan")
    q = P.quantize(w, P.E4M3, P.SCALE_BLOCK, P.ROLE_WEIGHT)
    torch.cuda.synchronize()
    check_block_weight_quant(w, q, P.E4M3)
    assert np.all(scales_of(q.rowwise)[128:256, 0] == 0xFF)


# ------------------------------------------------------- per-tensor scaling
@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("shape", [(256, 1536), (272, 400), (16, 16), (128, 2064)])
def test_tensor_quantize(shape, fmt):
    x = _t3(shape, 41 + shape[1], 0.01)
    q = P.quantize(x, fmt, P.SCALE_TENSOR, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_tensor_quant(x, q, fmt)


@pytest.mark.parametrize("fmt", FMTS)
@pytest.mark.parametrize("shape", [(32768, 1536), (4112, 3968)])
def test_tensor_quantize_many_tiles_per_cta(shape, fmt):
    """The per-tensor quantiser is persistent (two CTAs per SM, 304 on
    GB300): [32768, 1536] gives each CTA about ten 128 x 128 tiles, so the
    loop, the double-buffered loads and the reuse of the staging tiles run
    many times; [4112, 3968] adds ragged last row and column tiles.  Every
    byte, amax and scale_inv against the oracle."""
    x = _t3(shape, 160 + shape[1] + fmt, 2.0)
    check_tensor_quant(x, P.quantize(x, fmt, P.SCALE_TENSOR, P.ROLE_ACT), fmt)


def test_tensor_quantize_edge_cases():
    z = torch.zeros((32, 64), dtype=torch.bfloat16, device=DEV)
    q = P.quantize(z, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_tensor_quant(z, q, P.E4M3)
    assert host(q.rowwise.scale)[0] == 1.0
    tiny = torch.zeros((16, 32), dtype=torch.bfloat16, device=DEV)
    tiny.view(torch.int16)[0, 0] = 1          # smallest bf16 subnormal: 448/amax overflows -> FLT_MAX
    tiny.view(torch.int16)[5, 5] = -32767     # 0x8001
    q = P.quantize(tiny, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_tensor_quant(tiny, q, P.E4M3)
    bad = torch.ones((16, 32), dtype=torch.bfloat16, device=DEV)
    bad[3, 3] = float("-inf")
    q = P.quantize(bad, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT)
    torch.cuda.synchronize()
    check_tensor_quant(bad, q, P.E4M3)
    assert np.isnan(host(q.rowwise.scale)[0])


def test_tensor_quantize_empty():
    x = torch.empty((0, 64), dtype=torch.bfloat16, device=DEV)
    q = P.quantize(x, P.E4M3, P.SCALE_TENSOR, P.ROLE_ACT, transpose=False)
    torch.cuda.synchronize()
    assert int(host(q.amax)[0]) == 0 and host(q.rowwise.scale)[0] == 1.0


@pytest.mark.parametrize("fmt,with_t", [(P.E4M3, True), (P.E5M2, True), (P.E4M3, False)])
def test_grouped_weights_equal_the_single_calls(fmt, with_t):
    """puro_fp8_quantize_weights over more than one launch's worth of weights
    (70 entries: the four C5 shapes, an empty entry, many small ones, one
    with a non-finite block) writes the bytes puro_fp8_quantize writes for
    each weight; two of them are also checked against the oracle."""
    shapes = [(2048, 1536), (1536, 1536), (17920, 1536), (1536, 8960), (0, 128)] + [(128, 256), (384, 128)] * 32 + \
        [(256, 384)]
    entries, singles = [], []
    for i, (r, c) in enumerate(shapes):
        w = W.student_t3_f32((r, c), DEV, 4000 + i).mul_(0.02).to(torch.bfloat16) if r else \
            torch.empty((0, c), dtype=torch.bfloat16, device=DEV)
        if i == len(shapes) - 1:
            w[130, 200] = float("inf")  # a non-finite block
        q = P.quantize(torch.empty_like(w), fmt, P.SCALE_BLOCK, P.ROLE_WEIGHT, transpose=with_t) if r else \
            P.Quantized(P.FP8Operand(torch.empty((0, c), dtype=torch.uint8, device=DEV),
                                     torch.empty(16, dtype=torch.uint8, device=DEV)), None)
        entries.append((w, q))
        if r:
            singles.append(P.quantize(w, fmt, P.SCALE_BLOCK, P.ROLE_WEIGHT, transpose=with_t))
        else:
            singles.append(None)
    P.puro_fp8_quantize_weights(entries, fmt)
    torch.cuda.synchronize()
    for i, ((w, q), s) in enumerate(zip(entries, singles)):
        if s is None:
            continue
        assert torch.equal(q.rowwise.data, s.rowwise.data), f"entry {i}: codes"
        assert torch.equal(q.rowwise.scale, s.rowwise.scale), f"entry {i}: scales"
        if with_t:
            assert torch.equal(q.colwise.data, s.colwise.data), f"entry {i}: transposed codes"
            assert torch.equal(q.colwise.scale, s.colwise.scale), f"entry {i}: transposed scales"
    check_block_weight_quant(entries[1][0], entries[1][1], fmt)
    check_block_weight_quant(entries[-1][0], entries[-1][1], fmt)
