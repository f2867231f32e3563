"""Host-side checks of the C ABI (no GPU needed): the library builds and
loads, exports every entry point the header declares, the ctypes mirror of
puro_fp8_tensor_t has the C layout, and argument validation rejects bad
calls synchronously, before any CUDA work is enqueued."""
import ctypes
import os
import re
import subprocess

import numpy as np
import pytest
import torch

import paper_2608_27370_gb300 as P
from paper_2608_27370_gb300 import _build

BAD = P.PURO_ERR_INVALID_ARG
A = 0x100000  # a 16-byte aligned fake device address (never dereferenced)


@pytest.fixture(scope="module")
def lib():
    _build.build()
    return P.load_library()


def _declared_functions():
    text = open(P.HEADER_PATH).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(puro_\w+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = _declared_functions()
    for required in ("puro_fp8_amax", "puro_fp8_quantize", "puro_fp8_linear_fprop", "puro_fp8_linear_dgrad",
                     "puro_fp8_linear_wgrad", "puro_fp8_workspace_size", "puro_fp8_get_status",
                     "puro_bf16_linear_fprop", "puro_bf16_linear_dgrad", "puro_bf16_linear_wgrad"):
        assert required in names


def test_library_exports_every_declared_symbol(lib):
    for name in _declared_functions():
        assert hasattr(lib, name), name
        assert name in P._SIGNATURES, f"binding lacks {name}"


def test_struct_layout_matches_c(tmp_path):
    """Compile a probe against the header with the C compiler and compare."""
    src = tmp_path / "probe.c"
    src.write_text(
        '#include <stddef.h>\n#include <stdio.h>\n#include "puro_fp8.h"\n'
        "int main(void){printf(\"%zu %zu %zu %zu %zu %zu %zu %zu %zu\\n\", sizeof(puro_fp8_tensor_t),"
        "offsetof(puro_fp8_tensor_t,data),offsetof(puro_fp8_tensor_t,scale),offsetof(puro_fp8_tensor_t,rows),"
        "offsetof(puro_fp8_tensor_t,red),offsetof(puro_fp8_tensor_t,fmt),offsetof(puro_fp8_tensor_t,scaling),"
        "offsetof(puro_fp8_tensor_t,role),offsetof(puro_fp8_tensor_t,reserved));return 0;}\n")
    exe = tmp_path / "probe"
    subprocess.run(["gcc", "-std=c11", "-I", os.path.dirname(P.HEADER_PATH), str(src), "-o", str(exe)], check=True)
    got = [int(v) for v in subprocess.run([str(exe)], capture_output=True, text=True, check=True).stdout.split()]
    T = P.puro_fp8_tensor_t
    want = [ctypes.sizeof(T)] + [getattr(T, f).offset for f in
                                 ("data", "scale", "rows", "red", "fmt", "scaling", "role", "reserved")]
    assert got == want


def test_status_strings(lib):
    assert lib.puro_status_string(0) == b"PURO_OK"
    assert lib.puro_status_string(4) == b"PURO_ERR_TIMEOUT"


def test_amax_validation(lib):
    assert lib.puro_fp8_amax(A, 4, 8, None, None) == BAD           # no output word
    assert lib.puro_fp8_amax(A, -1, 8, A, None) == BAD             # negative extent
    assert lib.puro_fp8_amax(A + 2, 4, 8, A, None) == BAD          # misaligned input
    assert lib.puro_fp8_amax(None, 4, 8, A, None) == BAD           # null input
    assert lib.puro_fp8_amax(A, 4, 8, A + 2, None) == BAD          # misaligned output word


def test_quantize_validation(lib):
    q = lib.puro_fp8_quantize
    BLK, TEN, ACT, WGT = P.SCALE_BLOCK, P.SCALE_TENSOR, P.ROLE_ACT, P.ROLE_WEIGHT
    assert q(A, 128, 128, 7, BLK, ACT, None, A, A, A, A, None, None) == BAD       # bad format
    assert q(A, 128, 128, 0, 9, ACT, None, A, A, A, A, None, None) == BAD         # bad scaling
    assert q(A, 128, 128, 0, BLK, 5, None, A, A, A, A, None, None) == BAD         # bad role
    assert q(A, 130, 128, 0, BLK, ACT, None, A, A, A, A, None, None) == BAD       # ragged rows in BLOCK
    assert q(A, 128, 200, 0, BLK, WGT, None, A, A, A, A, None, None) == BAD       # ragged cols in BLOCK
    assert q(A, 128, 128, 0, BLK, ACT, A, A, A, A, A, None, None) == BAD          # amax given in BLOCK
    assert q(A, 128, 128, 0, BLK, ACT, None, A, A, A, None, None, None) == BAD    # q_t without scale_t
    assert q(A, 128, 128, 0, BLK, ACT, None, A + 8, A, None, None, None, None) == BAD  # misaligned q
    assert q(A, 128, 128, 0, TEN, ACT, None, A, A, None, None, None, None) == BAD  # TENSOR needs amax
    assert q(A, 128, 120, 0, TEN, ACT, A, A, A, None, None, None, None) == BAD     # TENSOR cols % 16
    assert q(A, 120, 128, 0, TEN, ACT, A, A, A, A, None, None, None) == BAD        # TENSOR rows % 16 with q_t
    assert q(None, 128, 128, 0, BLK, ACT, None, A, A, A, A, None, None) == BAD     # null input
    assert q(A, 128, 128, 0, BLK, ACT, None, None, A, None, None, None, None) == BAD  # null q
    # empty BLOCK tensors are a valid no-op that touches nothing
    assert q(None, 0, 128, 0, BLK, ACT, None, A, A, A, A, None, None) == P.PURO_OK


def _op(rows, red, scaling=P.SCALE_BLOCK, role=P.ROLE_ACT, fmt=0, data=A, scale=A, reserved=0):
    return P.puro_fp8_tensor_t(data, scale, rows, red, fmt, scaling, role, reserved)


def test_gemm_validation(lib):
    f = lib.puro_fp8_linear_fprop
    r = ctypes.byref
    x, w = _op(256, 384), _op(512, 384, role=P.ROLE_WEIGHT)
    assert f(r(x), r(w), None, None, 0, None, None) == BAD                       # no output
    assert f(r(x), r(w), A + 4, None, 0, None, None) == BAD                      # misaligned output
    assert f(r(x), r(_op(512, 256, role=P.ROLE_WEIGHT)), A, None, 0, None, None) == BAD  # K mismatch
    assert f(r(_op(256, 384, role=7)), r(w), A, None, 0, None, None) == BAD      # bad role
    assert f(r(x), r(_op(512, 384, scaling=P.SCALE_TENSOR)), A, None, 0, None, None) == BAD  # mixed scaling
    assert f(r(_op(200, 384)), r(w), A, None, 0, None, None) == BAD              # ragged BLOCK
    assert f(r(_op(256, 384, fmt=3)), r(w), A, None, 0, None, None) == BAD       # bad format
    assert f(r(_op(256, 384, reserved=1)), r(w), A, None, 0, None, None) == BAD  # reserved field
    assert f(r(_op(256, 384, data=0)), r(w), A, None, 0, None, None) == BAD      # null data
    assert f(r(_op(256, 384, scale=A + 1)), r(w), A, None, 0, None, None) == BAD  # misaligned scale
    assert f(r(_op(24, 40, scaling=P.SCALE_TENSOR)), r(_op(16, 40, scaling=P.SCALE_TENSOR)), A, None, 0, None,
             None) == BAD                                                         # TENSOR extents % 16
    assert f(None, r(w), A, None, 0, None, None) == BAD
    # empty output extent: valid no-op
    assert f(r(_op(0, 384)), r(w), A, None, 0, None, None) == P.PURO_OK


def test_dgrad_quantize_validation(lib):
    f = lib.puro_fp8_linear_dgrad_quantize
    r = ctypes.byref
    dy, wt = _op(256, 384), _op(512, 384, role=P.ROLE_WEIGHT)
    E4 = P.E4M3
    assert f(r(dy), r(wt), 2, None, A, A, A, A, None, None) == BAD             # bad output format
    assert f(r(dy), r(wt), E4, None, None, A, None, None, None, None) == BAD   # no rowwise codes
    assert f(r(dy), r(wt), E4, None, A, None, None, None, None, None) == BAD   # no rowwise scales
    assert f(r(dy), r(wt), E4, None, A, A, A, None, None, None) == BAD         # transposed codes without scales
    assert f(r(dy), r(wt), E4, None, A, A, None, A, None, None) == BAD         # scales without transposed codes
    assert f(r(dy), r(wt), E4, None, A + 8, A, None, None, None, None) == BAD  # misaligned codes
    assert f(r(dy), r(wt), E4, A + 2, A, A, None, None, None, None) == BAD     # misaligned dx
    assert f(r(dy), r(_op(512, 256, role=P.ROLE_WEIGHT)), E4, None, A, A, None, None, None, None) == BAD
    assert f(r(_op(256, 384, scaling=P.SCALE_TENSOR)), r(_op(512, 384, scaling=P.SCALE_TENSOR)), E4, None, A, A,
             None, None, None, None) == BAD                                     # BLOCK scaling only
    assert f(None, r(wt), E4, None, A, A, None, None, None, None) == BAD
    # an empty output extent is a valid no-op
    assert f(r(_op(0, 384)), r(wt), E4, None, A, A, A, A, None, None) == P.PURO_OK


def test_grouped_weight_quantize_validation(lib):
    f = lib.puro_fp8_quantize_weights
    W_ = P.puro_fp8_weight_t

    def table(*entries):
        t = (W_ * len(entries))()
        for i, e in enumerate(entries):
            t[i] = e
        return t

    good = W_(A, 256, 384, A, A, A, A)
    no_t = W_(A, 256, 384, A, A, None, None)
    assert f(None, 1, P.E4M3, None, None) == BAD                                   # no table
    assert f(table(good), -1, P.E4M3, None, None) == BAD                           # negative count
    assert f(table(good), 1, 5, None, None) == BAD                                 # bad format
    assert f(table(W_(A, 200, 384, A, A, A, A)), 1, P.E4M3, None, None) == BAD      # rows % 128
    assert f(table(good, no_t), 2, P.E4M3, None, None) == BAD                      # mixed transposed copies
    assert f(table(W_(A, 256, 384, A, A, A, None)), 1, P.E4M3, None, None) == BAD  # q_t without scale_t
    assert f(table(W_(A + 2, 256, 384, A, A, A, A)), 1, P.E4M3, None, None) == BAD  # misaligned input
    assert f(table(W_(A, 256, 384, None, A, A, A)), 1, P.E4M3, None, None) == BAD   # no codes buffer
    assert f(table(good, W_(A, 256, 384, A, A + 8, A, A)), 2, P.E4M3, None, None) == BAD  # checked before any launch
    # nothing to do: valid no-ops
    assert f(None, 0, P.E4M3, None, None) == P.PURO_OK
    assert f(table(W_(None, 0, 384, None, None, None, None)), 1, P.E4M3, None, None) == P.PURO_OK


def test_backward_validation(lib):
    f = lib.puro_fp8_linear_backward
    r = ctypes.byref
    # dY [256, 384], W^T [512, 384] -> dX [256, 512]; dY^T [384, 256], X^T [512, 256] -> dW [384, 512]
    dy, wt = _op(256, 384), _op(512, 384, role=P.ROLE_WEIGHT)
    dyt, xt = _op(384, 256), _op(512, 256)
    assert f(r(dy), r(wt), None, r(dyt), r(xt), A, None, 0, None, None) == BAD              # no dX
    assert f(r(dy), r(wt), A, r(dyt), r(xt), A + 4, None, 0, None, None) == BAD             # misaligned dW
    assert f(r(dy), r(wt), A, r(dyt), r(_op(512, 128)), A, None, 0, None, None) == BAD      # Wgrad reduction mismatch
    assert f(r(dy), r(_op(512, 256, role=P.ROLE_WEIGHT)), A, r(dyt), r(xt), A, None, 0, None, None) == BAD
    assert f(None, r(wt), A, r(dyt), r(xt), A, None, 0, None, None) == BAD
    # both empty: a valid no-op
    assert f(r(_op(0, 384)), r(wt), A, r(_op(0, 256)), r(xt), A, None, 0, None, None) == P.PURO_OK


def test_noalloc_wgrad_checks_arguments_before_the_scratch_limit(lib):
    # every call here is answered on the host before any CUDA call
    f = lib.puro_fp8_linear_wgrad_noalloc
    r = ctypes.byref
    big_dyt, big_xt = _op(2048, 32768), _op(1792, 32768)   # a valid split would need 58.7 MB > 40 MiB
    assert P.puro_fp8_workspace_size(2048, 1792, 32768) > 40 * 1024 * 1024
    assert f(r(big_dyt), r(big_xt), A, None, None) == P.PURO_ERR_UNSUPPORTED
    assert f(r(big_dyt), r(_op(1792, 32640)), A, None, None) == BAD          # reduction mismatch
    assert f(r(_op(2048, 32768, fmt=9)), r(big_xt), A, None, None) == BAD    # bad format
    assert f(r(big_dyt), r(big_xt), A + 4, None, None) == BAD               # misaligned dW
    assert f(r(big_dyt), r(_op(1792, 32768, scaling=P.SCALE_TENSOR)), A, None, None) == BAD  # mixed scaling
    assert f(None, r(big_xt), A, None, None) == BAD
    assert f(r(_op(0, 32768)), r(big_xt), A, None, None) == P.PURO_OK       # empty output: no-op


def test_backward_plan_groups_every_c5_and_c6_linear(lib):
    # host-only: with the bench's workspace (large enough for any split) the
    # Dgrad and the Wgrad of every linear share one launch -- the qkv and
    # o_proj Wgrads, which would split, join their Dgrads unsplit
    big = 1 << 30
    for M, shapes in ((32768, [(2048, 1536), (1536, 1536), (17920, 1536), (1536, 8960)]),
                      (8192, [(4096, 2048), (2048, 2048), (12288, 2048), (2048, 6144)])):
        for N, K in shapes:
            assert lib.puro_fp8_linear_backward_launches(M, N, K, big) == 1, (M, N, K)
            assert lib.puro_fp8_linear_backward_launches(M, N, K, 0) == 1, (M, N, K)
    assert lib.puro_fp8_linear_backward_launches(0, 2048, 1536, big) == 0
    # a Dgrad that splits its reduction (2 output tiles, reduction 32768) is
    # never grouped: its two launches (partials, reduction) plus the Wgrad's
    assert lib.puro_fp8_linear_backward_launches(512, 32768, 256, big) == 3
    assert lib.puro_fp8_linear_backward_launches(512, 32768, 256, 0) == 1  # no workspace: both unsplit, grouped


def test_bf16_gemm_validation(lib):
    assert lib.puro_bf16_linear_fprop(A, A, A, 12, 16, 16, None, None) == BAD   # M % 8
    assert lib.puro_bf16_linear_fprop(A, A + 2, A, 16, 16, 16, None, None) == BAD
    assert lib.puro_bf16_linear_dgrad(None, A, A, 16, 16, 16, None, None) == BAD
    assert lib.puro_bf16_linear_wgrad(A, A, A, 16, -8, 16, None, None) == BAD
    assert lib.puro_bf16_linear_fprop(A, A, A, 0, 16, 16, None, None) == P.PURO_OK


def test_scale_buffer_size(lib):
    assert lib.puro_fp8_scale_bytes(256, 1536) == 256 * 3 * 4      # 12 k-blocks -> 3 groups
    assert lib.puro_fp8_scale_bytes(128, 8960) == 128 * 18 * 4     # 70 k-blocks -> 18 groups
    assert lib.puro_fp8_scale_bytes(0, 128) == 0
    assert int(np.prod(P.scale_vec_shape(256, 8960))) == lib.puro_fp8_scale_bytes(256, 8960)


def test_workspace_size_plans_split_reductions(lib):
    # Wgrad of qkv / o_proj at 32768 tokens: 96 / 72 output tiles < 152 SMs
    assert lib.puro_fp8_workspace_size(2048, 1536, 32768) == 3 * 2048 * 1536 * 4
    assert lib.puro_fp8_workspace_size(1536, 1536, 32768) == 2 * 1536 * 1536 * 4
    # enough tiles, or too short a reduction: no split
    assert lib.puro_fp8_workspace_size(17920, 1536, 32768) == 0
    assert lib.puro_fp8_workspace_size(1536, 1536, 256) == 0
    assert lib.puro_fp8_workspace_size(0, 1536, 32768) == 0


def test_get_status_validation(lib):
    out = ctypes.c_int32(0)
    assert lib.puro_fp8_get_status(None, ctypes.byref(out), None) == BAD
    assert lib.puro_fp8_get_status(A, None, None) == BAD


@pytest.mark.skipif(torch.cuda.is_available(), reason="checks the no-GPU failure mode")
def test_valid_call_without_gpu_fails_loudly(lib):
    x, w = _op(256, 384), _op(512, 384, role=P.ROLE_WEIGHT)
    st = lib.puro_fp8_linear_fprop(ctypes.byref(x), ctypes.byref(w), A, None, 0, None, None)
    assert st == P.PURO_ERR_CUDA


def test_binding_refuses_host_tensors():
    x = torch.zeros(128, 128, dtype=torch.bfloat16)
    with pytest.raises(ValueError):
        P.puro_fp8_amax(x, torch.zeros(1, dtype=torch.int32))


def test_gemm_tile_knob_validates_on_the_host(lib):
    assert lib.puro_set_gemm_tile_n(192) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_set_gemm_tile_n(-1) == P.PURO_ERR_INVALID_ARG
    for v in (224, 256, 0):
        assert lib.puro_set_gemm_tile_n(v) == P.PURO_OK


def test_fused_rmsnorm_validates_on_the_host(lib):
    fake = 0x100000  # never dereferenced: every call below is refused before any CUDA call
    args = dict(gamma=None, eps=ctypes.c_float(1e-6), fmt=P.E4M3, rstd=fake, y=None, q=fake, scale=fake,
                q_t=None, scale_t=None, stream=None)

    def call(rows, cols, **kw):
        a = dict(args, **kw)
        return lib.puro_fp8_quantize_rmsnorm(fake, rows, cols, a["gamma"], a["eps"], a["fmt"], a["rstd"], a["y"],
                                             a["q"], a["scale"], a["q_t"], a["scale_t"], None, a["stream"])

    assert call(200, 256) == P.PURO_ERR_INVALID_ARG            # rows not a multiple of 128
    assert call(256, 200) == P.PURO_ERR_INVALID_ARG            # cols not a multiple of 128
    assert call(256, 256, fmt=7) == P.PURO_ERR_INVALID_ARG     # unknown format
    assert call(256, 256, eps=ctypes.c_float(-1.0)) == P.PURO_ERR_INVALID_ARG
    assert call(256, 256, q_t=fake) == P.PURO_ERR_INVALID_ARG  # transposed codes without their scales
    assert call(256, 256, rstd=fake + 2) == P.PURO_ERR_INVALID_ARG  # misaligned rstd
    assert call(0, 256) == P.PURO_OK                           # empty: nothing to do
    assert lib.puro_rmsnorm_bf16(fake, 4, 12, None, ctypes.c_float(1e-6), fake, fake, None) == P.PURO_ERR_INVALID_ARG


def test_fused_swiglu_validates_on_the_host(lib):
    fake = 0x100000  # never dereferenced: every call below is refused before any CUDA call

    def call(rows, cols, ld, fmt=P.E4M3, gate=fake, up=fake, y=None, q_t=None, scale_t=None):
        return lib.puro_fp8_quantize_swiglu(gate, up, rows, cols, ld, fmt, y, fake, fake, q_t, scale_t, None, None)

    assert call(200, 256, 512) == P.PURO_ERR_INVALID_ARG            # rows not a multiple of 128
    assert call(256, 200, 400) == P.PURO_ERR_INVALID_ARG            # cols not a multiple of 128
    assert call(256, 256, 128) == P.PURO_ERR_INVALID_ARG            # row stride shorter than a row
    assert call(256, 256, 260) == P.PURO_ERR_INVALID_ARG            # row stride not 16-byte aligned
    assert call(256, 256, 512, fmt=7) == P.PURO_ERR_INVALID_ARG     # unknown format
    assert call(256, 256, 512, q_t=fake) == P.PURO_ERR_INVALID_ARG  # transposed codes without their scales
    assert call(256, 256, 512, up=fake + 2) == P.PURO_ERR_INVALID_ARG  # misaligned up
    assert call(256, 256, 512, up=None) == P.PURO_ERR_INVALID_ARG
    assert call(0, 256, 512) == P.PURO_OK                           # empty: nothing to do
    assert lib.puro_swiglu_bf16(fake, fake, 4, 12, 16, fake, None) == P.PURO_ERR_INVALID_ARG  # cols % 8
    assert lib.puro_swiglu_bf16(fake, fake, 4, 16, 8, fake, None) == P.PURO_ERR_INVALID_ARG   # ld < cols
    assert lib.puro_swiglu_bf16(fake, fake, 0, 16, 16, fake, None) == P.PURO_OK


def test_muonh_validates_on_the_host(lib):
    fake = 0x100000  # never dereferenced: every call below is refused before any CUDA call
    ws = lib.puro_muonh_workspace_size(1 << 20)
    assert ws > 0 and ws % 24 == 0 and lib.puro_muonh_workspace_size(0) == 0
    # chunks of n/4096 values, clamped to [4096, 65536]: 24 bytes per chunk
    assert lib.puro_muonh_workspace_size(4096) == 24
    assert lib.puro_muonh_workspace_size(4100) == 48
    assert lib.puro_muonh_workspace_size(1 << 24) == 24 * 1024
    assert lib.puro_muonh_workspace_size(1 << 30) == 24 * (1 << 14)
    assert lib.puro_muonh_reduce(fake, fake, 6, fake, fake, ws, None) == P.PURO_ERR_INVALID_ARG  # n % 4
    assert lib.puro_muonh_reduce(fake + 8, fake, 1 << 20, fake, fake, ws, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_reduce(fake, fake, 1 << 20, fake, fake, ws - 8, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_apply(fake, fake, 1 << 20, fake, -1.0, 1.0, None, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_apply(fake, fake, 1 << 20, fake, 0.1, 0.0, None, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_apply(fake, fake, 1 << 20, fake, float("nan"), 1.0, None, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_apply(fake, fake, 1 << 20, fake, 0.1, 1.0, fake + 4, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_step(fake, fake, 0, 0.1, 1.0, fake, None, 0, None, None) == P.PURO_OK


def test_muonh_grouped_validates_on_the_host(lib):
    fake = 0x100000
    M = P.puro_muonh_matrix_t
    good = M(fake, fake + 0x10000, None, 1 << 16, 1.0)
    arr = (M * 3)(good, M(fake, fake, None, 6, 1.0), good)            # the middle one has n % 4 != 0
    assert lib.puro_muonh_step_grouped(arr, 3, 0.1, fake, fake, 1 << 20, None) == P.PURO_ERR_INVALID_ARG
    arr = (M * 2)(good, M(fake, fake, None, 1024, -1.0))               # negative radius
    assert lib.puro_muonh_step_grouped(arr, 2, 0.1, fake, fake, 1 << 20, None) == P.PURO_ERR_INVALID_ARG
    arr = (M * 2)(good, good)
    need = lib.puro_muonh_grouped_workspace_size(arr, 2)
    assert need == 2 * lib.puro_muonh_workspace_size(1 << 16)
    assert lib.puro_muonh_step_grouped(arr, 2, 0.1, fake, fake, need - 8, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_step_grouped(arr, 2, float("inf"), fake, fake, need, None) == P.PURO_ERR_INVALID_ARG
    assert lib.puro_muonh_step_grouped(arr, 0, 0.1, None, None, 0, None) == P.PURO_OK
    # launches of 128 matrices reuse the scratch: 200 matrices need the larger batch only
    big = (M * 200)(*([good] * 200))
    assert lib.puro_muonh_grouped_workspace_size(big, 200) == 128 * lib.puro_muonh_workspace_size(1 << 16)
