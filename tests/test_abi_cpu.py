"""The C-ABI library without a GPU: it builds, loads, exports every symbol that
include/dqt.h declares, and rejects bad arguments on the host before any CUDA
call.  No kernel is launched here."""
import ctypes as C
import os
import re

import pytest

from paper_2412_04787_gb300 import build as dqt_build
from paper_2412_04787_gb300 import dqt

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "dqt.h")


@pytest.fixture(scope="module")
def L():
    dqt_build.build()
    return dqt.lib()


def _declared():
    src = open(HEADER).read()
    src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
    return sorted(set(re.findall(r"\b(dqt_[a-z0-9_]+)\s*\(", src)))


def test_header_symbols_exported(L):
    names = _declared()
    assert len(names) >= 12
    assert sorted(dqt.EXPORTED) == names
    for n in names:
        assert hasattr(L, n), n  # dlsym succeeds


def test_hot_path_entry_points_present():
    for n in ["dqt_act_quant", "dqt_bitlinear_fwd", "dqt_bitlinear_bwd_dx",
              "dqt_bitlinear_bwd_dw_update", "dqt_sr_update"]:
        assert n in _declared()


def test_grid_for_bits(L):
    g = dqt.dqt_grid_t()
    assert L.dqt_grid_for_bits(C.c_float(1.58), C.byref(g)) == 0 and (g.qmin, g.qmax) == (-1, 1)
    for n in range(2, 9):
        assert L.dqt_grid_for_bits(C.c_float(n), C.byref(g)) == 0
        assert (g.qmin, g.qmax) == (-(2 ** (n - 1)), 2 ** (n - 1) - 1)
    for bad in (1.0, 9.0, 2.5):
        assert L.dqt_grid_for_bits(C.c_float(bad), C.byref(g)) == dqt.DQT_ERR_ARG


def test_status_strings(L):
    for s in range(6):
        assert L.dqt_status_string(s).startswith(b"DQT")
    assert L.dqt_status_string(99) == b"DQT: unknown status"


def _p(addr):
    return C.c_void_p(addr)


def test_argument_validation_without_launch(L):
    g = dqt.dqt_grid_t(-1, 1)
    A = _p(0x10000)  # never dereferenced: validation fails before any CUDA call
    # null pointers
    assert L.dqt_bitlinear_fwd(None, A, A, 1.0, g, 4, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dx(A, None, 1.0, 4, 8, 8, A, A, 1 << 20, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dx(A, A, 1.0, 4, 8, 8, A, None, 1 << 20, None) == dqt.DQT_ERR_ARG
    assert L.dqt_act_quant(A, 4, 8, None, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_act_quant_images(A, 4, 8, None, A, None, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_img(None, A, A, 1.0, g, 4, 8, 8, A, None, None, 0, None) == dqt.DQT_ERR_ARG
    # sizes
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, g, 0, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ARG
    assert L.dqt_act_quant(A, -1, 8, A, A, None) == dqt.DQT_ERR_ARG
    # the dX workspace must hold the weight's bf16 image
    assert L.dqt_bwd_dx_workspace_size(4, 8, 8) >= 8 * 8 * 2
    assert L.dqt_bitlinear_bwd_dx(A, A, 1.0, 4, 8, 8, A, A, 64, None) == dqt.DQT_ERR_ARG
    # K, N multiples of 8 and 16-byte alignment; the forward's workspace holds
    # both operands' bf16 images
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, g, 4, 12, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_fwd_workspace_size(4, 8, 8) >= (4 + 8) * 8 * 2
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, g, 4, 8, 8, A, None, A, 16, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_img(A, A, A, 1.0, g, 4, 12, 8, A, None, None, 0, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_bwd_dx(A, A, 1.0, 4, 8, 20, A, A, 1 << 20, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_bwd_dx_img(A, A, 1.0, 4, 8, 20, A, None, 0, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_fwd(_p(0x10004), A, A, 1.0, g, 4, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ALIGN
    # the forward's and dX's optional workspace for last-wave slice partials:
    # when a cut is planned (a shape whose tiles leave the last wave short),
    # a workspace below the size, or misaligned, is refused before any launch
    # (8192 x 2048 outputs: 256 pair tiles, 3.4 waves on 74 or 76 SM pairs)
    T, K, N = 8192, 5632, 2048
    need = L.dqt_fwd_img_workspace_size(T, K, N)
    assert need > 0
    assert L.dqt_bitlinear_fwd_img(A, A, A, 1.0, g, T, K, N, A, None, A, need - 16, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_img(A, A, A, 1.0, g, T, K, N, A, None, _p(0x10008), need, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_fwd_workspace_size(T, K, N) >= (T + N) * K * 2 + need
    T, N, K = 8192, 5632, 2048
    need = L.dqt_bwd_dx_img_workspace_size(T, N, K)
    assert need > 0
    assert L.dqt_bitlinear_bwd_dx_img(A, A, 1.0, T, N, K, A, A, need - 16, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bwd_dx_workspace_size(T, N, K) >= N * K * 2 + need
    # one pair tile, or a reduction shorter than 4096: nothing to cut
    assert L.dqt_fwd_img_workspace_size(256, 512, 256) == 0
    assert L.dqt_fwd_img_workspace_size(8192, 2048, 5632) == 0
    assert L.dqt_bwd_dx_img_workspace_size(8192, 2048, 5632) == 0
    # stacked weights: the split a positive multiple of 256 below N, both scales positive
    assert L.dqt_bitlinear_fwd_img_pair(A, A, A, 200, 1.0, 1.0, g, 4, 8, 512, A, None, None, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_img_pair(A, A, A, 512, 1.0, 1.0, g, 4, 8, 512, A, None, None, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_img_pair(A, A, A, 256, 1.0, 0.0, g, 4, 8, 512, A, None, None, 0, None) == dqt.DQT_ERR_ARG
    hp = dqt.adamw()
    sr = dqt.sr_stream()
    assert L.dqt_bitlinear_bwd_dw_update_img_pair(A, A, A, 100, 1.0, 1.0, A, A, hp, sr, sr, g, 4, 512, 8,
                                                  None, None, None, None, None, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dw_update_img_pair(A, A, None, 256, 1.0, 1.0, A, A, hp, sr, sr, g, 4, 512, 8,
                                                  None, None, None, None, None, 0, None) == dqt.DQT_ERR_ARG
    # the E4M3 image of wider codes is the split image: rows of K codes, K a
    # multiple of 16
    g8 = dqt.dqt_grid_t(-128, 127)
    assert L.dqt_bitlinear_bwd_dw_update_img_pair(A, A, A, 256, 1.0, 1.0, A, A, hp, sr, sr, g8, 4, 512, 8,
                                                  None, None, A, None, None, 0, None) == dqt.DQT_ERR_ALIGN
    # the stacked FP8 forward: the same split rule, and the E4M3-exact grid
    assert L.dqt_bitlinear_fwd_fp8_pair(A, A, A, 200, 1.0, 1.0, g, 4, 16, 512, A, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_fp8_pair(A, A, A, 256, 1.0, 0.0, g, 4, 16, 512, A, None, None) == dqt.DQT_ERR_ARG
    # wide grids take the split image: the reduction a multiple of 128
    assert L.dqt_bitlinear_fwd_fp8_pair(A, A, A, 256, 1.0, 1.0, g8, 4, 16, 512, A, None, None) == dqt.DQT_ERR_ALIGN
    # bad grid / scale
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, dqt.dqt_grid_t(2, 1), 4, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, dqt.dqt_grid_t(-129, 1), 4, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd(A, A, A, 0.0, g, 4, 8, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_ARG
    # int32 accumulator range: K * 128 * 128 must fit int32
    g8 = dqt.dqt_grid_t(-128, 127)
    assert L.dqt_bitlinear_fwd(A, A, A, 1.0, g8, 4, 1 << 17, 8, A, None, A, 1 << 24, None) == dqt.DQT_ERR_RANGE


def test_update_argument_validation(L):
    g = dqt.dqt_grid_t(-1, 1)
    A = _p(0x10000)
    hp = dqt.adamw()
    sr = dqt.sr_stream()
    ok = C.byref(hp), C.byref(sr)
    # partial state
    assert L.dqt_bitlinear_bwd_dw_update_img(A, A, A, 1.0, None, A, *ok, g, 4, 8, 8, None, None, None, None, None, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dw_update(A, A, A, A, 1.0, None, A, *ok, g, 4, 8, 16, None, None, A, 1 << 20, None) == dqt.DQT_ERR_ARG
    # gradient-only mode needs dW_out
    assert L.dqt_bitlinear_bwd_dw_update_img(A, A, None, 1.0, None, None, *ok, g, 4, 8, 8, None, None, None, None, None, 0, None) == dqt.DQT_ERR_ARG
    # an image of the updated codes needs the update
    assert L.dqt_bitlinear_bwd_dw_update_img(A, A, None, 1.0, None, None, *ok, g, 4, 8, 8, A, A, None, None, None, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dw_update_img(A, A, None, 1.0, None, None, *ok, g, 4, 8, 8, A, None, A, None, None, 0, None) == dqt.DQT_ERR_ARG
    # the split E4M3 image of wider codes needs K a multiple of 16
    assert L.dqt_bitlinear_bwd_dw_update_img(A, A, A, 1.0, A, A, *ok, dqt.dqt_grid_t(-128, 127), 4, 8, 8, None, None, A, None, None, 0, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_bwd_dw_update(A, A, A, None, 1.0, None, None, *ok, g, 4, 8, 16, None, None, A, 1 << 20, None) == dqt.DQT_ERR_ARG
    # the int8 call needs the X_tilde image in its workspace, 16-byte int8 rows
    assert L.dqt_bwd_dw_workspace_size(4, 8, 16) >= 4 * 16 * 2
    assert L.dqt_bitlinear_bwd_dw_update(A, A, A, A, 1.0, A, A, *ok, g, 4, 8, 16, None, None, A, 64, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dw_update(A, A, A, A, 1.0, A, A, *ok, g, 4, 8, 24, None, None, A, 1 << 20, None) == dqt.DQT_ERR_ALIGN
    bad = dqt.adamw(step=0)
    assert L.dqt_sr_update(A, A, 1.0, A, A, C.byref(bad), C.byref(sr), g, 16, None, None) == dqt.DQT_ERR_ARG
    bad = dqt.adamw(beta1=1.0)
    assert L.dqt_sr_update(A, A, 1.0, A, A, C.byref(bad), C.byref(sr), g, 16, None, None) == dqt.DQT_ERR_ARG
    badsr = dqt.sr_stream(round_mode=2)
    assert L.dqt_sr_update(A, A, 1.0, A, A, C.byref(hp), C.byref(badsr), g, 16, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_sr_update(A, A, -1.0, A, A, *ok, g, 16, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_sr_update(_p(0x10008), A, 1.0, A, A, *ok, g, 16, None, None) == dqt.DQT_ERR_ALIGN


def test_absmean_workspace(L):
    assert L.dqt_absmean_workspace_size() >= 8 * 1025
    s = C.c_float()
    A = _p(0x10000)
    assert L.dqt_absmean_init(A, 16, dqt.dqt_grid_t(-1, 1), A, C.byref(s), A, 8, None) == dqt.DQT_ERR_ARG


def test_fp8_argument_validation(L):
    A = _p(0x10000)
    t = dqt.dqt_grid_t(-1, 1)
    g8 = dqt.dqt_grid_t(-128, 127)
    # activations: K a multiple of 16, outputs required
    assert L.dqt_act_quant_fp8(A, 4, 24, A, A, None, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_act_quant_fp8(A, 4, 32, None, A, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_act_quant_fp8(A, 0, 32, A, A, None, None) == dqt.DQT_ERR_ARG
    # weight image: codes beyond 16 in magnitude are not exact in E4M3
    assert L.dqt_codes_to_fp8(A, 64, g8, A, None) == dqt.DQT_ERR_RANGE
    assert L.dqt_codes_to_fp8(A, 64, dqt.dqt_grid_t(-32, 31), A, None) == dqt.DQT_ERR_RANGE
    assert L.dqt_codes_to_fp8(A, 0, t, A, None) == dqt.DQT_ERR_ARG
    # forward
    assert L.dqt_bitlinear_fwd_fp8(A, A, A, 1.0, g8, 4, 32, 8, A, None, None) == dqt.DQT_ERR_ALIGN
    # the split image: K a multiple of 16
    assert L.dqt_codes_to_fp8_split(A, 4, 24, A, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_codes_to_fp8_split(A, 0, 32, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_fp8(A, A, A, 1.0, t, 4, 24, 8, A, None, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_fwd_fp8(A, A, A, 1.0, t, 4, 32, 12, A, None, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_bitlinear_fwd_fp8(A, A, A, 0.0, t, 4, 32, 8, A, None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_fwd_fp8(None, A, A, 1.0, t, 4, 32, 8, A, None, None) == dqt.DQT_ERR_ARG


def test_packed_and_adafactor_argument_validation(L):
    A = _p(0x10000)
    g = dqt.dqt_grid_t(-1, 1)
    hp = dqt.adamw()
    sr = dqt.sr_stream()
    af = dqt.adafactor()
    assert L.dqt_pack_ternary(None, 16, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_pack_ternary(_p(0x10004), 16, A, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_unpack_ternary(A, 0, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_packed_to_bf16(A, 16, _p(0x10002), None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_sr_update_packed(A, A, 1.0, A, None, C.byref(hp), C.byref(sr), 16, None,
                                  None) == dqt.DQT_ERR_ARG
    assert L.dqt_bitlinear_bwd_dw_update_packed(A, A, A, 1.0, A, A, C.byref(hp), C.byref(sr), 4,
                                                8, 12, None, None, None, 0, None) == dqt.DQT_ERR_ALIGN
    # Adafactor: workspace size, hyper-parameters, packed codes need the ternary grid
    assert L.dqt_adafactor_workspace_size(64, 64) > 0
    assert L.dqt_adafactor_workspace_size(0, 64) == 0
    assert L.dqt_bwd_dw_adafactor_workspace_size(128, 64, 64) >= 64 * 64 * 4
    nb = L.dqt_adafactor_workspace_size(64, 64)
    W = _p(0x100000)  # 256-byte aligned
    assert L.dqt_adafactor_stats(A, A, 0, 1.0, A, A, C.byref(dqt.adafactor(step=0)), 64, 64, A, A,
                                 A, W, nb, None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_stats(A, A, 0, 1.0, A, A, C.byref(dqt.adafactor(clip_d=0.0)), 64, 64,
                                 A, A, A, W, nb, None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_stats(A, A, 0, 1.0, A, A, C.byref(af), 64, 64, A, A, A, W, nb - 1,
                                 None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_stats(A, A, 0, 1.0, A, A, C.byref(af), 64, 64, None, A, A, W, nb,
                                 None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_stats(A, A, 0, 1.0, A, A, C.byref(af), 64, 64, A, A, A, _p(0x10010),
                                 nb, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_adafactor_apply(A, A, 1, A, A, A, 1, C.byref(sr), dqt.dqt_grid_t(-2, 1), 64, 64,
                                 None, None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_apply(A, A, 0, A, A, A, 0, C.byref(sr), g, 64, 64, None,
                                 None) == dqt.DQT_ERR_ARG
    assert L.dqt_adafactor_apply(A, A, 0, A, A, A, 1, C.byref(sr), g, 64, 66, None,
                                 None) == dqt.DQT_ERR_ALIGN


def test_decoder_support_argument_validation(L):
    A = _p(0x10000)
    # rotary embedding: D a multiple of 8, aligned pointers, inverse 0 or 1
    assert L.dqt_rope_bf16(None, A, A, 4, 4, 2, 64, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_rope_bf16(A, A, A, 0, 4, 2, 64, 0, None) == dqt.DQT_ERR_ARG
    assert L.dqt_rope_bf16(A, A, A, 4, 4, 2, 64, 2, None) == dqt.DQT_ERR_ARG
    assert L.dqt_rope_bf16(A, A, A, 4, 4, 2, 36, 0, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_rope_bf16(_p(0x10008), A, A, 4, 4, 2, 64, 0, None) == dqt.DQT_ERR_ALIGN
    # cross-entropy: V a multiple of 8, outputs required
    assert L.dqt_cross_entropy_fwd_bf16(A, A, 4, 36, A, A, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_cross_entropy_fwd_bf16(A, A, 4, 64, None, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_cross_entropy_fwd_bf16(A, A, 0, 64, A, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_cross_entropy_bwd_bf16(A, A, A, None, 4, 64, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_cross_entropy_bwd_bf16(A, A, A, A, 4, 64, _p(0x10004), None) == dqt.DQT_ERR_ALIGN
    # SwiGLU: n a multiple of 8, every pointer aligned
    assert L.dqt_swiglu_bf16(A, A, None, 64, None) == dqt.DQT_ERR_ARG
    assert L.dqt_swiglu_bf16(A, A, A, 12, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_swiglu_bwd_bf16(A, A, A, A, _p(0x10002), 64, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_swiglu_bwd_bf16(A, A, A, A, A, 0, None) == dqt.DQT_ERR_ARG
    # RMSNorm: D a multiple of 8 and at most 2048; the backward needs its workspace
    assert L.dqt_rmsnorm_bf16(A, A, C.c_float(1e-6), 4, 12, A, A, None) == dqt.DQT_ERR_ALIGN
    assert L.dqt_rmsnorm_bf16(A, A, C.c_float(1e-6), 4, 4096, A, A, None) == dqt.DQT_ERR_RANGE
    assert L.dqt_rmsnorm_bf16(A, A, C.c_float(-1.0), 4, 64, A, A, None) == dqt.DQT_ERR_ARG
    assert L.dqt_rmsnorm_bwd_workspace_size(4, 4096) == 0
    assert L.dqt_rmsnorm_bwd_bf16(A, A, A, A, 4, 64, A, A, None, 0, None) == dqt.DQT_ERR_ARG


def test_sr_stream_offset_validation(L):
    """elem0 of the SR stream: negative -> DQT_ERR_ARG, not a multiple of 4 ->
    DQT_ERR_ALIGN (one Philox block per four elements); Adafactor's calls need
    elem0 = 0.  The host block of constants records elem0 / 4."""
    g = dqt.dqt_grid_t(-1, 1)
    hp = dqt.adamw(lr=1e-3, step=1)
    out = (C.c_uint8 * 256)()
    n = L.dqt_update_consts_size()
    assert n <= 80  # fits the shared-memory slot the GEMM kernels copy it to
    ok = dqt.sr_stream(seed=1, tensor_id=2, elem0=1 << 36)
    assert L.dqt_update_consts(C.byref(hp), C.byref(ok), g, C.c_float(10.0), out, 256) == dqt.DQT_OK
    blk0 = int.from_bytes(bytes(out[n - 8: n]), "little")
    assert blk0 == (1 << 36) // 4
    for bad, rc in [(-4, dqt.DQT_ERR_ARG), (2, dqt.DQT_ERR_ALIGN), (6, dqt.DQT_ERR_ALIGN)]:
        sr = dqt.sr_stream(seed=1, tensor_id=2, elem0=bad)
        assert L.dqt_update_consts(C.byref(hp), C.byref(sr), g, C.c_float(10.0), out, 256) == rc
        A = _p(0x10000)
        assert L.dqt_sr_update(A, A, C.c_float(10.0), A, A, C.byref(hp), C.byref(sr), g, 64,
                               None, None) == rc
    sr = dqt.sr_stream(seed=1, tensor_id=2, elem0=16)
    A = _p(0x10000)
    assert L.dqt_adafactor_apply(A, A, 0, A, A, A, 1, C.byref(sr), g, 8, 8, None,
                                 None) == dqt.DQT_ERR_ARG


def test_dw_group_argument_validation(L):
    """The grouped weight-gradient call checks both problems on the host
    before it launches anything."""
    g = dqt.dqt_grid_t(-1, 1)
    hp = dqt.adamw()
    sr = dqt.sr_stream()
    a = 0x10000

    def prob(N=512, K=256, N0=0, W=a, sr1=None, W8=None):
        pr = dqt.dqt_dw_problem_t()
        pr.dY, pr.Xdq, pr.W, pr.m, pr.v = a, a, W, a, a
        pr.N, pr.K, pr.N0 = N, K, N0
        pr.s_w0, pr.s_w1 = 1.0, 1.0
        pr.sr0 = C.pointer(sr)
        pr.sr1 = C.pointer(sr1) if sr1 is not None else None
        pr.W8_next = W8
        return pr

    def call(p0, p1, n=2):
        arr = (dqt.dqt_dw_problem_t * 2)(p0, p1)
        return L.dqt_bitlinear_bwd_dw_update_group(arr, n, C.byref(hp), g, 4, None)

    assert L.dqt_bitlinear_bwd_dw_update_group(None, 2, C.byref(hp), g, 4, None) == dqt.DQT_ERR_ARG
    assert call(prob(), prob(), n=1) == dqt.DQT_ERR_ARG
    assert call(prob(), prob(W=None)) == dqt.DQT_ERR_ARG             # no codes
    assert call(prob(N0=256), prob()) == dqt.DQT_ERR_ARG             # stacked without sr1
    assert call(prob(N0=200, sr1=sr), prob()) == dqt.DQT_ERR_ARG     # split not on a tile
    assert call(prob(), prob(K=260)) == dqt.DQT_ERR_ALIGN            # K % 8
    assert call(prob(), prob(W=a + 4)) == dqt.DQT_ERR_ALIGN          # 16-byte alignment
    g8 = dqt.dqt_grid_t(-128, 127)
    arr = (dqt.dqt_dw_problem_t * 2)(prob(K=264, W8=a), prob())
    # the split E4M3 image of wide codes needs K % 16
    assert L.dqt_bitlinear_bwd_dw_update_group(arr, 2, C.byref(hp), g8, 4, None) == dqt.DQT_ERR_ALIGN
    bad = dqt.adamw(step=0)
    arr = (dqt.dqt_dw_problem_t * 2)(prob(), prob())
    assert L.dqt_bitlinear_bwd_dw_update_group(arr, 2, C.byref(bad), g, 4, None) == dqt.DQT_ERR_ARG
