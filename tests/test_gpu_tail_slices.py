"""The forward's and dX's last wave cut into reduction slices.

When a GEMM's 256 x 256 output tiles leave the last wave of the persistent
2-SM kernel short, the tiles of that wave are cut into slices of the
reduction whose fp32 partials go to the caller's workspace; the last slice
to finish a region adds them in slice order and applies the epilogue.  Forward: every partial is
an exact integer, so Y and the int32 accumulators equal the uncut kernel's
bit for bit (and the oracle's).  dX: a fixed fp32 order, reproducible, within
the dX tolerance of the fp64 oracle and within one bf16 rounding of the uncut
kernel.  Shapes: the LLaMA-MLP projections and a ragged one whose tail tiles
include the partial last row and column tiles.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2412_04787_gb300 import dqt, inputs

pytestmark = pytest.mark.gpu

REL_TOL = 2e-2


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2412_04787_gb300 import build
    build.build()
    dqt.lib()
    yield
    torch.cuda.synchronize()


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _tail_rows(T):
    """Rows of the last row tiles (where the cut tiles lie), the last row
    included, and one row of the first tile."""
    return np.unique(np.array([0, T - 1, T - 2, T - 255, T - 700, T - 1000, max(T - 1500, 1)]))


# (T, K, N, cut planned): the LLaMA-MLP down projection (256 output tiles for
# 76 SM pairs, a 5632-long reduction), a ragged shape whose last-wave tiles
# include the partial last row and column tiles, and the gate/up projection
# (704 tiles, a 2048-long reduction: no cut, the workspace size is 0)
FWD_SHAPES = [(8192, 5632, 2048, True), (4896, 4104, 1032, True), (8192, 2048, 5632, False)]


@pytest.mark.parametrize("T,K,N,cut", FWD_SHAPES)
def test_fwd_cut_equals_uncut_and_oracle(T, K, N, cut):
    assert (dqt.dqt_fwd_img_workspace_size(T, K, N) > 0) == cut
    X = inputs.normal((T, K), 1.0, seed=T + K, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=N)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    s_w = float(s_w)
    _, s_x, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    acc1 = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y1 = dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, s_w, (qmin, qmax), acc_out=acc1)
    acc0 = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y0 = dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, s_w, (qmin, qmax), acc_out=acc0, ws=False)
    dqt.dqt_check_device_status()
    assert torch.equal(acc1, acc0)
    assert torch.equal(Y1.view(torch.int16), Y0.view(torch.int16))
    rows = _tail_rows(T)
    q, s, _, _ = oracle.act_quant(bits(X[torch.from_numpy(rows)]))
    Yr, accr = oracle.fwd(q, s, c, np.float32(s_w))
    it = torch.from_numpy(rows).cuda()
    assert np.array_equal(acc1[it].cpu().numpy(), accr)
    assert np.array_equal(bits(Y1[it]), Yr)


def test_fwd_cut_through_int8_call():
    """The int8 call's workspace holds the cut's partials after the images:
    identical bytes to the image call."""
    T, K, N = 8192, 5632, 2048
    X = inputs.normal((T, K), 1.0, seed=5, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=6)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    Wc = torch.from_numpy(c).cuda()
    Y = dqt.dqt_bitlinear_fwd(Xq, s_x, Wc, float(s_w), (qmin, qmax))
    _, s_x2, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    Y2 = dqt.dqt_bitlinear_fwd_img(q_img, s_x2, dqt.dqt_codes_to_bf16(Wc), float(s_w), (qmin, qmax),
                                   ws=False)
    dqt.dqt_check_device_status()
    assert torch.equal(Y.view(torch.int16), Y2.view(torch.int16))


# (T, N, K, cut planned): dX's output is T x K, reduced over N
DX_SHAPES = [(8192, 5632, 2048, True), (4896, 4104, 1032, True), (8192, 2048, 5632, False)]


@pytest.mark.parametrize("T,N,K,cut", DX_SHAPES)
def test_dx_cut_reproducible_and_within_tolerance(T, N, K, cut):
    assert (dqt.dqt_bwd_dx_img_workspace_size(T, N, K) > 0) == cut
    dY = inputs.normal((T, N), 1e-2, seed=T + N, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=K)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    s_w = float(s_w)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    dYc = dY.cuda()
    dX1 = dqt.dqt_bitlinear_bwd_dx_img(dYc, W_img, s_w)
    dX2 = dqt.dqt_bitlinear_bwd_dx_img(dYc, W_img, s_w)
    dX0 = dqt.dqt_bitlinear_bwd_dx_img(dYc, W_img, s_w, ws=False)
    # the int8 call, whose workspace holds the weight image and the partials
    dX3 = dqt.dqt_bitlinear_bwd_dx(dYc, torch.from_numpy(c).cuda(), s_w)
    dqt.dqt_check_device_status()
    assert torch.equal(dX1.view(torch.int16), dX2.view(torch.int16))  # fixed summation order
    assert torch.equal(dX1.view(torch.int16), dX3.view(torch.int16))
    # against the uncut kernel: the same fp32 sums up to their order, so one
    # bf16 rounding step apart at most, with an absolute floor of 2^-16 of
    # the largest value for sums that cancel to near zero
    a = dX1.float()
    b = dX0.float()
    floor = float(torch.abs(b).max()) * 2.0 ** -16
    assert bool((torch.abs(a - b) <= torch.abs(b) * 2.0 ** -7 + floor).all())
    rows = _tail_rows(T)
    ref = oracle.bwd_dx(bits(dY[torch.from_numpy(rows)]), c, np.float32(s_w))
    got = dX1[torch.from_numpy(rows).cuda()].cpu().double().numpy()
    assert float(np.abs(got - ref).max() / np.abs(ref).max()) <= REL_TOL


def test_stale_workspace_words_never_count_as_slices():
    """The slice counters need no reset: each launch tags its counts, and the
    tag is spread over 48 bits with its top bit set, so words the workspace
    held before -- counts, small integers, other launches' counters -- never
    read as this launch's slices.  Here the workspace is filled with every
    small integer and with words whose tag field holds small launch numbers."""
    T, N, K = 8192, 5632, 2048
    need = dqt.dqt_bwd_dx_img_workspace_size(T, N, K)
    assert need > 0
    dY = inputs.normal((T, N), 1e-2, seed=31, dtype=torch.bfloat16).cuda()
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=32).numpy(), qmin, qmax)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    ref = dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, float(s_w), ws=False)
    words = need // 8
    i = torch.arange(words, dtype=torch.int64, device="cuda")
    for fill in (i + 65536,                 # counts 65536.. (tag field 1, 2, ...)
                 ((i % 64) << 16) | 1,      # tag field 0..63, one slice done
                 ((i % 64) << 16) | 2):     # tag field 0..63, two slices done
        ws = torch.empty(need, dtype=torch.uint8, device="cuda")
        ws.view(torch.int64)[:words] = fill
        got = dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, float(s_w), ws=ws)
        dqt.dqt_check_device_status()
        a, b = got.float(), ref.float()
        floor = float(torch.abs(b).max()) * 2.0 ** -16
        assert bool((torch.abs(a - b) <= torch.abs(b) * 2.0 ** -7 + floor).all())


def test_forward_then_dx_on_one_workspace():
    """A forward and a dX that cut their last waves on the same workspace,
    one after the other: the dX launch's counters start from the forward's
    leftovers, which carry another launch's tag and count as zero."""
    T, N, K = 8192, 5632, 2048  # dX reduces over N = 5632; the forward below over 5632 too
    need = max(dqt.dqt_bwd_dx_img_workspace_size(T, N, K), dqt.dqt_fwd_img_workspace_size(T, N, K))
    ws = torch.zeros(need, dtype=torch.uint8, device="cuda")
    qmin, qmax = oracle.grid(1.58)
    X = inputs.normal((T, N), 1.0, seed=41, dtype=torch.bfloat16)
    cf, sf, _ = oracle.absmean_init(inputs.normal((K, N), 0.02, seed=42).numpy(), qmin, qmax)
    _, s_x, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    Wf = dqt.dqt_codes_to_bf16(torch.from_numpy(cf).cuda())
    dY = inputs.normal((T, N), 1e-2, seed=43, dtype=torch.bfloat16).cuda()
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=44).numpy(), qmin, qmax)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    ref = dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, float(s_w), ws=False)
    for _ in range(3):
        dqt.dqt_bitlinear_fwd_img(q_img, s_x, Wf, float(sf), (qmin, qmax), ws=ws)
        got = dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, float(s_w), ws=ws)
        dqt.dqt_check_device_status()
        a, b = got.float(), ref.float()
        floor = float(torch.abs(b).max()) * 2.0 ** -16
        assert bool((torch.abs(a - b) <= torch.abs(b) * 2.0 ** -7 + floor).all())
