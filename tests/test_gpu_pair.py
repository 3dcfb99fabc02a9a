"""Two BitLinear weights that read the same input, stacked in one call (a
LLaMA MLP's gate and up projections): dqt_bitlinear_fwd_img_pair and
dqt_bitlinear_bwd_dw_update_img_pair; and the next-step weight image the
update writes (W_img_next).

Each weight keeps its own per-tensor scale (Eq. 2-3) and its own
stochastic-rounding stream (Philox elements counted from its own first
element), so the stacked calls must give, bit for bit, what two separate
calls give: the forward's Y and int32 accumulators, and the update's codes,
moments and changed-code count.  Both GEMM tilings; the split at whole
256-wide tiles.
"""
import numpy as np
import pytest
import torch

import oracle
from fused_rule import assert_fused_codes
from paper_2412_04787_gb300 import dqt, inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2412_04787_gb300 import build
    build.build()
    dqt.lib()
    yield
    dqt.dqt_set_gemm_tiles(0)
    torch.cuda.synchronize()


def _weights(N0, N1, K, bits, seed):
    qmin, qmax = oracle.grid(bits)
    c0, s0, _ = oracle.absmean_init(inputs.normal((N0, K), 0.02, seed=seed).numpy(), qmin, qmax)
    c1, s1, _ = oracle.absmean_init(inputs.normal((N1, K), 0.03, seed=seed + 1).numpy(), qmin, qmax)
    assert s0 != s1  # two different per-tensor scales
    return np.concatenate([c0, c1]), float(s0), float(s1), (qmin, qmax)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("T,K,N0,N1,bits", [(300, 264, 256, 264, 1.58), (1024, 2048, 5632, 5632, 1.58),
                                            (256, 1088, 512, 256, 8)])
def test_fwd_pair_equals_two_calls(mode, T, K, N0, N1, bits):
    dqt.dqt_set_gemm_tiles(mode)
    try:
        X = inputs.normal((T, K), 1.0, seed=T + K, dtype=torch.bfloat16)
        c, s0, s1, g = _weights(N0, N1, K, bits, seed=N0 + N1)
        _, s_x, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
        W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
        N = N0 + N1
        acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
        Y = dqt.dqt_bitlinear_fwd_img_pair(q_img, s_x, W_img, N0, s0, s1, g, acc_out=acc)
        acc0 = torch.empty((T, N0), dtype=torch.int32, device="cuda")
        acc1 = torch.empty((T, N1), dtype=torch.int32, device="cuda")
        Y0 = dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img[:N0], s0, g, acc_out=acc0)
        Y1 = dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img[N0:], s1, g, acc_out=acc1)
        dqt.dqt_check_device_status()
        assert torch.equal(acc[:, :N0], acc0) and torch.equal(acc[:, N0:], acc1)
        assert torch.equal(Y[:, :N0].contiguous().view(torch.int16), Y0.view(torch.int16))
        assert torch.equal(Y[:, N0:].contiguous().view(torch.int16), Y1.view(torch.int16))
        # and the oracle on two rows, the second weight's scale included
        rows = np.array([0, T - 1])
        Xb = X[torch.from_numpy(rows)].contiguous().view(torch.int16).numpy().view(np.uint16)
        q, s, _, _ = oracle.act_quant(Xb)
        Yr, accr = oracle.fwd(q, s, c[N0:], np.float32(s1))
        it = torch.from_numpy(rows).cuda()
        assert np.array_equal(acc[it][:, N0:].cpu().numpy(), accr)
        assert np.array_equal(Y[it][:, N0:].contiguous().view(torch.int16).cpu().numpy().view(np.uint16), Yr)
    finally:
        dqt.dqt_set_gemm_tiles(0)


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("T,K,N0,N1,bits,step", [(256, 512, 256, 264, 1.58, 1),
                                                 (1024, 2048, 5632, 5632, 1.58, 3),
                                                 (512, 264, 512, 256, 8, 2)])
def test_dw_update_pair_equals_two_calls(mode, T, K, N0, N1, bits, step):
    dqt.dqt_set_gemm_tiles(mode)
    try:
        N = N0 + N1
        X = inputs.normal((T, K), 1.0, seed=T, dtype=torch.bfloat16)
        dY = inputs.normal((T, N), 1e-2, seed=T + 1, dtype=torch.bfloat16).cuda()
        c, s0, s1, g = _weights(N0, N1, K, bits, seed=K)
        _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
        if step > 1:
            m0 = inputs.normal((N, K), 1e-4, seed=7).cuda()
            v0 = inputs.normal((N, K), 1e-4, seed=8).square().cuda()
        else:
            m0 = torch.zeros((N, K), device="cuda")
            v0 = torch.zeros((N, K), device="cuda")
        hp = dqt.adamw(lr=1e-3, weight_decay=0.01, step=step)
        sr0 = dqt.sr_stream(seed=1234, tensor_id=4)
        sr1 = dqt.sr_stream(seed=1234, tensor_id=5)
        W = torch.from_numpy(c).cuda()
        m, v = m0.clone(), v0.clone()
        ch = torch.zeros(1, dtype=torch.int64, device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s0, s1, m, v, hp, sr0, sr1, g,
                                                 changed_out=ch, ws=False)
        # two separate calls on the halves (no token slicing on either side:
        # the same tiles, the same fp32 sums)
        Wa = torch.from_numpy(c[:N0]).cuda()
        Wb = torch.from_numpy(c[N0:]).cuda()
        ma, va = m0[:N0].clone(), v0[:N0].clone()
        mb, vb = m0[N0:].clone(), v0[N0:].clone()
        ch2 = torch.zeros(1, dtype=torch.int64, device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img(dY[:, :N0].contiguous(), Xdq, Wa, s0, ma, va, hp, sr0, g,
                                            changed_out=ch2, ws=False)
        dqt.dqt_bitlinear_bwd_dw_update_img(dY[:, N0:].contiguous(), Xdq, Wb, s1, mb, vb, hp, sr1, g,
                                            changed_out=ch2, ws=False)
        dqt.dqt_check_device_status()
        assert torch.equal(W[:N0], Wa) and torch.equal(W[N0:], Wb)
        assert torch.equal(m[:N0], ma) and torch.equal(m[N0:], mb)
        assert torch.equal(v[:N0], va) and torch.equal(v[N0:], vb)
        assert int(ch.item()) == int(ch2.item())
        assert int(ch.item()) > 0
    finally:
        dqt.dqt_set_gemm_tiles(0)


def test_dw_update_pair_with_token_slices():
    """A stacked update whose output leaves the last wave short (token slices
    and the streaming tail update): the second weight's rows in the tail take
    its own constants and element count — equal to the slice-free call up to
    the gradient's fp32 summation order (the fused-update rule)."""
    T, K, N0, N1 = 4096, 2048, 2816 - 256, 2816 + 256  # 22 x 8 = 176 output tiles
    N = N0 + N1
    assert dqt.dqt_bwd_dw_img_workspace_size(T, N, K) > 0
    X = inputs.normal((T, K), 1.0, seed=3, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=4, dtype=torch.bfloat16).cuda()
    c, s0, s1, g = _weights(N0, N1, K, 1.58, seed=9)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    hp = dqt.adamw(lr=1e-3, step=1)
    sr0 = dqt.sr_stream(seed=77, tensor_id=0)
    sr1 = dqt.sr_stream(seed=77, tensor_id=1)
    outs = []
    for ws in (None, False):
        W = torch.from_numpy(c).cuda()
        m = torch.zeros((N, K), device="cuda")
        v = torch.zeros((N, K), device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s0, s1, m, v, hp, sr0, sr1, g, ws=ws)
        outs.append(W)
    dqt.dqt_check_device_status()
    assert_fused_codes(outs[0].cpu().numpy(), outs[1].cpu().numpy(), "pair, sliced vs unsliced")


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("T,K,N,bits", [(4096, 2048, 5632, 1.58),  # 176 tiles: token slices + tail kernel
                                        (256, 512, 520, 8),        # one wave, ragged N
                                        (4096, 512, 512, 1.58)])   # split-T path (few tiles)
def test_dw_update_writes_next_image(mode, T, K, N, bits):
    """W_img_next: the update also writes the bf16 image of the codes it
    writes, byte for byte what dqt_codes_to_bf16 makes of them."""
    dqt.dqt_set_gemm_tiles(mode)
    try:
        X = inputs.normal((T, K), 1.0, seed=T + N, dtype=torch.bfloat16)
        dY = inputs.normal((T, N), 1e-2, seed=T + 7, dtype=torch.bfloat16).cuda()
        qmin, qmax = oracle.grid(bits)
        c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=N).numpy(), qmin, qmax)
        _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
        W = torch.from_numpy(c).cuda()
        m = torch.zeros((N, K), device="cuda")
        v = torch.zeros((N, K), device="cuda")
        img = torch.full((N, K), float("nan"), dtype=torch.bfloat16, device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img(dY, Xdq, W, float(s_w), m, v, dqt.adamw(lr=1e-2),
                                            dqt.sr_stream(seed=3), (qmin, qmax), W_img_next=img)
        dqt.dqt_check_device_status()
        assert not torch.equal(W.cpu(), torch.from_numpy(c))  # the update moved codes
        assert torch.equal(img.view(torch.int16), dqt.dqt_codes_to_bf16(W).view(torch.int16))
    finally:
        dqt.dqt_set_gemm_tiles(0)


def test_dw_update_pair_writes_next_image():
    T, K, N0, N1 = 1024, 2048, 5632, 5632
    N = N0 + N1
    X = inputs.normal((T, K), 1.0, seed=11, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=12, dtype=torch.bfloat16).cuda()
    c, s0, s1, g = _weights(N0, N1, K, 1.58, seed=13)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    W = torch.from_numpy(c).cuda()
    m = torch.zeros((N, K), device="cuda")
    v = torch.zeros((N, K), device="cuda")
    img = torch.empty((N, K), dtype=torch.bfloat16, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s0, s1, m, v, dqt.adamw(lr=1e-2),
                                             dqt.sr_stream(seed=1), dqt.sr_stream(seed=1, tensor_id=1),
                                             g, W_img_next=img)
    dqt.dqt_check_device_status()
    assert torch.equal(img.view(torch.int16), dqt.dqt_codes_to_bf16(W).view(torch.int16))


@pytest.mark.parametrize("T,K,N0,N1", [(300, 272, 256, 264), (1024, 2048, 5632, 5632)])
def test_fwd_fp8_pair_equals_two_calls(T, K, N0, N1):
    """The stacked FP8 forward: each half of the output with its own scale,
    equal to two dqt_bitlinear_fwd_fp8 calls (the same fp32 sums per tile)."""
    X = inputs.normal((T, K), 1.0, seed=T + 3, dtype=torch.bfloat16).cuda()
    c, s0, s1, g = _weights(N0, N1, K, 1.58, seed=N0 + 7)
    q8, s8, _ = dqt.dqt_act_quant_fp8(X, want_xdq=False)
    W8 = dqt.dqt_codes_to_fp8(torch.from_numpy(c).cuda(), g)
    N = N0 + N1
    acc = torch.empty((T, N), dtype=torch.float32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_fp8_pair(q8, s8, W8, N0, s0, s1, g, acc_out=acc)
    acc0 = torch.empty((T, N0), dtype=torch.float32, device="cuda")
    acc1 = torch.empty((T, N1), dtype=torch.float32, device="cuda")
    Y0 = dqt.dqt_bitlinear_fwd_fp8(q8, s8, W8[:N0], s0, g, acc_out=acc0)
    Y1 = dqt.dqt_bitlinear_fwd_fp8(q8, s8, W8[N0:], s1, g, acc_out=acc1)
    dqt.dqt_check_device_status()
    assert torch.equal(acc[:, :N0].view(torch.int32), acc0.view(torch.int32))
    assert torch.equal(acc[:, N0:].view(torch.int32), acc1.view(torch.int32))
    assert torch.equal(Y[:, :N0].contiguous().view(torch.int16), Y0.view(torch.int16))
    assert torch.equal(Y[:, N0:].contiguous().view(torch.int16), Y1.view(torch.int16))


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("T,K,N", [(4096, 2048, 5632),   # token slices + tail kernel
                                   (256, 512, 520),      # one wave, ragged N
                                   (4096, 512, 512)])    # split-T path
def test_dw_update_writes_next_e4m3_image(mode, T, K, N):
    """W8_next: the update also writes the E4M3 image of the codes it writes,
    byte for byte what dqt_codes_to_fp8 makes of them (with the bf16 image
    beside it)."""
    dqt.dqt_set_gemm_tiles(mode)
    try:
        X = inputs.normal((T, K), 1.0, seed=T + N + 1, dtype=torch.bfloat16)
        dY = inputs.normal((T, N), 1e-2, seed=T + 9, dtype=torch.bfloat16).cuda()
        qmin, qmax = oracle.grid(1.58)
        c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=N + 1).numpy(), qmin, qmax)
        _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
        W = torch.from_numpy(c).cuda()
        m = torch.zeros((N, K), device="cuda")
        v = torch.zeros((N, K), device="cuda")
        img = torch.full((N, K), float("nan"), dtype=torch.bfloat16, device="cuda")
        img8 = torch.full((N, K), 0x7F, dtype=torch.uint8, device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img(dY, Xdq, W, float(s_w), m, v, dqt.adamw(lr=1e-2),
                                            dqt.sr_stream(seed=5), (qmin, qmax), W_img_next=img,
                                            W8_next=img8)
        dqt.dqt_check_device_status()
        assert not torch.equal(W.cpu(), torch.from_numpy(c))
        assert torch.equal(img8, dqt.dqt_codes_to_fp8(W, (qmin, qmax)))
        assert torch.equal(img.view(torch.int16), dqt.dqt_codes_to_bf16(W).view(torch.int16))
    finally:
        dqt.dqt_set_gemm_tiles(0)


def test_dw_update_pair_writes_next_e4m3_image():
    T, K, N0, N1 = 1024, 2048, 5632, 5632
    N = N0 + N1
    X = inputs.normal((T, K), 1.0, seed=21, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=22, dtype=torch.bfloat16).cuda()
    c, s0, s1, g = _weights(N0, N1, K, 1.58, seed=23)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    W = torch.from_numpy(c).cuda()
    m = torch.zeros((N, K), device="cuda")
    v = torch.zeros((N, K), device="cuda")
    img8 = torch.empty((N, K), dtype=torch.uint8, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s0, s1, m, v, dqt.adamw(lr=1e-2),
                                             dqt.sr_stream(seed=2), dqt.sr_stream(seed=2, tensor_id=1),
                                             g, W8_next=img8)
    dqt.dqt_check_device_status()
    assert torch.equal(img8, dqt.dqt_codes_to_fp8(W, g))


@pytest.mark.parametrize("mode", [0, 1])
@pytest.mark.parametrize("T,K,N,bits", [(4096, 2048, 5632, 8),   # token slices + tail kernel
                                        (256, 512, 520, 6),      # one wave, ragged N
                                        (4096, 512, 512, 8)])    # split-T path
def test_dw_update_writes_next_split_e4m3_image(mode, T, K, N, bits):
    """W8_next for codes wider than 16 in magnitude: the update writes the
    split E4M3 image [N, 2K] of the codes it writes, byte for byte what
    dqt_codes_to_fp8_split makes of them."""
    dqt.dqt_set_gemm_tiles(mode)
    try:
        X = inputs.normal((T, K), 1.0, seed=T + N + 2, dtype=torch.bfloat16)
        dY = inputs.normal((T, N), 1e-2, seed=T + 10, dtype=torch.bfloat16).cuda()
        qmin, qmax = oracle.grid(bits)
        c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=N + 2).numpy(), qmin, qmax)
        _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
        W = torch.from_numpy(c).cuda()
        m = torch.zeros((N, K), device="cuda")
        v = torch.zeros((N, K), device="cuda")
        img8 = torch.full((N, 2 * K), 0x7F, dtype=torch.uint8, device="cuda")
        dqt.dqt_bitlinear_bwd_dw_update_img(dY, Xdq, W, float(s_w), m, v, dqt.adamw(lr=1e-2),
                                            dqt.sr_stream(seed=6), (qmin, qmax), W8_next=img8)
        dqt.dqt_check_device_status()
        assert not torch.equal(W.cpu(), torch.from_numpy(c))
        assert torch.equal(img8, dqt.dqt_codes_to_fp8_split(W))
    finally:
        dqt.dqt_set_gemm_tiles(0)


@pytest.mark.parametrize("T,K,N0,N1", [(1024, 2048, 5632, 5632),  # token slices + tail kernel
                                       (4096, 512, 256, 256)])    # split-T path, one slab pass each
def test_dw_update_pair_writes_next_split_e4m3_image(T, K, N0, N1):
    N = N0 + N1
    X = inputs.normal((T, K), 1.0, seed=31, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=32, dtype=torch.bfloat16).cuda()
    c, s0, s1, g = _weights(N0, N1, K, 8, seed=33)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    W = torch.from_numpy(c).cuda()
    m = torch.zeros((N, K), device="cuda")
    v = torch.zeros((N, K), device="cuda")
    img = torch.empty((N, K), dtype=torch.bfloat16, device="cuda")
    img8 = torch.full((N, 2 * K), 0x7F, dtype=torch.uint8, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s0, s1, m, v, dqt.adamw(lr=1e-2),
                                             dqt.sr_stream(seed=4), dqt.sr_stream(seed=4, tensor_id=1),
                                             g, W_img_next=img, W8_next=img8)
    dqt.dqt_check_device_status()
    assert torch.equal(img8, dqt.dqt_codes_to_fp8_split(W))
    assert torch.equal(img.view(torch.int16), dqt.dqt_codes_to_bf16(W).view(torch.int16))


def _state(N, K, seed):
    m = inputs.normal((N, K), 1e-4, seed=seed).cuda()
    v = inputs.normal((N, K), 1e-4, seed=seed + 1).abs().square().cuda()
    return m, v


# (T, K0, N0 split, N1 rest of the stacked problem, K1, N of the second
# problem, bits): the LLaMA-MLP pair (gate + up stacked, and down) at 2048
# tokens, and a ragged one (partial tiles in rows, columns and tokens)
GROUP_CASES = [(2048, 2048, 5632, 5632, 5632, 2048, 1.58),
               (2048, 2048, 5632, 5632, 5632, 2048, 8),
               (300, 272, 256, 264, 264, 520, 1.58)]


@pytest.mark.parametrize("T,K0,Na,Nb,K1,N1,bits", GROUP_CASES)
def test_dw_update_group_equals_separate_calls(T, K0, Na, Nb, K1, N1, bits):
    """One launch over both problems' tiles: codes, moments, next-step images
    and changed counts equal the stacked call and the single call made
    separately with whole tiles (ws=False), bit for bit."""
    N0 = Na + Nb
    c0, s0, s1, g = _weights(Na, Nb, K0, bits, seed=T + 1)
    qmin, qmax = g
    c1, s2, _ = oracle.absmean_init(inputs.normal((N1, K1), 0.02, seed=T + 5).numpy(), qmin, qmax)
    s2 = float(s2)
    X0 = inputs.normal((T, K0), 1.0, seed=T + 2, dtype=torch.bfloat16).cuda()
    X1 = inputs.normal((T, K1), 1.0, seed=T + 3, dtype=torch.bfloat16).cuda()
    dY0 = inputs.normal((T, N0), 1e-2, seed=T + 4, dtype=torch.bfloat16).cuda()
    dY1 = inputs.normal((T, N1), 1e-2, seed=T + 6, dtype=torch.bfloat16).cuda()
    _, _, _, Xd0 = dqt.dqt_act_quant_images(X0, want=("Xdq",))
    _, _, _, Xd1 = dqt.dqt_act_quant_images(X1, want=("Xdq",))
    m0, v0 = _state(N0, K0, T + 7)
    m1, v1 = _state(N1, K1, T + 9)
    hp = dqt.adamw(lr=1e-2, weight_decay=0.01, step=3)
    sra, srb, src = dqt.sr_stream(seed=8), dqt.sr_stream(seed=8, tensor_id=1), dqt.sr_stream(seed=8, tensor_id=2)
    w8 = 2 if dqt.fp8_split_grid(g) else 1
    out = []
    for grouped in (True, False):
        W0, W1 = torch.from_numpy(c0).cuda(), torch.from_numpy(c1).cuda()
        M0, V0, M1, V1 = m0.clone(), v0.clone(), m1.clone(), v1.clone()
        i0 = torch.empty((N0, K0), dtype=torch.bfloat16, device="cuda")
        i1 = torch.empty((N1, K1), dtype=torch.bfloat16, device="cuda")
        e0 = torch.empty((N0, K0 * w8), dtype=torch.uint8, device="cuda")
        e1 = torch.empty((N1, K1 * w8), dtype=torch.uint8, device="cuda")
        ch = torch.zeros(2, dtype=torch.int64, device="cuda")
        if grouped:
            dqt.dqt_bitlinear_bwd_dw_update_group(
                [dict(dY=dY0, Xdq=Xd0, W=W0, m=M0, v=V0, N0=Na, s_w0=s0, s_w1=s1, sr0=sra, sr1=srb,
                      W_img_next=i0, W8_next=e0, changed_out=ch[0:1]),
                 dict(dY=dY1, Xdq=Xd1, W=W1, m=M1, v=V1, s_w0=s2, sr0=src, W_img_next=i1,
                      W8_next=e1, changed_out=ch[1:2])], hp, g)
        else:
            dqt.dqt_bitlinear_bwd_dw_update_img_pair(dY0, Xd0, W0, Na, s0, s1, M0, V0, hp, sra, srb, g,
                                                     changed_out=ch[0:1], ws=False, W_img_next=i0,
                                                     W8_next=e0)
            dqt.dqt_bitlinear_bwd_dw_update_img(dY1, Xd1, W1, s2, M1, V1, hp, src, g,
                                                changed_out=ch[1:2], ws=False, W_img_next=i1,
                                                W8_next=e1)
        dqt.dqt_check_device_status()
        out.append([W0, W1, M0, V0, M1, V1, i0, i1, e0, e1, ch])
    names = ["W0", "W1", "m0", "v0", "m1", "v1", "img0", "img1", "e4m3_0", "e4m3_1", "changed"]
    for n, a, b in zip(names, out[0], out[1]):
        a = a.view(torch.int16) if a.dtype == torch.bfloat16 else a
        b = b.view(torch.int16) if b.dtype == torch.bfloat16 else b
        assert torch.equal(a, b), n
    assert int(out[0][-1][0]) > 0 and int(out[0][-1][1]) > 0
    assert not torch.equal(out[0][0].cpu(), torch.from_numpy(c0))
