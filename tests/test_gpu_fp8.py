"""GPU parity of the FP8-environment forward (Sec. 4.1 hardware paragraph,
Sec. 4.3) against the CPU oracle on the same seeded inputs.

Rules:
  * bit-exact: the E4M3 activation bytes, s_x8, the dequantised bf16 image and
    the E4M3 weight image;
  * forward: the products value(Xq8) * c are exact, only the fp32 accumulation
    rounds.  Any order of K - 1 fp32 additions stays within
    (K - 1) * 2^-24 * sum_k |value(Xq8[t,k]) c[n,k]| of the exact sum, so the
    fp32 accumulators are held to that bound against the oracle's exact sum,
    and Y to one bf16 ulp of the oracle's Y plus the same bound scaled by
    1 / (s_x8 s_w).
Shapes span several 256 x 256 pair tiles with ragged tails, the three
activation-kernel variants (rows up to 2048, up to 8192 and beyond), and the
LLaMA-MLP sizes (T = 8192, H = 2048, I = 5632) on sampled rows.
"""
import numpy as np
import pytest
import torch

import oracle
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
    torch.cuda.synchronize()


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _x(T, K, seed):
    X = inputs.normal((T, K), 1.0, seed=seed, dtype=torch.bfloat16)
    if T > 3:
        X[1] = 0.0                    # all-zero token: amax floor, +0 codes
        X[2, 0] = 4.0
        X[2, 1:] = -1e-6              # tiny negatives round to -0
        X[3, : K // 2] = 0.25         # values landing on ties after scaling
    return X


@pytest.mark.parametrize("T,K", [(256, 512), (37, 272), (1, 16), (300, 5632), (64, 16400),
                                 (8192, 2048)])
def test_act_quant_fp8_bit_exact(T, K):
    X = _x(T, K, seed=T + K)
    q8, s8, xdq = oracle.act_quant_fp8(bits(X))
    g8, gs, gx = dqt.dqt_act_quant_fp8(X.cuda())
    assert (gs.cpu().numpy() == s8).all()
    assert (g8.cpu().numpy() == q8).all()
    assert (bits(gx) == xdq).all()


@pytest.mark.parametrize("bits_w,numel", [(1.58, 512 * 512), (1.58, 1000003), (4, 4099), (5, 65536)])
def test_codes_to_fp8_bit_exact(bits_w, numel):
    qmin, qmax = oracle.grid(bits_w)
    g = torch.Generator().manual_seed(numel)
    c = torch.randint(qmin, qmax + 1, (numel,), generator=g, dtype=torch.int8)
    ref = oracle.codes_to_e4m3(c.numpy())
    got = dqt.dqt_codes_to_fp8(c.cuda(), (qmin, qmax)).cpu().numpy()
    assert (got == ref).all()


def test_codes_to_fp8_rejects_wide_grids():
    c = torch.zeros(64, dtype=torch.int8, device="cuda")
    with pytest.raises(dqt.DQTError) as e:
        dqt.dqt_codes_to_fp8(c, 8)
    assert e.value.status == dqt.DQT_ERR_RANGE


def _check_fwd(q8, s8, c, s_w, Y_gpu, acc_gpu, rows=None):
    """Oracle forward on the given token rows, compared under the rules above."""
    q8r = q8 if rows is None else q8[rows]
    s8r = s8 if rows is None else s8[rows]
    Y_ref, acc_ref = oracle.fwd_fp8(q8r, s8r, c, s_w)
    xv = np.vectorize(oracle.e4m3_value)(q8r)
    mag = np.abs(xv) @ np.abs(c.astype(np.float64)).T
    K = q8.shape[1]
    bound = (K - 1) * 2.0 ** -24 * mag
    acc_g = acc_gpu if rows is None else acc_gpu[rows]
    err = np.abs(acc_g.astype(np.float64) - acc_ref)
    assert (err <= bound).all(), float((err / np.maximum(bound, 1e-300)).max())
    a_t = (np.float32(1.0) / (s8r.astype(np.float32) * np.float32(s_w))).astype(np.float64)
    y_ref = torch.from_numpy(Y_ref.view(np.int16)).view(torch.bfloat16).double().numpy()
    Yg = Y_gpu if rows is None else Y_gpu[rows]
    y_gpu = torch.from_numpy(Yg.view(np.int16)).view(torch.bfloat16).double().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(y_ref), 1e-38))) - 7)
    tol = ulp + a_t[:, None] * bound * 1.01
    assert (np.abs(y_gpu - y_ref) <= tol).all()
    # how far the hardware's accumulation is from exact (bit-identical Y is common)
    return float((err / np.maximum(mag, 1e-300)).max()), float((Y_ref == Yg).mean())


@pytest.mark.parametrize("T,K,N,bits_w", [(256, 512, 512, 1.58), (300, 272, 520, 1.58),
                                          (129, 144, 264, 5), (1, 16, 8, 1.58),
                                          (520, 1040, 776, 2)])
def test_fwd_fp8(T, K, N, bits_w):
    X = _x(T, K, seed=3 * T + K)
    W0 = inputs.normal((N, K), 0.02, seed=N + 7)
    qmin, qmax = oracle.grid(bits_w)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    q8, s8, _ = oracle.act_quant_fp8(bits(X))
    W8 = dqt.dqt_codes_to_fp8(torch.from_numpy(c).cuda(), (qmin, qmax))
    acc = torch.empty((T, N), dtype=torch.float32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_fp8(torch.from_numpy(q8).cuda(), torch.from_numpy(s8).cuda(), W8,
                                  float(s_w), (qmin, qmax), acc_out=acc)
    rel, same = _check_fwd(q8, s8, c, float(s_w), bits(Y), acc.cpu().numpy())
    assert rel < 1e-5 and same > 0.9, (rel, same)


def test_fwd_fp8_llama_mlp_sampled_rows():
    """gate/up shape of the MLP step (T = 8192, K = 2048, N = 5632), ternary,
    through the whole FP8 forward (activation kernel, weight image, GEMM)."""
    T, K, N = 8192, 2048, 5632
    X = inputs.normal((T, K), 1.0, seed=101, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=103)
    qmin, qmax = -1, 1
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    g8, gs, _ = dqt.dqt_act_quant_fp8(X.cuda(), want_xdq=False)
    W8 = dqt.dqt_codes_to_fp8(torch.from_numpy(c).cuda(), (qmin, qmax))
    acc = torch.empty((T, N), dtype=torch.float32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_fp8(g8, gs, W8, float(s_w), (qmin, qmax), acc_out=acc)
    rows = np.array([0, 1, 255, 256, 4097, 8190, 8191])
    q8, s8, _ = oracle.act_quant_fp8(bits(X[rows]))
    assert (g8.cpu().numpy()[rows] == q8).all() and (gs.cpu().numpy()[rows] == s8).all()
    Yb = bits(Y)[rows]
    accg = acc.cpu().numpy()[rows]
    _check_fwd(q8, s8, c, float(s_w), Yb, accg)


def test_fwd_fp8_matches_integer_path_on_integer_values():
    """When every E4M3 activation value is an integer of magnitude <= 16 and
    the per-token scale is the same on both paths, the FP8 forward and the
    exact integer forward compute the same sums: here value(Xq8) = Xq."""
    T, K, N = 128, 1024, 256
    g = torch.Generator().manual_seed(5)
    q = torch.randint(-16, 17, (T, K), generator=g, dtype=torch.int8)
    q8 = oracle.codes_to_e4m3(q.numpy())
    s = np.full(T, 3.0, np.float32)
    W0 = inputs.normal((N, K), 0.02, seed=9)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), -1, 1)
    W8 = dqt.dqt_codes_to_fp8(torch.from_numpy(c).cuda(), (-1, 1))
    acc = torch.empty((T, N), dtype=torch.float32, device="cuda")
    Y8 = dqt.dqt_bitlinear_fwd_fp8(torch.from_numpy(q8).cuda(), torch.from_numpy(s).cuda(), W8,
                                   float(s_w), (-1, 1), acc_out=acc)
    Y_int, acc_int = oracle.fwd(q.numpy(), s, c, s_w)
    assert (acc.cpu().numpy() == acc_int.astype(np.float32)).all()
    assert (bits(Y8) == Y_int).all()


def _split_halves(c):
    """The split of codes c = 16 h + l (h = c >> 4, l = c & 15)."""
    c = c.astype(np.int32)
    return 16 * (c >> 4), c & 15


@pytest.mark.parametrize("N,K", [(64, 16), (520, 256), (1000, 2048)])
def test_codes_to_fp8_split_exact(N, K):
    g = torch.Generator().manual_seed(N + K)
    c = torch.randint(-128, 128, (N, K), generator=g, dtype=torch.int8)
    h16, l = _split_halves(c.numpy())
    ref = np.concatenate([oracle.codes_to_e4m3(h16.astype(np.int16)),
                          oracle.codes_to_e4m3(l.astype(np.int16))], axis=1)
    got = dqt.dqt_codes_to_fp8_split(c.cuda()).cpu().numpy()
    assert (got == ref).all()
    # both halves are exact: their values add back to the codes
    v = np.vectorize(oracle.e4m3_value)(got).astype(np.float64)
    assert (v[:, :K] + v[:, K:] == c.numpy().astype(np.float64)).all()


def _check_fwd_split(q8, s8, c, s_w, Y_gpu, acc_gpu, rows=None):
    """The split forward: 2K exact products in fp32, so the accumulators are
    held to (2K - 1) 2^-24 sum_k |value(Xq8)| (|16 h| + |l|) of the exact sum
    (the oracle's, over value(Xq8) c) and Y to one bf16 ulp plus that bound
    scaled by 1 / (s_x8 s_w)."""
    q8r = q8 if rows is None else q8[rows]
    s8r = s8 if rows is None else s8[rows]
    Y_ref, acc_ref = oracle.fwd_fp8(q8r, s8r, c, s_w)
    xv = np.vectorize(oracle.e4m3_value)(q8r)
    h16, l = _split_halves(c)
    mag = np.abs(xv) @ (np.abs(h16) + np.abs(l)).astype(np.float64).T
    K = q8.shape[1]
    bound = (2 * K - 1) * 2.0 ** -24 * mag
    acc_g = acc_gpu if rows is None else acc_gpu[rows]
    err = np.abs(acc_g.astype(np.float64) - acc_ref)
    assert (err <= bound).all(), float((err / np.maximum(bound, 1e-300)).max())
    a_t = (np.float32(1.0) / (s8r.astype(np.float32) * np.float32(s_w))).astype(np.float64)
    y_ref = torch.from_numpy(Y_ref.view(np.int16)).view(torch.bfloat16).double().numpy()
    Yg = Y_gpu if rows is None else Y_gpu[rows]
    y_gpu = torch.from_numpy(Yg.view(np.int16)).view(torch.bfloat16).double().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(y_ref), 1e-38))) - 7)
    assert (np.abs(y_gpu - y_ref) <= ulp + a_t[:, None] * bound * 1.01).all()
    return float((Y_ref == Yg).mean())


@pytest.mark.parametrize("T,K,N,bits_w", [(256, 512, 512, 8), (300, 256, 520, 8), (129, 384, 264, 6)])
def test_fwd_fp8_split_codes(T, K, N, bits_w):
    """6- to 8-bit codes through the FP8 forward: the split image, the
    activation row read for both halves."""
    X = _x(T, K, seed=5 * T + K)
    W0 = inputs.normal((N, K), 0.02, seed=N + 11)
    qmin, qmax = oracle.grid(bits_w)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    q8, s8, _ = oracle.act_quant_fp8(bits(X))
    W8 = dqt.dqt_codes_to_fp8_split(torch.from_numpy(c).cuda())
    acc = torch.empty((T, N), dtype=torch.float32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_fp8(torch.from_numpy(q8).cuda(), torch.from_numpy(s8).cuda(), W8,
                                  float(s_w), (qmin, qmax), acc_out=acc)
    dqt.dqt_check_device_status()
    same = _check_fwd_split(q8, s8, c, float(s_w), bits(Y), acc.cpu().numpy())
    assert same > 0.8, same


def test_fwd_fp8_split_llama_mlp_sampled_rows_and_pair():
    """8-bit codes at the MLP's gate/up shape (T = 8192, K = 2048, N = 2 x
    5632 stacked, one scale per weight), on sampled rows; the stacked call
    equals two calls bit for bit."""
    T, K, N0 = 8192, 2048, 5632
    X = inputs.normal((T, K), 1.0, seed=111, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(8)
    c0, s0, _ = oracle.absmean_init(inputs.normal((N0, K), 0.02, seed=113).numpy(), qmin, qmax)
    c1, s1, _ = oracle.absmean_init(inputs.normal((N0, K), 0.03, seed=114).numpy(), qmin, qmax)
    c = np.concatenate([c0, c1])
    g8, gs, _ = dqt.dqt_act_quant_fp8(X.cuda(), want_xdq=False)
    W8 = dqt.dqt_codes_to_fp8_split(torch.from_numpy(c).cuda())
    acc = torch.empty((T, 2 * N0), dtype=torch.float32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_fp8_pair(g8, gs, W8, N0, float(s0), float(s1), (qmin, qmax), acc_out=acc)
    acc1 = torch.empty((T, N0), dtype=torch.float32, device="cuda")
    Y1 = dqt.dqt_bitlinear_fwd_fp8(g8, gs, W8[N0:], float(s1), (qmin, qmax), acc_out=acc1)
    dqt.dqt_check_device_status()
    assert torch.equal(acc[:, N0:].view(torch.int32), acc1.view(torch.int32))
    assert torch.equal(Y[:, N0:].contiguous().view(torch.int16), Y1.view(torch.int16))
    rows = np.array([0, 1, 255, 256, 4097, 8191])
    q8, s8, _ = oracle.act_quant_fp8(bits(X[rows]))
    assert (g8.cpu().numpy()[rows] == q8).all()
    _check_fwd_split(q8, s8, c0, float(s0), bits(Y[:, :N0].contiguous())[rows], acc.cpu().numpy()[rows, :N0])


def test_layer_keeps_split_image_across_steps():
    """A DQTBitLinear on 8-bit codes with the E4M3 forward: its update writes
    the split image of the new codes into the layer's cached operand, so the
    next forward converts nothing and reads exactly the image of the new
    codes (and gives the forward of a freshly converted image, bit for bit)."""
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    T, K, N = 384, 256, 520
    layer = DQTBitLinear(K, N, bits=8, lr=1e-2, seed=5, tensor_id=1, init_seed=9, act="fp8")
    assert layer.w8_split
    X = inputs.normal((T, K), 1.0, seed=12, dtype=torch.bfloat16).cuda()
    dY = inputs.normal((T, N), 1e-2, seed=13, dtype=torch.bfloat16).cuda()
    c0 = layer.codes.clone()
    for _ in range(2):
        layer(X.requires_grad_(True)).backward(dY)
    torch.cuda.synchronize()
    assert not torch.equal(layer.codes, c0)
    assert layer._img8_version == layer.codes._version  # kept current by the update
    img8 = layer.image_fp8()
    assert torch.equal(img8, dqt.dqt_codes_to_fp8_split(layer.codes))
    q8, s8, _ = dqt.dqt_act_quant_fp8(X.detach(), want_xdq=False)
    y = layer(X.detach())
    y_ref = dqt.dqt_bitlinear_fwd_fp8(q8, s8, dqt.dqt_codes_to_fp8_split(layer.codes),
                                      float(layer.s_w), layer.grid_tuple)
    dqt.dqt_check_device_status()
    assert torch.equal(y.view(torch.int16), y_ref.view(torch.int16))
