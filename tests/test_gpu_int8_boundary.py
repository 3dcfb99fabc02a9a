"""GPU parity of the hot-path entry points that take int8 codes (the C-ABI
boundary: dqt_act_quant, dqt_bitlinear_fwd, dqt_bitlinear_bwd_dx,
dqt_bitlinear_bwd_dw_update) against the CPU oracle, and against the same
GEMMs on bf16 operand images (the *_img calls).

Rules as for the image path:
  * bit-exact: codes and s_x of the activation quantiser; the forward's int32
    accumulators and Y; the forward, dX, the weight gradient and the fused
    update equal the *_img calls bit for bit (the calls' workspace passes
    write the images dqt_act_quant_images and dqt_codes_to_bf16 write);
  * dX, dW: max relative error <= 2e-2 against the fp64 oracle;
  * fused update: at most 1e-4 of the codes differ from the oracle's update of
    the bf16-environment gradient, each by one grid step.
"""
import numpy as np
import pytest
import torch

import oracle
from fused_rule import assert_fused_codes
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


def rel_err(gpu, ref):
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.abs(gpu - ref).max() / np.abs(ref).max())


def problem(T, K, N, bits_w, seed=1):
    X = inputs.normal((T, K), 1.0, seed=seed, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=seed + 1, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(bits_w)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=seed + 2).numpy(), qmin,
                                    qmax)
    return X, dY, c, float(s_w), (qmin, qmax)


# ---------------------------------------------------------------------------
# activation codes: 2 bytes read, 1 byte written per element
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,K", [(256, 512), (37, 264), (1, 8), (8192, 2048), (300, 5632),
                                 (1000, 1088), (3, 24584)])
def test_act_quant_codes_only(T, K):
    X = inputs.normal((T, K), 1.0, seed=T * 7 + K, dtype=torch.bfloat16)
    if T > 2:
        X[1] = 0.0
        X[2, : K // 2] = 0.5
    q, s, _, _ = oracle.act_quant(bits(X))
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    torch.cuda.synchronize()
    assert np.array_equal(Xq.cpu().numpy(), q)
    assert np.array_equal(s_x.cpu().numpy().view(np.uint32), s.view(np.uint32))


@pytest.mark.parametrize("T,K", [(256, 512), (37, 272), (8192, 5632), (300, 2048), (3, 49168)])
def test_codes_to_xdq_is_the_act_quant_image(T, K):
    """The X_tilde conversion the weight-gradient call runs: bf16(q / s_x),
    bit for bit the oracle's image."""
    X = inputs.normal((T, K), 1.0, seed=T + K, dtype=torch.bfloat16)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    xdq = dqt.dqt_codes_to_xdq(Xq, s_x)
    torch.cuda.synchronize()
    _, _, _, xd = oracle.act_quant(bits(X))
    assert np.array_equal(bits(xdq), xd)


# ---------------------------------------------------------------------------
# forward on int8 operands (their bf16 images made in the call's workspace)
# ---------------------------------------------------------------------------
def _fwd_i8(T, K, N, bits_w, rows=None, seed=1):
    X, _, c, s_w, g = problem(T, K, N, bits_w, seed)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    Wc = torch.from_numpy(c).cuda()
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd(Xq, s_x, Wc, s_w, g, acc_out=acc)
    # the image path on the same codes
    _, s_x2, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    acc2 = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y2 = dqt.dqt_bitlinear_fwd_img(q_img, s_x2, dqt.dqt_codes_to_bf16(Wc), s_w, g, acc_out=acc2)
    dqt.dqt_check_device_status()
    assert torch.equal(acc, acc2) and torch.equal(Y.view(torch.int16), Y2.view(torch.int16))
    rows = np.arange(T) if rows is None else rows
    q, s, _, _ = oracle.act_quant(bits(X[torch.from_numpy(rows)]))
    Yr, accr = oracle.fwd(q, s, c, np.float32(s_w))
    it = torch.from_numpy(rows).cuda()
    assert np.array_equal(acc[it].cpu().numpy(), accr)
    assert np.array_equal(bits(Y[it]), Yr)


@pytest.mark.parametrize("bits_w", [1.58, 4, 8])
def test_fwd_int8_config1(bits_w):
    _fwd_i8(256, 512, 512, bits_w)


@pytest.mark.parametrize("T,K,N", [(300, 264, 520), (129, 72, 264), (1, 8, 8), (200, 64, 24),
                                   (37, 48, 8), (513, 1040, 776)])
def test_fwd_int8_ragged(T, K, N):
    _fwd_i8(T, K, N, 1.58, seed=T)
    _fwd_i8(T, K, N, 8, seed=T + 1)


@pytest.mark.parametrize("K", [1088, 2048, 5632])
def test_fwd_int8_8bit_drained_chunks(K):
    """8-bit codes, K > 1024: exact fp32 chunks drained into int32 sums."""
    _fwd_i8(160, K, 272, 8, seed=K)


def test_fwd_int8_adversarial_magnitudes():
    """Sums far above 2^24: every product ~ -2^14, codes at the int8 ends."""
    T, K, N = 130, 4096, 264
    g = torch.Generator().manual_seed(5)
    q = torch.randint(120, 128, (T, K), dtype=torch.int32, generator=g)
    q[0, :64] = -128  # the most negative activation code
    c = -torch.randint(120, 129, (N, K), dtype=torch.int32, generator=g).clamp(-128, 127)
    s_x = torch.full((T,), 1.0, dtype=torch.float32)
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd(q.to(torch.int8).cuda(), s_x.cuda(), c.to(torch.int8).cuda(), 1.0,
                              (-128, 127), acc_out=acc)
    dqt.dqt_check_device_status()
    ref = q.to(torch.int64) @ c.to(torch.int64).T
    assert ref.abs().max() > 2 ** 24
    assert torch.equal(acc.cpu().to(torch.int64), ref)
    Yr, _ = oracle.fwd(q.numpy().astype(np.int8), s_x.numpy(), c.numpy().astype(np.int8), 1.0)
    assert np.array_equal(bits(Y), Yr)


@pytest.mark.parametrize("which", ["gate_up", "down"])
def test_fwd_int8_llama_mlp_sampled_rows(which):
    T, H, I = 8192, 2048, 5632
    K, N = (H, I) if which == "gate_up" else (I, H)
    _fwd_i8(T, K, N, 1.58, rows=np.array([0, 1, 127, 128, 1000, 4095, 4096, 8190, 8191]), seed=11)


def test_fwd_int8_output_beyond_int32_sampled():
    """T x N = 524293 x 4096 > 2^31 outputs (row 524288 starts at 2^31)."""
    T, K, N = (1 << 19) + 5, 64, 4096
    X = inputs.normal((T, K), 1.0, seed=41, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=42).numpy(), qmin, qmax)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd(Xq, s_x, torch.from_numpy(c).cuda(), float(s_w), (qmin, qmax),
                              acc_out=acc)
    dqt.dqt_check_device_status()
    rows = np.array([0, 1, T // 2, 524287, 524288, T - 2, T - 1])
    q, s, _, _ = oracle.act_quant(bits(X[torch.from_numpy(rows)]))
    Yr, accr = oracle.fwd(q, s, c, np.float32(s_w))
    it = torch.from_numpy(rows).cuda()
    assert np.array_equal(acc[it].cpu().numpy(), accr)
    assert np.array_equal(bits(Y[it]), Yr)


# ---------------------------------------------------------------------------
# dX from int8 weight codes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,N,K,bits_w", [(256, 512, 512, 1.58), (300, 520, 264, 8),
                                          (64, 24, 200, 4), (8192, 5632, 2048, 1.58)])
def test_bwd_dx_int8(T, N, K, bits_w):
    X, dY, c, s_w, g = problem(T, K, N, bits_w, seed=N + K)
    Wc = torch.from_numpy(c).cuda()
    dX = dqt.dqt_bitlinear_bwd_dx(dY.cuda(), Wc, s_w)
    dX2 = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), dqt.dqt_codes_to_bf16(Wc), s_w)
    dqt.dqt_check_device_status()
    assert torch.equal(dX.view(torch.int16), dX2.view(torch.int16))
    rows = np.arange(T) if T <= 512 else np.array([0, 129, 4097, 8191])
    ref = oracle.bwd_dx(bits(dY)[rows], c, np.float32(s_w))
    assert rel_err(dX.cpu().double().numpy()[rows], ref) <= REL_TOL


# ---------------------------------------------------------------------------
# weight gradient + update from int8 activation codes
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,K,N,bits_w,step", [(256, 512, 512, 1.58, 1), (300, 272, 520, 8, 3),
                                               (8192, 256, 256, 4, 2)])
def test_bwd_dw_update_int8(T, K, N, bits_w, step):
    X, dY, c, s_w, g = problem(T, K, N, bits_w, seed=T + 3)
    qmin, qmax = g
    if step > 1:
        m = inputs.normal((N, K), 1e-4, seed=T + 5)
        v = inputs.normal((N, K), 1e-4, seed=T + 6).square()
    else:
        m = torch.zeros((N, K))
        v = torch.zeros((N, K))
    hp = dqt.adamw(lr=1e-3, step=step)
    sr = dqt.sr_stream(seed=1234, tensor_id=2)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    W1, m1, v1 = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    dW1 = torch.empty((N, K), dtype=torch.float32, device="cuda")
    ch1 = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update(dY.cuda(), Xq, s_x, W1, s_w, m1, v1, hp, sr, g, dW_out=dW1,
                                    changed_out=ch1)
    # the image path with the same (full) token-slice workspace
    _, _, _, xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    W2, m2, v2 = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    dW2 = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), xdq, W2, s_w, m2, v2, hp, sr, g, dW_out=dW2)
    dqt.dqt_check_device_status()
    assert torch.equal(dW1, dW2)
    assert torch.equal(W1, W2) and torch.equal(m1, m2) and torch.equal(v1, v2)
    # against the oracle
    q, s, _, xd = oracle.act_quant(bits(X))
    assert rel_err(dW1.cpu().numpy(), oracle.bwd_dw(bits(dY), q, s)) <= REL_TOL
    gref = oracle.bwd_dw_bf16x(bits(dY), xd).astype(np.float32)
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, step, s_w)
    c1, m_r, _, n_ch = oracle.update(gref, c, m.numpy(), v.numpy(), k, qmin, qmax, 1234, step, 2)
    assert_fused_codes(W1.cpu().numpy(), c1)
    assert np.abs(m1.cpu().numpy() - m_r).max() <= 1e-3 * np.abs(m_r).max()
    assert int(ch1.item()) == int((W1.cpu().numpy() != c).sum())


def test_bwd_dw_int8_image_only_workspace_and_gradient_only():
    """A workspace of exactly the X_tilde image runs the single fused kernel;
    gradient-only calls (W, m, v absent) write dW_out alone."""
    T, K, N = 512, 256, 264
    X, dY, c, s_w, g = problem(T, K, N, 1.58, seed=9)
    Xq, s_x = dqt.dqt_act_quant(X.cuda())
    dW = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update(dY.cuda(), Xq, s_x, None, s_w, None, None, None, None, g,
                                    dW_out=dW, ws=False)
    dqt.dqt_check_device_status()
    q, s, _, xd = oracle.act_quant(bits(X))
    assert rel_err(dW.cpu().numpy(), oracle.bwd_dw(bits(dY), q, s)) <= REL_TOL
    ref_b = oracle.bwd_dw_bf16x(bits(dY), xd)
    floor = 1e-2 * np.abs(ref_b).max()
    assert (np.abs(dW.cpu().numpy() - ref_b) / np.maximum(np.abs(ref_b), floor)).max() <= REL_TOL
