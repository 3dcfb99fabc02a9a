"""GPU parity: the CUDA path (through the C ABI) against the CPU oracle on the
same seeded inputs.

Rules:
  * bit-exact: activation codes, s_x, the bf16 operand images, the int32 forward
    accumulators, the forward output Y (same fp32 formula on both sides), the
    weight image, and the standalone SR update (codes, m, v) given identical
    fp32 gradients and the same Philox stream;
  * dX, dW: max relative error <= 2e-2 against the fp64 oracle, normwise
    (max |gpu - ref| / max |ref|); in addition, elementwise (floored at 1% of
    max |ref|) <= 2e-2 against the oracle fed the same operands: dX always,
    dW against the oracle that holds X_tilde as its bf16 image (the BF16
    environment the kernel computes in);
  * fused dW + update, against the oracle update fed the bf16-environment
    gradient: at most 1e-4 of the codes differ (floored count), each by
    exactly one grid step (the fp32 gradient differs in summation order, the
    uniform is the same); moments within 1e-3 relative (normwise).
Shapes span several 128 x 256 tiles with ragged tails; the full LLaMA-MLP
sizes (T=8192, H=2048, I=5632) are checked on sampled rows.
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
    """Max relative error, normwise: max |gpu - ref| / max |ref|."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    return float(np.abs(gpu - ref).max() / np.abs(ref).max())


def elem_err(gpu, ref):
    """Elementwise relative error, floored at 1% of max |ref| (near-zero sums)."""
    gpu = np.asarray(gpu, np.float64)
    ref = np.asarray(ref, np.float64)
    floor = 1e-2 * np.abs(ref).max()
    return float((np.abs(gpu - ref) / np.maximum(np.abs(ref), floor)).max())


def problem(T, K, N, bits_w, seed=1):
    X = inputs.normal((T, K), 1.0, seed=seed, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=seed + 1, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=seed + 2)
    qmin, qmax = oracle.grid(bits_w)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    return X, dY, W0, c, float(s_w), (qmin, qmax)


# ---------------------------------------------------------------------------
# act_quant (bit-exact)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,K", [(256, 512), (37, 264), (1, 8), (300, 5632), (8192, 2048),
                                 (129, 72), (5, 16384), (3, 24584)])
def test_act_quant_bit_exact(T, K):
    X = inputs.normal((T, K), 1.0, seed=T + K, dtype=torch.bfloat16)
    if T > 2:
        X[1] = 0.0  # all-zero row: amax floor
        X[2, : K // 2] = 0.5  # ties at .5 after scaling
    q, s, qi, xd = oracle.act_quant(bits(X))
    Xq, s_x, Xq_img, Xdq = dqt.dqt_act_quant_images(X.cuda())
    torch.cuda.synchronize()
    assert np.array_equal(Xq.cpu().numpy(), q)
    assert np.array_equal(s_x.cpu().numpy().view(np.uint32), s.view(np.uint32))
    assert np.array_equal(bits(Xq_img), qi)
    assert np.array_equal(bits(Xdq), xd)


def test_act_quant_beyond_int32_sampled():
    """T x K = 262147 x 8192 > 2^31 elements (row 262144 starts at element
    2^31): codes, s_x and both images bit-exact on sampled rows."""
    T, K = (1 << 18) + 3, 8192
    X = inputs.normal((T, K), 1.0, seed=45, dtype=torch.bfloat16)
    Xq, s_x, Xq_img, Xdq = dqt.dqt_act_quant_images(X.cuda())
    torch.cuda.synchronize()
    rows = np.array([0, 1, T // 2, 262143, 262144, T - 1])
    q, s, qi, xd = oracle.act_quant(bits(X[torch.from_numpy(rows)]))
    it = torch.from_numpy(rows).cuda()
    assert np.array_equal(Xq[it].cpu().numpy(), q)
    assert np.array_equal(s_x[it].cpu().numpy().view(np.uint32), s.view(np.uint32))
    assert np.array_equal(bits(Xq_img[it]), qi)
    assert np.array_equal(bits(Xdq[it]), xd)


def test_act_quant_partial_outputs():
    X = inputs.normal((64, 128), 1.0, seed=3, dtype=torch.bfloat16)
    q, s, qi, xd = oracle.act_quant(bits(X))
    _, s_x, Xq_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    torch.cuda.synchronize()
    assert np.array_equal(bits(Xq_img), qi)
    assert np.array_equal(s_x.cpu().numpy(), s)


# ---------------------------------------------------------------------------
# weight image and AbsMean init
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("n", [1, 15, 16, 4099, 512 * 512])
def test_codes_to_bf16_exact(n):
    c = torch.randint(-128, 128, (n,), dtype=torch.int8, generator=torch.Generator().manual_seed(n))
    img = dqt.dqt_codes_to_bf16(c.cuda())
    torch.cuda.synchronize()
    assert torch.equal(img.cpu().float(), c.float())


@pytest.mark.parametrize("bits_w", [1.58, 4, 8])
def test_absmean_init_matches_oracle(bits_w):
    W0 = inputs.normal((512, 520), 0.02, seed=7)
    qmin, qmax = oracle.grid(bits_w)
    c_ref, s_ref, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    codes, s_w = dqt.dqt_absmean_init(W0.cuda(), (qmin, qmax))
    torch.cuda.synchronize()
    # fp64 sums in a different (fixed) order: s_w agrees to the last fp32 ulp
    assert abs(s_w - float(s_ref)) <= np.spacing(np.float32(s_ref))
    # the codes are Eq. 4 at the scale the GPU found, bit for bit, always
    want = oracle.quantize_weights(W0.numpy(), np.float32(s_w), qmin, qmax)
    assert np.array_equal(codes.cpu().numpy(), want)
    if s_w == float(s_ref):
        assert np.array_equal(want, c_ref)


# ---------------------------------------------------------------------------
# forward (bit-exact int32 accumulators and Y)
# ---------------------------------------------------------------------------
def _fwd_check(T, K, N, bits_w, rows=None, seed=1):
    X, dY, W0, c, s_w, g = problem(T, K, N, bits_w, seed)
    Xg = X.cuda()
    _, s_x, Xq_img, _ = dqt.dqt_act_quant_images(Xg, want=("Xq_img",))
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_img(Xq_img, s_x, W_img, s_w, g, acc_out=acc)
    dqt.dqt_check_device_status()
    q, s, _, _ = oracle.act_quant(bits(X))
    if rows is None:
        rows = np.arange(T)
    Yr, accr = oracle.fwd(q[rows], s[rows], c, np.float32(s_w))
    assert np.array_equal(acc.cpu().numpy()[rows], accr)
    assert np.array_equal(bits(Y)[rows], Yr)


@pytest.mark.parametrize("bits_w", [1.58, 8])
def test_fwd_config1(bits_w):
    _fwd_check(256, 512, 512, bits_w)


@pytest.mark.parametrize("T,K,N", [(300, 264, 520), (129, 72, 264), (1, 8, 8), (200, 64, 24)])
def test_fwd_ragged(T, K, N):
    _fwd_check(T, K, N, 1.58, seed=T)
    _fwd_check(T, K, N, 4, seed=T + 1)


@pytest.mark.parametrize("K", [1088, 2048, 5632])
def test_fwd_8bit_exact_chunked(K):
    """8-bit codes with K > 1024: the kernel drains exact fp32 chunks into int32."""
    _fwd_check(160, K, 272, 8, seed=K)


def test_fwd_adversarial_magnitudes():
    """Partial sums far above 2^24: all-large codes make every product ~ -2^14."""
    T, K, N = 130, 4096, 264
    g = torch.Generator().manual_seed(5)
    q = torch.randint(120, 128, (T, K), dtype=torch.int32, generator=g)
    c = -torch.randint(120, 129, (N, K), dtype=torch.int32, generator=g)
    s_x = torch.full((T,), 1.0, dtype=torch.float32)
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_img(q.to(torch.bfloat16).cuda(), s_x.cuda(), c.to(torch.bfloat16).cuda(),
                                  1.0, (-128, 127), acc_out=acc)
    dqt.dqt_check_device_status()
    ref = q.to(torch.int64) @ c.to(torch.int64).T
    assert ref.abs().max() > 2**24
    assert torch.equal(acc.cpu().to(torch.int64), ref)
    Yr, accr = oracle.fwd(q.numpy().astype(np.int8), s_x.numpy(), c.clamp(-128, 127).numpy().astype(np.int8), 1.0)
    assert np.array_equal(bits(Y), Yr)


def test_fwd_output_beyond_int32_sampled():
    """Y and the int32 accumulators with T x N = 524293 x 4096 > 2^31 elements
    (row 524288 starts at element 2^31): sampled rows on both sides of it."""
    T, K, N = (1 << 19) + 5, 64, 4096
    X = inputs.normal((T, K), 1.0, seed=41, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=42)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    _, s_x, Xq_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_img(Xq_img, s_x, W_img, float(s_w), (qmin, qmax), acc_out=acc)
    dqt.dqt_check_device_status()
    rows = np.array([0, 1, T // 2, 524287, 524288, T - 2, T - 1])
    q, s, _, _ = oracle.act_quant(bits(X[torch.from_numpy(rows)]))
    Yr, accr = oracle.fwd(q, s, c, np.float32(s_w))
    it = torch.from_numpy(rows).cuda()
    assert np.array_equal(acc[it].cpu().numpy(), accr)
    assert np.array_equal(bits(Y[it]), Yr)


@pytest.mark.parametrize("which", ["gate_up", "down"])
def test_fwd_llama_mlp_sampled_rows(which):
    T, H, I = 8192, 2048, 5632
    K, N = (H, I) if which == "gate_up" else (I, H)
    rows = np.array([0, 1, 127, 128, 1000, 4095, 4096, 8190, 8191])
    _fwd_check(T, K, N, 1.58, rows=rows, seed=11)


# ---------------------------------------------------------------------------
# backward dX and dW (tolerance against fp64)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,N,K", [(256, 512, 512), (300, 520, 264), (64, 24, 200)])
def test_bwd_dx(T, N, K):
    X, dY, W0, c, s_w, g = problem(T, K, N, 1.58, seed=N)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    dX = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), W_img, s_w)
    dqt.dqt_check_device_status()
    ref = oracle.bwd_dx(bits(dY), c, np.float32(s_w))
    assert rel_err(dX.cpu().double().numpy(), ref) <= REL_TOL
    assert elem_err(dX.cpu().double().numpy(), ref) <= REL_TOL


def test_bwd_dx_output_beyond_int32_sampled():
    """dX of T x K = 524293 x 4096 > 2^31 elements: sampled rows on both sides
    of element 2^31, within the fp64 tolerance."""
    T, N, K = (1 << 19) + 5, 64, 4096
    dY = inputs.normal((T, N), 1e-2, seed=43, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=44)
    qmin, qmax = oracle.grid(1.58)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    dX = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), W_img, float(s_w))
    dqt.dqt_check_device_status()
    rows = np.array([0, 1, T // 2, 524287, 524288, T - 2, T - 1])
    ref = oracle.bwd_dx(bits(dY[torch.from_numpy(rows)]), c, np.float32(s_w))
    got = dX[torch.from_numpy(rows).cuda()].cpu().double().numpy()
    assert rel_err(got, ref) <= REL_TOL
    assert elem_err(got, ref) <= REL_TOL


@pytest.mark.parametrize("T,N,K", [(256, 512, 512), (300, 520, 264), (77, 24, 200)])
def test_bwd_dw_gradient(T, N, K):
    X, dY, W0, c, s_w, g = problem(T, K, N, 1.58, seed=K)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    dW = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, None, s_w, None, None, None, None, g, dW_out=dW)
    dqt.dqt_check_device_status()
    q, s, _, xd = oracle.act_quant(bits(X))
    ref = oracle.bwd_dw(bits(dY), q, s)
    assert rel_err(dW.cpu().numpy(), ref) <= REL_TOL
    ref_b = oracle.bwd_dw_bf16x(bits(dY), xd)
    assert elem_err(dW.cpu().numpy(), ref_b) <= REL_TOL


def test_bwd_llama_mlp_sampled_rows():
    T, H, I = 8192, 2048, 5632
    X, dY, W0, c, s_w, g = problem(T, H, I, 1.58, seed=21)
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    dX = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), W_img, s_w)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    dW = torch.empty((I, H), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, None, s_w, None, None, None, None, g, dW_out=dW)
    dqt.dqt_check_device_status()
    trows = np.array([0, 129, 4097, 8191])
    ref = oracle.bwd_dx(bits(dY)[trows], c, np.float32(s_w))
    assert rel_err(dX.cpu().double().numpy()[trows], ref) <= REL_TOL
    q, s, _, xd = oracle.act_quant(bits(X))
    nrows = np.array([0, 255, 256, 5631])
    ref = oracle.bwd_dw(bits(dY), q, s, rows=nrows)
    assert rel_err(dW.cpu().numpy()[nrows], ref) <= REL_TOL
    ref_b = oracle.bwd_dw_bf16x(bits(dY), xd, rows=nrows)
    assert elem_err(dW.cpu().numpy()[nrows], ref_b) <= REL_TOL


# ---------------------------------------------------------------------------
# standalone SR update (bit-exact)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("bits_w,numel,step,round_mode", [
    (1.58, 512 * 512, 1, 0), (8, 512 * 512, 1, 0), (8, 1_000_003, 7, 0), (4, 4099, 3, 0),
    (8, 65536, 2, 1), (1.58, 3, 1, 0)])
def test_sr_update_bit_exact(bits_w, numel, step, round_mode):
    qmin, qmax = oracle.grid(bits_w)
    W0 = inputs.normal((numel,), 0.02, seed=numel)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    grad = inputs.normal((numel,), 1e-3, seed=numel + 1)
    m = inputs.normal((numel,), 1e-4, seed=numel + 2) if step > 1 else torch.zeros(numel)
    v = inputs.normal((numel,), 1e-4, seed=numel + 3).square() if step > 1 else torch.zeros(numel)
    hp = dqt.adamw(lr=1e-3, weight_decay=0.01 if step > 1 else 0.0, step=step)
    sr = dqt.sr_stream(seed=1234, tensor_id=3, round_mode=round_mode)
    Wg, mg, vg = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    changed = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_sr_update(grad.cuda(), Wg, s_w, mg, vg, hp, sr, (qmin, qmax), changed_out=changed)
    dqt.dqt_check_device_status()
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, step, s_w)
    c1, m1, v1, n_ch = oracle.update(grad.numpy(), c, m.numpy(), v.numpy(), k, qmin, qmax,
                                     1234, step, 3, round_mode)
    assert np.array_equal(Wg.cpu().numpy(), c1.ravel())
    assert np.array_equal(mg.cpu().numpy().view(np.uint32), m1.ravel().view(np.uint32))
    assert np.array_equal(vg.cpu().numpy().view(np.uint32), v1.ravel().view(np.uint32))
    assert int(changed.item()) == n_ch


def test_sr_update_beyond_int32_sampled():
    """The largest update size: 2^31 + 6 weights (past the int32 index range,
    with a ragged tail), ternary codes from the AbsMean init of N(0, 0.02),
    AdamW step 1.  Bit-exact against the oracle on sampled 4096-element rows
    (both ends, both sides of element 2^31, random rows) and on the six tail
    elements, each at its global element index (Philox counter e / 4)."""
    numel = (1 << 31) + 6
    qmin, qmax = oracle.grid(1.58)
    W0 = inputs.normal((numel,), 0.02, seed=31)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    del W0
    grad = inputs.normal((numel,), 1e-3, seed=32)
    hp = dqt.adamw(lr=1e-3, step=1)
    sr = dqt.sr_stream(seed=1234, tensor_id=5)
    Wg = torch.from_numpy(c).cuda()
    gg = grad.cuda()
    mg = torch.zeros(numel, dtype=torch.float32, device="cuda")
    vg = torch.zeros(numel, dtype=torch.float32, device="cuda")
    dqt.dqt_sr_update(gg, Wg, s_w, mg, vg, hp, sr, (qmin, qmax))
    dqt.dqt_check_device_status()
    del gg
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, 1, s_w)
    g_np = grad.numpy()
    K = 4096
    last_full = numel // K - 1  # row 524287 ends at element 2^31 - 1
    rng = np.random.default_rng(7)
    rows = np.unique(np.concatenate([[0, 1, last_full - 1, last_full],
                                     rng.integers(0, last_full, 28)])).astype(np.int64)
    cases = [(rows, K), (np.arange(1 << 30, (1 << 30) + 3, dtype=np.int64), 2)]
    for rws, kk in cases:
        idx = (rws[:, None] * kk + np.arange(kk)[None, :]).ravel()
        assert idx.max() < numel
        zeros = np.zeros(idx.size, np.float32)
        c1, m1, v1, _ = oracle.update(g_np[idx].reshape(-1, kk), c[idx], zeros, zeros, k,
                                      qmin, qmax, 1234, 1, 5, 0, rows=rws)
        it = torch.from_numpy(idx).cuda()
        assert np.array_equal(Wg[it].cpu().numpy(), c1.ravel())
        assert np.array_equal(mg[it].cpu().numpy().view(np.uint32), m1.ravel().view(np.uint32))
        assert np.array_equal(vg[it].cpu().numpy().view(np.uint32), v1.ravel().view(np.uint32))


# ---------------------------------------------------------------------------
# fused dW GEMM + AdamW + SR
# ---------------------------------------------------------------------------
def _fused(T, K, N, bits_w, step, seed, rows=None):
    X, dY, W0, c, s_w, g = problem(T, K, N, bits_w, seed)
    qmin, qmax = g
    if step > 1:
        m = inputs.normal((N, K), 1e-4, seed=seed + 5)
        v = inputs.normal((N, K), 1e-4, seed=seed + 6).square()
    else:
        m = torch.zeros((N, K))
        v = torch.zeros((N, K))
    hp = dqt.adamw(lr=1e-3, step=step)
    sr = dqt.sr_stream(seed=1234, tensor_id=1)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    Wg, mg, vg = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    dW = torch.empty((N, K), dtype=torch.float32, device="cuda")
    changed = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, Wg, s_w, mg, vg, hp, sr, g, dW_out=dW,
                                        changed_out=changed)
    dqt.dqt_check_device_status()
    q, s, _, xd = oracle.act_quant(bits(X))
    if rows is None:
        rows = np.arange(N)
    # the gradient the kernel's epilogue sees: X_tilde held in bf16 (BF16
    # environment), reduced in fp64 here and rounded once to fp32
    gref = oracle.bwd_dw_bf16x(bits(dY), xd, rows=rows).astype(np.float32)
    # and the paper-exact gradient (X_tilde = q / s_x in fp64) is within 2e-2
    gex = oracle.bwd_dw(bits(dY), q, s, rows=rows)
    assert rel_err(dW.cpu().numpy()[rows], gex) <= REL_TOL
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, step, s_w)
    c1, m1, v1, _ = oracle.update(gref, c[rows], m.numpy()[rows], v.numpy()[rows], k, qmin, qmax,
                                  1234, step, 1, 0, rows=rows)
    assert_fused_codes(Wg.cpu().numpy()[rows], c1)
    mr = mg.cpu().numpy()[rows]
    vr = vg.cpu().numpy()[rows]
    assert np.abs(mr - m1).max() <= 1e-3 * np.abs(m1).max()
    assert np.abs(vr - v1).max() <= 1e-3 * np.abs(v1).max()
    return Wg, dW, c, s_w, m, v, hp, sr, g, changed, mg, vg


@pytest.mark.parametrize("bits_w,step", [(1.58, 1), (8, 1), (8, 5), (1.58, 5)])
def test_fused_update_config1(bits_w, step):
    _fused(256, 512, 512, bits_w, step, seed=31)


def test_fused_update_ragged():
    _fused(300, 264, 520, 4, 2, seed=41)


def test_fused_update_llama_mlp_sampled_rows():
    # rows from the first waves of tiles and from the last, partly idle, wave
    _fused(8192, 2048, 5632, 1.58, 1, seed=51,
           rows=np.array([0, 127, 128, 3000, 4864, 5200, 5631]))
    _fused(8192, 5632, 2048, 1.58, 2, seed=52, rows=np.array([0, 1535, 1536, 1800, 2047]))


def test_fused_update_beyond_int32_sampled():
    """The fused dW + AdamW + SR call on N x K = 65544 x 32768 > 2^31 weights
    (row 65536 starts at element 2^31; the last tile row holds 8 ragged rows),
    T = 256 tokens: sampled weight rows on both sides of element 2^31, each
    at its global element index."""
    T, K, N = 256, 32768, 65544
    X = inputs.normal((T, K), 1.0, seed=61, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=62, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(1.58)
    W0 = inputs.normal((N, K), 0.02, seed=63)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    del W0
    hp = dqt.adamw(lr=1e-3, step=1)
    sr = dqt.sr_stream(seed=1234, tensor_id=6)
    _, _, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    Wg = torch.from_numpy(c).cuda()
    mg = torch.zeros((N, K), dtype=torch.float32, device="cuda")
    vg = torch.zeros((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, Wg, float(s_w), mg, vg, hp, sr, (qmin, qmax))
    dqt.dqt_check_device_status()
    rows = np.array([0, 1, 40000, 65535, 65536, 65543])
    _, _, _, xd = oracle.act_quant(bits(X))
    gref = oracle.bwd_dw_bf16x(bits(dY), xd, rows=rows).astype(np.float32)
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, 1, s_w)
    zeros = np.zeros((rows.size, K), np.float32)
    c1, m1, _, _ = oracle.update(gref, c[rows], zeros, zeros, k, qmin, qmax, 1234, 1, 6, 0,
                                 rows=rows)
    it = torch.from_numpy(rows).cuda()
    assert_fused_codes(Wg[it].cpu().numpy(), c1)
    mr = mg[it].cpu().numpy()
    assert np.abs(mr - m1).max() <= 1e-3 * np.abs(m1).max()


def test_fused_equals_standalone_on_same_gradient():
    """Fused epilogue and standalone kernel draw the same uniforms for the same
    element and evaluate the update in the same IEEE operations: given the
    fused kernel's own fp32 gradient, codes, moments and the changed-code
    count are identical, bit for bit (at one ragged shape as well)."""
    for T, K, N, seed in ((256, 512, 512, 61), (256, 264, 520, 62)):
        Wg, dW, c, s_w, m, v, hp, sr, g, changed, mg, vg = _fused(T, K, N, 8, 3, seed=seed)
        W2, m2, v2 = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
        ch2 = torch.zeros(1, dtype=torch.int64, device="cuda")
        dqt.dqt_sr_update(dW.reshape(-1), W2.reshape(-1), s_w, m2.reshape(-1), v2.reshape(-1), hp,
                          sr, g, changed_out=ch2)
        dqt.dqt_check_device_status()
        assert torch.equal(W2, Wg)
        assert torch.equal(m2.view(torch.int32), mg.view(torch.int32))
        assert torch.equal(v2.view(torch.int32), vg.view(torch.int32))
        assert int(ch2.item()) == int(changed.item())


def test_update_frequency_counter_ternary_step1():
    """Sec. 5.2 hook: the changed-code counter equals the number of codes that
    moved, and at step 1 the ternary rate is close to lr * s_w per movable code."""
    Wg, dW, c, s_w, m, v, hp, sr, g, changed, _, _ = _fused(256, 512, 512, 1.58, 1, seed=71)
    moved = int((Wg.cpu().numpy() != c).sum())
    assert int(changed.item()) == moved
    rate = moved / c.size
    assert 0.2 * 1e-3 * s_w < rate < 1e-3 * s_w * 1.2


# ---------------------------------------------------------------------------
# both GEMM tilings (2-SM pair tiles are the default; 1-SM tiles forced here)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("mode", [0, 1])
def test_both_tilings_agree_with_oracle(mode):
    dqt.dqt_set_gemm_tiles(mode)
    try:
        _fwd_check(300, 264, 520, 1.58, seed=91)
        _fwd_check(513, 512, 264, 4, seed=92)
        X, dY, W0, c, s_w, g = problem(300, 264, 520, 1.58, seed=93)
        W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
        dX = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), W_img, s_w)
        dqt.dqt_check_device_status()
        ref = oracle.bwd_dx(bits(dY), c, np.float32(s_w))
        assert elem_err(dX.cpu().double().numpy(), ref) <= REL_TOL
        _fused(300, 264, 520, 8, 3, seed=94)
    finally:
        dqt.dqt_set_gemm_tiles(0)


def test_tilings_bit_identical():
    """Same per-element arithmetic, same reduction order within a tile: the two
    tilings give bit-identical forward outputs and identical fused updates."""
    outs = []
    for mode in (0, 1):
        dqt.dqt_set_gemm_tiles(mode)
        try:
            X, dY, W0, c, s_w, g = problem(520, 512, 776, 1.58, seed=95)
            _, s_x, q_img, xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img", "Xdq"))
            W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
            Y = dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, s_w, g)
            dX = dqt.dqt_bitlinear_bwd_dx_img(dY.cuda(), W_img, s_w)
            dW = torch.empty((776, 512), dtype=torch.float32, device="cuda")
            # unsplit on both tilings (the split-T path sums in another order)
            dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), xdq, None, s_w, None, None, None, None, g,
                                                dW_out=dW, ws=False)
            dqt.dqt_check_device_status()
            outs.append((Y.cpu(), dX.cpu(), dW.cpu()))
        finally:
            dqt.dqt_set_gemm_tiles(0)
    assert torch.equal(outs[0][0], outs[1][0])
    assert torch.equal(outs[0][1], outs[1][1])
    assert torch.equal(outs[0][2], outs[1][2])


# ---------------------------------------------------------------------------
# split-T weight gradient (small outputs, long token reductions)
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("T,K,N,bits_w", [(8192, 256, 256, 1.58), (2048, 264, 520, 8),
                                           (4096, 768, 768, 4)])
def test_split_t_dw_update(T, K, N, bits_w):
    assert dqt.dqt_bwd_dw_img_workspace_size(T, N, K) > 0  # the shape takes the split path
    X, dY, W0, c, s_w, g = problem(T, K, N, bits_w, seed=T + N)
    qmin, qmax = g
    m = inputs.normal((N, K), 1e-4, seed=T + 5)
    v = inputs.normal((N, K), 1e-4, seed=T + 6).square()
    hp = dqt.adamw(lr=1e-3, step=2)
    sr = dqt.sr_stream(seed=1234, tensor_id=6)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    Wg, mg, vg = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    dW = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, Wg, s_w, mg, vg, hp, sr, g, dW_out=dW)
    dW2 = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, None, s_w, None, None, None, None, g, dW_out=dW2)
    dqt.dqt_check_device_status()
    assert torch.equal(dW, dW2)  # the gradient-only split path sums the same slabs
    q, s, _, xd = oracle.act_quant(bits(X))
    gref = oracle.bwd_dw_bf16x(bits(dY), xd)
    assert elem_err(dW.cpu().numpy(), gref) <= REL_TOL
    assert rel_err(dW.cpu().numpy(), oracle.bwd_dw(bits(dY), q, s)) <= REL_TOL
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, 2, s_w)
    c1, m1, v1, _ = oracle.update(gref.astype(np.float32), c, m.numpy(), v.numpy(), k, qmin, qmax,
                                  1234, 2, 6, 0)
    assert_fused_codes(Wg.cpu().numpy(), c1)
    assert np.abs(mg.cpu().numpy() - m1).max() <= 1e-3 * np.abs(m1).max()
    assert np.abs(vg.cpu().numpy() - v1).max() <= 1e-3 * np.abs(v1).max()
    # and the standalone update on the split path's own summed gradient is the
    # same update, bit for bit
    W3, m3, v3 = torch.from_numpy(c).cuda(), m.clone().cuda(), v.clone().cuda()
    dqt.dqt_sr_update(dW.view(-1), W3.view(-1), s_w, m3.view(-1), v3.view(-1), hp, sr, g)
    dqt.dqt_check_device_status()
    assert torch.equal(W3, Wg) and torch.equal(m3, mg) and torch.equal(v3, vg)


def test_split_t_matches_unsplit_within_tolerance():
    T, K, N = 8192, 256, 512
    X, dY, W0, c, s_w, g = problem(T, K, N, 1.58, seed=77)
    _, s_x, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    a = torch.empty((N, K), dtype=torch.float32, device="cuda")
    b = torch.empty((N, K), dtype=torch.float32, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, None, s_w, None, None, None, None, g, dW_out=a)
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, None, s_w, None, None, None, None, g, dW_out=b,
                                        ws=False)
    dqt.dqt_check_device_status()
    # fp32 summation order only (a wrong token slice would be an O(1) error)
    assert elem_err(a.cpu().numpy(), b.cpu().double().numpy()) <= 2e-3
