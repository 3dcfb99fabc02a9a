"""GPU parity of the 2-bit packed ternary storage (Sec. 1) and of Adafactor
with stochastic rounding (Sec. 4.3) against the CPU oracle.

Rules:
  * bit-exact: packing and unpacking, the operand images built from packed
    codes, the standalone AdamW + SR update on packed codes (codes, m, v), and
    the Adafactor per-element step given the oracle's statistics (R, C, Rbar,
    step, decay uploaded to the device) -- the same fp32 operations on both
    sides;
  * the fused dW + update on packed codes equals the same kernel on int8 codes
    bit for bit (only the code storage differs);
  * Adafactor statistics (fp32 sums in a fixed tree on the GPU, fp64 in the
    oracle): R, C and the scalars within 1e-5 relative;
  * the whole dW + Adafactor step against the oracle fed the bf16-environment
    gradient: at most 1e-4 of the codes differ (floored count), each by one
    grid step, at every step, the oracle starting each step from the GPU's
    codes and statistics.
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
    torch.cuda.synchronize()


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def _ternary(n, seed):
    g = torch.Generator().manual_seed(seed)
    return torch.randint(-1, 2, (n,), generator=g, dtype=torch.int8)


# ---------------------------------------------------------------------------
# packed ternary
# ---------------------------------------------------------------------------
@pytest.mark.parametrize("n", [1, 5, 16, 1023, 1000003, 1 << 20])
def test_pack_unpack_bit_exact(n):
    c = _ternary(n, n)
    ref = oracle.pack_ternary(c.numpy())
    p = dqt.dqt_pack_ternary(c.cuda())
    assert (p.cpu().numpy() == ref).all()
    back = dqt.dqt_unpack_ternary(torch.from_numpy(ref).cuda(), n)
    assert (back.cpu().numpy() == c.numpy()).all()


@pytest.mark.parametrize("N,K", [(512, 512), (264, 520), (1, 8)])
def test_packed_images_bit_exact(N, K):
    c = _ternary(N * K, N + K).view(N, K)
    p = torch.from_numpy(oracle.pack_ternary(c.numpy())).cuda()
    img = dqt.dqt_packed_to_bf16(p, (N, K))
    want = np.vectorize(oracle.f32_to_bf16_bits)(c.numpy().astype(np.float32)).astype(np.uint16)
    assert (bits(img) == want).all()
    w8 = dqt.dqt_packed_to_fp8(p, (N, K))
    assert (w8.cpu().numpy() == oracle.codes_to_e4m3(c.numpy())).all()


@pytest.mark.parametrize("numel,step", [(3, 1), (4099, 2), (1000003, 5)])
def test_sr_update_packed_bit_exact(numel, step):
    c0 = _ternary(numel, 7 + numel).numpy()
    g = inputs.normal((numel,), 1e-3, seed=numel).numpy()
    m0 = inputs.normal((numel,), 1e-4, seed=numel + 1).numpy()
    v0 = np.square(inputs.normal((numel,), 1e-4, seed=numel + 2).numpy())
    s_w = 62.7
    hp = dqt.adamw(lr=1e-3, weight_decay=0.01, step=step)
    sr = dqt.sr_stream(seed=99, tensor_id=3)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.01, step, np.float32(s_w))
    c1, m1, v1, ch = oracle.update(g.reshape(1, -1), c0, m0, v0, k, -1, 1, 99, step, 3)
    p = torch.from_numpy(oracle.pack_ternary(c0)).cuda()
    m = torch.from_numpy(m0).cuda()
    v = torch.from_numpy(v0).cuda()
    changed = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_sr_update_packed(torch.from_numpy(g).cuda(), p, s_w, m, v, hp, sr, changed_out=changed)
    assert (p.cpu().numpy() == oracle.pack_ternary(c1.ravel())).all()
    assert (m.cpu().numpy() == m1.ravel()).all() and (v.cpu().numpy() == v1.ravel()).all()
    assert int(changed.item()) == ch


@pytest.mark.parametrize("T,K,N,ws", [(256, 512, 512, False), (300, 264, 520, False),
                                      (4096, 768, 768, None)])
def test_fused_dw_update_packed_equals_int8(T, K, N, ws):
    """Same kernel, int8 vs packed code storage: identical codes, m, v."""
    X = inputs.normal((T, K), 1.0, seed=T, dtype=torch.bfloat16).cuda()
    dY = inputs.normal((T, N), 1e-2, seed=T + 1, dtype=torch.bfloat16).cuda()
    c0, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=T + 2).numpy(), -1, 1)
    _, s_x, _, xdq = dqt.dqt_act_quant_images(X, want=("Xdq",))
    hp = dqt.adamw(lr=1e-3, step=1)
    sr = dqt.sr_stream(seed=5, tensor_id=1)
    W = torch.from_numpy(c0).cuda()
    m = torch.zeros((N, K), device="cuda")
    v = torch.zeros((N, K), device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, W, float(s_w), m, v, hp, sr, (-1, 1), ws=ws)
    Wp = torch.from_numpy(oracle.pack_ternary(c0)).cuda()
    m2 = torch.zeros((N, K), device="cuda")
    v2 = torch.zeros((N, K), device="cuda")
    ch = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_packed(dY, xdq, Wp, float(s_w), m2, v2, hp, sr,
                                           changed_out=ch, ws=ws)
    got = oracle.unpack_ternary(Wp.cpu().numpy(), N * K).reshape(N, K)
    assert (got == W.cpu().numpy()).all()
    assert torch.equal(m, m2) and torch.equal(v, v2)
    assert int(ch.item()) == int((got != c0).sum())


# ---------------------------------------------------------------------------
# Adafactor
# ---------------------------------------------------------------------------
def _af_problem(N, K, bits_w, seed):
    qmin, qmax = oracle.grid(bits_w)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=seed).numpy(), qmin, qmax)
    return c, float(s_w), (qmin, qmax)


HPS = [dict(lr=1e-3), dict(lr=1e-2, relative_step=True, scale_parameter=True, weight_decay=0.1),
       dict(lr=5e-3, clip_d=0.5)]


@pytest.mark.parametrize("N,K", [(512, 512), (264, 520), (5632, 2048)])
@pytest.mark.parametrize("hpi", [0, 1, 2])
def test_adafactor_stats(N, K, hpi):
    c, s_w, grid = _af_problem(N, K, 1.58, seed=N + hpi)
    hpo = oracle.AdafactorHP(**HPS[hpi])
    R = np.zeros(N, np.float32)
    Cc = np.zeros(K, np.float32)
    Rg = torch.zeros(N, device="cuda")
    Cg = torch.zeros(K, device="cuda")
    for t in (1, 2, 3):
        g = inputs.normal((N, K), 1e-3, seed=10 * t + hpi).numpy()
        if t == 2:
            g[N // 2, K // 3] = 0.5  # an outlier: update clipping is active
        R, Cc, st = oracle.adafactor_stats(g, c, s_w, R, Cc, t, hpo)
        ag, bg, sc = dqt.dqt_adafactor_stats(torch.from_numpy(g).cuda(), torch.from_numpy(c).cuda(),
                                             s_w, Rg, Cg, dqt.adafactor(step=t, **HPS[hpi]))
        assert np.allclose(Rg.cpu().numpy(), R, rtol=1e-5, atol=0)
        assert np.allclose(Cg.cpu().numpy(), Cc, rtol=1e-5, atol=0)
        assert np.allclose(ag.cpu().numpy(), st["a"], rtol=1e-5, atol=0)
        assert np.allclose(bg.cpu().numpy(), st["b"], rtol=1e-5, atol=0)
        s = sc.cpu().numpy().astype(np.float64)
        for i, key in enumerate(["rbar", "step", "decay", "rms_u", "rms_x", "alpha"]):
            if key == "rms_x" and not HPS[hpi].get("scale_parameter"):
                assert s[i] == 0.0  # the codes are read only for parameter scaling
                continue
            assert s[i] == pytest.approx(float(st[key]), rel=1e-5), (t, key)


@pytest.mark.parametrize("N,K,bits_w,packed,round_mode", [
    (512, 512, 1.58, False, 0), (512, 512, 1.58, True, 0), (264, 520, 4, False, 0),
    (264, 520, 1.58, True, 1), (5632, 2048, 1.58, True, 0), (2048, 5632, 8, False, 0)])
def test_adafactor_apply_bit_exact(N, K, bits_w, packed, round_mode):
    """The per-element step given the oracle's statistics."""
    c, s_w, (qmin, qmax) = _af_problem(N, K, bits_w, seed=K)
    g = inputs.normal((N, K), 1e-3, seed=N).numpy()
    hpo = oracle.AdafactorHP(lr=1e-2)
    R, Cc, st = oracle.adafactor_stats(g, c, s_w, np.zeros(N), np.zeros(K), 1, hpo)
    c1, ch = oracle.adafactor_apply(g, c, st["a"], st["b"], st["step"], st["decay"], qmin, qmax,
                                    77, 1, 9, round_mode)
    scal = torch.tensor([np.float32(st["rbar"]), st["step"], st["decay"], 0, 0, 0, 0, 0],
                        dtype=torch.float32, device="cuda")
    W = torch.from_numpy(oracle.pack_ternary(c) if packed else c).cuda()
    changed = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_adafactor_apply(torch.from_numpy(g).cuda(), W, torch.from_numpy(st["a"]).cuda(),
                            torch.from_numpy(st["b"]).cuda(), scal, 1,
                            dqt.sr_stream(seed=77, tensor_id=9, round_mode=round_mode),
                            (qmin, qmax), packed=packed, changed_out=changed)
    got = oracle.unpack_ternary(W.cpu().numpy(), N * K).reshape(N, K) if packed else W.cpu().numpy()
    assert (got == c1).all()
    assert int(changed.item()) == ch


@pytest.mark.parametrize("T,K,N,bits_w,packed", [(256, 512, 512, 1.58, False),
                                                 (300, 264, 520, 1.58, True),
                                                 (512, 768, 768, 8, False)])
def test_bwd_dw_adafactor(T, K, N, bits_w, packed):
    """dW on the tensor cores + statistics + step, against the oracle fed the
    bf16-environment gradient, over two steps.  Each step is checked on its
    own: the oracle starts from the GPU's codes and R, C after the step
    before, so a difference of step 1 is not carried into step 2."""
    X = inputs.normal((T, K), 1.0, seed=T, dtype=torch.bfloat16)
    c, s_w, (qmin, qmax) = _af_problem(N, K, bits_w, seed=N)
    Xg = X.cuda()
    _, s_x, _, xdq = dqt.dqt_act_quant_images(Xg, want=("Xdq",))
    xd = bits(xdq)
    Rg = torch.zeros(N, device="cuda")
    Cg = torch.zeros(K, device="cuda")
    W = torch.from_numpy(oracle.pack_ternary(c) if packed else c.copy()).cuda()
    hpo = oracle.AdafactorHP(lr=1e-2)
    for t in (1, 2):
        # the GPU state the step starts from, which the oracle starts from too
        cur = (oracle.unpack_ternary(W.cpu().numpy(), N * K).reshape(N, K) if packed
               else W.cpu().numpy().copy())
        R0, C0 = Rg.cpu().numpy().copy(), Cg.cpu().numpy().copy()
        dY = inputs.normal((T, N), 1e-2, seed=100 * t + T, dtype=torch.bfloat16)
        g = oracle.bwd_dw_bf16x(bits(dY), xd).astype(np.float32)
        R, Cc, st = oracle.adafactor_stats(g, cur, s_w, R0, C0, t, hpo)
        ref, _ = oracle.adafactor_apply(g, cur, st["a"], st["b"], st["step"], st["decay"], qmin,
                                        qmax, 4, t, 2)
        dqt.dqt_bitlinear_bwd_dw_adafactor(dY.cuda(), xdq, W, s_w, Rg, Cg,
                                           dqt.adafactor(lr=1e-2, step=t),
                                           dqt.sr_stream(seed=4, tensor_id=2), (qmin, qmax),
                                           packed=packed)
        got = (oracle.unpack_ternary(W.cpu().numpy(), N * K).reshape(N, K) if packed
               else W.cpu().numpy())
        assert_fused_codes(got, ref, what="step %d" % t)
        assert np.allclose(Rg.cpu().numpy(), R, rtol=1e-4) and np.allclose(Cg.cpu().numpy(), Cc, rtol=1e-4)
