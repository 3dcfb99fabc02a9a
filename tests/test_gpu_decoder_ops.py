"""Decoder-support kernels (not part of the DQT method) against references on
the same inputs: the rotary embedding bit-exact against the same formula in
separately rounded fp32 torch operations (and its backward against autograd
through that formula); the token cross-entropy against F.cross_entropy on the
fp32 upcast of the same bf16 logits; the SwiGLU gate and RMSNorm (outputs and
all gradients) against fp64 within one bf16 rounding, and close to PyTorch's
own silu * up and rms_norm."""
import pytest
import torch
import torch.nn.functional as F

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


def _table(S, D, theta=10000.0):
    inv = 1.0 / (theta ** (torch.arange(0, D, 2, dtype=torch.float32, device="cuda") / D))
    ang = torch.outer(torch.arange(S, dtype=torch.float32, device="cuda"), inv)
    return torch.stack((torch.cos(ang), torch.sin(ang)), dim=-1).contiguous()


def _rope_ref(x, cs, sign=1.0):
    """y[2i] = x[2i] c - x[2i+1] s, y[2i+1] = x[2i] s + x[2i+1] c, each op one
    fp32 rounding, then bf16 (nearest-even)."""
    xf = x.float()
    xe, xo = xf[..., 0::2], xf[..., 1::2]
    c = cs[None, :, None, :, 0]
    s = cs[None, :, None, :, 1] * sign
    ye = xe * c - xo * s
    yo = xe * s + xo * c
    return torch.stack((ye, yo), dim=-1).flatten(-2).to(torch.bfloat16)


@pytest.mark.parametrize("B,S,H,D", [(2, 37, 3, 64), (1, 1, 1, 8), (3, 128, 12, 64), (2, 16, 4, 128)])
def test_rope_matches_fp32_formula(B, S, H, D):
    x = inputs.normal((B, S, H, D), 1.0, seed=S + D, dtype=torch.bfloat16).cuda()
    cs = _table(S, D)
    y = dqt.dqt_rope_bf16(x, cs)
    assert torch.equal(y, _rope_ref(x, cs))
    yi = dqt.dqt_rope_bf16(x, cs, inverse=True)
    assert torch.equal(yi, _rope_ref(x, cs, -1.0))
    # rotating back recovers x up to the two bf16 roundings
    back = dqt.dqt_rope_bf16(y, cs, inverse=True).float()
    assert (back - x.float()).abs().max() <= 2 ** -7 * x.float().abs().max()


def test_rope_backward_is_the_transpose():
    from paper_2412_04787_gb300.decoder import _Rope
    B, S, H, D = 2, 24, 4, 64
    x = inputs.normal((B, S, H, D), 1.0, seed=3, dtype=torch.bfloat16).cuda().requires_grad_()
    g = inputs.normal((B, S, H, D), 1.0, seed=4, dtype=torch.bfloat16).cuda()
    cs = _table(S, D)
    _Rope.apply(x, cs).backward(g)
    # d/dx of the rotation: the rotation by -theta applied to g
    assert torch.equal(x.grad, _rope_ref(g, cs, -1.0))
    # and it agrees with autograd through the fp32 formula (to bf16 rounding)
    xr = x.detach().float().requires_grad_()
    xe, xo = xr[..., 0::2], xr[..., 1::2]
    c, s = cs[None, :, None, :, 0], cs[None, :, None, :, 1]
    torch.stack((xe * c - xo * s, xe * s + xo * c), dim=-1).flatten(-2).backward(g.float())
    assert (x.grad.float() - xr.grad).abs().max() <= 2 ** -8 * xr.grad.abs().max()


@pytest.mark.parametrize("M,V", [(64, 512), (300, 32000), (7, 8)])
def test_cross_entropy_matches_torch(M, V):
    from paper_2412_04787_gb300.decoder import _TokenCrossEntropy
    logits = (inputs.normal((M, V), 2.0, seed=M, dtype=torch.bfloat16)).cuda().requires_grad_()
    gen = torch.Generator().manual_seed(V)
    tg = torch.randint(0, V, (M,), generator=gen)
    if M > 4:
        tg[3] = -100  # ignored row, as F.cross_entropy's default ignore_index
    tg = tg.cuda()
    loss = _TokenCrossEntropy.apply(logits, tg)
    loss.backward()
    ref_in = logits.detach().float().requires_grad_()
    ref = F.cross_entropy(ref_in, tg)
    ref.backward()
    assert abs(loss.item() - ref.item()) <= 1e-5 * abs(ref.item())
    gref = ref_in.grad
    # the kernel rounds its fp32 gradient to bf16 once; fp32 rounding
    # differences may flip that rounding: within one bf16 ulp (2^-7 relative)
    err = (logits.grad.float() - gref).abs()
    assert (err <= 2 ** -7 * gref.abs() + 1e-12).all()
    if M > 4:
        assert torch.count_nonzero(logits.grad[3]) == 0


def test_cross_entropy_row_values():
    """lse and the row loss of a hand-checkable row: logits (0, ln 3, 0, 0, ...)."""
    V = 8
    row = torch.zeros(1, V)
    row[0, 1] = float(torch.log(torch.tensor(3.0)))
    logits = row.to(torch.bfloat16).cuda()
    lse, loss = dqt.dqt_cross_entropy_fwd_bf16(logits, torch.tensor([1], device="cuda"))
    x1 = logits.float()[0, 1].item()
    expect = float(torch.log(torch.tensor(7.0 + torch.exp(torch.tensor(x1)).item())))
    assert abs(lse.item() - expect) <= 1e-6
    assert abs(loss.item() - (expect - x1)) <= 1e-6


@pytest.mark.parametrize("shape", [(8,), (3, 40), (64, 5632)])
def test_swiglu_matches_fp64(shape):
    from paper_2412_04787_gb300.decoder import _SwiGLU
    g = inputs.normal(shape, 2.0, seed=1, dtype=torch.bfloat16).cuda().requires_grad_()
    u = inputs.normal(shape, 1.0, seed=2, dtype=torch.bfloat16).cuda().requires_grad_()
    dh = inputs.normal(shape, 1.0, seed=3, dtype=torch.bfloat16).cuda()
    h = _SwiGLU.apply(g, u)
    h.backward(dh)
    gd, ud, hd = g.detach().double(), u.detach().double(), dh.double()
    s = torch.sigmoid(gd)
    ref_h = gd * s * ud
    ref_dg = hd * ud * s * (1 + gd * (1 - s))
    ref_du = hd * gd * s
    # one rounding of an fp32 evaluation to bf16: within one bf16 ulp
    for got, ref in ((h, ref_h), (g.grad, ref_dg), (u.grad, ref_du)):
        err = (got.double() - ref).abs()
        assert (err <= 2 ** -7 * ref.abs() + 1e-30).all()
    # and close to PyTorch's own silu(g) * u (which rounds silu(g) to bf16 first)
    ref_t = F.silu(g.detach()) * u.detach()
    assert ((h.float() - ref_t.float()).abs() <= 2 ** -6 * ref_t.float().abs() + 1e-30).all()


@pytest.mark.parametrize("rows,D", [(1, 8), (37, 768), (300, 2048), (64, 1288)])
def test_rmsnorm_matches_fp64(rows, D):
    from paper_2412_04787_gb300.decoder import _RMSNorm
    eps = 1e-6
    x = inputs.normal((rows, D), 1.0, seed=rows + D, dtype=torch.bfloat16).cuda().requires_grad_()
    w = (1.0 + inputs.normal((D,), 0.1, seed=D, dtype=torch.float32)).to(torch.bfloat16).cuda()
    w.requires_grad_()
    dy = inputs.normal((rows, D), 1.0, seed=rows, dtype=torch.bfloat16).cuda()
    y = _RMSNorm.apply(x, w, eps)
    y.backward(dy)
    xd, wd, gd = x.detach().double(), w.detach().double(), dy.double()
    r = 1.0 / torch.sqrt((xd * xd).mean(dim=1, keepdim=True) + eps)
    ref_y = xd * r * wd
    assert ((y.double() - ref_y).abs() <= 2 ** -7 * ref_y.abs() + 1e-30).all()
    # dx = r w dy - x r^3 mean(w dy x): bounded relative to its two terms
    t1 = r * wd * gd
    t2 = xd * r ** 3 * (wd * gd * xd).mean(dim=1, keepdim=True)
    err = (x.grad.double() - (t1 - t2)).abs()
    assert (err <= 2 ** -7 * (t1.abs() + t2.abs()) + 1e-6).all()
    # dw = sum over rows of dy x r (fp32 sums in a fixed order, one bf16 rounding)
    terms = gd * xd * r
    ref_dw = terms.sum(dim=0)
    err = (w.grad.double() - ref_dw).abs()
    assert (err <= 2 ** -7 * ref_dw.abs() + 1e-5 * terms.abs().sum(dim=0)).all()
    # the decoder's module agrees with PyTorch's own rms_norm to bf16 rounding
    ref_t = F.rms_norm(x.detach(), (D,), w.detach(), eps)
    assert ((y.float() - ref_t.float()).abs() <= 2 ** -6 * ref_t.float().abs() + 1e-6).all()


def test_rmsnorm_gain_gradient_is_deterministic():
    from paper_2412_04787_gb300.decoder import _RMSNorm
    x = inputs.normal((4096, 768), 1.0, seed=9, dtype=torch.bfloat16).cuda()
    w = torch.ones(768, dtype=torch.bfloat16, device="cuda")
    dy = inputs.normal((4096, 768), 1.0, seed=10, dtype=torch.bfloat16).cuda()
    grads = []
    for _ in range(2):
        xi, wi = x.clone().requires_grad_(), w.clone().requires_grad_()
        _RMSNorm.apply(xi, wi, 1e-6).backward(dy)
        grads.append((xi.grad, wi.grad))
    assert torch.equal(grads[0][0], grads[1][0]) and torch.equal(grads[0][1], grads[1][1])
