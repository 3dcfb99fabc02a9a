"""DQTBitLinear (the torch module over the C ABI) and the LLaMA-structured DQT
decoder.

* The module's forward is the oracle's BitLinear forward bit for bit; its
  backward returns dX within the dX tolerance and leaves the codes where the
  oracle's DQT update (Eq. 5, fed the bf16-environment weight gradient) puts
  them, to the fused-update tolerance.
* state_dict carries the whole DQT state: reload + step == continue.
* A small decoder trained on a fixed batch lowers its loss with ternary and
  8-bit weights (Sec. 4.2: training with only low-precision weights
  converges), and its BitLinear codes move.  With round-to-nearest instead of
  stochastic rounding (the Sec. 5.1 ablation) and lr * s_w < 1/2, no code can
  ever move: the update is lost, as the paper observes.
"""
import io
import os

import numpy as np
import pytest
import torch

import oracle
from fused_rule import assert_fused_codes
from paper_2412_04787_gb300 import inputs

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _cuda():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from paper_2412_04787_gb300 import build
    build.build()


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


@pytest.mark.parametrize("bits_w", [1.58, 8])
def test_bitlinear_module_matches_oracle(bits_w):
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    T, K, N = 300, 264, 520
    layer = DQTBitLinear(K, N, bits=bits_w, lr=1e-3, seed=99, tensor_id=4, init_seed=7)
    qmin, qmax = layer.grid_tuple
    # the layer starts from the oracle's AbsMean codes of a seeded W0
    c0, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=7).numpy(), qmin, qmax)
    layer.codes.copy_(torch.from_numpy(c0))
    layer.s_w = float(s_w)
    X = inputs.normal((T, K), 1.0, seed=1, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=2, dtype=torch.bfloat16)
    x = X.cuda().requires_grad_(True)
    y = layer(x)
    torch.cuda.synchronize()
    q, s, _, xd = oracle.act_quant(bits(X))
    Yr, _ = oracle.fwd(q, s, c0, np.float32(layer.s_w))
    assert np.array_equal(bits(y), Yr)
    y.backward(dY.cuda())
    torch.cuda.synchronize()
    dXr = oracle.bwd_dx(bits(dY), c0, np.float32(layer.s_w))
    err = np.abs(x.grad.cpu().double().numpy() - dXr).max() / np.abs(dXr).max()
    assert err <= 2e-2
    g = oracle.bwd_dw_bf16x(bits(dY), xd).astype(np.float32)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, layer.s_w)
    z = np.zeros((N, K), np.float32)
    c1, m1, _, _ = oracle.update(g, c0, z, z, k, qmin, qmax, 99, 1, 4)
    cg = layer.codes.cpu().numpy().astype(np.int32)
    assert_fused_codes(cg, c1)
    assert layer.step == 1 and int(layer.changed.item()) == int((cg != c0).sum())


def test_module_backward_in_a_fresh_process():
    """The first CUDA work of the autograd worker thread of a fresh process is
    this library's dX GEMM, whose tensor-map encoder (a driver call) needs a
    context bound in that thread: a process of its own, so that no earlier test
    has already bound one there."""
    import subprocess
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    code = (
        "import torch\n"
        "from paper_2412_04787_gb300.bitlinear import DQTBitLinear\n"
        "layer = DQTBitLinear(264, 520, bits=1.58, seed=3, tensor_id=1, init_seed=5)\n"
        "x = torch.randn(300, 264, device='cuda', dtype=torch.bfloat16, requires_grad=True)\n"
        "layer(x).backward(torch.randn(300, 520, device='cuda', dtype=torch.bfloat16))\n"
        "torch.cuda.synchronize()\n"
        "assert x.grad is not None and int(layer.step) == 1\n"
        "print('ok')\n")
    r = subprocess.run([sys.executable, "-c", code], cwd=root, capture_output=True, text=True,
                       timeout=600)
    assert r.returncode == 0 and "ok" in r.stdout, r.stderr[-3000:]


def test_bitlinear_state_dict_resume():
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    K, N = 128, 256
    a = DQTBitLinear(K, N, bits=4, seed=5, tensor_id=1, init_seed=11)
    b = DQTBitLinear(K, N, bits=4, seed=5, tensor_id=1, init_seed=12)  # different init
    xs = [inputs.normal((64, K), 1.0, seed=20 + i, dtype=torch.bfloat16).cuda() for i in range(2)]
    gs = [inputs.normal((64, N), 1e-2, seed=30 + i, dtype=torch.bfloat16).cuda() for i in range(2)]
    a(xs[0].requires_grad_(True)).backward(gs[0])
    buf = io.BytesIO()
    torch.save(a.state_dict(), buf)
    buf.seek(0)
    b.load_state_dict(torch.load(buf, weights_only=False))
    assert b.step == 1 and b.s_w == a.s_w
    for layer in (a, b):
        layer(xs[1].clone().requires_grad_(True)).backward(gs[1])
    torch.cuda.synchronize()
    for name in ("codes", "m", "v"):
        assert torch.equal(getattr(a, name), getattr(b, name)), name


def _train(bits_w, round_mode=0, steps=40, act="int8", optimizer="adamw", packed=False, lr=2e-3):
    from paper_2412_04787_gb300.decoder import DecoderConfig, DQTDecoder
    torch.manual_seed(0)
    cfg = DecoderConfig(layers=2, hidden=128, heads=4, ffn=256, vocab=512, bits=bits_w,
                        lr=lr, seed=7, act=act, optimizer=optimizer, packed=packed)
    model = DQTDecoder(cfg)
    for m in model.bitlinear_layers():
        m.round_mode = round_mode
    opt = torch.optim.AdamW(model.dense_parameters(), lr=2e-3)
    g = torch.Generator().manual_seed(3)
    ids = torch.randint(0, cfg.vocab, (4, 65), generator=g).cuda()
    codes0 = [m.int8_codes().clone() for m in model.bitlinear_layers()]
    losses = []
    for _ in range(steps):
        loss = model(ids[:, :-1], ids[:, 1:])
        loss.backward()
        opt.step()
        opt.zero_grad(set_to_none=True)
        losses.append(float(loss.detach()))
    moved = sum(int((m.int8_codes() != c).sum()) for m, c in zip(model.bitlinear_layers(), codes0))
    return losses, moved, model


@pytest.mark.parametrize("bits_w", [1.58, 8])
def test_decoder_trains_with_low_bit_weights(bits_w):
    losses, moved, model = _train(bits_w)
    assert all(np.isfinite(losses))
    assert losses[-1] < 0.8 * losses[0], (losses[0], losses[-1])
    assert moved > 0
    for m in model.bitlinear_layers():
        lo, hi = m.grid_tuple
        c = m.int8_codes()
        assert int(c.min()) >= lo and int(c.max()) <= hi


@pytest.mark.parametrize("packed", [False, True])
def test_decoder_trains_with_adafactor(packed):
    """Sec. 4.3: DQT with the memory-efficient Adafactor optimiser (here with
    2-bit packed ternary codes as well) still trains."""
    losses, moved, model = _train(1.58, optimizer="adafactor", packed=packed, lr=1e-2)
    assert all(m.optimizer == "adafactor" and m.packed == packed for m in model.bitlinear_layers())
    assert all(np.isfinite(losses))
    assert losses[-1] < 0.8 * losses[0], (losses[0], losses[-1])
    assert moved > 0


def test_packed_module_equals_int8_module():
    """AdamW on packed ternary codes: the same forward, dX and codes as on int8 codes."""
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    T, K, N = 256, 264, 520
    a = DQTBitLinear(K, N, bits=1.58, seed=3, tensor_id=2, init_seed=5)
    b = DQTBitLinear(K, N, bits=1.58, seed=3, tensor_id=2, init_seed=5, packed=True)
    assert b.codes.numel() == (N * K + 3) // 4
    assert torch.equal(a.codes, b.int8_codes())
    for i in range(2):
        X = inputs.normal((T, K), 1.0, seed=40 + i, dtype=torch.bfloat16).cuda()
        dY = inputs.normal((T, N), 1e-2, seed=50 + i, dtype=torch.bfloat16).cuda()
        xa = X.clone().requires_grad_(True)
        xb = X.clone().requires_grad_(True)
        ya, yb = a(xa), b(xb)
        assert torch.equal(ya, yb)
        ya.backward(dY)
        yb.backward(dY)
        assert torch.equal(xa.grad, xb.grad)
        assert torch.equal(a.codes, b.int8_codes()) and torch.equal(a.m, b.m) and torch.equal(a.v, b.v)


def test_adafactor_module_matches_oracle():
    """optimizer="adafactor": after one backward the codes are the oracle's
    Adafactor + SR step of the bf16-environment gradient (fused tolerance)."""
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    T, K, N = 300, 264, 520
    layer = DQTBitLinear(K, N, bits=4, lr=1e-2, seed=8, tensor_id=6, init_seed=9,
                         optimizer="adafactor")
    qmin, qmax = layer.grid_tuple
    c0, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=9).numpy(), qmin, qmax)
    layer.codes.copy_(torch.from_numpy(c0))
    layer.s_w = float(s_w)
    X = inputs.normal((T, K), 1.0, seed=1, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=2, dtype=torch.bfloat16)
    layer(X.cuda().requires_grad_(True)).backward(dY.cuda())
    torch.cuda.synchronize()
    _, _, _, xd = oracle.act_quant(bits(X))
    g = oracle.bwd_dw_bf16x(bits(dY), xd).astype(np.float32)
    hp = oracle.AdafactorHP(lr=1e-2)
    R, Cc, st = oracle.adafactor_stats(g, c0, np.float32(layer.s_w), np.zeros(N), np.zeros(K), 1, hp)
    c1, _ = oracle.adafactor_apply(g, c0, st["a"], st["b"], st["step"], st["decay"], qmin, qmax,
                                   8, 1, 6)
    cg = layer.codes.cpu().numpy().astype(np.int32)
    assert_fused_codes(cg, c1)
    assert np.allclose(layer.R.cpu().numpy(), R, rtol=1e-4)


def test_decoder_trains_in_fp8_environment():
    """The same decoder with the E4M3 BitLinear forward (Sec. 4.3: DQT stays
    robust when moving to the FP8 environment)."""
    losses, moved, model = _train(1.58, act="fp8")
    assert all(m.act == "fp8" for m in model.bitlinear_layers())
    assert all(np.isfinite(losses))
    assert losses[-1] < 0.8 * losses[0], (losses[0], losses[-1])
    assert moved > 0


def test_bitlinear_module_fp8_matches_oracle():
    """act="fp8": the forward is the oracle's E4M3 forward (fp32-accumulation
    bound), and the update is the oracle's DQT update fed the weight gradient
    of the E4M3 dequantised activation (fused-update tolerance)."""
    from paper_2412_04787_gb300.bitlinear import DQTBitLinear
    T, K, N = 300, 272, 520
    layer = DQTBitLinear(K, N, bits=1.58, lr=1e-3, seed=99, tensor_id=4, init_seed=7, act="fp8")
    qmin, qmax = layer.grid_tuple
    c0, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=7).numpy(), qmin, qmax)
    layer.codes.copy_(torch.from_numpy(c0))
    layer.s_w = float(s_w)
    X = inputs.normal((T, K), 1.0, seed=1, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=2, dtype=torch.bfloat16)
    x = X.cuda().requires_grad_(True)
    y = layer(x)
    torch.cuda.synchronize()
    q8, s8, xd = oracle.act_quant_fp8(bits(X))
    Yr, acc = oracle.fwd_fp8(q8, s8, c0, np.float32(layer.s_w))
    xv = np.vectorize(oracle.e4m3_value)(q8)
    mag = np.abs(xv) @ np.abs(c0.astype(np.float64)).T
    a_t = (np.float32(1.0) / (s8 * np.float32(layer.s_w))).astype(np.float64)
    y_ref = torch.from_numpy(Yr.view(np.int16)).view(torch.bfloat16).double().numpy()
    y_gpu = y.detach().double().cpu().numpy()
    ulp = np.exp2(np.floor(np.log2(np.maximum(np.abs(y_ref), 1e-38))) - 7)
    assert (np.abs(y_gpu - y_ref) <= ulp + a_t[:, None] * (K - 1) * 2.0 ** -24 * mag * 1.01).all()
    y.backward(dY.cuda())
    torch.cuda.synchronize()
    g = oracle.bwd_dw_bf16x(bits(dY), xd).astype(np.float32)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, layer.s_w)
    z = np.zeros((N, K), np.float32)
    c1, _, _, _ = oracle.update(g, c0, z, z, k, qmin, qmax, 99, 1, 4)
    cg = layer.codes.cpu().numpy().astype(np.int32)
    assert_fused_codes(cg, c1)


def test_round_to_nearest_loses_small_updates():
    """Ternary, lr * s_w < 1/2: |x - c| <= lr * s_w * |u| with |u| <= ~1 at
    these steps, so rint(x) == c and no BitLinear code ever moves."""
    losses, moved, model = _train(1.58, round_mode=1, steps=10)
    assert max(m.lr * m.s_w for m in model.bitlinear_layers()) < 0.5
    assert moved == 0


def test_device_consts_update_matches_host_path():
    """The _dev entry points with the constants block in device memory give
    exactly the host-constant path's codes and moments (fused and standalone)."""
    from paper_2412_04787_gb300 import dqt
    T, K, N = 256, 264, 520
    qmin, qmax = oracle.grid(8)
    c0, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=3).numpy(), qmin, qmax)
    X = inputs.normal((T, K), 1.0, seed=4, dtype=torch.bfloat16).cuda()
    dY = inputs.normal((T, N), 1e-2, seed=5, dtype=torch.bfloat16).cuda()
    _, s_x, _, xdq = dqt.dqt_act_quant_images(X, want=("Xdq",))
    hp = dqt.adamw(lr=1e-3, weight_decay=0.01, step=3)
    sr = dqt.sr_stream(seed=11, tensor_id=2)
    blk = dqt.dqt_update_consts(hp, sr, (qmin, qmax), float(s_w))
    dev = blk.cuda()
    m0 = inputs.normal((N, K), 1e-4, seed=6).cuda()
    v0 = inputs.normal((N, K), 1e-4, seed=7).square().cuda()
    a = [torch.from_numpy(c0).cuda(), m0.clone(), v0.clone()]
    b = [torch.from_numpy(c0).cuda(), m0.clone(), v0.clone()]
    dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, a[0], float(s_w), a[1], a[2], hp, sr, (qmin, qmax))
    dqt.dqt_bitlinear_bwd_dw_update_dev(dY, xdq, b[0], b[1], b[2], dev)
    g = inputs.normal((N * K,), 1e-3, seed=8).cuda()
    dqt.dqt_sr_update(g, a[0].view(-1), float(s_w), a[1].view(-1), a[2].view(-1), hp, sr, (qmin, qmax))
    dqt.dqt_sr_update_dev(g, b[0].view(-1), b[1].view(-1), b[2].view(-1), dev)
    dqt.dqt_check_device_status()
    for x, y in zip(a, b):
        assert torch.equal(x, y)


def test_graph_replayed_decoder_equals_eager():
    """Whole training steps captured once in a CUDA graph and replayed with a
    new step each time (constants uploaded from the pinned block) leave the
    model in exactly the state eager steps do."""
    from paper_2412_04787_gb300.decoder import DecoderConfig, DQTDecoder

    def make():
        cfg = DecoderConfig(layers=2, hidden=128, heads=4, ffn=256, vocab=512, bits=1.58,
                            lr=2e-3, seed=9)
        model = DQTDecoder(cfg)
        model.enable_graph_updates()
        opt = torch.optim.AdamW(model.dense_parameters(), lr=2e-3, capturable=True)
        return model, opt

    g = torch.Generator().manual_seed(4)
    batches = [torch.randint(0, 512, (4, 65), generator=g).cuda() for _ in range(6)]

    def eager_step(model, opt, ids, slot):
        model.prepare_step(slot)
        model.upload_update_consts(slot)
        loss = model(ids[:, :-1], ids[:, 1:])
        loss.backward()
        opt.step()
        opt.zero_grad(set_to_none=True)

    ea, oa = make()
    for i, ids in enumerate(batches):
        eager_step(ea, oa, ids, i % 2)

    gb, ob = make()
    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        for i, ids in enumerate(batches[:2]):
            eager_step(gb, ob, ids, i % 2)
    torch.cuda.current_stream().wait_stream(side)
    static_ids = batches[2].clone()
    graph = torch.cuda.CUDAGraph()
    ob.zero_grad(set_to_none=True)
    with torch.cuda.graph(graph):
        loss = gb(static_ids[:, :-1], static_ids[:, 1:])
        loss.backward()
        ob.step()
    for i, ids in enumerate(batches[2:], start=2):
        static_ids.copy_(ids)
        gb.prepare_step(i % 2)
        gb.upload_update_consts(i % 2)
        graph.replay()
    torch.cuda.synchronize()
    for la, lb in zip(ea.bitlinear_layers(), gb.bitlinear_layers()):
        assert la.step == lb.step == 6
        assert torch.equal(la.codes, lb.codes)
        assert torch.equal(la.m, lb.m) and torch.equal(la.v, lb.v)
