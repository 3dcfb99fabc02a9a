"""Checkpoint / resume: the DQT state is the int8 codes, the fp32 moments and
(seed, step).  The uniforms of stochastic rounding are keyed by (seed, step,
tensor id, element), and every kernel reduces in a fixed order, so two steps
run straight through and one step, a save/reload through host memory, then
the second step give bit-identical state; repeating a step from the same
state gives the same result."""
import io

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


def _layer(bits_w, T=320, K=264, N=520, seed=3):
    qmin, qmax = oracle.grid(bits_w)
    W0 = inputs.normal((N, K), 0.02, seed=seed)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    X = [inputs.normal((T, K), 1.0, seed=seed + 10 + i, dtype=torch.bfloat16).cuda() for i in range(2)]
    dY = [inputs.normal((T, N), 1e-2, seed=seed + 20 + i, dtype=torch.bfloat16).cuda() for i in range(2)]
    state = {"W": torch.from_numpy(c).cuda(), "m": torch.zeros((N, K), device="cuda"),
             "v": torch.zeros((N, K), device="cuda")}
    return (qmin, qmax), float(s_w), X, dY, state


def _step(g, s_w, X, dY, state, step):
    _, s_x, q_img, xdq = dqt.dqt_act_quant_images(X, want=("Xq_img", "Xdq"))
    W_img = dqt.dqt_codes_to_bf16(state["W"])
    dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, s_w, g)
    dqt.dqt_bitlinear_bwd_dx_img(dY, W_img, s_w)
    dqt.dqt_bitlinear_bwd_dw_update_img(dY, xdq, state["W"], s_w, state["m"], state["v"],
                                        dqt.adamw(lr=1e-3, step=step),
                                        dqt.sr_stream(seed=77, tensor_id=5), g)
    dqt.dqt_check_device_status()


@pytest.mark.parametrize("bits_w", [1.58, 8])
def test_resume_is_bit_exact(bits_w):
    g, s_w, X, dY, a = _layer(bits_w)
    _, _, _, _, b = _layer(bits_w)
    # straight through
    _step(g, s_w, X[0], dY[0], a, 1)
    _step(g, s_w, X[1], dY[1], a, 2)
    # step, checkpoint to host bytes, reload into fresh tensors, step
    _step(g, s_w, X[0], dY[0], b, 1)
    buf = io.BytesIO()
    torch.save({k: v.cpu() for k, v in b.items()}, buf)
    buf.seek(0)
    restored = {k: v.cuda() for k, v in torch.load(buf).items()}
    _step(g, s_w, X[1], dY[1], restored, 2)
    for k in ("W", "m", "v"):
        assert torch.equal(a[k], restored[k]), k
    assert (a["W"].cpu().numpy() != _layer(bits_w)[4]["W"].cpu().numpy()).any()


def test_repeated_step_is_deterministic():
    g, s_w, X, dY, a = _layer(4)
    _, _, _, _, b = _layer(4)
    _step(g, s_w, X[0], dY[0], a, 3)
    _step(g, s_w, X[0], dY[0], b, 3)
    for k in ("W", "m", "v"):
        assert torch.equal(a[k], b[k]), k
