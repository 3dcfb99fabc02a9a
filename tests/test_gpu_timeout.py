"""Failure detection on the GPU without a fault: a bounded device wait that
runs out is reported to the host as DQT_ERR_TIMEOUT, the kernel returns, and
the CUDA context stays usable (the next launch is bit-exact again).

The wait limit is set to zero, so the epilogue's first wait for the tensor
cores (tens of microseconds of MMAs at K = 8192) gives up after about a
microsecond: a wait on a flag that has not been set yet."""
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
    yield
    dqt.dqt_set_wait_limit_ns(2_000_000_000)


def _bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def test_timeout_reported_and_context_survives():
    T, K, N = 1024, 8192, 1024  # a tile's MMAs take tens of microseconds
    X = inputs.normal((T, K), 1.0, seed=5, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=6)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), -1, 1)
    _, s_x, q_img, _ = dqt.dqt_act_quant_images(X.cuda(), want=("Xq_img",))
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    dqt.dqt_check_device_status()

    dqt.dqt_set_wait_limit_ns(0)
    try:
        dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, float(s_w), (-1, 1))
        with pytest.raises(dqt.DQTError) as err:
            dqt.dqt_check_device_status()
        assert err.value.status == dqt.DQT_ERR_TIMEOUT
    finally:
        dqt.dqt_set_wait_limit_ns(2_000_000_000)

    # the record is cleared and the context is usable: a normal launch is exact
    acc = torch.empty((T, N), dtype=torch.int32, device="cuda")
    dqt.dqt_bitlinear_fwd_img(q_img, s_x, W_img, float(s_w), (-1, 1), acc_out=acc)
    dqt.dqt_check_device_status()
    q, s, _, _ = oracle.act_quant(_bits(X))
    rows = np.array([0, 511, 1023])
    _, accr = oracle.fwd(q[rows], s[rows], c, np.float32(s_w))
    assert np.array_equal(acc.cpu().numpy()[rows], accr)
