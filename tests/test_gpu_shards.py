"""Sharded updates on the GPU: the global element offset of the SR stream
(dqt_sr_t.elem0) and the data-parallel exchange of paper_2412_04787_gb300/dp.py.

Element e of a weight draws the Philox uniform of its global index e, so a
rank that updates the shard [a, b) with elem0 = a writes exactly the codes,
moments and changed-code count that the whole-tensor update writes there.
Checked bit for bit through the C ABI for int8 codes, 2-bit packed codes and
device-resident constants, and the fused weight-gradient path with an offset
against the standalone update with the same offset; then the exchange itself
over a one-rank NCCL group (reduce-scatter, the library's update of the
shard, all-gather) against the plain update.  The multi-rank host logic of
the exchange is covered on CPU gloo ranks.
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


def _state(numel, bits, step, seed):
    qmin, qmax = oracle.grid(bits)
    c, s_w, _ = oracle.absmean_init(inputs.normal((numel,), 0.02, seed=seed).numpy(), qmin, qmax)
    g = inputs.normal((numel,), 1e-3, seed=seed + 1)
    if step > 1:
        m = inputs.normal((numel,), 1e-4, seed=seed + 2)
        v = inputs.normal((numel,), 1e-4, seed=seed + 3).square()
    else:
        m = torch.zeros(numel)
        v = torch.zeros(numel)
    return torch.from_numpy(c), float(s_w), g, m, v, (qmin, qmax)


@pytest.mark.parametrize("numel,cut,bits,step", [(1_000_003, 499_968, 8, 3),
                                                  (262_144 + 7, 131_072 + 64, 1.58, 1),
                                                  (4099, 16, 4, 2)])
def test_sr_update_halves_equal_whole(numel, cut, bits, step):
    c, s_w, g, m, v, grid = _state(numel, bits, step, seed=numel % 1000)
    hp = dqt.adamw(lr=1e-3, weight_decay=0.01, step=step)
    W1, m1, v1 = c.cuda(), m.clone().cuda(), v.clone().cuda()
    ch1 = torch.zeros(1, dtype=torch.int64, device="cuda")
    dqt.dqt_sr_update(g.cuda(), W1, s_w, m1, v1, hp, dqt.sr_stream(seed=9, tensor_id=4), grid,
                      changed_out=ch1)
    W2, m2, v2, gg = c.cuda(), m.clone().cuda(), v.clone().cuda(), g.cuda()
    ch2 = torch.zeros(1, dtype=torch.int64, device="cuda")
    for lo, hi in [(0, cut), (cut, numel)]:
        dqt.dqt_sr_update(gg[lo:hi], W2[lo:hi], s_w, m2[lo:hi], v2[lo:hi], hp,
                          dqt.sr_stream(seed=9, tensor_id=4, elem0=lo), grid, changed_out=ch2)
    dqt.dqt_check_device_status()
    assert torch.equal(W1, W2) and torch.equal(m1, m2) and torch.equal(v1, v2)
    assert int(ch1.item()) == int(ch2.item())
    # and the oracle's shard update gives the second half's codes
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, step, s_w)
    c_ref, _, _, _ = oracle.update_shard(g.numpy()[cut:], c.numpy()[cut:], m.numpy()[cut:],
                                         v.numpy()[cut:], k, grid[0], grid[1], 9, step, 4, cut)
    assert np.array_equal(W2[cut:].cpu().numpy(), c_ref)


def test_packed_and_device_constant_halves_equal_whole():
    numel, cut = 65_536 * 4 + 12, 131_072  # the cut is a 16-byte boundary of the packed codes
    c, s_w, g, m, v, grid = _state(numel, 1.58, 2, seed=17)
    hp = dqt.adamw(lr=1e-3, step=2)
    sr = dqt.sr_stream(seed=5, tensor_id=2)
    P1 = dqt.dqt_pack_ternary(c.cuda())
    m1, v1 = m.clone().cuda(), v.clone().cuda()
    dqt.dqt_sr_update_packed(g.cuda(), P1, s_w, m1, v1, hp, sr)
    P2 = dqt.dqt_pack_ternary(c.cuda())
    m2, v2, gg = m.clone().cuda(), v.clone().cuda(), g.cuda()
    for lo, hi in [(0, cut), (cut, numel)]:
        dqt.dqt_sr_update_packed(gg[lo:hi], P2[lo // 4: (hi + 3) // 4], s_w, m2[lo:hi], v2[lo:hi],
                                 hp, dqt.sr_stream(seed=5, tensor_id=2, elem0=lo))
    # device-resident constants carry the offset too
    W3, m3, v3 = c.cuda(), m.clone().cuda(), v.clone().cuda()
    for lo, hi in [(0, cut), (cut, numel)]:
        blk = dqt.dqt_update_consts(hp, dqt.sr_stream(seed=5, tensor_id=2, elem0=lo), grid, s_w)
        dev = blk.cuda()
        dqt.dqt_sr_update_dev(gg[lo:hi], W3[lo:hi], m3[lo:hi], v3[lo:hi], dev)
        torch.cuda.synchronize()
    dqt.dqt_check_device_status()
    assert torch.equal(P1, P2) and torch.equal(m1, m2) and torch.equal(v1, v2)
    assert torch.equal(dqt.dqt_unpack_ternary(P1, numel), W3)
    assert torch.equal(m1, m3) and torch.equal(v1, v3)


def test_fused_update_with_offset_equals_standalone():
    """A weight that is a block of a larger flat parameter (elem0 = its first
    element): the fused dW + update and the standalone update of the fused
    kernel's own gradient, both with the offset, give the same codes."""
    T, K, N = 256, 512, 520
    X = inputs.normal((T, K), 1.0, seed=3, dtype=torch.bfloat16)
    dY = inputs.normal((T, N), 1e-2, seed=4, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(8)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=5).numpy(), qmin, qmax)
    s_w = float(s_w)
    hp = dqt.adamw(lr=1e-3, step=1)
    sr = dqt.sr_stream(seed=11, tensor_id=7, elem0=3 * N * K)
    _, _, _, Xdq = dqt.dqt_act_quant_images(X.cuda(), want=("Xdq",))
    W1 = torch.from_numpy(c).cuda()
    m1 = torch.zeros((N, K), device="cuda")
    v1 = torch.zeros((N, K), device="cuda")
    dW = torch.empty((N, K), device="cuda")
    dqt.dqt_bitlinear_bwd_dw_update_img(dY.cuda(), Xdq, W1, s_w, m1, v1, hp, sr, (qmin, qmax),
                                        dW_out=dW, ws=False)
    W2 = torch.from_numpy(c).cuda()
    m2 = torch.zeros((N, K), device="cuda")
    v2 = torch.zeros((N, K), device="cuda")
    dqt.dqt_sr_update(dW.view(-1), W2.view(-1), s_w, m2.view(-1), v2.view(-1), hp, sr,
                      (qmin, qmax))
    dqt.dqt_check_device_status()
    assert torch.equal(W1, W2)
    # the offset changes the stream: without it some codes differ
    W3 = torch.from_numpy(c).cuda()
    dqt.dqt_sr_update(dW.view(-1), W3.view(-1), s_w, torch.zeros(N * K, device="cuda"),
                      torch.zeros(N * K, device="cuda"), hp, dqt.sr_stream(seed=11, tensor_id=7),
                      (qmin, qmax))
    torch.cuda.synchronize()
    assert not torch.equal(W1, W3)


def test_exchange_over_one_rank_nccl_group(tmp_path):
    """The data-parallel exchange on the GPU with NCCL (one rank): the
    reduce-scatter and all-gather are copies, the shard is the whole weight,
    and the result is the library's plain update, bit for bit."""
    import torch.distributed as dist
    from paper_2412_04787_gb300 import dp
    if dist.is_initialized():
        pytest.skip("a process group already exists")
    dist.init_process_group("nccl", init_method="file://" + str(tmp_path / "pg"), rank=0,
                            world_size=1)
    try:
        N, K = 520, 264
        c, s_w, g, m, v, grid = _state(N * K, 8, 1, seed=29)
        upd = dp.DataParallelUpdater(c.view(N, K).cuda())
        hp = dqt.adamw(lr=1e-3, step=1)
        sr = dqt.sr_stream(seed=3, tensor_id=1)
        upd.grad_view().copy_(g.view(N, K).cuda())
        out = upd.step(s_w, hp, sr, grid)
        W = c.cuda()
        dqt.dqt_sr_update(g.cuda(), W, s_w, torch.zeros(N * K, device="cuda"),
                          torch.zeros(N * K, device="cuda"), hp, sr, grid)
        dqt.dqt_check_device_status()
        assert torch.equal(out.reshape(-1), W)
    finally:
        dist.destroy_process_group()
