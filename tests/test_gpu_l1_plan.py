"""Row L1 bounds of the activation codes and the exact forward that plans its
fp32 chunks from them (dqt_act_quant_l1, dqt_bitlinear_fwd_l1).

The bounds are a plain function of the oracle's codes (max over 128-row
blocks of each row's sum of |q| over 1024-column blocks), and the forward's
int32 sums and Y must equal the oracle's exactly.  The exactness cases use
odd products (q = 127, c = -127), so that a chunk whose partial sums passed
2^24 would lose its lowest bit: a plan that merged one column block too many
fails them.
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
    dqt.dqt_set_gemm_tiles(0)
    torch.cuda.synchronize()


def bits(t):
    return t.detach().cpu().contiguous().view(torch.int16).numpy().view(np.uint16)


def l1_bounds(q):
    """max over each 128-row block of sum |q| over each 1024-column block."""
    q = np.abs(q.astype(np.int64))
    T, K = q.shape
    nrb, ncb = -(-T // 128), -(-K // 1024)
    out = np.zeros((nrb, ncb), np.int64)
    for j in range(ncb):
        s = q[:, 1024 * j:1024 * (j + 1)].sum(axis=1)
        for b in range(nrb):
            out[b, j] = s[128 * b:128 * (b + 1)].max()
    return out


# persistent (K <= 2048), rows (K <= 8192) and general (K > 8192) kernels;
# ragged T and K
@pytest.mark.parametrize("T,K", [(1, 8), (37, 264), (300, 2048), (129, 3000), (260, 5632),
                                 (130, 17416)])
def test_act_quant_l1_matches_codes(T, K):
    X = inputs.normal((T, K), 1.0, seed=T * 7 + K, dtype=torch.bfloat16)
    if T > 3:
        X[1] = 0.0
        X[2] = 1.0  # every code 127
        X[3, ::3] = 8.0
    q, s, qi, xd = oracle.act_quant(bits(X))
    Xq, s_x, Xq_img, Xdq, blk = dqt.dqt_act_quant_l1(X.cuda(), want=("Xq", "Xq_img", "Xdq"))
    torch.cuda.synchronize()
    assert dqt.dqt_act_l1_count(T, K) == blk.numel()
    assert np.array_equal(blk.cpu().numpy().astype(np.int64), l1_bounds(q))
    # the codes and images are those of dqt_act_quant
    assert np.array_equal(Xq.cpu().numpy(), q)
    assert np.array_equal(s_x.cpu().numpy().view(np.uint32), s.view(np.uint32))
    assert np.array_equal(bits(Xq_img), qi)
    assert np.array_equal(bits(Xdq), xd)


def test_act_quant_l1_overwrites_stale_bounds():
    X = inputs.normal((256, 2048), 1.0, seed=11, dtype=torch.bfloat16).cuda()
    blk = torch.full((2, 2), 1 << 30, dtype=torch.int32, device="cuda")
    q, _, _, _ = oracle.act_quant(bits(X))
    dqt.dqt_act_quant_l1(X, blk_l1=blk)
    torch.cuda.synchronize()
    assert np.array_equal(blk.cpu().numpy().astype(np.int64), l1_bounds(q))


def _fwd_l1_check(X, c, s_w, grid):
    T, K = X.shape
    Xg = X.cuda()
    _, s_x, Xq_img, _, blk = dqt.dqt_act_quant_l1(Xg, want=("Xq_img",))
    W_img = dqt.dqt_codes_to_bf16(torch.from_numpy(c).cuda())
    acc = torch.empty((T, c.shape[0]), dtype=torch.int32, device="cuda")
    Y = dqt.dqt_bitlinear_fwd_l1(Xq_img, s_x, W_img, s_w, grid, blk, acc_out=acc)
    acc0 = torch.empty_like(acc)
    Y0 = dqt.dqt_bitlinear_fwd(Xq_img, s_x, W_img, s_w, grid, acc_out=acc0)
    dqt.dqt_check_device_status()
    q, s, _, _ = oracle.act_quant(bits(X))
    Yr, accr = oracle.fwd(q, s, c, np.float32(s_w))
    assert np.array_equal(acc.cpu().numpy(), accr)
    assert np.array_equal(bits(Y), Yr)
    assert torch.equal(acc, acc0) and torch.equal(Y, Y0)
    return q


@pytest.mark.parametrize("K", [1088, 2048, 3000, 5632])
def test_fwd_l1_random_8bit(K):
    T, N = 300, 264
    X = inputs.normal((T, K), 1.0, seed=K + 1, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=K + 2)
    qmin, qmax = oracle.grid(8)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    _fwd_l1_check(X, c, float(s_w), (qmin, qmax))


def _rows(kind, n, K, seed):
    if kind == "worst":  # |q| = 127 everywhere: each column block is its own chunk
        return torch.ones((n, K), dtype=torch.bfloat16)
    if kind == "half":  # 472 codes of 127 per 1024 columns: two blocks per chunk
        x = torch.zeros((n, K), dtype=torch.bfloat16)
        cols = torch.arange(K)
        x[:, (cols % 1024) < 472] = 1.0
        return x
    return inputs.normal((n, K), 1.0, seed=seed, dtype=torch.bfloat16)


@pytest.mark.parametrize("K", [2048, 3000, 5632])
def test_fwd_l1_planned_chunks_stay_exact(K):
    """Tiles of 256 rows with different plans: 'half' + random rows (two
    blocks per chunk), 'worst' + 'half' (one block per chunk), random rows
    only (several blocks per chunk), and a ragged last tile.  Codes -127 on
    the first half of the outputs make every product odd and every partial sum
    as large as the plan allows."""
    blocks = ["half", "random", "worst", "half", "random"]
    X = torch.cat([_rows(k, 128, K, seed=31 + i) for i, k in enumerate(blocks)])[:600]
    T, N = X.shape[0], 264
    g = torch.Generator().manual_seed(K)
    c = torch.randint(-128, 128, (N, K), dtype=torch.int32, generator=g)
    c[: N // 2] = -127
    c = c.numpy().astype(np.int8)
    q = _fwd_l1_check(X, c, 50.0, (-128, 127))
    # the worst rows' sums are far past 2^24 and odd-sensitive
    full = q.astype(np.int64) @ c.astype(np.int64).T
    assert np.abs(full).max() > 2 ** 24


def test_fwd_l1_4bit_long_reduction():
    """4-bit codes drain only past K = 16384; the plan then takes one chunk."""
    T, K, N = 200, 17416, 136
    X = inputs.normal((T, K), 1.0, seed=5, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=6)
    qmin, qmax = oracle.grid(4)
    c, s_w, _ = oracle.absmean_init(W0.numpy(), qmin, qmax)
    _fwd_l1_check(X, c, float(s_w), (qmin, qmax))


def test_fwd_l1_one_sm_tiles_ignore_the_plan():
    T, K, N = 160, 3000, 264
    X = torch.cat([_rows("worst", 64, K, 0), _rows("half", 96, K, 0)])
    g = torch.Generator().manual_seed(9)
    c = torch.randint(-128, 128, (N, K), dtype=torch.int8, generator=g).numpy()
    dqt.dqt_set_gemm_tiles(1)
    try:
        _fwd_l1_check(X, c, 40.0, (-128, 127))
    finally:
        dqt.dqt_set_gemm_tiles(0)
