"""Pins of the packed-ternary and Adafactor oracle functions against facts
fixed outside the oracle: hand-worked packings (tests/golden/), closed forms
of Adafactor's schedules and of its factored second moment (exact for a
rank-one squared gradient, whose first step is then a sign step), its
invariances (gradient scale, row/column marginals, update clipping to RMS d),
and PyTorch's own torch.optim.Adafactor (an independent implementation of
the same optimiser) on the dense target.  No GPU is needed.
"""
import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2412_04787_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


# --------------------------------------------------------------------------
# packed ternary
# --------------------------------------------------------------------------
def test_pack_hand_examples():
    with open(os.path.join(GOLDEN, "packed_ternary_examples.json")) as f:
        cases = json.load(f)["cases"]
    for case in cases:
        c = np.array(case["codes"], np.int8)
        want = [int(b, 16) for b in case["bytes"]]
        assert list(oracle.pack_ternary(c)) == want, case
        assert list(oracle.unpack_ternary(np.array(want, np.uint8), c.size)) == list(c)


@pytest.mark.parametrize("n", [1, 3, 4, 5, 1023, 4096])
def test_pack_roundtrip_and_size(n):
    rng = np.random.default_rng(n)
    c = rng.integers(-1, 2, n).astype(np.int8)
    p = oracle.pack_ternary(c)
    assert p.size == (n + 3) // 4
    assert (oracle.unpack_ternary(p, n) == c).all()
    # bit-level definition, re-derived with integer arithmetic
    for e in rng.integers(0, n, 16):
        f = (int(p[e // 4]) >> (2 * (e % 4))) & 3
        assert {0: 0, 1: 1, 3: -1}[f] == c[e]


def test_packed_size_of_a_1b_model():
    """1e9 ternary weights: 0.25 GB packed (the paper's 0.2 GB is log2(3) bits)."""
    assert (10 ** 9 + 3) // 4 == 250_000_000
    assert abs(10 ** 9 * math.log2(3) / 8 / 1e9 - 0.198) < 1e-3


# --------------------------------------------------------------------------
# Adafactor schedules
# --------------------------------------------------------------------------
def test_adafactor_schedules_closed_form():
    hp = oracle.AdafactorHP(decay_rate=-0.8, relative_step=True)
    b2, omb2, rho = oracle.adafactor_consts(1, hp)
    assert b2 == 0.0 and omb2 == 1.0 and rho == np.float32(1e-2)   # min(1e-2, 1/sqrt(1))
    b2, omb2, rho = oracle.adafactor_consts(2, hp)
    assert b2 == np.float32(1 - 2 ** -0.8) and omb2 == np.float32(2 ** -0.8)
    assert oracle.adafactor_consts(10 ** 4, hp)[2] == np.float32(1e-2)
    assert oracle.adafactor_consts(4 * 10 ** 4, hp)[2] == np.float32(5e-3)   # 1/sqrt(t)
    hpw = oracle.AdafactorHP(relative_step=True, warmup_init=True)
    assert oracle.adafactor_consts(100, hpw)[2] == np.float32(1e-4)          # 1e-6 t
    assert oracle.adafactor_consts(7, oracle.AdafactorHP(lr=3e-4))[2] == np.float32(3e-4)


def _rank1(N, K, seed):
    rng = np.random.default_rng(seed)
    a = rng.uniform(0.5, 2.0, N) * rng.choice([-1, 1], N)
    b = rng.uniform(0.5, 2.0, K) * rng.choice([-1, 1], K)
    return (np.outer(a, b) * 1e-3).astype(np.float32)


def test_rank_one_first_step_is_a_sign_step():
    """t = 1: beta2_1 = 0, so R and C are this gradient's row and column means
    of g^2.  For a rank-one g^2 the factored estimate R C / mean(R) equals g^2
    exactly, every normalised update is sign(g), RMS = 1 (no clipping), and
    x = c - s_w * lr * sign(g)."""
    N, K = 24, 40
    g = _rank1(N, K, 1)
    c = np.random.default_rng(2).integers(-1, 2, (N, K)).astype(np.int8)
    s_w = 60.0
    hp = oracle.AdafactorHP(lr=1e-2, eps1=0.0)
    R, C, st = oracle.adafactor_stats(g, c, s_w, np.zeros(N), np.zeros(K), 1, hp)
    V = np.outer(R.astype(np.float64), C.astype(np.float64)) / st["rbar"]
    g64 = g.astype(np.float64)
    assert np.allclose(V, g64 * g64, rtol=1e-6)
    assert abs(st["rms_u"] - 1.0) < 1e-6
    rho = np.float64(np.float32(1e-2))  # the step size is an fp32 constant
    assert st["alpha"] == rho and st["step"] == np.float32(s_w * rho)
    x = oracle.adafactor_x(g, c, st["a"], st["b"], st["step"], st["decay"])
    assert np.allclose(x, c - 0.6 * np.sign(g), atol=1e-5)
    # round to nearest moves every code one step against its gradient's sign, where the grid allows
    c1, _ = oracle.adafactor_apply(g, c, st["a"], st["b"], st["step"], st["decay"], -1, 1,
                                   0, 1, 0, round_mode=1)
    want = np.clip(np.rint(c - 0.6 * np.sign(g)), -1, 1)
    assert (c1 == want).all()


def test_factored_moment_marginals():
    """At t = 1 the factored estimate keeps the row and column means of g^2 + eps1:
    mean_k V[n,k] = R[n] and mean_n V[n,k] = C[k]."""
    N, K = 33, 70
    g = inputs.normal((N, K), 1e-3, seed=5).numpy()
    c = np.zeros((N, K), np.int8)
    R, C, st = oracle.adafactor_stats(g, c, 10.0, np.zeros(N), np.zeros(K), 1, oracle.AdafactorHP())
    V = np.outer(R.astype(np.float64), C.astype(np.float64)) / st["rbar"]
    assert np.allclose(V.mean(axis=1), R, rtol=1e-6)
    assert np.allclose(V.mean(axis=0), C, rtol=1e-6)
    sq = g.astype(np.float64) ** 2 + 1e-30
    assert np.allclose(R, sq.mean(axis=1), rtol=1e-6) and np.allclose(C, sq.mean(axis=0), rtol=1e-6)


def test_factors_are_the_inverse_square_root_of_the_estimate():
    """a[n] b[k] = 1 / sqrt(R[n] C[k] / Rbar): the rank-one estimate's inverse
    square root splits into a row and a column factor."""
    N, K = 40, 24
    g = inputs.normal((N, K), 1e-3, seed=15).numpy()
    R, C, st = oracle.adafactor_stats(g, np.zeros((N, K), np.int8), 10.0, np.zeros(N), np.zeros(K),
                                      1, oracle.AdafactorHP())
    V = np.outer(R.astype(np.float64), C.astype(np.float64)) / st["rbar"]
    ab = np.outer(st["a"].astype(np.float64), st["b"].astype(np.float64))
    assert np.allclose(ab, 1.0 / np.sqrt(V), rtol=1e-6)
    assert st["rbar"] == np.float32(R.astype(np.float64).mean())


def test_moment_ema_over_steps():
    """R_t = b2_t R_{t-1} + (1 - b2_t) mean_k(g_t^2 + eps1), b2_t = 1 - t^-0.8."""
    N, K = 8, 16
    R = np.zeros(N, np.float32)
    C = np.zeros(K, np.float32)
    c = np.zeros((N, K), np.int8)
    hp = oracle.AdafactorHP()
    Rr = np.zeros(N)
    for t in range(1, 5):
        g = inputs.normal((N, K), 1e-3, seed=10 + t).numpy()
        R, C, _ = oracle.adafactor_stats(g, c, 10.0, R, C, t, hp)
        b2 = 1 - t ** -0.8
        Rr = b2 * Rr + (1 - b2) * (g.astype(np.float64) ** 2 + 1e-30).mean(axis=1)
        assert np.allclose(R, Rr, rtol=1e-5), t


def test_gradient_scale_invariance():
    """Scaling g by a power of two scales R, C, Rbar and V exactly, leaves
    g / sqrt(V) unchanged bit for bit, and so the codes (eps1 = 0)."""
    N, K = 20, 48
    g = inputs.normal((N, K), 1e-3, seed=7).numpy()
    c = np.random.default_rng(3).integers(-1, 2, (N, K)).astype(np.int8)
    hp = oracle.AdafactorHP(lr=5e-3, eps1=0.0)
    outs = []
    for scale in (1.0, 4.0):
        R, C, st = oracle.adafactor_stats(g * np.float32(scale), c, 40.0, np.zeros(N), np.zeros(K), 1, hp)
        x = oracle.adafactor_x(g * np.float32(scale), c, st["a"], st["b"], st["step"], st["decay"])
        cc, _ = oracle.adafactor_apply(g * np.float32(scale), c, st["a"], st["b"], st["step"],
                                       st["decay"], -1, 1, 1234, 1, 3)
        outs.append((x, cc, st["rms_u"]))
    assert (outs[0][0] == outs[1][0]).all() and (outs[0][1] == outs[1][1]).all()
    assert outs[0][2] == pytest.approx(outs[1][2], rel=1e-12)


def test_update_clipping_to_rms_d():
    """A gradient with one huge entry has RMS(g / sqrt(V)) > d; the applied
    update is divided by RMS / d, so its RMS is exactly d."""
    N, K = 16, 32
    g = inputs.normal((N, K), 1e-3, seed=9).numpy()
    g[3, 5] = 1.0
    c = np.zeros((N, K), np.int8)
    for d in (1.0, 0.5):
        hp = oracle.AdafactorHP(lr=1e-2, clip_d=d)
        R, C, st = oracle.adafactor_stats(g, c, 20.0, np.zeros(N), np.zeros(K), 1, hp)
        assert st["rms_u"] > d
        x = oracle.adafactor_x(g, c, st["a"], st["b"], st["step"], st["decay"]).astype(np.float64)
        upd = -x / (20.0 * 1e-2)  # the normalised update actually applied
        assert math.sqrt((upd ** 2).mean()) == pytest.approx(d, rel=1e-5)


def test_parameter_scale_and_weight_decay():
    """alpha = rho * max(eps2, RMS(W)), RMS(W) = sqrt(mean c^2) / s_w for the
    code-domain weight; decay = 1 - wd * alpha multiplies the codes."""
    N, K = 10, 20
    c = np.random.default_rng(4).integers(-1, 2, (N, K)).astype(np.int8)
    g = inputs.normal((N, K), 1e-3, seed=11).numpy()
    s_w = 25.0
    hp = oracle.AdafactorHP(lr=1e-2, scale_parameter=True, weight_decay=0.1)
    _, _, st = oracle.adafactor_stats(g, c, s_w, np.zeros(N), np.zeros(K), 1, hp)
    rms_x = math.sqrt((c.astype(np.float64) ** 2).mean()) / s_w
    assert st["rms_x"] == pytest.approx(rms_x, rel=1e-12)
    assert st["alpha"] == pytest.approx(1e-2 * max(1e-3, rms_x), rel=1e-7)  # rho is fp32
    assert st["decay"] == np.float32(1 - 0.1 * st["alpha"])
    hp0 = oracle.AdafactorHP(lr=1e-2, scale_parameter=True)
    c0 = np.zeros((N, K), np.int8)
    assert oracle.adafactor_stats(g, c0, s_w, np.zeros(N), np.zeros(K), 1, hp0)[2]["alpha"] == \
        pytest.approx(1e-2 * 1e-3)  # RMS 0: eps2 floor


def test_descent_direction():
    """Without weight decay the dense target moves against the gradient."""
    N, K = 12, 24
    g = inputs.normal((N, K), 1e-3, seed=13).numpy()
    c = np.random.default_rng(5).integers(-1, 2, (N, K)).astype(np.int8)
    R, C, st = oracle.adafactor_stats(g, c, 30.0, np.zeros(N), np.zeros(K), 1, oracle.AdafactorHP())
    x = oracle.adafactor_x(g, c, st["a"], st["b"], st["step"], st["decay"])
    d = x - c
    assert (np.sign(d[g != 0]) == -np.sign(g[g != 0])).all()


@pytest.mark.skipif(not hasattr(torch.optim, "Adafactor"), reason="torch without Adafactor")
def test_matches_torch_adafactor_dense_target():
    """torch.optim.Adafactor (relative step min(lr, 1/sqrt(t)), parameter
    scaling, clipping d, beta2_t = 1 - t^-0.8, eps1 as a clamp) on the dense
    weight W = c / s_w: over three steps its parameter change equals the
    oracle's (x - c) / s_w, with eps1 ~ 0 and no weight decay on both sides."""
    N, K = 16, 40
    s_w = 30.0
    c = np.random.default_rng(6).integers(-1, 2, (N, K)).astype(np.int8)
    W = torch.tensor(c.astype(np.float64) / s_w, requires_grad=True)
    opt = torch.optim.Adafactor([W], lr=1e-2, beta2_decay=-0.8, eps=(1e-30, 1e-3), d=1.0,
                                weight_decay=0.0)
    hp = oracle.AdafactorHP(lr=1e-2, eps1=0.0, eps2=1e-3, clip_d=1.0, relative_step=True,
                            scale_parameter=True)
    R = np.zeros(N, np.float32)
    C = np.zeros(K, np.float32)
    cur = c.copy()
    for t in range(1, 4):
        g = inputs.normal((N, K), 1e-3, seed=20 + t).numpy()
        W.grad = torch.tensor(g.astype(np.float64))
        before = W.detach().clone()
        opt.step()
        dW = (W.detach() - before).numpy()
        R, C, st = oracle.adafactor_stats(g, cur, s_w, R, C, t, hp)
        x = oracle.adafactor_x(g, cur, st["a"], st["b"], st["step"], st["decay"])
        ours = (x.astype(np.float64) - cur) / s_w
        # x is fp32 near the integer c: (x - c) / s_w is exact to 2^-24 |x| / s_w
        assert np.allclose(ours, dW, rtol=1e-5, atol=2.0 ** -23 / s_w), t
        # keep both sides on the same weight: torch's W stays dense, the
        # oracle's codes do not move (the comparison is of one step's target)
        with torch.no_grad():
            W.copy_(torch.tensor(cur.astype(np.float64) / s_w))


# --------------------------------------------------------------------------
# The factored evaluation u = (g a[n]) b[k] against Shazeer & Stern's printed
# form u = g / sqrt(R[n] C[k] / Rbar): in fp32 (the same quantity in another
# order of rounded operations) and in fp64, over edge inputs.
# --------------------------------------------------------------------------
# (name, gradient scale, log-spread of row scales, of column scales, steps)
AF_EDGE_CASES = [
    ("typical, step 1", 1e-3, 0.0, 0.0, 1),
    ("rows and columns spread over 2.6 decades", 1e-3, 3.0, 3.0, 1),
    ("spread, step 5", 1e-3, 3.0, 3.0, 5),
    ("eps1 dominates (g^2 << 1e-30)", 1e-16, 0.0, 0.0, 1),
    ("eps1 dominates with spread, step 3", 1e-16, 3.0, 3.0, 3),
    ("large gradients, wide spread", 1.0, 5.0, 5.0, 2),
]


def _af_edge(case, N=64, K=96):
    name, gs, rs, cs, steps = case
    r = np.random.default_rng(len(name) * 1000 + steps)
    g = (r.normal(0, 1, (N, K)) * gs * np.exp(r.uniform(-rs, rs, (N, 1)))
         * np.exp(r.uniform(-cs, cs, (1, K)))).astype(np.float32)
    c = r.integers(-1, 2, (N, K)).astype(np.int8)
    hp = oracle.AdafactorHP(lr=1e-2)
    R, Cc = np.zeros(N, np.float32), np.zeros(K, np.float32)
    for t in range(1, steps + 1):
        R, Cc, st = oracle.adafactor_stats(g, c, np.float32(62.66), R, Cc, t, hp)
    return g, c, R, Cc, st, steps


@pytest.mark.parametrize("case", AF_EDGE_CASES, ids=[c[0] for c in AF_EDGE_CASES])
def test_factored_u_equals_printed_form(case):
    """Relative to the fp64 value of g / sqrt(R C / Rbar) (same fp32 R, C,
    Rbar): the factored form rounds R/Rbar, two square roots, two
    reciprocals and two products -- below 7 * 2^-24 of |u| (a square root
    halves its input's error), bound 8 here; the printed fp32 form rounds the
    product, the quotient, the square root and the division -- below 4 *
    2^-24, bound 5, wherever R[n] C[k] is a normal fp32 number (below that
    the printed form underflows and only the factored one is defined); the
    two fp32 forms then differ by at most 13 * 2^-24 of |u|."""
    g, c, R, Cc, st, _ = _af_edge(case)
    uf = oracle.adafactor_u(g, st["a"], st["b"])
    ut = oracle.adafactor_u_textbook(g, R, Cc, st["rbar"])
    rbar = float(np.float32(st["rbar"]))
    V = R.astype(np.float64)[:, None] * Cc.astype(np.float64)[None, :] / rbar
    u64 = g.astype(np.float64) / np.sqrt(V)
    ulp24 = np.abs(u64) * 2.0 ** -24 + 1e-45
    assert (np.abs(uf - u64) <= 8 * ulp24).all()
    normal = np.abs(R.astype(np.float64)[:, None] * Cc[None, :]) >= np.finfo(np.float32).tiny
    assert (np.abs(ut - u64) <= 5 * ulp24)[normal].all()
    assert (np.abs(uf.astype(np.float64) - ut) <= 13 * ulp24)[normal].all()
    if case[1] >= 1e-3:
        assert normal.all()  # the comparison covers every element there


def test_factored_and_printed_forms_flip_few_stochastic_roundings():
    """Under the same Philox stream, codes from x = c decay - step u with the
    factored u and with the printed-form u (where it is defined) differ in at
    most 1e-4 of the elements, each by exactly one grid step."""
    total = flips = 0
    for case in AF_EDGE_CASES:
        g, c, R, Cc, st, t = _af_edge(case)
        N, K = g.shape
        uf = oracle.adafactor_u(g, st["a"], st["b"])
        ut = oracle.adafactor_u_textbook(g, R, Cc, st["rbar"])
        normal = np.abs(R.astype(np.float64)[:, None] * Cc[None, :]) >= np.finfo(np.float32).tiny
        # x in separately rounded fp32 operations (numpy float32 forms no FMA)
        cd = c.astype(np.float32) * st["decay"]
        xf = cd - st["step"] * uf
        xt = cd - st["step"] * ut
        # the oracle's own apply reproduces xf's rounding exactly
        c_apply, _ = oracle.adafactor_apply(g, c, st["a"], st["b"], st["step"], st["decay"],
                                            -1, 1, 77, t, 9)
        words = np.array([oracle.sr_word(77, t, 9, e) for e in range(N * K)], np.uint32)
        U = ((words >> 8).astype(np.float64) * 2.0 ** -24).astype(np.float32)
        cf = np.clip(oracle.sr_batch(xf.ravel(), U), -1, 1)
        ctb = np.clip(oracle.sr_batch(xt.ravel(), U), -1, 1)
        assert np.array_equal(cf, c_apply.ravel())
        m = normal.ravel()
        diff = cf[m] != ctb[m]
        assert (np.abs(cf[m] - ctb[m])[diff] == 1).all()
        total += int(m.sum())
        flips += int(diff.sum())
    assert total > 0
    assert flips <= int(1e-4 * total), (flips, total)
