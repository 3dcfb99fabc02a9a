"""Pins of the CPU oracle against what the paper and mathematics fix.

Each test checks the oracle against something other than itself: values the
paper prints, hand-worked examples (tests/golden/), closed forms, exact
enumeration, textbook library routines (numpy matmul, torch.optim.AdamW) and
published Philox known-answer vectors.  No GPU is needed.
"""
import ctypes
import json
import math
import os
import zlib

import numpy as np
import pytest
import torch

import oracle
from paper_2412_04787_gb300 import inputs

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _golden(name):
    with open(os.path.join(GOLDEN, name)) as f:
        return json.load(f)


def _bf16_bits(values):
    return inputs.bf16_bits(torch.tensor(values, dtype=torch.float32).to(torch.bfloat16))


# --------------------------------------------------------------------------
# Philox4x32-10
# --------------------------------------------------------------------------
def test_philox_known_answer_vectors():
    for vec in _golden("philox_kat.json")["vectors"]:
        ctr = [int(h, 16) for h in vec["ctr"]]
        key = [int(h, 16) for h in vec["key"]]
        out = [int(h, 16) for h in vec["out"]]
        assert list(oracle.philox4x32_10(ctr, key)) == out


def test_philox_matches_curand_host_generator_block0():
    """cuRAND's host Philox4_32_10 generator emits Philox(counter 0, key = seed) first."""
    path = "/usr/local/cuda/lib64/libcurand.so"
    if not os.path.exists(path):
        pytest.skip("libcurand not present")
    L = ctypes.CDLL(path)
    for seed in [0, 1234, 0x0123456789ABCDEF, 2**64 - 1]:
        gen = ctypes.c_void_p()
        if L.curandCreateGeneratorHost(ctypes.byref(gen), 161) != 0:
            pytest.skip("cuRAND host generator unavailable")
        assert L.curandSetPseudoRandomGeneratorSeed(gen, ctypes.c_ulonglong(seed)) == 0
        out = np.zeros(4, np.uint32)
        assert L.curandGenerate(gen, out.ctypes.data_as(ctypes.c_void_p), ctypes.c_size_t(4)) == 0
        L.curandDestroyGenerator(gen)
        ref = oracle.philox4x32_10([0, 0, 0, 0], [seed & 0xFFFFFFFF, seed >> 32])
        assert (out == ref).all(), seed


def test_sr_word_counter_mapping():
    """Element e uses counter (e>>2, step, tensor id) and word e&3."""
    seed, step, tid = 0x1122334455667788, 7, 3
    for e in [0, 1, 2, 3, 4, 5, 1023, 2**33 + 6]:
        blk = e >> 2
        words = oracle.philox4x32_10([blk & 0xFFFFFFFF, blk >> 32, step, tid],
                                     [seed & 0xFFFFFFFF, seed >> 32])
        assert oracle.sr_word(seed, step, tid, e) == int(words[e & 3])


def test_uniform_is_24_bit_grid():
    assert oracle.uniform_from_word(0) == 0.0
    assert oracle.uniform_from_word(0xFFFFFFFF) == 1.0 - 2.0**-24
    assert oracle.uniform_from_word(0x80000000) == 0.5
    assert oracle.uniform_from_word(0x000000FF) == 0.0  # low 8 bits dropped


def test_philox_stream_uniformity_chi2():
    n = 1 << 16
    u = np.array([oracle.uniform_from_word(oracle.sr_word(99, 1, 0, e)) for e in range(n)])
    hist, _ = np.histogram(u, bins=64, range=(0.0, 1.0))
    exp = n / 64
    chi2 = float(((hist - exp) ** 2 / exp).sum())
    # 63 degrees of freedom: mean 63, sd ~11.2; 130 is > 6 sd out.
    assert chi2 < 130.0, chi2


# --------------------------------------------------------------------------
# Eq. 3 grid
# --------------------------------------------------------------------------
def test_grid_paper_values():
    facts = _golden("paper_facts.json")
    for key in ("grid_8bit", "grid_ternary"):
        f = facts[key]
        assert oracle.grid(f["bits"]) == (f["qmin"], f["qmax"])


def test_grid_eq3_all_integer_widths():
    for n in range(2, 9):
        assert oracle.grid(n) == (-(2 ** (n - 1)), 2 ** (n - 1) - 1)
    for bad in (1, 9, 2.5):
        with pytest.raises(ValueError):
            oracle.grid(bad)


# --------------------------------------------------------------------------
# Eq. 1 stochastic rounding
# --------------------------------------------------------------------------
ALL_U = (np.arange(1 << 24, dtype=np.float64) * 2.0**-24).astype(np.float32)


def _p_up_exact(x):
    """P(SR(x) = floor(x)+1) by enumerating every value of the 24-bit uniform."""
    xs = np.full(ALL_U.shape, x, np.float32)
    out = oracle.sr_batch(xs, ALL_U)
    f = math.floor(float(np.float32(x)))
    assert set(np.unique(out)) <= {f, f + 1}
    return float((out == f + 1).mean())


def test_sr_paper_example():
    """Sec. 5: -1 + 0.02 goes to 0 with probability 2%, else to -1."""
    f = _golden("paper_facts.json")["sr_example"]
    xs = np.full(ALL_U.shape, f["x"], np.float32)
    out = oracle.sr_batch(xs, ALL_U)
    assert set(np.unique(out)) == {f["down_to"], f["p_up_to"]}
    assert abs((out == f["p_up_to"]).mean() - f["p_up"]) < 1e-6


@pytest.mark.parametrize("x", [0.25, -0.25, 2.75, -3.125, 0.5, 126.9, -127.3, 1e-3, -1e-3])
def test_sr_probabilities_eq1(x):
    """Eq. 1: P(floor) = ceil(x) - x, so P(ceil) = x - floor(x) (to the 2^-24 grid)."""
    xf = float(np.float32(x))
    r = xf - math.floor(xf)
    assert abs(_p_up_exact(x) - r) <= 2.0**-24


@pytest.mark.parametrize("x", [-3.0, 0.0, 5.0, -128.0, 127.0])
def test_sr_integer_fixed_point(x):
    xs = np.full(4096, x, np.float32)
    u = np.linspace(0, 1 - 2**-24, 4096, dtype=np.float32)
    assert (oracle.sr_batch(xs, u) == int(x)).all()


def test_sr_unbiased_and_variance_monte_carlo():
    """E[SR(x)] = x and Var = r(1-r) (Sec. 5: zero-mean noise, bounded variance)."""
    xs = np.array([0.3, -1.7, 2.02, -0.98], np.float32)
    n = 200_000
    e = np.arange(n, dtype=np.int64)
    words = np.array([oracle.sr_word(4242, 1, 0, int(i)) for i in e], np.uint64)
    u = ((words >> 8).astype(np.float64) * 2.0**-24).astype(np.float32)
    for x in xs:
        out = oracle.sr_batch(np.full(n, x, np.float32), u).astype(np.float64)
        r = float(x) - math.floor(float(x))
        sigma = math.sqrt(r * (1 - r) / n)
        assert abs(out.mean() - float(x)) < 5 * sigma + 1e-6
        assert abs(out.var() - r * (1 - r)) < 0.01


def test_sr_brute_force_small_tensor_expectation():
    """Exact enumeration for a 3-element tensor: every rounding outcome, with its
    probability as the product of per-element probabilities, sums to 1 and has
    expectation x elementwise (values chosen on the 2^-8 grid, exact in fp32)."""
    x = np.array([0.25, -1.75, 3.5], np.float32)
    p_up = [_p_up_exact(v) for v in x]
    floors = np.floor(x.astype(np.float64))
    total = 0.0
    mean = np.zeros(3)
    for mask in range(8):
        bits = np.array([(mask >> i) & 1 for i in range(3)])
        p = np.prod([p_up[i] if bits[i] else 1 - p_up[i] for i in range(3)])
        total += p
        mean += p * (floors + bits)
    assert abs(total - 1.0) < 1e-12
    assert np.allclose(mean, x.astype(np.float64), atol=1e-12)


# --------------------------------------------------------------------------
# Eq. 2-4 AbsMean initialisation
# --------------------------------------------------------------------------
def test_absmean_hand_examples():
    for case in _golden("absmean_examples.json")["cases"]:
        qmin, qmax = oracle.grid(case["bits"])
        codes, s, am = oracle.absmean_init(np.array(case["W"], np.float32), qmin, qmax)
        assert abs(am - case["absmean"]) < 1e-7, case
        assert abs(float(s) - case["s"]) < 1e-5 * case["s"], case
        assert codes.tolist() == case["codes"], case
        # Eq. 4 on its own, at the worked scale, gives the worked codes
        q = oracle.quantize_weights(np.array(case["W"], np.float32), s, qmin, qmax)
        assert q.tolist() == case["codes"], case


def test_quantize_weights_is_round_half_even_then_clip():
    """Eq. 4 at a given fp32 scale against numpy's rint (half-to-even) and clip
    of the fp32 product, over random weights and a scale whose products land
    on exact .5 ties."""
    W = np.concatenate([inputs.normal((4096,), 0.02, seed=12).numpy(),
                        np.arange(-20, 21, dtype=np.float32) * 0.25]).astype(np.float32)
    for s, (qmin, qmax) in [(np.float32(62.66), (-1, 1)), (np.float32(6.0), (-128, 127)),
                            (np.float32(2.0), (-8, 7))]:
        want = np.clip(np.rint(W * s), qmin, qmax).astype(np.int8)
        assert np.array_equal(oracle.quantize_weights(W, s, qmin, qmax), want)


def test_absmean_statistics_gaussian():
    """For N(0, sigma) weights AbsMean -> sigma sqrt(2/pi); ternary codes are
    {-1,0,1} with P(0) = P(|z| < sqrt(2/pi)/2): w s rounds to 0 when
    |w| < AbsMean/2 = sigma sqrt(2/pi)/2."""
    W0 = inputs.normal((512, 512), 0.02, seed=3).numpy()
    codes, s, am = oracle.absmean_init(W0, -1, 1)
    assert abs(am - 0.02 * math.sqrt(2 / math.pi)) < 2e-4
    assert set(np.unique(codes)) == {-1, 0, 1}
    p0 = math.erf(math.sqrt(2 / math.pi) / 2 / math.sqrt(2))
    assert abs((codes == 0).mean() - p0) < 0.01


# --------------------------------------------------------------------------
# Sec. 3.2 activation quantisation
# --------------------------------------------------------------------------
def test_act_quant_hand_examples():
    for case in _golden("act_quant_examples.json")["cases"]:
        X = _bf16_bits([case["x"]])
        q, s, qi, xd = oracle.act_quant(X)
        assert abs(float(s[0]) - case["s_x"]) <= 1e-6 * case["s_x"], case
        assert q[0].tolist() == case["q"], case
        # the code image is the code itself in bf16
        img = torch.from_numpy(qi.view(np.int16).copy()).view(torch.bfloat16).float()
        assert img[0].tolist() == [float(v) for v in case["q"]]


def test_act_quant_properties_random():
    X = inputs.normal((37, 200), 1.0, seed=11, dtype=torch.bfloat16)
    q, s, qi, xd = oracle.act_quant(inputs.bf16_bits(X))
    xf = X.float().numpy().astype(np.float64)
    amax = np.abs(xf).max(axis=1)
    assert np.allclose(s, 127.0 / amax, rtol=1e-6)
    assert (np.abs(q).max(axis=1) == 127).all()  # the row max maps to +-127
    # |x s - q| <= 1/2 (nearest) and the dequantised image is q/s in bf16
    assert (np.abs(xf * s[:, None].astype(np.float64) - q) <= 0.5 + 1e-4).all()
    deq = torch.from_numpy(xd.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    ref = q / s[:, None].astype(np.float64)
    assert np.allclose(deq, ref, rtol=2.0**-8, atol=0)


# --------------------------------------------------------------------------
# Sec. 3.2 forward and backward: reduce to textbook matmul
# --------------------------------------------------------------------------
def _small_problem(T=19, K=40, N=24, bits=1.58, seed=5):
    X = inputs.normal((T, K), 1.0, seed=seed, dtype=torch.bfloat16)
    W0 = inputs.normal((N, K), 0.02, seed=seed + 1).numpy()
    dY = inputs.normal((T, N), 1e-2, seed=seed + 2, dtype=torch.bfloat16)
    qmin, qmax = oracle.grid(bits)
    c, s_w, _ = oracle.absmean_init(W0, qmin, qmax)
    q, s_x, _, _ = oracle.act_quant(inputs.bf16_bits(X))
    return X, dY, c, s_w, q, s_x


@pytest.mark.parametrize("bits", [1.58, 8])
def test_fwd_is_integer_matmul(bits):
    X, dY, c, s_w, q, s_x = _small_problem(bits=bits)
    Y, acc = oracle.fwd(q, s_x, c, s_w)
    ref = q.astype(np.int64) @ c.astype(np.int64).T
    assert (acc == ref).all()
    yref = ref / (s_x.astype(np.float64)[:, None] * np.float64(s_w))
    y = torch.from_numpy(Y.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    assert np.allclose(y, yref, rtol=2.0**-8, atol=1e-30)


def test_fwd_rejects_int32_overflow():
    q = np.full((1, 140000), 127, np.int8)
    c = np.full((1, 140000), 127, np.int8)
    with pytest.raises(OverflowError):
        oracle.fwd(q, np.ones(1, np.float32), c, 1.0)


def test_bwd_dx_dw_are_textbook_matmul():
    X, dY, c, s_w, q, s_x = _small_problem(T=23, K=48, N=32, bits=4)
    dYf = dY.double().numpy()
    Wt = c.astype(np.float64) / np.float64(s_w)
    dX = oracle.bwd_dx(inputs.bf16_bits(dY), c, s_w)
    assert np.allclose(dX, dYf @ Wt, rtol=1e-12, atol=1e-15)
    Xt = q.astype(np.float64) / s_x.astype(np.float64)[:, None]
    dW = oracle.bwd_dw(inputs.bf16_bits(dY), q, s_x)
    assert dW.shape == (32, 48)
    assert np.allclose(dW, dYf.T @ Xt, rtol=1e-12, atol=1e-15)
    rows = np.array([31, 0, 7])
    assert np.array_equal(oracle.bwd_dw(inputs.bf16_bits(dY), q, s_x, rows=rows), dW[rows])
    # BF16 environment: X_tilde held as bf16(q / s_x)
    _, _, _, xd = oracle.act_quant(inputs.bf16_bits(X))
    Xb = torch.from_numpy(xd.view(np.int16).copy()).view(torch.bfloat16).double().numpy()
    dWb = oracle.bwd_dw_bf16x(inputs.bf16_bits(dY), xd)
    assert np.allclose(dWb, dYf.T @ Xb, rtol=1e-12, atol=1e-15)
    assert np.abs(dWb - dW).max() <= 2.0**-8 * np.abs(dW).max()


# --------------------------------------------------------------------------
# Sec. 4.1 AdamW, against torch.optim.AdamW in fp64
# --------------------------------------------------------------------------
@pytest.mark.parametrize("wd", [0.0, 0.1])
def test_adamw_matches_torch_adamw(wd):
    # the oracle takes its hyper-parameters as fp32 values: give torch the same
    f32 = lambda a: float(np.float32(a))  # noqa: E731
    lr, b1, b2, eps, wd = f32(1e-3), f32(0.9), f32(0.999), f32(1e-8), f32(wd)
    n = 4096
    c = np.random.default_rng(0).integers(-128, 128, n).astype(np.int8)
    s_w = np.float32(40.0)
    p = torch.tensor(c.astype(np.float64) / float(s_w), requires_grad=True)
    opt = torch.optim.AdamW([p], lr=lr, betas=(b1, b2), eps=eps, weight_decay=wd)
    m = np.zeros(n, np.float32)
    v = np.zeros(n, np.float32)
    cur = c.copy()
    for step in range(1, 4):
        g = inputs.normal((n,), 1e-3, seed=100 + step).numpy()
        p.grad = torch.tensor(g.astype(np.float64))
        opt.step()
        k = oracle.adamw_consts(lr, b1, b2, eps, wd, step, s_w)
        x, m, v = oracle.adamw_x(g, cur, m, v, k)
        st = opt.state[p]
        # fp32 vs fp64: a few fp32 roundings, scaled by the moment's magnitude
        # (b1 m and (1-b1) g may cancel, so the bound is absolute, not relative)
        em, ev = st["exp_avg"].numpy(), st["exp_avg_sq"].numpy()
        assert np.abs(m - em).max() <= 1e-6 * np.abs(em).max()
        assert np.abs(v - ev).max() <= 1e-6 * np.abs(ev).max()
        assert np.allclose(x, p.detach().numpy() * float(s_w), rtol=0, atol=2e-5 * 128)
        # next step starts from the torch weights, which are on the grid here
        cur = np.round(p.detach().numpy() * float(s_w)).astype(np.int8)
        with torch.no_grad():
            p.copy_(torch.tensor(cur.astype(np.float64) / float(s_w)))


def test_adamw_step1_closed_form():
    """At step 1 with zero moments: m = (1-b1) g, v = (1-b2) g^2, and the update
    direction is g / (|g| + eps), so x = c - lr s_w g/(|g|+eps) (no decay)."""
    g = inputs.normal((1000,), 1e-2, seed=8).numpy()
    c = np.zeros(1000, np.int8)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, 50.0)
    x, m, v = oracle.adamw_x(g, c, np.zeros(1000, np.float32), np.zeros(1000, np.float32), k)
    g64 = g.astype(np.float64)
    assert np.allclose(m, 0.1 * g64, rtol=1e-6)
    assert np.allclose(v, 0.001 * g64 * g64, rtol=1e-6)
    assert np.allclose(x, -0.05 * g64 / (np.abs(g64) + 1e-8), rtol=1e-5)


# --------------------------------------------------------------------------
# Sec. 4.1 AdamW: the one-division form used by the update (m' / (sqrt(v') k1
# + k2)) against the textbook order (m_hat = m'/bc1, v_hat = v'/bc2,
# m_hat / (sqrt(v_hat) + eps)), each in separately rounded fp32 operations,
# and both against the same formula in fp64, over edge inputs.
# --------------------------------------------------------------------------
_F32 = lambda a: float(np.float32(a))  # noqa: E731
# (name, scale of g, scale of m, scale of sqrt(v), step, weight decay, lr)
ADAMW_EDGE_CASES = [
    ("zero gradient and moments", 0.0, 0.0, 0.0, 1, 0.0, 1e-3),
    ("step 1 from zero moments", 1e-3, 0.0, 0.0, 1, 0.0, 1e-3),
    ("v = 0, m != 0", 0.0, 1e-4, 0.0, 3, 0.0, 1e-3),
    ("v << eps^2 (eps dominates)", 1e-12, 1e-12, 1e-13, 5, 0.0, 1e-3),
    ("sqrt(v_hat) ~ eps", 1e-8, 1e-8, 1e-8, 5, 0.0, 1e-3),
    ("typical, weight decay", 1e-3, 1e-4, 1e-4, 7, 0.01, 1e-3),
    ("step 100", 1e-3, 1e-4, 1e-4, 100, 0.0, 1e-3),
    ("step 10^4, wd 0.1, lr 1e-2", 1e-3, 1e-4, 1e-4, 10_000, 0.1, 1e-2),
    ("large gradients", 1.0, 1.0, 1.0, 2, 0.0, 1e-3),
    ("subnormal moments", 1e-20, 1e-20, 1e-20, 2, 0.0, 1e-3),
]


def _adamw_edge(case, bits, n=20000):
    name, gs, ms, vs, step, wd, lr = case
    r = np.random.default_rng(zlib.crc32(f"{name}/{bits}".encode()))
    qmin, qmax = oracle.grid(bits)
    c = r.integers(qmin, qmax + 1, n).astype(np.int8)
    # s_w of AbsMean-quantised N(0, 0.02) weights: qmax / (0.02 sqrt(2/pi))
    s_w = np.float32(qmax / (0.02 * math.sqrt(2.0 / math.pi)))
    g = (r.normal(0, 1, n) * gs).astype(np.float32)
    m = (r.normal(0, 1, n) * ms).astype(np.float32)
    v = np.square(r.normal(0, 1, n) * vs).astype(np.float32)
    k = oracle.adamw_consts(lr, 0.9, 0.999, 1e-8, wd, step, s_w)
    kt = oracle.adamw_textbook_consts(lr, 0.9, 0.999, 1e-8, wd, step, s_w)
    return c, s_w, g, m, v, k, kt, (qmin, qmax), (step, wd, lr)


def _ulp(x):
    return np.spacing(np.abs(np.asarray(x, np.float32))).astype(np.float64)


@pytest.mark.parametrize("bits", [1.58, 8])
@pytest.mark.parametrize("case", ADAMW_EDGE_CASES, ids=[c[0] for c in ADAMW_EDGE_CASES])
def test_adamw_one_division_form_equals_textbook_order(case, bits):
    """The two orders share m' and v' bit for bit.  Their u differ only by
    rounding: the textbook order rounds m_hat, v_hat, sqrt, the sum and the
    quotient; the one-division form rounds sqrt, the product with k1, the sum
    and the quotient, plus k1 and k2 themselves -- at most 6 roundings each, a
    relative difference below 12 * 2^-24 of u (a square root halves its
    input's error).  Through x = c decay - lrs u that is at most
    (12 + 2 + 2) * 2^-24 of the step |lrs u| (the product and its ulp on
    either side) plus one ulp of x on either side.  The bound below, 20 ulps
    of 2^-24 |step| plus 3 ulps of x, holds with margin for every element."""
    c, s_w, g, m, v, k, kt, _, _ = _adamw_edge(case, bits)
    xr, mr, vr = oracle.adamw_x(g, c, m, v, k)
    xt, mt, vt = oracle.adamw_x_textbook(g, c, m, v, kt)
    assert np.array_equal(mr.view(np.uint32), mt.view(np.uint32))
    assert np.array_equal(vr.view(np.uint32), vt.view(np.uint32))
    A = (c.astype(np.float32) * kt[7]).astype(np.float64)  # c decay, rounded alike
    step_mag = np.abs(A - xt.astype(np.float64))
    d = np.abs(xr.astype(np.float64) - xt.astype(np.float64))
    bound = 20 * 2.0 ** -24 * step_mag + 3 * _ulp(xt) + 1e-37
    assert (d <= bound).all(), float((d / bound).max())
    # most elements agree bit for bit
    assert np.mean(d == 0) >= 0.5


@pytest.mark.parametrize("bits", [1.58, 8])
@pytest.mark.parametrize("case", ADAMW_EDGE_CASES, ids=[c[0] for c in ADAMW_EDGE_CASES])
def test_adamw_both_orders_match_fp64(case, bits):
    """Both fp32 orders against AdamW's dense target evaluated in fp64 from the
    same hyper-parameters (as fp32 values) and the same new moments: within
    8 * 2^-24 of the step, 2^-24 |c| (the rounding of c decay and of its
    constant) and one ulp of x."""
    c, s_w, g, m, v, k, kt, _, (step, wd, lr) = _adamw_edge(case, bits)
    xr, _, _ = oracle.adamw_x(g, c, m, v, k)
    xt, mt, vt = oracle.adamw_x_textbook(g, c, m, v, kt)
    b1, b2, eps, lr, wd = _F32(0.9), _F32(0.999), _F32(1e-8), _F32(lr), _F32(wd)
    bc1 = 1.0 - b1 ** step
    bc2 = 1.0 - b2 ** step
    u = (mt.astype(np.float64) / bc1) / (np.sqrt(vt.astype(np.float64) / bc2) + eps)
    x64 = c.astype(np.float64) * (1.0 - lr * wd) - lr * float(s_w) * u
    bound = (8 * 2.0 ** -24 * np.abs(lr * float(s_w) * u)
             + 2.0 ** -24 * np.abs(c.astype(np.float64)) + _ulp(xt) + 1e-37)
    assert (np.abs(xr - x64) <= bound).all()
    assert (np.abs(xt - x64) <= bound).all()


def test_adamw_orders_flip_few_stochastic_roundings():
    """Under the same Philox stream, the update with the one-division AdamW and
    the update with the textbook order round to the same codes except where a
    uniform falls between their two dense targets: over all edge cases at
    most 1e-4 of the codes differ, each by exactly one grid step."""
    total = flips = 0
    for case in ADAMW_EDGE_CASES:
        for bits in (1.58, 8):
            c, s_w, g, m, v, k, kt, (qmin, qmax), (step, _, _) = _adamw_edge(case, bits)
            cr, mr, vr, _ = oracle.update(g, c, m, v, k, qmin, qmax, 1234, step, 3)
            ct, mt, vt, _ = oracle.update(g, c, m, v, kt, qmin, qmax, 1234, step, 3,
                                          textbook=True)
            assert np.array_equal(mr, mt) and np.array_equal(vr, vt)
            diff = cr != ct
            assert (np.abs(cr.astype(np.int32) - ct.astype(np.int32))[diff] == 1).all()
            total += diff.size
            flips += int(diff.sum())
    assert flips <= int(1e-4 * total), (flips, total)


# --------------------------------------------------------------------------
# Eq. 5 update
# --------------------------------------------------------------------------
def _update_case(N=16, K=64, bits=1.58, seed=21, step=1):
    qmin, qmax = oracle.grid(bits)
    W0 = inputs.normal((N, K), 0.02, seed=seed).numpy()
    c, s_w, _ = oracle.absmean_init(W0, qmin, qmax)
    g = inputs.normal((N, K), 1e-3, seed=seed + 1).numpy()
    m = np.zeros((N, K), np.float32)
    v = np.zeros((N, K), np.float32)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, step, s_w)
    return c, s_w, g, m, v, k, qmin, qmax


def test_update_is_sr_of_adamw_target():
    c, s_w, g, m, v, k, qmin, qmax = _update_case(bits=8)
    c1, m1, v1, changed = oracle.update(g, c, m, v, k, qmin, qmax, 77, 1, 5)
    x, mx, vx = oracle.adamw_x(g, c, m, v, k)
    assert np.array_equal(m1.ravel(), mx) and np.array_equal(v1.ravel(), vx)
    f = np.floor(x.astype(np.float64))
    out = c1.ravel().astype(np.int64)
    clamped = np.clip(f, qmin, qmax)
    clamped_up = np.clip(f + 1, qmin, qmax)
    assert ((out == clamped) | (out == clamped_up)).all()
    assert changed == int((c1 != c).sum())


def test_update_round_to_nearest_ablation():
    c, s_w, g, m, v, k, qmin, qmax = _update_case(bits=8)
    c1, _, _, _ = oracle.update(g, c, m, v, k, qmin, qmax, 77, 1, 5, round_mode=1)
    x, _, _ = oracle.adamw_x(g, c, m, v, k)
    assert np.array_equal(c1.ravel(), np.clip(np.rint(x), qmin, qmax).astype(np.int8))


def test_update_clamps_to_grid():
    c = np.array([[1, -1, 1, -1]], np.int8)
    g = np.array([[-1.0, 1.0, -1.0, 1.0]], np.float32)  # pushes outward
    k = oracle.adamw_consts(1.0, 0.9, 0.999, 1e-8, 0.0, 1, 10.0)  # lr s_w = 10
    c1, _, _, _ = oracle.update(g, c, np.zeros_like(g), np.zeros_like(g), k, -1, 1, 1, 1, 0)
    assert c1.tolist() == [[1, -1, 1, -1]]


def test_update_rows_map_to_global_indices_and_shards_agree():
    """The uniform of element (n,k) depends only on its global flat index, so
    updating row blocks (shards) gives the same codes as the whole tensor."""
    c, s_w, g, m, v, k, qmin, qmax = _update_case(N=12, K=32, bits=4)
    full, mf, vf, _ = oracle.update(g, c, m, v, k, qmin, qmax, 9, 3, 2)
    parts = []
    for lo, hi in [(0, 5), (5, 12)]:
        rows = np.arange(lo, hi)
        p, _, _, _ = oracle.update(g[lo:hi], c[lo:hi], m[lo:hi], v[lo:hi], k, qmin, qmax,
                                   9, 3, 2, rows=rows)
        parts.append(p)
    assert np.array_equal(np.concatenate(parts), full)


def test_update_expected_code_monte_carlo():
    """Averaged over seeds, the new code equals the clamped dense target x."""
    c, s_w, g, m, v, k, qmin, qmax = _update_case(N=2, K=8, bits=8)
    x, _, _ = oracle.adamw_x(g, c, m, v, k)
    acc = np.zeros(16)
    S = 4000
    for seed in range(S):
        c1, _, _, _ = oracle.update(g, c, m, v, k, qmin, qmax, seed, 1, 0)
        acc += c1.ravel()
    # outside [Q_n, Q_p] both rounding outcomes clamp to the same end, so the
    # expectation is exactly clip(x, Q_n, Q_p)
    r = np.where((x > qmin) & (x < qmax), x - np.floor(x), 0.0)
    sigma = np.sqrt(r * (1 - r) / S) + 1e-9
    assert (np.abs(acc / S - np.clip(x, qmin, qmax)) < 5 * sigma + 1e-6).all()
    assert ((x > qmin) & (x < qmax)).sum() >= 4  # some elements are interior


def test_update_step1_change_rate_ternary():
    """Ternary, step 1, no decay: x = c - lr s_w g/(|g|+eps), so a code moves
    with probability lr s_w unless the move would leave [-1, 1]."""
    W0 = inputs.normal((256, 256), 0.02, seed=3).numpy()
    c, s_w, _ = oracle.absmean_init(W0, -1, 1)
    g = inputs.normal((256, 256), 1e-2, seed=4).numpy()
    z = np.zeros_like(g)
    k = oracle.adamw_consts(1e-3, 0.9, 0.999, 1e-8, 0.0, 1, s_w)
    c1, _, _, changed = oracle.update(g, c, z, z, k, -1, 1, 1234, 1, 0)
    movable = ~(((c == 1) & (g < 0)) | ((c == -1) & (g > 0)))
    p = 1e-3 * float(s_w)
    expect = movable.sum() * p
    assert abs(changed - expect) < 5 * math.sqrt(expect) + 1
