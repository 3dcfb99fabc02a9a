"""Pins of the FP8-environment oracle functions (Sec. 4.1 hardware paragraph,
Sec. 4.3: training with 8-bit floating-point operands) against facts fixed
outside the oracle: the E4M3 format's definition worked by hand
(tests/golden/e4m3_examples.json), PyTorch's own float8_e4m3fn conversion (an
independent implementation of the same format and rounding), and numpy's
fp64 matrix product for the forward.  No GPU is needed.
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
E4M3 = getattr(torch, "float8_e4m3fn", None)


def _golden():
    with open(os.path.join(GOLDEN, "e4m3_examples.json")) as f:
        return json.load(f)


def _torch_decode(b):
    return torch.from_numpy(np.asarray(b, np.uint8)).view(E4M3).to(torch.float64).numpy()


def _torch_encode(x):
    return torch.from_numpy(np.asarray(x, np.float32)).to(E4M3).view(torch.uint8).numpy()


def test_e4m3_hand_values():
    g = _golden()
    for d in g["decode"]:
        v = oracle.e4m3_value(int(d["byte"], 16))
        if d["value"] == "nan":
            assert math.isnan(v), d
        else:
            assert v == d["value"], d
    for e in g["encode"]:
        assert oracle.e4m3_from_f32(e["x"]) == int(e["byte"], 16), e
    for w in g["weight_codes"]:
        assert oracle.codes_to_e4m3(np.array([w["code"]], np.int8))[0] == int(w["byte"], 16), w


@pytest.mark.skipif(E4M3 is None, reason="torch without float8_e4m3fn")
def test_e4m3_decode_matches_torch_all_bytes():
    ours = np.array([oracle.e4m3_value(b) for b in range(256)])
    ref = _torch_decode(np.arange(256))
    nan = np.isnan(ref)
    assert (np.isnan(ours) == nan).all() and nan.sum() == 2
    assert (ours[~nan] == ref[~nan]).all()
    # every finite byte round-trips
    for b in range(256):
        if not nan[b]:
            assert oracle.e4m3_from_f32(ours[b]) == b or (b == 0x80 and ours[b] == 0.0)


@pytest.mark.skipif(E4M3 is None, reason="torch without float8_e4m3fn")
def test_e4m3_encode_matches_torch():
    rng = np.random.default_rng(7)
    mags = np.exp2(rng.uniform(-12.0, np.log2(448.0), 20000)).astype(np.float32)
    x = mags * rng.choice([-1.0, 1.0], mags.size).astype(np.float32)
    # every midpoint between adjacent finite magnitudes (the ties) and its
    # two fp32 neighbours
    vals = np.array([oracle.e4m3_value(b) for b in range(0x7F)])
    mids = ((vals[:-1] + vals[1:]) / 2).astype(np.float32)
    near = np.concatenate([mids, np.nextafter(mids, np.float32(0)), np.nextafter(mids, np.float32(1e9))])
    x = np.concatenate([x, near, -near, vals.astype(np.float32)]).astype(np.float32)
    x = x[np.abs(x) <= 448.0]
    ours = np.array([oracle.e4m3_from_f32(v) for v in x], np.uint8)
    ref = _torch_encode(x)
    bad = np.nonzero(ours != ref)[0]
    assert bad.size == 0, [(float(x[i]), hex(ours[i]), hex(ref[i])) for i in bad[:5]]


def test_e4m3_saturates_and_keeps_sign():
    assert oracle.e4m3_from_f32(float("inf")) == 0x7E
    assert oracle.e4m3_from_f32(float("-inf")) == 0xFE
    assert oracle.e4m3_from_f32(449.0) == 0x7E
    assert oracle.e4m3_from_f32(-0.0) == 0x80
    assert oracle.e4m3_from_f32(0.0) == 0x00


def test_weight_codes_exact_up_to_16():
    c = np.arange(-16, 17, dtype=np.int8)
    b = oracle.codes_to_e4m3(c)
    assert [oracle.e4m3_value(int(v)) for v in b] == [float(v) for v in c]
    # 17 needs five significant bits: not representable
    assert oracle.e4m3_value(oracle.e4m3_from_f32(17.0)) != 17.0


def test_act_quant_fp8_hand_examples():
    for case in _golden()["act_quant"]:
        X = inputs.bf16_bits(torch.tensor([case["x"]], dtype=torch.float32).to(torch.bfloat16))
        q8, s8, xdq = oracle.act_quant_fp8(X)
        assert np.float32(s8[0]) == np.float32(case["s8"]), case
        assert [int(h, 16) for h in case["q8"]] == list(q8[0]), case
        assert [int(h, 16) for h in case["xdq_bits"]] == list(xdq[0]), case


@pytest.mark.skipif(E4M3 is None, reason="torch without float8_e4m3fn")
def test_act_quant_fp8_matches_torch_scaled_cast():
    """Per-token amax scaling followed by PyTorch's own fp8 cast (the products
    never exceed 448 by more than rounding, where both saturate or agree)."""
    T, K = 64, 96
    Xb = inputs.normal((T, K), 1.0, seed=11, dtype=torch.bfloat16)
    Xb[3] = 0  # an all-zero token
    Xb[5, 7] = 1e-30
    q8, s8, xdq = oracle.act_quant_fp8(inputs.bf16_bits(Xb))
    X = Xb.float()
    amax = X.abs().amax(dim=1).clamp_min(1e-5)
    s = torch.tensor(448.0) / amax
    assert (s.numpy() == s8).all()
    p = (X * s[:, None]).clamp(-448.0, 448.0)
    ref = p.to(E4M3)
    assert (ref.view(torch.uint8).numpy() == q8).all()
    ref_xdq = (ref.float() / s[:, None]).to(torch.bfloat16)
    assert (inputs.bf16_bits(ref_xdq) == xdq).all()


def test_fwd_fp8_matches_fp64_matmul():
    T, K, N = 48, 160, 40
    Xb = inputs.normal((T, K), 1.0, seed=21, dtype=torch.bfloat16)
    q8, s8, _ = oracle.act_quant_fp8(inputs.bf16_bits(Xb))
    W0 = inputs.normal((N, K), 0.02, seed=22).numpy()
    for qmin, qmax in [(-1, 1), (-16, 15), (-128, 127)]:
        c, s_w, _ = oracle.absmean_init(W0, qmin, qmax)
        Y, acc = oracle.fwd_fp8(q8, s8, c, s_w)
        xv = np.vectorize(oracle.e4m3_value)(q8)  # decoded by the format definition
        ref = xv @ c.astype(np.float64).T
        assert (acc == ref).all()  # every partial sum is exact in fp64
        a_t = np.float32(1.0) / (s8.astype(np.float32) * np.float32(s_w))
        yf = ref.astype(np.float32) * a_t[:, None]
        assert (inputs.bf16_bits(torch.from_numpy(yf).to(torch.bfloat16)) == Y).all()


def test_fwd_fp8_wide_codes_split_exactly():
    """Codes beyond 16 in magnitude reach the E4M3 forward as 16 (c >> 4) and
    c & 15: both are E4M3 values (decoded by the format definition) and they
    add back to c for every int8 code, so the exact sum over value(q8) c is
    the sum over the two halves."""
    c = np.arange(-128, 128, dtype=np.int32)
    h16, l = 16 * (c >> 4), c & 15
    vh = np.vectorize(oracle.e4m3_value)(oracle.codes_to_e4m3(h16.astype(np.int8)))
    vl = np.vectorize(oracle.e4m3_value)(oracle.codes_to_e4m3(l.astype(np.int8)))
    assert (vh == h16).all() and (vl == l).all() and (vh + vl == c).all()
