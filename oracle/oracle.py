"""ctypes front end of the C oracle (test infrastructure only).

Every function mirrors one step of the DQT BitLinear training step as the
paper states it (Zhao et al., "Direct Quantized Training of Language Models
with Stochastic Rounding"):

* ``sr``/``sr_batch``          -- Eq. 1, stochastic rounding
* ``grid``                     -- Eq. 3, the n-bit grid [Q_n, Q_p]
* ``absmean_init``             -- Eq. 2-4, AbsMean scale and initial codes
* ``quantize_weights``         -- Eq. 4 alone, for a given scale
* ``act_quant``                -- Sec. 3.2, 8-bit per-token absmax activations
* ``fwd``                      -- Sec. 3.2, BitLinear forward (exact int accumulation)
* ``bwd_dx`` / ``bwd_dw``      -- Sec. 3.2, backward w.r.t. input and low-bit weight (fp64)
* ``bwd_dw_bf16x``             -- Sec. 4.1/4.3, the weight gradient with X_tilde in bf16
* ``adamw_consts``/``adamw_x`` -- Sec. 4.1, AdamW producing the dense target W'
  (``adamw_textbook_consts``/``adamw_x_textbook``: the textbook evaluation order)
* ``update``                   -- Eq. 5, W_hat = SR(W') clamped onto the grid
* ``update_shard``             -- Eq. 5 on a flat shard at a global element offset
* ``pack_ternary``/``unpack_ternary`` -- Sec. 1, 2-bit packed ternary storage
* ``adafactor_consts``/``adafactor_stats``/``adafactor_x``/``adafactor_apply``
                               -- Sec. 4.3, Adafactor (factored second moment) + SR
* ``e4m3_value``/``e4m3_from_f32``/``act_quant_fp8``/``fwd_fp8``
                               -- Sec. 4.1/4.3 FP8 environment: E4M3 activations
                                  and the forward on E4M3 operands

bf16 tensors are passed as ``numpy.uint16`` arrays holding the raw bits.
"""
import ctypes as C
import numpy as np

from .build_oracle import build

_lib = None

_f32p = C.POINTER(C.c_float)
_f64p = C.POINTER(C.c_double)
_i8p = C.POINTER(C.c_int8)
_i32p = C.POINTER(C.c_int32)
_i64p = C.POINTER(C.c_int64)
_u16p = C.POINTER(C.c_uint16)
_u32p = C.POINTER(C.c_uint32)
_u8p = C.POINTER(C.c_uint8)


def lib():
    global _lib
    if _lib is None:
        L = C.CDLL(build())
        L.dqt_oracle_f32_to_bf16.argtypes = [C.c_float]
        L.dqt_oracle_f32_to_bf16.restype = C.c_uint16
        L.dqt_oracle_philox4x32_10.argtypes = [_u32p, _u32p, _u32p]
        L.dqt_oracle_philox4x32_10.restype = None
        L.dqt_oracle_sr_word.argtypes = [C.c_uint64, C.c_int64, C.c_uint32, C.c_int64]
        L.dqt_oracle_sr_word.restype = C.c_uint32
        L.dqt_oracle_uniform_from_word.argtypes = [C.c_uint32]
        L.dqt_oracle_uniform_from_word.restype = C.c_float
        L.dqt_oracle_sr.argtypes = [C.c_float, C.c_float]
        L.dqt_oracle_sr.restype = C.c_int32
        L.dqt_oracle_sr_batch.argtypes = [_f32p, _f32p, _i32p, C.c_int64]
        L.dqt_oracle_sr_batch.restype = None
        L.dqt_oracle_grid.argtypes = [C.c_int32, _i32p, _i32p]
        L.dqt_oracle_grid.restype = C.c_int
        L.dqt_oracle_absmean_init.argtypes = [_f32p, C.c_int64, C.c_int32, C.c_int32,
                                              _i8p, _f32p, _f64p]
        L.dqt_oracle_absmean_init.restype = C.c_int
        L.dqt_oracle_act_quant.argtypes = [_u16p, C.c_int64, C.c_int64, _i8p, _f32p,
                                           _u16p, _u16p]
        L.dqt_oracle_act_quant.restype = None
        L.dqt_oracle_fwd.argtypes = [_i8p, _f32p, _i8p, C.c_float, C.c_int64, C.c_int64,
                                     C.c_int64, _u16p, _i32p]
        L.dqt_oracle_fwd.restype = C.c_int
        L.dqt_oracle_bwd_dx.argtypes = [_u16p, _i8p, C.c_float, C.c_int64, C.c_int64,
                                        C.c_int64, _f64p]
        L.dqt_oracle_bwd_dx.restype = None
        L.dqt_oracle_bwd_dw.argtypes = [_u16p, _i8p, _f32p, C.c_int64, C.c_int64,
                                        C.c_int64, _i64p, C.c_int64, _f64p]
        L.dqt_oracle_bwd_dw.restype = None
        L.dqt_oracle_bwd_dw_bf16x.argtypes = [_u16p, _u16p, C.c_int64, C.c_int64, C.c_int64,
                                              _i64p, C.c_int64, _f64p]
        L.dqt_oracle_bwd_dw_bf16x.restype = None
        L.dqt_oracle_adamw_consts.argtypes = [C.c_float, C.c_float, C.c_float, C.c_float,
                                              C.c_float, C.c_int64, C.c_float, _f32p]
        L.dqt_oracle_adamw_consts.restype = None
        L.dqt_oracle_adamw_x.argtypes = [_f32p, _i8p, _f32p, _f32p, _f32p, C.c_int64, _f32p]
        L.dqt_oracle_adamw_x.restype = None
        L.dqt_oracle_update.argtypes = [_f32p, _i8p, _f32p, _f32p, _f32p, C.c_int32,
                                        C.c_int32, C.c_uint64, C.c_int64, C.c_uint32,
                                        C.c_int32, _i64p, C.c_int64, C.c_int64]
        L.dqt_oracle_update.restype = C.c_int64
        L.dqt_oracle_adamw_textbook_consts.argtypes = [C.c_float, C.c_float, C.c_float,
                                                       C.c_float, C.c_float, C.c_int64,
                                                       C.c_float, _f32p]
        L.dqt_oracle_adamw_textbook_consts.restype = None
        L.dqt_oracle_adamw_x_textbook.argtypes = [_f32p, _i8p, _f32p, _f32p, _f32p, C.c_int64,
                                                  _f32p]
        L.dqt_oracle_adamw_x_textbook.restype = None
        L.dqt_oracle_update_shard.argtypes = [_f32p, _i8p, _f32p, _f32p, _f32p, C.c_int32,
                                              C.c_int32, C.c_uint64, C.c_int64, C.c_uint32,
                                              C.c_int32, C.c_int64, C.c_int64]
        L.dqt_oracle_update_shard.restype = C.c_int64
        L.dqt_oracle_update_textbook.argtypes = L.dqt_oracle_update.argtypes
        L.dqt_oracle_update_textbook.restype = C.c_int64
        L.dqt_oracle_quantize_weights.argtypes = [_f32p, C.c_int64, C.c_float, C.c_int32,
                                                  C.c_int32, _i8p]
        L.dqt_oracle_quantize_weights.restype = None
        L.dqt_oracle_adafactor_u_textbook.argtypes = [_f32p, _f32p, _f32p, C.c_float,
                                                      C.c_int64, C.c_int64, _f32p]
        L.dqt_oracle_adafactor_u_textbook.restype = None
        L.dqt_oracle_adafactor_u.argtypes = [_f32p, _f32p, _f32p, C.c_int64, C.c_int64, _f32p]
        L.dqt_oracle_adafactor_u.restype = None
        L.dqt_oracle_e4m3_value.argtypes = [C.c_uint8]
        L.dqt_oracle_e4m3_value.restype = C.c_double
        L.dqt_oracle_e4m3_from_f32.argtypes = [C.c_float]
        L.dqt_oracle_e4m3_from_f32.restype = C.c_uint8
        L.dqt_oracle_codes_to_e4m3.argtypes = [_i8p, C.c_int64, _u8p]
        L.dqt_oracle_codes_to_e4m3.restype = None
        L.dqt_oracle_act_quant_fp8.argtypes = [_u16p, C.c_int64, C.c_int64, _u8p, _f32p, _u16p]
        L.dqt_oracle_act_quant_fp8.restype = None
        L.dqt_oracle_fwd_fp8.argtypes = [_u8p, _f32p, _i8p, C.c_float, C.c_int64, C.c_int64,
                                         C.c_int64, _u16p, _f64p]
        L.dqt_oracle_fwd_fp8.restype = C.c_int
        L.dqt_oracle_pack_ternary.argtypes = [_i8p, C.c_int64, _u8p]
        L.dqt_oracle_pack_ternary.restype = None
        L.dqt_oracle_unpack_ternary.argtypes = [_u8p, C.c_int64, _i8p]
        L.dqt_oracle_unpack_ternary.restype = None
        L.dqt_oracle_adafactor_consts.argtypes = [C.c_int64, C.c_float, C.c_float, C.c_int32,
                                                  C.c_int32, _f32p, _f32p, _f32p]
        L.dqt_oracle_adafactor_consts.restype = None
        L.dqt_oracle_adafactor_stats.argtypes = [_f32p, _i8p, C.c_int64, C.c_int64, C.c_float,
                                                 _f32p, _f32p, C.c_float, C.c_float, C.c_float,
                                                 C.c_float, C.c_float, C.c_float, C.c_int32,
                                                 C.c_float, _f32p, _f32p, _f64p, _f32p, _f32p]
        L.dqt_oracle_adafactor_stats.restype = None
        L.dqt_oracle_adafactor_x.argtypes = [_f32p, _i8p, _f32p, _f32p, C.c_float, C.c_float,
                                             C.c_int64, C.c_int64, _f32p]
        L.dqt_oracle_adafactor_x.restype = None
        L.dqt_oracle_adafactor_apply.argtypes = [_f32p, _i8p, _f32p, _f32p, C.c_float,
                                                 C.c_float, C.c_int64, C.c_int64, C.c_int32,
                                                 C.c_int32, C.c_uint64, C.c_int64, C.c_uint32,
                                                 C.c_int32]
        L.dqt_oracle_adafactor_apply.restype = C.c_int64
        _lib = L
    return _lib


def _p(a, ct):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ct)


def _c(a, dt):
    return np.ascontiguousarray(a, dtype=dt)


# --------------------------------------------------------------------------
# scalars and small helpers
# --------------------------------------------------------------------------
def f32_to_bf16_bits(x: float) -> int:
    return int(lib().dqt_oracle_f32_to_bf16(float(x)))


def philox4x32_10(ctr, key):
    c = _c(ctr, np.uint32)
    k = _c(key, np.uint32)
    out = np.zeros(4, np.uint32)
    lib().dqt_oracle_philox4x32_10(_p(c, _u32p), _p(k, _u32p), _p(out, _u32p))
    return out


def sr_word(seed: int, step: int, tensor_id: int, e: int) -> int:
    return int(lib().dqt_oracle_sr_word(seed, step, tensor_id, e))


def uniform_from_word(w: int) -> float:
    return float(lib().dqt_oracle_uniform_from_word(w))


def sr(x: float, u: float) -> int:
    return int(lib().dqt_oracle_sr(x, u))


def sr_batch(x, u):
    x = _c(x, np.float32)
    u = _c(u, np.float32)
    assert x.shape == u.shape
    out = np.empty(x.shape, np.int32)
    lib().dqt_oracle_sr_batch(_p(x, _f32p), _p(u, _f32p), _p(out, _i32p), x.size)
    return out


def grid(bits: float):
    """Eq. 3 grid for ``bits`` in {1.58, 2, ..., 8}; returns (Q_n, Q_p)."""
    bx = int(round(bits * 100))
    qmin = C.c_int32()
    qmax = C.c_int32()
    if lib().dqt_oracle_grid(bx, C.byref(qmin), C.byref(qmax)) != 0:
        raise ValueError("unsupported bit width %r" % bits)
    return qmin.value, qmax.value


# --------------------------------------------------------------------------
# Eq. 2-4
# --------------------------------------------------------------------------
def absmean_init(W0, qmin: int, qmax: int):
    """Returns (codes int8, s_w float32, absmean float64)."""
    W = _c(W0, np.float32)
    codes = np.empty(W.shape, np.int8)
    s = C.c_float()
    am = C.c_double()
    rc = lib().dqt_oracle_absmean_init(_p(W, _f32p), W.size, qmin, qmax,
                                       _p(codes, _i8p), C.byref(s), C.byref(am))
    if rc != 0:
        raise ValueError("absmean_init failed (%d)" % rc)
    return codes, np.float32(s.value), am.value


def quantize_weights(W, s_w, qmin: int, qmax: int):
    """Eq. 4 alone: Clip[Round(W * s_w), qmin, qmax] for a given fp32 scale."""
    W = _c(W, np.float32)
    codes = np.empty(W.shape, np.int8)
    lib().dqt_oracle_quantize_weights(_p(W, _f32p), W.size, float(np.float32(s_w)), qmin, qmax,
                                      _p(codes, _i8p))
    return codes


# --------------------------------------------------------------------------
# Sec. 3.2 activation quantisation
# --------------------------------------------------------------------------
def act_quant(X_bits):
    """X_bits: uint16 [T, K] raw bf16.  Returns (q int8, s_x f32, q_img u16, xdq u16)."""
    X = _c(X_bits, np.uint16)
    T, K = X.shape
    q = np.empty((T, K), np.int8)
    s = np.empty(T, np.float32)
    qi = np.empty((T, K), np.uint16)
    xd = np.empty((T, K), np.uint16)
    lib().dqt_oracle_act_quant(_p(X, _u16p), T, K, _p(q, _i8p), _p(s, _f32p),
                               _p(qi, _u16p), _p(xd, _u16p))
    return q, s, qi, xd


# --------------------------------------------------------------------------
# Sec. 3.2 forward / backward
# --------------------------------------------------------------------------
def fwd(q, s_x, c, s_w):
    """Returns (Y bf16 bits u16 [T,N], acc int32 [T,N])."""
    q = _c(q, np.int8)
    s_x = _c(s_x, np.float32)
    c = _c(c, np.int8)
    T, K = q.shape
    N, K2 = c.shape
    assert K == K2 and s_x.shape == (T,)
    Y = np.empty((T, N), np.uint16)
    acc = np.empty((T, N), np.int32)
    ov = lib().dqt_oracle_fwd(_p(q, _i8p), _p(s_x, _f32p), _p(c, _i8p), float(s_w),
                              T, K, N, _p(Y, _u16p), _p(acc, _i32p))
    if ov:
        raise OverflowError("int32 accumulator overflow")
    return Y, acc


def bwd_dx(dY_bits, c, s_w):
    dY = _c(dY_bits, np.uint16)
    c = _c(c, np.int8)
    T, N = dY.shape
    N2, K = c.shape
    assert N == N2
    dX = np.empty((T, K), np.float64)
    lib().dqt_oracle_bwd_dx(_p(dY, _u16p), _p(c, _i8p), float(s_w), T, N, K,
                            _p(dX, _f64p))
    return dX


def bwd_dw(dY_bits, q, s_x, rows=None):
    dY = _c(dY_bits, np.uint16)
    q = _c(q, np.int8)
    s_x = _c(s_x, np.float32)
    T, N = dY.shape
    T2, K = q.shape
    assert T == T2
    rows = np.arange(N, dtype=np.int64) if rows is None else _c(rows, np.int64)
    dW = np.empty((rows.size, K), np.float64)
    lib().dqt_oracle_bwd_dw(_p(dY, _u16p), _p(q, _i8p), _p(s_x, _f32p), T, N, K,
                            _p(rows, _i64p), rows.size, _p(dW, _f64p))
    return dW


def bwd_dw_bf16x(dY_bits, xdq_bits, rows=None):
    """dW with X_tilde held as the bf16 image bf16(q/s_x) (BF16 environment)."""
    dY = _c(dY_bits, np.uint16)
    xd = _c(xdq_bits, np.uint16)
    T, N = dY.shape
    T2, K = xd.shape
    assert T == T2
    rows = np.arange(N, dtype=np.int64) if rows is None else _c(rows, np.int64)
    dW = np.empty((rows.size, K), np.float64)
    lib().dqt_oracle_bwd_dw_bf16x(_p(dY, _u16p), _p(xd, _u16p), T, N, K, _p(rows, _i64p),
                                  rows.size, _p(dW, _f64p))
    return dW


# --------------------------------------------------------------------------
# Sec. 4.1 AdamW and Eq. 5 update
# --------------------------------------------------------------------------
def adamw_consts(lr, b1, b2, eps, wd, step, s_w):
    out = np.empty(9, np.float32)
    lib().dqt_oracle_adamw_consts(lr, b1, b2, eps, wd, step, float(s_w), _p(out, _f32p))
    return out


def adamw_x(g, c, m, v, consts):
    """Returns (x, m', v'): the dense code-domain target and the new moments."""
    g = _c(g, np.float32).ravel()
    c = _c(c, np.int8).ravel()
    m = _c(m, np.float32).ravel().copy()
    v = _c(v, np.float32).ravel().copy()
    x = np.empty_like(g)
    k = _c(consts, np.float32)
    lib().dqt_oracle_adamw_x(_p(g, _f32p), _p(c, _i8p), _p(m, _f32p), _p(v, _f32p),
                             _p(k, _f32p), g.size, _p(x, _f32p))
    return x, m, v


def adamw_textbook_consts(lr, b1, b2, eps, wd, step, s_w):
    """Constants of the textbook-order AdamW: b1, b2, 1-b1, 1-b2, bc1, bc2, eps,
    1 - lr wd, lr s_w (each rounded once to fp32)."""
    out = np.empty(9, np.float32)
    lib().dqt_oracle_adamw_textbook_consts(lr, b1, b2, eps, wd, step, float(s_w),
                                           _p(out, _f32p))
    return out


def adamw_x_textbook(g, c, m, v, tconsts):
    """As adamw_x, with m_hat = m'/bc1, v_hat = v'/bc2, m_hat/(sqrt(v_hat)+eps)."""
    g = _c(g, np.float32).ravel()
    c = _c(c, np.int8).ravel()
    m = _c(m, np.float32).ravel().copy()
    v = _c(v, np.float32).ravel().copy()
    x = np.empty_like(g)
    k = _c(tconsts, np.float32)
    lib().dqt_oracle_adamw_x_textbook(_p(g, _f32p), _p(c, _i8p), _p(m, _f32p), _p(v, _f32p),
                                      _p(k, _f32p), g.size, _p(x, _f32p))
    return x, m, v


def update(g, c, m, v, consts, qmin, qmax, seed, step, tensor_id, round_mode=0,
           rows=None, textbook=False):
    """Eq. 5 over an [Nr, K] block.  Returns (c', m', v', changed).  With
    textbook=True the AdamW step is the textbook-order form and ``consts``
    come from adamw_textbook_consts."""
    g = _c(g, np.float32)
    if g.ndim == 1:
        g = g.reshape(1, -1)
    Nr, K = g.shape
    c = _c(c, np.int8).reshape(Nr, K).copy()
    m = _c(m, np.float32).reshape(Nr, K).copy()
    v = _c(v, np.float32).reshape(Nr, K).copy()
    k = _c(consts, np.float32)
    if rows is not None:
        rows = _c(rows, np.int64)
        assert rows.size == Nr
        rp = _p(rows, _i64p)
    else:
        rp = None
    fn = lib().dqt_oracle_update_textbook if textbook else lib().dqt_oracle_update
    changed = fn(_p(g, _f32p), _p(c, _i8p), _p(m, _f32p), _p(v, _f32p), _p(k, _f32p), qmin,
                 qmax, seed, step, tensor_id, round_mode, rp, Nr, K)
    return c, m, v, int(changed)


def update_shard(g, c, m, v, consts, qmin, qmax, seed, step, tensor_id, elem0,
                 round_mode=0):
    """Eq. 5 on a flat shard: element i is global element elem0 + i of the
    weight tensor.  Returns (c', m', v', changed) as flat arrays."""
    g = _c(g, np.float32).ravel()
    n = g.size
    c = _c(c, np.int8).ravel().copy()
    m = _c(m, np.float32).ravel().copy()
    v = _c(v, np.float32).ravel().copy()
    assert c.size == n and m.size == n and v.size == n
    k = _c(consts, np.float32)
    changed = lib().dqt_oracle_update_shard(_p(g, _f32p), _p(c, _i8p), _p(m, _f32p),
                                            _p(v, _f32p), _p(k, _f32p), qmin, qmax, seed, step,
                                            tensor_id, round_mode, int(elem0), n)
    return c, m, v, int(changed)


# --------------------------------------------------------------------------
# Sec. 4.1/4.3 FP8 environment
# --------------------------------------------------------------------------
def e4m3_value(b: int) -> float:
    """The real value of the E4M3 byte b (NaN for the NaN patterns)."""
    return float(lib().dqt_oracle_e4m3_value(int(b) & 0xFF))


def e4m3_from_f32(p: float) -> int:
    """Nearest-even E4M3 byte of the fp32 value p, saturating at +-448."""
    return int(lib().dqt_oracle_e4m3_from_f32(float(p)))


def codes_to_e4m3(c):
    c = _c(c, np.int8)
    out = np.empty(c.shape, np.uint8)
    lib().dqt_oracle_codes_to_e4m3(_p(c, _i8p), c.size, _p(out, _u8p))
    return out


def act_quant_fp8(X_bits):
    """X_bits: uint16 [T, K] raw bf16.  Returns (q8 u8 E4M3 bytes, s8 f32, xdq u16)."""
    X = _c(X_bits, np.uint16)
    T, K = X.shape
    q8 = np.empty((T, K), np.uint8)
    s = np.empty(T, np.float32)
    xd = np.empty((T, K), np.uint16)
    lib().dqt_oracle_act_quant_fp8(_p(X, _u16p), T, K, _p(q8, _u8p), _p(s, _f32p),
                                   _p(xd, _u16p))
    return q8, s, xd


def fwd_fp8(q8, s8, c, s_w):
    """Returns (Y bf16 bits u16 [T,N], acc float64 [T,N], exact)."""
    q8 = _c(q8, np.uint8)
    s8 = _c(s8, np.float32)
    c = _c(c, np.int8)
    T, K = q8.shape
    N, K2 = c.shape
    assert K == K2 and s8.shape == (T,)
    Y = np.empty((T, N), np.uint16)
    acc = np.empty((T, N), np.float64)
    lib().dqt_oracle_fwd_fp8(_p(q8, _u8p), _p(s8, _f32p), _p(c, _i8p), float(s_w),
                             T, K, N, _p(Y, _u16p), _p(acc, _f64p))
    return Y, acc


# --------------------------------------------------------------------------
# Sec. 1: 2-bit packed ternary storage
# --------------------------------------------------------------------------
def pack_ternary(c):
    """int8 ternary codes -> uint8 [ceil(n/4)], code e in bits 2(e%4)..2(e%4)+1."""
    c = _c(c, np.int8).ravel()
    out = np.empty((c.size + 3) // 4, np.uint8)
    lib().dqt_oracle_pack_ternary(_p(c, _i8p), c.size, _p(out, _u8p))
    return out


def unpack_ternary(p, n):
    p = _c(p, np.uint8).ravel()
    assert p.size >= (n + 3) // 4
    out = np.empty(n, np.int8)
    lib().dqt_oracle_unpack_ternary(_p(p, _u8p), n, _p(out, _i8p))
    return out


# --------------------------------------------------------------------------
# Sec. 4.3: Adafactor (Shazeer & Stern 2018) + SR, no first moment
# --------------------------------------------------------------------------
class AdafactorHP:
    """Adafactor hyper-parameters (defaults: a fixed step size lr, no
    parameter scaling, eps1 = 1e-30 added to g^2, eps2 = 1e-3, update
    clipping d = 1, beta2_t = 1 - t^-0.8, no weight decay)."""

    def __init__(self, lr=1e-3, eps1=1e-30, eps2=1e-3, clip_d=1.0, decay_rate=-0.8,
                 weight_decay=0.0, relative_step=False, scale_parameter=False,
                 warmup_init=False):
        self.lr, self.eps1, self.eps2, self.clip_d = lr, eps1, eps2, clip_d
        self.decay_rate, self.weight_decay = decay_rate, weight_decay
        self.relative_step, self.scale_parameter = relative_step, scale_parameter
        self.warmup_init = warmup_init


def adafactor_consts(t, hp):
    """(b2, omb2, rho) of step t, each rounded once to fp32."""
    b2, omb2, rho = C.c_float(), C.c_float(), C.c_float()
    lib().dqt_oracle_adafactor_consts(int(t), hp.lr, hp.decay_rate, int(hp.relative_step),
                                      int(hp.warmup_init), C.byref(b2), C.byref(omb2),
                                      C.byref(rho))
    return np.float32(b2.value), np.float32(omb2.value), np.float32(rho.value)


def adafactor_stats(g, c, s_w, R, C_, t, hp):
    """Returns (R', C', st) with st = dict(rbar, rms_u, rms_x, alpha, step, decay, a, b):
    R', C' fp32 state, a [N] and b [K] the fp32 inverse-square-root factors."""
    g = _c(g, np.float32)
    N, K = g.shape
    c = _c(c, np.int8).reshape(N, K)
    R = _c(R, np.float32).copy()
    Cc = _c(C_, np.float32).copy()
    assert R.shape == (N,) and Cc.shape == (K,)
    b2, omb2, rho = adafactor_consts(t, hp)
    a = np.empty(N, np.float32)
    b = np.empty(K, np.float32)
    out4 = np.empty(4, np.float64)
    step, decay = C.c_float(), C.c_float()
    lib().dqt_oracle_adafactor_stats(_p(g, _f32p), _p(c, _i8p), N, K, float(s_w), _p(R, _f32p),
                                     _p(Cc, _f32p), b2, omb2, rho, hp.eps1, hp.eps2, hp.clip_d,
                                     int(hp.scale_parameter), hp.weight_decay, _p(a, _f32p),
                                     _p(b, _f32p), _p(out4, _f64p), C.byref(step),
                                     C.byref(decay))
    st = {"rbar": out4[0], "rms_u": out4[1], "rms_x": out4[2], "alpha": out4[3],
          "step": np.float32(step.value), "decay": np.float32(decay.value), "a": a, "b": b}
    return R, Cc, st


def adafactor_u(g, a, b):
    """The factored form's u = (g a[n]) b[k] for every element of g [N, K]."""
    g = _c(g, np.float32)
    N, K = g.shape
    a = _c(a, np.float32)
    b = _c(b, np.float32)
    u = np.empty((N, K), np.float32)
    lib().dqt_oracle_adafactor_u(_p(g, _f32p), _p(a, _f32p), _p(b, _f32p), N, K, _p(u, _f32p))
    return u


def adafactor_u_textbook(g, R, C_, rbar):
    """The printed form u = g / sqrt(R[n] C[k] / Rbar), fp32 operations."""
    g = _c(g, np.float32)
    N, K = g.shape
    R = _c(R, np.float32)
    Cc = _c(C_, np.float32)
    u = np.empty((N, K), np.float32)
    lib().dqt_oracle_adafactor_u_textbook(_p(g, _f32p), _p(R, _f32p), _p(Cc, _f32p),
                                          float(np.float32(rbar)), N, K, _p(u, _f32p))
    return u


def adafactor_x(g, c, a, b, step, decay):
    g = _c(g, np.float32)
    N, K = g.shape
    c = _c(c, np.int8).reshape(N, K)
    a = _c(a, np.float32)
    b = _c(b, np.float32)
    x = np.empty((N, K), np.float32)
    lib().dqt_oracle_adafactor_x(_p(g, _f32p), _p(c, _i8p), _p(a, _f32p), _p(b, _f32p),
                                 float(step), float(decay), N, K, _p(x, _f32p))
    return x


def adafactor_apply(g, c, a, b, step, decay, qmin, qmax, seed, t, tensor_id, round_mode=0):
    """Returns (c', changed)."""
    g = _c(g, np.float32)
    N, K = g.shape
    c = _c(c, np.int8).reshape(N, K).copy()
    a = _c(a, np.float32)
    b = _c(b, np.float32)
    ch = lib().dqt_oracle_adafactor_apply(_p(g, _f32p), _p(c, _i8p), _p(a, _f32p), _p(b, _f32p),
                                          float(step), float(decay), N, K, qmin, qmax, seed, t,
                                          tensor_id, round_mode)
    return c, int(ch)
