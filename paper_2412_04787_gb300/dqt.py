"""Python binding of the DQT C ABI (``include/dqt.h``), argument marshalling only.

Every function has the name of the C entry point it calls, takes CUDA torch
tensors, checks dtype / device / contiguity / shape, and passes raw device
pointers and the current CUDA stream to ``libdqt.so``.  All arithmetic runs in
the library's CUDA kernels; if the library is missing, loading it raises.
"""
import ctypes as C
import os

import torch

_LIB_PATH = os.path.join(os.path.dirname(os.path.abspath(__file__)), "libdqt.so")
_lib = None

DQT_OK, DQT_ERR_ARG, DQT_ERR_ALIGN, DQT_ERR_CUDA, DQT_ERR_TIMEOUT, DQT_ERR_RANGE = range(6)

# Every symbol include/dqt.h declares.
EXPORTED = [
    "dqt_grid_for_bits", "dqt_status_string", "dqt_check_device_status",
    "dqt_set_wait_limit_ns", "dqt_absmean_workspace_size", "dqt_absmean_init",
    "dqt_act_quant", "dqt_codes_to_bf16", "dqt_bitlinear_fwd", "dqt_bitlinear_bwd_dx",
    "dqt_bitlinear_bwd_dw_update", "dqt_sr_update", "dqt_absmean_init_noalloc",
    "dqt_set_gemm_tiles", "dqt_update_consts_size", "dqt_update_consts",
    "dqt_bitlinear_bwd_dw_update_dev", "dqt_sr_update_dev", "dqt_bwd_dw_workspace_size",
    "dqt_act_quant_fp8", "dqt_codes_to_fp8", "dqt_codes_to_fp8_split", "dqt_bitlinear_fwd_fp8",
    "dqt_bitlinear_fwd_fp8_pair",
    "dqt_pack_ternary", "dqt_unpack_ternary", "dqt_packed_to_bf16", "dqt_packed_to_fp8",
    "dqt_sr_update_packed", "dqt_bitlinear_bwd_dw_update_packed",
    "dqt_adafactor_workspace_size", "dqt_adafactor_stats", "dqt_adafactor_apply",
    "dqt_bwd_dw_adafactor_workspace_size", "dqt_bitlinear_bwd_dw_adafactor",
    "dqt_rope_bf16", "dqt_cross_entropy_fwd_bf16", "dqt_cross_entropy_bwd_bf16",
    "dqt_swiglu_bf16", "dqt_swiglu_bwd_bf16", "dqt_rmsnorm_bf16",
    "dqt_rmsnorm_bwd_workspace_size", "dqt_rmsnorm_bwd_bf16",
    "dqt_act_quant_images", "dqt_bitlinear_fwd_img", "dqt_bitlinear_bwd_dx_img",
    "dqt_bwd_dx_workspace_size", "dqt_bitlinear_bwd_dw_update_img",
    "dqt_bwd_dw_img_workspace_size", "dqt_codes_to_xdq", "dqt_fwd_workspace_size",
    "dqt_fwd_img_workspace_size", "dqt_bwd_dx_img_workspace_size",
    "dqt_bitlinear_fwd_img_pair", "dqt_bitlinear_bwd_dw_update_img_pair",
    "dqt_bitlinear_bwd_dx_img_ld", "dqt_bitlinear_bwd_dw_update_group",
]


class DQTError(RuntimeError):
    def __init__(self, status, where):
        self.status = status
        super().__init__("%s: %s" % (where, lib().dqt_status_string(status).decode()))


class dqt_grid_t(C.Structure):
    _fields_ = [("qmin", C.c_int32), ("qmax", C.c_int32)]


class dqt_adamw_t(C.Structure):
    _fields_ = [("lr", C.c_float), ("beta1", C.c_float), ("beta2", C.c_float),
                ("eps", C.c_float), ("weight_decay", C.c_float), ("step", C.c_int64)]


class dqt_sr_t(C.Structure):
    _fields_ = [("seed", C.c_uint64), ("tensor_id", C.c_uint32), ("round_mode", C.c_int32),
                ("elem0", C.c_int64)]


class dqt_dw_problem_t(C.Structure):
    _fields_ = [("dY", C.c_void_p), ("Xdq", C.c_void_p), ("W", C.c_void_p), ("m", C.c_void_p),
                ("v", C.c_void_p), ("N", C.c_int64), ("K", C.c_int64), ("N0", C.c_int64),
                ("s_w0", C.c_float), ("s_w1", C.c_float), ("sr0", C.POINTER(dqt_sr_t)),
                ("sr1", C.POINTER(dqt_sr_t)), ("W_img_next", C.c_void_p), ("W8_next", C.c_void_p),
                ("changed_out", C.c_void_p)]


class dqt_adafactor_t(C.Structure):
    _fields_ = [("lr", C.c_float), ("eps1", C.c_float), ("eps2", C.c_float),
                ("clip_d", C.c_float), ("decay_rate", C.c_float), ("weight_decay", C.c_float),
                ("step", C.c_int64), ("relative_step", C.c_int32),
                ("scale_parameter", C.c_int32), ("warmup_init", C.c_int32), ("pad", C.c_int32)]


_vp, _i64, _f32, _sz = C.c_void_p, C.c_int64, C.c_float, C.c_size_t


def lib():
    """Load libdqt.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(_LIB_PATH):
            raise RuntimeError("libdqt.so is not built (run __graft_entry__.build()); "
                               "the DQT library has no CPU fallback")
        L = C.CDLL(_LIB_PATH)
        L.dqt_grid_for_bits.argtypes = [_f32, C.POINTER(dqt_grid_t)]
        L.dqt_status_string.argtypes = [C.c_int]
        L.dqt_status_string.restype = C.c_char_p
        L.dqt_check_device_status.argtypes = [_vp]
        L.dqt_set_wait_limit_ns.argtypes = [C.c_uint64]
        L.dqt_set_gemm_tiles.argtypes = [C.c_int]
        L.dqt_absmean_workspace_size.argtypes = []
        L.dqt_absmean_workspace_size.restype = _sz
        L.dqt_absmean_init.argtypes = [_vp, _i64, dqt_grid_t, _vp, C.POINTER(C.c_float), _vp,
                                       _sz, _vp]
        L.dqt_absmean_init_noalloc.argtypes = [_vp, _i64, dqt_grid_t, _vp,
                                               C.POINTER(C.c_float), _vp]
        L.dqt_act_quant.argtypes = [_vp, _i64, _i64, _vp, _vp, _vp]
        L.dqt_act_quant_images.argtypes = [_vp, _i64, _i64, _vp, _vp, _vp, _vp, _vp]
        L.dqt_codes_to_bf16.argtypes = [_vp, _i64, _vp, _vp]
        L.dqt_codes_to_xdq.argtypes = [_vp, _vp, _i64, _i64, _vp, _vp]
        L.dqt_bitlinear_fwd.argtypes = [_vp, _vp, _vp, _f32, dqt_grid_t, _i64, _i64, _i64, _vp,
                                        _vp, _vp, _sz, _vp]
        L.dqt_fwd_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_fwd_workspace_size.restype = _sz
        L.dqt_bitlinear_fwd_img.argtypes = [_vp, _vp, _vp, _f32, dqt_grid_t, _i64, _i64, _i64,
                                            _vp, _vp, _vp, _sz, _vp]
        L.dqt_bitlinear_fwd_img_pair.argtypes = [_vp, _vp, _vp, _i64, _f32, _f32, dqt_grid_t, _i64,
                                                 _i64, _i64, _vp, _vp, _vp, _sz, _vp]
        L.dqt_bitlinear_bwd_dw_update_img_pair.argtypes = [
            _vp, _vp, _vp, _i64, _f32, _f32, _vp, _vp, C.POINTER(dqt_adamw_t),
            C.POINTER(dqt_sr_t), C.POINTER(dqt_sr_t), dqt_grid_t, _i64, _i64, _i64, _vp, _vp,
            _vp, _vp, _vp, _sz, _vp]
        L.dqt_bitlinear_bwd_dw_update_group.argtypes = [
            C.POINTER(dqt_dw_problem_t), C.c_int, C.POINTER(dqt_adamw_t), dqt_grid_t, _i64, _vp]
        L.dqt_fwd_img_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_fwd_img_workspace_size.restype = _sz
        L.dqt_bitlinear_bwd_dx.argtypes = [_vp, _vp, _f32, _i64, _i64, _i64, _vp, _vp, _sz, _vp]
        L.dqt_bitlinear_bwd_dx_img.argtypes = [_vp, _vp, _f32, _i64, _i64, _i64, _vp, _vp, _sz,
                                               _vp]
        L.dqt_bitlinear_bwd_dx_img_ld.argtypes = [_vp, _i64, _vp, _f32, _i64, _i64, _i64, _vp, _vp,
                                                  _sz, _vp]
        L.dqt_bwd_dx_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_bwd_dx_workspace_size.restype = _sz
        L.dqt_bwd_dx_img_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_bwd_dx_img_workspace_size.restype = _sz
        L.dqt_bitlinear_bwd_dw_update.argtypes = [_vp, _vp, _vp, _vp, _f32, _vp, _vp,
                                                  C.POINTER(dqt_adamw_t), C.POINTER(dqt_sr_t),
                                                  dqt_grid_t, _i64, _i64, _i64, _vp, _vp, _vp,
                                                  _sz, _vp]
        L.dqt_bitlinear_bwd_dw_update_img.argtypes = [_vp, _vp, _vp, _f32, _vp, _vp,
                                                      C.POINTER(dqt_adamw_t),
                                                      C.POINTER(dqt_sr_t), dqt_grid_t, _i64,
                                                      _i64, _i64, _vp, _vp, _vp, _vp, _vp, _sz,
                                                      _vp]
        L.dqt_bwd_dw_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_bwd_dw_workspace_size.restype = _sz
        L.dqt_bwd_dw_img_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_bwd_dw_img_workspace_size.restype = _sz
        L.dqt_sr_update.argtypes = [_vp, _vp, _f32, _vp, _vp, C.POINTER(dqt_adamw_t),
                                    C.POINTER(dqt_sr_t), dqt_grid_t, _i64, _vp, _vp]
        L.dqt_update_consts_size.argtypes = []
        L.dqt_update_consts_size.restype = _sz
        L.dqt_update_consts.argtypes = [C.POINTER(dqt_adamw_t), C.POINTER(dqt_sr_t), dqt_grid_t,
                                        _f32, _vp, _sz]
        L.dqt_bitlinear_bwd_dw_update_dev.argtypes = [_vp, _vp, _vp, _vp, _vp, _vp, _i64, _i64,
                                                      _i64, _vp, _vp, _vp, _vp, _vp, _sz, _vp]
        L.dqt_sr_update_dev.argtypes = [_vp, _vp, _vp, _vp, _vp, _i64, _vp, _vp]
        L.dqt_act_quant_fp8.argtypes = [_vp, _i64, _i64, _vp, _vp, _vp, _vp]
        L.dqt_codes_to_fp8.argtypes = [_vp, _i64, dqt_grid_t, _vp, _vp]
        L.dqt_codes_to_fp8_split.argtypes = [_vp, _i64, _i64, _vp, _vp]
        L.dqt_bitlinear_fwd_fp8.argtypes = [_vp, _vp, _vp, _f32, dqt_grid_t, _i64, _i64, _i64,
                                            _vp, _vp, _vp]
        L.dqt_bitlinear_fwd_fp8_pair.argtypes = [_vp, _vp, _vp, _i64, _f32, _f32, dqt_grid_t, _i64,
                                                 _i64, _i64, _vp, _vp, _vp]
        for name in ("dqt_pack_ternary", "dqt_unpack_ternary", "dqt_packed_to_bf16",
                     "dqt_packed_to_fp8"):
            getattr(L, name).argtypes = [_vp, _i64, _vp, _vp]
        L.dqt_sr_update_packed.argtypes = [_vp, _vp, _f32, _vp, _vp, C.POINTER(dqt_adamw_t),
                                           C.POINTER(dqt_sr_t), _i64, _vp, _vp]
        L.dqt_bitlinear_bwd_dw_update_packed.argtypes = [_vp, _vp, _vp, _f32, _vp, _vp,
                                                         C.POINTER(dqt_adamw_t),
                                                         C.POINTER(dqt_sr_t), _i64, _i64, _i64,
                                                         _vp, _vp, _vp, _sz, _vp]
        L.dqt_adafactor_workspace_size.argtypes = [_i64, _i64]
        L.dqt_adafactor_workspace_size.restype = _sz
        L.dqt_adafactor_stats.argtypes = [_vp, _vp, C.c_int32, _f32, _vp, _vp,
                                          C.POINTER(dqt_adafactor_t), _i64, _i64, _vp, _vp, _vp,
                                          _vp, _sz, _vp]
        L.dqt_adafactor_apply.argtypes = [_vp, _vp, C.c_int32, _vp, _vp, _vp, _i64,
                                          C.POINTER(dqt_sr_t), dqt_grid_t, _i64, _i64, _vp, _vp]
        L.dqt_bwd_dw_adafactor_workspace_size.argtypes = [_i64, _i64, _i64]
        L.dqt_bwd_dw_adafactor_workspace_size.restype = _sz
        L.dqt_bitlinear_bwd_dw_adafactor.argtypes = [_vp, _vp, _vp, C.c_int32, _f32, _vp, _vp,
                                                     C.POINTER(dqt_adafactor_t),
                                                     C.POINTER(dqt_sr_t), dqt_grid_t, _i64, _i64,
                                                     _i64, _vp, _vp, _sz, _vp]
        L.dqt_rope_bf16.argtypes = [_vp, _vp, _vp, _i64, _i64, _i64, _i64, C.c_int32, _vp]
        L.dqt_cross_entropy_fwd_bf16.argtypes = [_vp, _vp, _i64, _i64, _vp, _vp, _vp]
        L.dqt_cross_entropy_bwd_bf16.argtypes = [_vp, _vp, _vp, _vp, _i64, _i64, _vp, _vp]
        L.dqt_swiglu_bf16.argtypes = [_vp, _vp, _vp, _i64, _vp]
        L.dqt_swiglu_bwd_bf16.argtypes = [_vp, _vp, _vp, _vp, _vp, _i64, _vp]
        L.dqt_rmsnorm_bf16.argtypes = [_vp, _vp, _f32, _i64, _i64, _vp, _vp, _vp]
        L.dqt_rmsnorm_bwd_workspace_size.argtypes = [_i64, _i64]
        L.dqt_rmsnorm_bwd_workspace_size.restype = _sz
        L.dqt_rmsnorm_bwd_bf16.argtypes = [_vp, _vp, _vp, _vp, _i64, _i64, _vp, _vp, _vp, _sz,
                                           _vp]
        for name in EXPORTED:
            if name not in ("dqt_status_string", "dqt_absmean_workspace_size",
                            "dqt_update_consts_size", "dqt_bwd_dw_workspace_size",
                            "dqt_bwd_dw_img_workspace_size", "dqt_bwd_dx_workspace_size",
                            "dqt_fwd_workspace_size", "dqt_fwd_img_workspace_size",
                            "dqt_bwd_dx_img_workspace_size",
                            "dqt_adafactor_workspace_size",
                            "dqt_bwd_dw_adafactor_workspace_size",
                            "dqt_rmsnorm_bwd_workspace_size"):
                getattr(L, name).restype = C.c_int
        _lib = L
    return _lib


def _check(rc, where):
    if rc != DQT_OK:
        raise DQTError(rc, where)


def _ptr(t):
    return None if t is None else C.c_void_p(t.data_ptr())


def _need(t, name, dtype, shape=None):
    if t is None:
        raise ValueError("%s is required" % name)
    if not t.is_cuda:
        raise ValueError("%s must be a CUDA tensor" % name)
    if t.dtype != dtype:
        raise ValueError("%s must be %s, got %s" % (name, dtype, t.dtype))
    if not t.is_contiguous():
        raise ValueError("%s must be contiguous" % name)
    if shape is not None and tuple(t.shape) != tuple(shape):
        raise ValueError("%s must have shape %s, got %s" % (name, tuple(shape), tuple(t.shape)))
    return t


def _opt(t, name, dtype, shape):
    return None if t is None else _need(t, name, dtype, shape)


def _stream(stream=None):
    s = torch.cuda.current_stream() if stream is None else stream
    return C.c_void_p(s.cuda_stream)


def grid(bits):
    """Eq. 3 grid for ``bits`` (1.58 or 2..8) as a dqt_grid_t."""
    g = dqt_grid_t()
    _check(lib().dqt_grid_for_bits(float(bits), C.byref(g)), "dqt_grid_for_bits")
    return g


def _grid(g):
    if isinstance(g, dqt_grid_t):
        return g
    if isinstance(g, (tuple, list)):
        return dqt_grid_t(int(g[0]), int(g[1]))
    return grid(g)


def adamw(lr=1e-3, beta1=0.9, beta2=0.999, eps=1e-8, weight_decay=0.0, step=1):
    return dqt_adamw_t(lr, beta1, beta2, eps, weight_decay, step)


def sr_stream(seed=1234, tensor_id=0, round_mode=0, elem0=0):
    """The SR stream of a tensor; elem0 = global index of the call's first
    element (a data-parallel shard's offset into the flat weight)."""
    return dqt_sr_t(seed, tensor_id, round_mode, elem0)


# ---------------------------------------------------------------------------
# entry points
# ---------------------------------------------------------------------------
def dqt_check_device_status(stream=None):
    _check(lib().dqt_check_device_status(_stream(stream)), "device status")


def dqt_set_wait_limit_ns(ns):
    _check(lib().dqt_set_wait_limit_ns(int(ns)), "dqt_set_wait_limit_ns")


def dqt_set_gemm_tiles(mode):
    """0 = 2-SM 256x256 tiles (default), 1 = 1-SM 128x256 tiles."""
    _check(lib().dqt_set_gemm_tiles(int(mode)), "dqt_set_gemm_tiles")


def dqt_absmean_init(W0, bits_or_grid, codes=None, stream=None):
    """Eq. 2-4.  Returns (codes int8, s_w float)."""
    _need(W0, "W0", torch.float32)
    g = _grid(bits_or_grid)
    codes = torch.empty(W0.shape, dtype=torch.int8, device=W0.device) if codes is None else \
        _need(codes, "codes", torch.int8, W0.shape)
    nws = lib().dqt_absmean_workspace_size()
    ws = torch.empty(nws, dtype=torch.uint8, device=W0.device)
    s = C.c_float()
    _check(lib().dqt_absmean_init(_ptr(W0), W0.numel(), g, _ptr(codes), C.byref(s), _ptr(ws),
                                  nws, _stream(stream)), "dqt_absmean_init")
    return codes, float(s.value)


def dqt_act_quant(X, Xq=None, s_x=None, stream=None):
    """Sec. 3.2 activation codes: returns (Xq int8 [T, K], s_x fp32 [T])."""
    _need(X, "X", torch.bfloat16)
    if X.dim() != 2:
        raise ValueError("X must be [T, K]")
    T, K = X.shape
    if Xq is None:
        Xq = torch.empty((T, K), dtype=torch.int8, device=X.device)
    if s_x is None:
        s_x = torch.empty(T, dtype=torch.float32, device=X.device)
    _need(Xq, "Xq", torch.int8, (T, K))
    _need(s_x, "s_x", torch.float32, (T,))
    _check(lib().dqt_act_quant(_ptr(X), T, K, _ptr(Xq), _ptr(s_x), _stream(stream)),
           "dqt_act_quant")
    return Xq, s_x


def dqt_act_quant_images(X, Xq=None, s_x=None, Xq_img=None, Xdq=None,
                         want=("Xq", "Xq_img", "Xdq"), stream=None):
    """Activation codes and the bf16 operand images of the *_img calls.
    Outputs not passed are allocated if named in ``want``.  Returns (Xq, s_x,
    Xq_img, Xdq), None for outputs not produced."""
    _need(X, "X", torch.bfloat16)
    if X.dim() != 2:
        raise ValueError("X must be [T, K]")
    T, K = X.shape
    dev = X.device
    if Xq is None and "Xq" in want:
        Xq = torch.empty((T, K), dtype=torch.int8, device=dev)
    if Xq_img is None and "Xq_img" in want:
        Xq_img = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    if Xdq is None and "Xdq" in want:
        Xdq = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    if s_x is None:
        s_x = torch.empty(T, dtype=torch.float32, device=dev)
    _opt(Xq, "Xq", torch.int8, (T, K))
    _need(s_x, "s_x", torch.float32, (T,))
    _opt(Xq_img, "Xq_img", torch.bfloat16, (T, K))
    _opt(Xdq, "Xdq", torch.bfloat16, (T, K))
    _check(lib().dqt_act_quant_images(_ptr(X), T, K, _ptr(Xq), _ptr(s_x), _ptr(Xq_img),
                                      _ptr(Xdq), _stream(stream)), "dqt_act_quant_images")
    return Xq, s_x, Xq_img, Xdq


def dqt_codes_to_bf16(W, W_img=None, stream=None):
    _need(W, "W", torch.int8)
    if W_img is None:
        W_img = torch.empty(W.shape, dtype=torch.bfloat16, device=W.device)
    _need(W_img, "W_img", torch.bfloat16, W.shape)
    _check(lib().dqt_codes_to_bf16(_ptr(W), W.numel(), _ptr(W_img), _stream(stream)),
           "dqt_codes_to_bf16")
    return W_img


def dqt_codes_to_xdq(Xq, s_x, Xdq=None, stream=None):
    """X_tilde = bf16(Xq / s_x), the weight-gradient operand image."""
    _need(Xq, "Xq", torch.int8)
    T, K = Xq.shape
    _need(s_x, "s_x", torch.float32, (T,))
    if Xdq is None:
        Xdq = torch.empty((T, K), dtype=torch.bfloat16, device=Xq.device)
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _check(lib().dqt_codes_to_xdq(_ptr(Xq), _ptr(s_x), T, K, _ptr(Xdq), _stream(stream)),
           "dqt_codes_to_xdq")
    return Xdq


def dqt_fwd_workspace_size(T, K, N):
    return int(lib().dqt_fwd_workspace_size(T, K, N))


def dqt_bitlinear_fwd(Xq, s_x, W, s_w, bits_or_grid, Y=None, acc_out=None, ws=None, stream=None):
    """Sec. 3.2 forward from the int8 codes; `ws` (uint8 CUDA tensor of
    dqt_fwd_workspace_size bytes) receives their bf16 images, allocated if None."""
    _need(Xq, "Xq", torch.int8)
    T, K = Xq.shape
    _need(W, "W", torch.int8)
    N = W.shape[0]
    _need(W, "W", torch.int8, (N, K))
    _need(s_x, "s_x", torch.float32, (T,))
    if Y is None:
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=Xq.device)
    _need(Y, "Y", torch.bfloat16, (T, N))
    _opt(acc_out, "acc_out", torch.int32, (T, N))
    if ws is None:
        ws = torch.empty(lib().dqt_fwd_workspace_size(T, K, N), dtype=torch.uint8,
                         device=Xq.device)
    _need(ws, "ws", torch.uint8)
    _check(lib().dqt_bitlinear_fwd(_ptr(Xq), _ptr(s_x), _ptr(W), float(s_w),
                                   _grid(bits_or_grid), T, K, N, _ptr(Y), _ptr(acc_out),
                                   _ptr(ws), ws.numel(), _stream(stream)), "dqt_bitlinear_fwd")
    return Y


def _tail_workspace(need, device, ws):
    """Optional workspace of the GEMM calls whose last wave may be cut into
    slices: None allocates the `need` bytes, False passes none."""
    if ws is False or need == 0:
        return None, 0
    if ws is None:
        ws = torch.empty(need, dtype=torch.uint8, device=device)
    _need(ws, "ws", torch.uint8)
    return ws, ws.numel()


def dqt_fwd_img_workspace_size(T, K, N):
    return int(lib().dqt_fwd_img_workspace_size(T, K, N))


def dqt_bitlinear_fwd_img(Xq_img, s_x, W_img, s_w, bits_or_grid, Y=None, acc_out=None,
                          ws=None, stream=None):
    """The forward on the bf16 operand images; `ws` (uint8 CUDA tensor of
    dqt_fwd_img_workspace_size bytes) holds last-wave slice partials:
    allocated if None, none if False."""
    _need(Xq_img, "Xq_img", torch.bfloat16)
    T, K = Xq_img.shape
    _need(W_img, "W_img", torch.bfloat16)
    N = W_img.shape[0]
    _need(W_img, "W_img", torch.bfloat16, (N, K))
    _need(s_x, "s_x", torch.float32, (T,))
    if Y is None:
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=Xq_img.device)
    _need(Y, "Y", torch.bfloat16, (T, N))
    _opt(acc_out, "acc_out", torch.int32, (T, N))
    ws, nws = _tail_workspace(lib().dqt_fwd_img_workspace_size(T, K, N), Xq_img.device, ws)
    _check(lib().dqt_bitlinear_fwd_img(_ptr(Xq_img), _ptr(s_x), _ptr(W_img), float(s_w),
                                       _grid(bits_or_grid), T, K, N, _ptr(Y), _ptr(acc_out),
                                       _ptr(ws), nws, _stream(stream)), "dqt_bitlinear_fwd_img")
    return Y


def dqt_bitlinear_fwd_img_pair(Xq_img, s_x, W_img, N0, s_w0, s_w1, bits_or_grid, Y=None,
                               acc_out=None, ws=None, stream=None):
    """Two weights that read the same input, stacked along N (rows [0, N0)
    of W_img the first's code image, scale s_w0; the rest the second's, s_w1):
    Y [T, N] holds both outputs side by side.  `ws` as dqt_bitlinear_fwd_img."""
    _need(Xq_img, "Xq_img", torch.bfloat16)
    T, K = Xq_img.shape
    _need(W_img, "W_img", torch.bfloat16)
    N = W_img.shape[0]
    _need(W_img, "W_img", torch.bfloat16, (N, K))
    _need(s_x, "s_x", torch.float32, (T,))
    if Y is None:
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=Xq_img.device)
    _need(Y, "Y", torch.bfloat16, (T, N))
    _opt(acc_out, "acc_out", torch.int32, (T, N))
    ws, nws = _tail_workspace(lib().dqt_fwd_img_workspace_size(T, K, N), Xq_img.device, ws)
    _check(lib().dqt_bitlinear_fwd_img_pair(_ptr(Xq_img), _ptr(s_x), _ptr(W_img), int(N0),
                                            float(s_w0), float(s_w1), _grid(bits_or_grid), T, K, N,
                                            _ptr(Y), _ptr(acc_out), _ptr(ws), nws, _stream(stream)),
           "dqt_bitlinear_fwd_img_pair")
    return Y


def dqt_bwd_dx_workspace_size(T, N, K):
    return int(lib().dqt_bwd_dx_workspace_size(T, N, K))


def dqt_bwd_dx_img_workspace_size(T, N, K):
    return int(lib().dqt_bwd_dx_img_workspace_size(T, N, K))


def dqt_bitlinear_bwd_dx(dY, W, s_w, dX=None, ws=None, stream=None):
    """dX = dY W_tilde from the int8 codes; `ws` (uint8 CUDA tensor of
    dqt_bwd_dx_workspace_size bytes) receives their bf16 image, allocated if
    None."""
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(W, "W", torch.int8)
    K = W.shape[1]
    _need(W, "W", torch.int8, (N, K))
    if dX is None:
        dX = torch.empty((T, K), dtype=torch.bfloat16, device=dY.device)
    _need(dX, "dX", torch.bfloat16, (T, K))
    nws = lib().dqt_bwd_dx_workspace_size(T, N, K)
    if ws is None:
        ws = torch.empty(nws, dtype=torch.uint8, device=dY.device)
    _need(ws, "ws", torch.uint8)
    _check(lib().dqt_bitlinear_bwd_dx(_ptr(dY), _ptr(W), float(s_w), T, N, K, _ptr(dX),
                                      _ptr(ws), ws.numel(), _stream(stream)),
           "dqt_bitlinear_bwd_dx")
    return dX


def dqt_bitlinear_bwd_dx_img(dY, W_img, s_w, dX=None, ws=None, stream=None):
    """dX on the weight's bf16 image; `ws` as for dqt_bitlinear_fwd_img
    (dqt_bwd_dx_img_workspace_size bytes).  dY may be a view of whole rows'
    column range (e.g. one weight's half of a stacked output's gradient):
    its rows are then read in place, dY.stride(0) elements apart."""
    if dY is not None and dY.dim() == 2 and dY.stride(1) == 1 and dY.stride(0) > dY.shape[1]:
        ldy = dY.stride(0)  # rows of a wider tensor
        if not dY.is_cuda or dY.dtype != torch.bfloat16:
            raise ValueError("dY must be a bf16 CUDA tensor")
    else:
        _need(dY, "dY", torch.bfloat16)
        ldy = dY.shape[1]
    T, N = dY.shape
    _need(W_img, "W_img", torch.bfloat16)
    K = W_img.shape[1]
    _need(W_img, "W_img", torch.bfloat16, (N, K))
    if dX is None:
        dX = torch.empty((T, K), dtype=torch.bfloat16, device=dY.device)
    _need(dX, "dX", torch.bfloat16, (T, K))
    ws, nws = _tail_workspace(lib().dqt_bwd_dx_img_workspace_size(T, N, K), dY.device, ws)
    _check(lib().dqt_bitlinear_bwd_dx_img_ld(_ptr(dY), ldy, _ptr(W_img), float(s_w), T, N, K,
                                             _ptr(dX), _ptr(ws), nws, _stream(stream)),
           "dqt_bitlinear_bwd_dx_img")
    return dX


def _dw_workspace(T, N, K, device, ws):
    if ws is False:
        return None, 0
    need = lib().dqt_bwd_dw_img_workspace_size(T, N, K)
    if need == 0:
        return None, 0
    if ws is None:
        ws = torch.empty(need, dtype=torch.uint8, device=device)
    _need(ws, "ws", torch.uint8)
    return ws, ws.numel()


def dqt_bwd_dw_workspace_size(T, N, K):
    return int(lib().dqt_bwd_dw_workspace_size(T, N, K))


def dqt_bwd_dw_img_workspace_size(T, N, K):
    return int(lib().dqt_bwd_dw_img_workspace_size(T, N, K))


def dqt_bitlinear_bwd_dw_update(dY, Xq, s_x, W, s_w, m, v, hp, sr, bits_or_grid, dW_out=None,
                                changed_out=None, ws=None, stream=None):
    """Weight gradient from the int8 activation codes + AdamW + stochastic
    rounding; W, m, v updated in place (W = m = v = None: dW_out only).
    `ws`: uint8 CUDA tensor of at least the X_tilde image (T K 2 bytes,
    rounded up to 256) -- dqt_bwd_dw_workspace_size bytes also enable the
    token-sliced reduction; None allocates the full size, False only the
    image (the single fused kernel)."""
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xq, "Xq", torch.int8)
    K = Xq.shape[1]
    _need(Xq, "Xq", torch.int8, (T, K))
    _need(s_x, "s_x", torch.float32, (T,))
    _opt(W, "W", torch.int8, (N, K))
    _opt(m, "m", torch.float32, (N, K))
    _opt(v, "v", torch.float32, (N, K))
    _opt(dW_out, "dW_out", torch.float32, (N, K))
    _opt(changed_out, "changed_out", torch.int64, (1,))
    if ws is None or ws is False:
        n = (lib().dqt_bwd_dw_workspace_size(T, N, K) if ws is None
             else (T * K * 2 + 255) // 256 * 256)
        ws = torch.empty(n, dtype=torch.uint8, device=dY.device)
    _need(ws, "ws", torch.uint8)
    _check(lib().dqt_bitlinear_bwd_dw_update(
        _ptr(dY), _ptr(Xq), _ptr(s_x), _ptr(W), float(s_w), _ptr(m), _ptr(v),
        C.byref(hp) if hp is not None else None, C.byref(sr) if sr is not None else None,
        _grid(bits_or_grid), T, N, K, _ptr(dW_out), _ptr(changed_out), _ptr(ws), ws.numel(),
        _stream(stream)), "dqt_bitlinear_bwd_dw_update")
    return W


def dqt_bitlinear_bwd_dw_update_img(dY, Xdq, W, s_w, m, v, hp, sr, bits_or_grid, dW_out=None,
                                    changed_out=None, ws=None, stream=None, W_img_next=None,
                                    W8_next=None):
    """Fused dW GEMM + AdamW + stochastic rounding on the X_tilde image Xdq;
    W, m, v updated in place.  With W = m = v = None only dW_out is computed.
    `ws`: split-T workspace (uint8 CUDA tensor of dqt_bwd_dw_img_workspace_size
    bytes); None allocates it when the shape benefits, False forces the single
    fused kernel.  W_img_next (bf16 [N, K]) and W8_next (uint8, E4M3: [N, K],
    or the split image [N, 2K] for grids beyond 16 in magnitude) receive the
    images of the updated codes (not images this step still reads)."""
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xdq, "Xdq", torch.bfloat16)
    K = Xdq.shape[1]
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _opt(W, "W", torch.int8, (N, K))
    _opt(m, "m", torch.float32, (N, K))
    _opt(v, "v", torch.float32, (N, K))
    _opt(dW_out, "dW_out", torch.float32, (N, K))
    _opt(W_img_next, "W_img_next", torch.bfloat16, (N, K))
    _opt(W8_next, "W8_next", torch.uint8, (N, 2 * K if fp8_split_grid(bits_or_grid) else K))
    _opt(changed_out, "changed_out", torch.int64, (1,))
    ws, nws = _dw_workspace(T, N, K, dY.device, ws)
    _check(lib().dqt_bitlinear_bwd_dw_update_img(
        _ptr(dY), _ptr(Xdq), _ptr(W), float(s_w), _ptr(m), _ptr(v),
        C.byref(hp) if hp is not None else None, C.byref(sr) if sr is not None else None,
        _grid(bits_or_grid), T, N, K, _ptr(dW_out), _ptr(W_img_next), _ptr(W8_next),
        _ptr(changed_out), _ptr(ws), nws, _stream(stream)), "dqt_bitlinear_bwd_dw_update_img")
    return W


def dqt_bitlinear_bwd_dw_update_img_pair(dY, Xdq, W, N0, s_w0, s_w1, m, v, hp, sr0, sr1,
                                         bits_or_grid, dW_out=None, changed_out=None, ws=None,
                                         stream=None, W_img_next=None, W8_next=None):
    """The fused dW + update of two stacked weights (rows [0, N0) of W, m, v
    and columns [0, N0) of dY the first's, with s_w0 and sr0; the rest the
    second's, with s_w1 and sr1).  `ws` as dqt_bitlinear_bwd_dw_update_img."""
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xdq, "Xdq", torch.bfloat16)
    K = Xdq.shape[1]
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _need(W, "W", torch.int8, (N, K))
    _need(m, "m", torch.float32, (N, K))
    _need(v, "v", torch.float32, (N, K))
    _opt(dW_out, "dW_out", torch.float32, (N, K))
    _opt(W_img_next, "W_img_next", torch.bfloat16, (N, K))
    _opt(W8_next, "W8_next", torch.uint8, (N, 2 * K if fp8_split_grid(bits_or_grid) else K))
    _opt(changed_out, "changed_out", torch.int64, (1,))
    ws, nws = _dw_workspace(T, N, K, dY.device, ws)
    _check(lib().dqt_bitlinear_bwd_dw_update_img_pair(
        _ptr(dY), _ptr(Xdq), _ptr(W), int(N0), float(s_w0), float(s_w1), _ptr(m), _ptr(v),
        C.byref(hp), C.byref(sr0), C.byref(sr1), _grid(bits_or_grid), T, N, K, _ptr(dW_out),
        _ptr(W_img_next), _ptr(W8_next), _ptr(changed_out), _ptr(ws), nws, _stream(stream)),
           "dqt_bitlinear_bwd_dw_update_img_pair")
    return W


def dqt_bitlinear_bwd_dw_update_group(problems, hp, bits_or_grid, stream=None):
    """Two weight-gradient + update problems over the same tokens in one
    persistent launch.  `problems`: two dicts with dY, Xdq, W, m, v, s_w0 and
    sr0, and optionally N0 (two stacked weights, with s_w1 and sr1),
    W_img_next, W8_next and changed_out, as for
    dqt_bitlinear_bwd_dw_update_img(_pair).  Results equal the two calls
    made with ws=False."""
    if len(problems) != 2:
        raise ValueError("two problems")
    arr = (dqt_dw_problem_t * 2)()
    keep = []
    T0 = None
    split = fp8_split_grid(bits_or_grid)
    for i, pr in enumerate(problems):
        dY = _need(pr["dY"], "dY", torch.bfloat16)
        T, N = dY.shape
        Xdq = _need(pr["Xdq"], "Xdq", torch.bfloat16)
        K = Xdq.shape[1]
        _need(Xdq, "Xdq", torch.bfloat16, (T, K))
        if T0 is not None and T != T0:
            raise ValueError("the problems must share T")
        T0 = T
        _need(pr["W"], "W", torch.int8, (N, K))
        _need(pr["m"], "m", torch.float32, (N, K))
        _need(pr["v"], "v", torch.float32, (N, K))
        _opt(pr.get("W_img_next"), "W_img_next", torch.bfloat16, (N, K))
        _opt(pr.get("W8_next"), "W8_next", torch.uint8, (N, 2 * K if split else K))
        _opt(pr.get("changed_out"), "changed_out", torch.int64, (1,))
        sr0, sr1 = pr["sr0"], pr.get("sr1")
        keep += [sr0, sr1]
        a = arr[i]
        a.dY, a.Xdq = dY.data_ptr(), Xdq.data_ptr()
        a.W, a.m, a.v = pr["W"].data_ptr(), pr["m"].data_ptr(), pr["v"].data_ptr()
        a.N, a.K, a.N0 = N, K, int(pr.get("N0", 0))
        a.s_w0, a.s_w1 = float(pr["s_w0"]), float(pr.get("s_w1", 0.0))
        a.sr0 = C.pointer(sr0)
        a.sr1 = C.pointer(sr1) if sr1 is not None else None
        for f in ("W_img_next", "W8_next", "changed_out"):
            t = pr.get(f)
            setattr(a, f, t.data_ptr() if t is not None else None)
    _check(lib().dqt_bitlinear_bwd_dw_update_group(arr, 2, C.byref(hp), _grid(bits_or_grid), T0,
                                                   _stream(stream)),
           "dqt_bitlinear_bwd_dw_update_group")
    del keep


def dqt_sr_update(grad, W, s_w, m, v, hp, sr, bits_or_grid, changed_out=None, stream=None):
    _need(grad, "grad", torch.float32)
    n = grad.numel()
    _need(W, "W", torch.int8)
    _need(m, "m", torch.float32)
    _need(v, "v", torch.float32)
    if W.numel() != n or m.numel() != n or v.numel() != n:
        raise ValueError("grad, W, m, v must have the same number of elements")
    _opt(changed_out, "changed_out", torch.int64, (1,))
    _check(lib().dqt_sr_update(_ptr(grad), _ptr(W), float(s_w), _ptr(m), _ptr(v), C.byref(hp),
                               C.byref(sr), _grid(bits_or_grid), n, _ptr(changed_out),
                               _stream(stream)), "dqt_sr_update")
    return W


def dqt_update_consts(hp, sr, bits_or_grid, s_w, out=None):
    """Host block of update constants (a uint8 tensor, pinned if `out` is None)."""
    n = lib().dqt_update_consts_size()
    if out is None:
        out = torch.empty(n, dtype=torch.uint8).pin_memory()
    if out.device.type != "cpu" or out.numel() < n or not out.is_contiguous():
        raise ValueError("out must be a contiguous host uint8 tensor of >= %d bytes" % n)
    _check(lib().dqt_update_consts(C.byref(hp), C.byref(sr), _grid(bits_or_grid), float(s_w),
                                   C.c_void_p(out.data_ptr()), out.numel()), "dqt_update_consts")
    return out


def dqt_bitlinear_bwd_dw_update_dev(dY, Xdq, W, m, v, consts_dev, dW_out=None, changed_out=None,
                                    ws=None, stream=None, W_img_next=None, W8_next=None):
    """As dqt_bitlinear_bwd_dw_update_img with the update constants read from
    the device block `consts_dev` (uint8 CUDA tensor) when the kernel runs."""
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xdq, "Xdq", torch.bfloat16)
    K = Xdq.shape[1]
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _need(W, "W", torch.int8, (N, K))
    _need(m, "m", torch.float32, (N, K))
    _need(v, "v", torch.float32, (N, K))
    _need(consts_dev, "consts_dev", torch.uint8)
    _opt(dW_out, "dW_out", torch.float32, (N, K))
    _opt(W_img_next, "W_img_next", torch.bfloat16, (N, K))
    _opt(W8_next, "W8_next", torch.uint8, (N, K))
    _opt(changed_out, "changed_out", torch.int64, (1,))
    ws, nws = _dw_workspace(T, N, K, dY.device, ws)
    _check(lib().dqt_bitlinear_bwd_dw_update_dev(
        _ptr(dY), _ptr(Xdq), _ptr(W), _ptr(m), _ptr(v), _ptr(consts_dev), T, N, K, _ptr(dW_out),
        _ptr(W_img_next), _ptr(W8_next), _ptr(changed_out), _ptr(ws), nws, _stream(stream)),
           "dqt_bitlinear_bwd_dw_update_dev")
    return W


def dqt_sr_update_dev(grad, W, m, v, consts_dev, changed_out=None, stream=None):
    _need(grad, "grad", torch.float32)
    n = grad.numel()
    _need(W, "W", torch.int8)
    _need(m, "m", torch.float32)
    _need(v, "v", torch.float32)
    _need(consts_dev, "consts_dev", torch.uint8)
    if W.numel() != n or m.numel() != n or v.numel() != n:
        raise ValueError("grad, W, m, v must have the same number of elements")
    _opt(changed_out, "changed_out", torch.int64, (1,))
    _check(lib().dqt_sr_update_dev(_ptr(grad), _ptr(W), _ptr(m), _ptr(v), _ptr(consts_dev), n,
                                   _ptr(changed_out), _stream(stream)), "dqt_sr_update_dev")
    return W


# --------------------------------------------------------------------------
# FP8 environment (Sec. 4.1/4.3): E4M3 bytes travel as torch.uint8 tensors.
# --------------------------------------------------------------------------
def dqt_act_quant_fp8(X, Xq8=None, s_x8=None, Xdq=None, want_xdq=True, stream=None):
    """E4M3 activations with per-token scale 448 / max(amax, 1e-5).  Returns
    (Xq8 uint8, s_x8 fp32, Xdq bf16 or None)."""
    _need(X, "X", torch.bfloat16)
    if X.dim() != 2:
        raise ValueError("X must be [T, K]")
    T, K = X.shape
    dev = X.device
    if Xq8 is None:
        Xq8 = torch.empty((T, K), dtype=torch.uint8, device=dev)
    if s_x8 is None:
        s_x8 = torch.empty(T, dtype=torch.float32, device=dev)
    if Xdq is None and want_xdq:
        Xdq = torch.empty((T, K), dtype=torch.bfloat16, device=dev)
    _need(Xq8, "Xq8", torch.uint8, (T, K))
    _need(s_x8, "s_x8", torch.float32, (T,))
    _opt(Xdq, "Xdq", torch.bfloat16, (T, K))
    _check(lib().dqt_act_quant_fp8(_ptr(X), T, K, _ptr(Xq8), _ptr(s_x8), _ptr(Xdq),
                                   _stream(stream)), "dqt_act_quant_fp8")
    return Xq8, s_x8, Xdq


def dqt_codes_to_fp8(W, bits_or_grid, W8=None, stream=None):
    _need(W, "W", torch.int8)
    if W8 is None:
        W8 = torch.empty(W.shape, dtype=torch.uint8, device=W.device)
    _need(W8, "W8", torch.uint8, W.shape)
    _check(lib().dqt_codes_to_fp8(_ptr(W), W.numel(), _grid(bits_or_grid), _ptr(W8),
                                  _stream(stream)), "dqt_codes_to_fp8")
    return W8


def dqt_codes_to_fp8_split(W, W8=None, stream=None):
    """E4M3 split image [N, 2K] of int8 codes [N, K] of any width: 16 (c >> 4)
    in the first half of each row, c & 15 in the second."""
    _need(W, "W", torch.int8)
    if W.dim() != 2:
        raise ValueError("W must be [N, K]")
    N, K = W.shape
    if W8 is None:
        W8 = torch.empty((N, 2 * K), dtype=torch.uint8, device=W.device)
    _need(W8, "W8", torch.uint8, (N, 2 * K))
    _check(lib().dqt_codes_to_fp8_split(_ptr(W), N, K, _ptr(W8), _stream(stream)),
           "dqt_codes_to_fp8_split")
    return W8


def fp8_split_grid(bits_or_grid):
    """Whether the E4M3 forward takes the split weight image [N, 2K] for this
    grid (codes beyond 16 in magnitude)."""
    g = _grid(bits_or_grid)
    return g.qmin < -16 or g.qmax > 16


def dqt_bitlinear_fwd_fp8(Xq8, s_x8, W8, s_w, bits_or_grid, Y=None, acc_out=None, stream=None):
    """The E4M3 forward; W8 [N, K] (dqt_codes_to_fp8), or [N, 2K]
    (dqt_codes_to_fp8_split) for grids beyond 16 in magnitude."""
    _need(Xq8, "Xq8", torch.uint8)
    T, K = Xq8.shape
    _need(W8, "W8", torch.uint8)
    N = W8.shape[0]
    _need(W8, "W8", torch.uint8, (N, 2 * K if fp8_split_grid(bits_or_grid) else K))
    _need(s_x8, "s_x8", torch.float32, (T,))
    if Y is None:
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=Xq8.device)
    _need(Y, "Y", torch.bfloat16, (T, N))
    _opt(acc_out, "acc_out", torch.float32, (T, N))
    _check(lib().dqt_bitlinear_fwd_fp8(_ptr(Xq8), _ptr(s_x8), _ptr(W8), float(s_w),
                                       _grid(bits_or_grid), T, K, N, _ptr(Y), _ptr(acc_out),
                                       _stream(stream)), "dqt_bitlinear_fwd_fp8")
    return Y


def dqt_bitlinear_fwd_fp8_pair(Xq8, s_x8, W8, N0, s_w0, s_w1, bits_or_grid, Y=None, acc_out=None,
                               stream=None):
    """The FP8 forward of two stacked weights: rows [0, N0) of W8 and columns
    [0, N0) of Y the first weight's (scale s_w0), the rest the second's."""
    _need(Xq8, "Xq8", torch.uint8)
    T, K = Xq8.shape
    _need(W8, "W8", torch.uint8)
    N = W8.shape[0]
    _need(W8, "W8", torch.uint8, (N, 2 * K if fp8_split_grid(bits_or_grid) else K))
    _need(s_x8, "s_x8", torch.float32, (T,))
    if Y is None:
        Y = torch.empty((T, N), dtype=torch.bfloat16, device=Xq8.device)
    _need(Y, "Y", torch.bfloat16, (T, N))
    _opt(acc_out, "acc_out", torch.float32, (T, N))
    _check(lib().dqt_bitlinear_fwd_fp8_pair(_ptr(Xq8), _ptr(s_x8), _ptr(W8), int(N0), float(s_w0),
                                            float(s_w1), _grid(bits_or_grid), T, K, N, _ptr(Y),
                                            _ptr(acc_out), _stream(stream)),
           "dqt_bitlinear_fwd_fp8_pair")
    return Y


# --------------------------------------------------------------------------
# 2-bit packed ternary codes (uint8 tensors of ceil(numel / 4) bytes)
# --------------------------------------------------------------------------
def packed_size(numel):
    return (int(numel) + 3) // 4


def dqt_pack_ternary(codes, packed=None, stream=None):
    _need(codes, "codes", torch.int8)
    n = codes.numel()
    if packed is None:
        packed = torch.empty(packed_size(n), dtype=torch.uint8, device=codes.device)
    _need(packed, "packed", torch.uint8, (packed_size(n),))
    _check(lib().dqt_pack_ternary(_ptr(codes), n, _ptr(packed), _stream(stream)),
           "dqt_pack_ternary")
    return packed


def dqt_unpack_ternary(packed, numel, codes=None, stream=None):
    _need(packed, "packed", torch.uint8, (packed_size(numel),))
    if codes is None:
        codes = torch.empty(int(numel), dtype=torch.int8, device=packed.device)
    _need(codes, "codes", torch.int8)
    if codes.numel() != numel:
        raise ValueError("codes must hold numel elements")
    _check(lib().dqt_unpack_ternary(_ptr(packed), int(numel), _ptr(codes), _stream(stream)),
           "dqt_unpack_ternary")
    return codes


def _numel(shape):
    n = 1
    for d in shape:
        n *= int(d)
    return n


def dqt_packed_to_bf16(packed, shape, W_img=None, stream=None):
    n = _numel(shape)
    _need(packed, "packed", torch.uint8, (packed_size(n),))
    if W_img is None:
        W_img = torch.empty(tuple(shape), dtype=torch.bfloat16, device=packed.device)
    _need(W_img, "W_img", torch.bfloat16, tuple(shape))
    _check(lib().dqt_packed_to_bf16(_ptr(packed), n, _ptr(W_img), _stream(stream)),
           "dqt_packed_to_bf16")
    return W_img


def dqt_packed_to_fp8(packed, shape, W8=None, stream=None):
    n = _numel(shape)
    _need(packed, "packed", torch.uint8, (packed_size(n),))
    if W8 is None:
        W8 = torch.empty(tuple(shape), dtype=torch.uint8, device=packed.device)
    _need(W8, "W8", torch.uint8, tuple(shape))
    _check(lib().dqt_packed_to_fp8(_ptr(packed), n, _ptr(W8), _stream(stream)),
           "dqt_packed_to_fp8")
    return W8


def dqt_sr_update_packed(grad, Wp, s_w, m, v, hp, sr, changed_out=None, stream=None):
    _need(grad, "grad", torch.float32)
    n = grad.numel()
    _need(Wp, "Wp", torch.uint8, (packed_size(n),))
    _need(m, "m", torch.float32)
    _need(v, "v", torch.float32)
    if m.numel() != n or v.numel() != n:
        raise ValueError("m and v must have grad's size")
    _opt(changed_out, "changed_out", torch.int64, None)
    _check(lib().dqt_sr_update_packed(_ptr(grad), _ptr(Wp), float(s_w), _ptr(m), _ptr(v),
                                      C.byref(hp), C.byref(sr), n, _ptr(changed_out),
                                      _stream(stream)), "dqt_sr_update_packed")


def dqt_bitlinear_bwd_dw_update_packed(dY, Xdq, Wp, s_w, m, v, hp, sr, dW_out=None,
                                       changed_out=None, ws=None, stream=None):
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xdq, "Xdq", torch.bfloat16)
    K = Xdq.shape[1]
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _need(Wp, "Wp", torch.uint8, (packed_size(N * K),))
    _need(m, "m", torch.float32, (N, K))
    _need(v, "v", torch.float32, (N, K))
    _opt(dW_out, "dW_out", torch.float32, (N, K))
    _opt(changed_out, "changed_out", torch.int64, None)
    ws_t, ws_n = _dw_workspace(T, N, K, dY.device, ws)
    _check(lib().dqt_bitlinear_bwd_dw_update_packed(
        _ptr(dY), _ptr(Xdq), _ptr(Wp), float(s_w), _ptr(m), _ptr(v), C.byref(hp), C.byref(sr),
        T, N, K, _ptr(dW_out), _ptr(changed_out), _ptr(ws_t), ws_n, _stream(stream)),
        "dqt_bitlinear_bwd_dw_update_packed")


# --------------------------------------------------------------------------
# Adafactor with stochastic rounding
# --------------------------------------------------------------------------
def adafactor(lr=1e-3, eps1=1e-30, eps2=1e-3, clip_d=1.0, decay_rate=-0.8, weight_decay=0.0,
              step=1, relative_step=False, scale_parameter=False, warmup_init=False):
    return dqt_adafactor_t(lr, eps1, eps2, clip_d, decay_rate, weight_decay, step,
                           int(relative_step), int(scale_parameter), int(warmup_init), 0)


def _codes_arg(W, packed, N, K):
    if packed:
        _need(W, "W", torch.uint8, (packed_size(N * K),))
    else:
        _need(W, "W", torch.int8, (N, K))


def dqt_adafactor_stats(G, W, s_w, R, C_, hp, packed=False, a_out=None, b_out=None,
                        scalars_out=None, ws=None, stream=None):
    """Returns (a [N], b [K], scalars {Rbar, step, decay, rms_u, rms_x, alpha, 0, 0}),
    all device fp32."""
    _need(G, "G", torch.float32)
    N, K = G.shape
    _codes_arg(W, packed, N, K)
    _need(R, "R", torch.float32, (N,))
    _need(C_, "C", torch.float32, (K,))
    dev = G.device
    a_out = torch.empty(N, dtype=torch.float32, device=dev) if a_out is None else a_out
    b_out = torch.empty(K, dtype=torch.float32, device=dev) if b_out is None else b_out
    if scalars_out is None:
        scalars_out = torch.zeros(8, dtype=torch.float32, device=dev)
    _need(a_out, "a_out", torch.float32, (N,))
    _need(b_out, "b_out", torch.float32, (K,))
    _need(scalars_out, "scalars_out", torch.float32, (8,))
    nb = lib().dqt_adafactor_workspace_size(N, K)
    if ws is None:
        ws = torch.empty(nb, dtype=torch.uint8, device=dev)
    _need(ws, "ws", torch.uint8)
    _check(lib().dqt_adafactor_stats(_ptr(G), _ptr(W), int(packed), float(s_w), _ptr(R),
                                     _ptr(C_), C.byref(hp), N, K, _ptr(a_out), _ptr(b_out),
                                     _ptr(scalars_out), _ptr(ws), ws.numel(), _stream(stream)),
           "dqt_adafactor_stats")
    return a_out, b_out, scalars_out


def dqt_adafactor_apply(G, W, a, b, scalars, step_t, sr, bits_or_grid, packed=False,
                        changed_out=None, stream=None):
    _need(G, "G", torch.float32)
    N, K = G.shape
    _codes_arg(W, packed, N, K)
    _need(a, "a", torch.float32, (N,))
    _need(b, "b", torch.float32, (K,))
    _need(scalars, "scalars", torch.float32)
    _opt(changed_out, "changed_out", torch.int64, None)
    _check(lib().dqt_adafactor_apply(_ptr(G), _ptr(W), int(packed), _ptr(a), _ptr(b),
                                     _ptr(scalars), int(step_t), C.byref(sr),
                                     _grid(bits_or_grid), N, K, _ptr(changed_out),
                                     _stream(stream)), "dqt_adafactor_apply")


def dqt_bwd_dw_adafactor_workspace_size(T, N, K):
    return int(lib().dqt_bwd_dw_adafactor_workspace_size(T, N, K))


def dqt_bitlinear_bwd_dw_adafactor(dY, Xdq, W, s_w, R, C_, hp, sr, bits_or_grid, packed=False,
                                   changed_out=None, ws=None, stream=None):
    _need(dY, "dY", torch.bfloat16)
    T, N = dY.shape
    _need(Xdq, "Xdq", torch.bfloat16)
    K = Xdq.shape[1]
    _need(Xdq, "Xdq", torch.bfloat16, (T, K))
    _codes_arg(W, packed, N, K)
    _need(R, "R", torch.float32, (N,))
    _need(C_, "C", torch.float32, (K,))
    _opt(changed_out, "changed_out", torch.int64, None)
    if ws is None:
        ws = torch.empty(dqt_bwd_dw_adafactor_workspace_size(T, N, K), dtype=torch.uint8,
                         device=dY.device)
    _need(ws, "ws", torch.uint8)
    _check(lib().dqt_bitlinear_bwd_dw_adafactor(
        _ptr(dY), _ptr(Xdq), _ptr(W), int(packed), float(s_w), _ptr(R), _ptr(C_), C.byref(hp),
        C.byref(sr), _grid(bits_or_grid), T, N, K, _ptr(changed_out), _ptr(ws), ws.numel(),
        _stream(stream)), "dqt_bitlinear_bwd_dw_adafactor")


# ---------------------------------------------------------------------------
# decoder support (not part of the DQT method)
# ---------------------------------------------------------------------------
def dqt_rope_bf16(x, cos_sin, inverse=False, y=None, stream=None):
    """Rotary embedding of x bf16 [B, S, H, D] (contiguous) with the (cos, sin)
    table fp32 [S, D/2, 2]; inverse rotates by -theta.  Returns y (new unless given)."""
    _need(x, "x", torch.bfloat16)
    if x.dim() != 4:
        raise ValueError("x must be [B, S, H, D]")
    B, S, H, D = x.shape
    _need(cos_sin, "cos_sin", torch.float32, (S, D // 2, 2))
    y = torch.empty_like(x) if y is None else _need(y, "y", torch.bfloat16, x.shape)
    _check(lib().dqt_rope_bf16(_ptr(x), _ptr(y), _ptr(cos_sin), B * S, S, H, D, int(bool(inverse)),
                               _stream(stream)), "dqt_rope_bf16")
    return y


def dqt_cross_entropy_fwd_bf16(logits, targets, stream=None):
    """Per-row log-sum-exp and loss of bf16 logits [M, V] against int64 targets
    [M].  Returns (lse, row_loss), fp32 [M] each."""
    _need(logits, "logits", torch.bfloat16)
    M, V = logits.shape
    _need(targets, "targets", torch.int64, (M,))
    lse = torch.empty(M, dtype=torch.float32, device=logits.device)
    row_loss = torch.empty(M, dtype=torch.float32, device=logits.device)
    _check(lib().dqt_cross_entropy_fwd_bf16(_ptr(logits), _ptr(targets), M, V, _ptr(lse),
                                            _ptr(row_loss), _stream(stream)),
           "dqt_cross_entropy_fwd_bf16")
    return lse, row_loss


def dqt_cross_entropy_bwd_bf16(logits, targets, lse, scale, dlogits=None, stream=None):
    """Gradient of the loss w.r.t. bf16 logits [M, V]: (softmax - onehot) * scale[0]
    (scale: fp32 device tensor of one element)."""
    _need(logits, "logits", torch.bfloat16)
    M, V = logits.shape
    _need(targets, "targets", torch.int64, (M,))
    _need(lse, "lse", torch.float32, (M,))
    _need(scale, "scale", torch.float32, (1,))
    dlogits = torch.empty_like(logits) if dlogits is None else \
        _need(dlogits, "dlogits", torch.bfloat16, (M, V))
    _check(lib().dqt_cross_entropy_bwd_bf16(_ptr(logits), _ptr(targets), _ptr(lse), _ptr(scale), M,
                                            V, _ptr(dlogits), _stream(stream)),
           "dqt_cross_entropy_bwd_bf16")
    return dlogits


def dqt_swiglu_bf16(g, u, h=None, stream=None):
    """h = silu(g) * u (fp32 inside, one bf16 rounding); g, u contiguous bf16 of one shape."""
    _need(g, "g", torch.bfloat16)
    _need(u, "u", torch.bfloat16, g.shape)
    h = torch.empty_like(g) if h is None else _need(h, "h", torch.bfloat16, g.shape)
    _check(lib().dqt_swiglu_bf16(_ptr(g), _ptr(u), _ptr(h), g.numel(), _stream(stream)),
           "dqt_swiglu_bf16")
    return h


def dqt_swiglu_bwd_bf16(g, u, dh, stream=None):
    """(dg, du) of h = silu(g) * u for the upstream gradient dh."""
    _need(g, "g", torch.bfloat16)
    _need(u, "u", torch.bfloat16, g.shape)
    _need(dh, "dh", torch.bfloat16, g.shape)
    dg, du = torch.empty_like(g), torch.empty_like(g)
    _check(lib().dqt_swiglu_bwd_bf16(_ptr(g), _ptr(u), _ptr(dh), _ptr(dg), _ptr(du), g.numel(),
                                     _stream(stream)), "dqt_swiglu_bwd_bf16")
    return dg, du


def dqt_rmsnorm_bf16(x, w, eps, stream=None):
    """RMSNorm of x bf16 [rows, D] with gain w bf16 [D].  Returns (y, rstd)."""
    _need(x, "x", torch.bfloat16)
    rows, D = x.shape
    _need(w, "w", torch.bfloat16, (D,))
    y = torch.empty_like(x)
    rstd = torch.empty(rows, dtype=torch.float32, device=x.device)
    _check(lib().dqt_rmsnorm_bf16(_ptr(x), _ptr(w), float(eps), rows, D, _ptr(y), _ptr(rstd),
                                  _stream(stream)), "dqt_rmsnorm_bf16")
    return y, rstd


def dqt_rmsnorm_bwd_bf16(x, w, rstd, dy, stream=None):
    """(dx, dw) of the RMSNorm above for the upstream gradient dy [rows, D]."""
    _need(x, "x", torch.bfloat16)
    rows, D = x.shape
    _need(w, "w", torch.bfloat16, (D,))
    _need(rstd, "rstd", torch.float32, (rows,))
    _need(dy, "dy", torch.bfloat16, (rows, D))
    dx = torch.empty_like(x)
    dw = torch.empty_like(w)
    nws = lib().dqt_rmsnorm_bwd_workspace_size(rows, D)
    ws = torch.empty(max(nws, 16), dtype=torch.uint8, device=x.device)
    _check(lib().dqt_rmsnorm_bwd_bf16(_ptr(x), _ptr(w), _ptr(rstd), _ptr(dy), rows, D, _ptr(dx),
                                      _ptr(dw), _ptr(ws), nws, _stream(stream)),
           "dqt_rmsnorm_bwd_bf16")
    return dx, dw
