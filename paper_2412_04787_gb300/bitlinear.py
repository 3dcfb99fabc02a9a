"""DQT BitLinear as a torch module (argument marshalling over the C ABI).

A ``DQTBitLinear`` layer holds only what DQT keeps (Sec. 3.2): the n-bit
integer codes of its weight (int8), the per-tensor scale s_w fixed at
initialisation (Eq. 2-4), and AdamW's two moments (Sec. 4.1).  There is no
high-precision weight and no weight gradient tensor:

* forward: 8-bit per-token activation codes (``dqt_act_quant``), the exact
  bf16 image of the weight codes (``dqt_codes_to_bf16``) and the integer GEMM
  (``dqt_bitlinear_fwd``);
* backward: dX through W_tilde (``dqt_bitlinear_bwd_dx``), then the weight
  gradient is reduced on the tensor cores and consumed in the same kernel by
  the AdamW step and stochastic rounding onto the grid
  (``dqt_bitlinear_bwd_dw_update``, Eq. 1 and Eq. 5): the layer is updated
  during its own backward.

With ``act="fp8"`` (the FP8 environment of Sec. 4.3) the forward quantises
activations to E4M3 bytes (``dqt_act_quant_fp8``), converts the codes to their
exact E4M3 image (``dqt_codes_to_fp8``, grids up to 5 bits) and runs the GEMM
on the 8-bit floating-point tensor cores (``dqt_bitlinear_fwd_fp8``); the
backward is the same.

``optimizer="adafactor"`` replaces AdamW's two fp32 moments by Adafactor's
factored row and column statistics (Sec. 4.3), and ``packed=True`` keeps
ternary codes 2 bits each (Sec. 1); the two together leave 0.25 byte of
state per weight plus N + K floats.

Consequences: one backward per forward (no gradient accumulation across
micro-batches, no weight sharing between calls), and ``optimizer.step()`` is
not needed for these layers.  The state is ordinary module buffers, so
``state_dict()`` checkpoints it (codes, m, v as buffers; s_w, step, seed and
tensor id as extra state).
"""
import weakref

import torch

from . import dqt

__all__ = ["DQTBitLinear"]


# Sibling layers that read the same activation (q, k and v; gate and up)
# share its quantisation: the last input quantised is remembered by object
# identity and version counter, so a new or modified tensor is never mistaken
# for it (a freed tensor's memory reused by a new one is a different object).
class _QuantCache:
    ref = None
    version = -1
    act = None
    result = None


def _quantised(x, x2, act):
    c = _QuantCache
    try:
        version = x._version
    except RuntimeError:  # inference tensors keep no version counter: no sharing
        version = None
    if (version is not None and c.ref is not None and c.ref() is x and c.version == version
            and c.act == act):
        return c.result
    if act == "fp8":
        res = dqt.dqt_act_quant_fp8(x2)
    else:
        res = dqt.dqt_act_quant_images(x2, want=("Xq_img", "Xdq"))
    if version is not None:
        c.ref, c.version, c.act, c.result = weakref.ref(x), version, act, res
    else:
        c.ref, c.result = None, None
    return res


class _BitLinearFn(torch.autograd.Function):
    @staticmethod
    def forward(ctx, x, anchor, layer):
        K, N = layer.in_features, layer.out_features
        x2 = x.reshape(-1, K)
        if x2.dtype != torch.bfloat16:
            x2 = x2.to(torch.bfloat16)
        x2 = x2.contiguous()
        if layer.act == "fp8":
            q8, s_x, xdq = _quantised(x, x2, "fp8")
            y = dqt.dqt_bitlinear_fwd_fp8(q8, s_x, layer.image_fp8(), float(layer.s_w),
                                          layer.grid_tuple)
            w_img = None  # dX needs the bf16 image: taken in backward
        else:
            _, s_x, q_img, xdq = _quantised(x, x2, "int8")
            # the weight's code image serves the forward and, kept until the
            # backward, dX (the codes change only after dX, in the update)
            w_img = layer.image_bf16()
            y = dqt.dqt_bitlinear_fwd_img(q_img, s_x, w_img, float(layer.s_w), layer.grid_tuple)
        ctx.save_for_backward(xdq, w_img)
        ctx.layer = layer
        ctx.in_shape = x.shape
        ctx.in_dtype = x.dtype
        return y.reshape(*x.shape[:-1], N)

    @staticmethod
    def backward(ctx, dy):
        xdq, w_img = ctx.saved_tensors
        layer = ctx.layer
        N = layer.out_features
        dy2 = dy.reshape(-1, N)
        if dy2.dtype != torch.bfloat16:
            dy2 = dy2.to(torch.bfloat16)
        dy2 = dy2.contiguous()
        # the codes have not changed since the forward
        if w_img is None:
            w_img = layer.image_bf16()
        dx = dqt.dqt_bitlinear_bwd_dx_img(dy2, w_img, float(layer.s_w))
        if layer.update_in_backward:
            layer._dqt_update(dy2, xdq)
        return dx.reshape(ctx.in_shape).to(ctx.in_dtype), None, None


class DQTBitLinear(torch.nn.Module):
    """y = X_tilde W_tilde^T with W_tilde = codes / s_w, trained by DQT.

    bits: 1.58 (ternary) or an integer width 2..8 (Eq. 3).  The dense initial
    weight is drawn N(0, init_std) from ``init_seed`` and quantised once with
    AbsMean (Eq. 2-4) on the device.  ``lr``, ``betas``, ``eps`` and
    ``weight_decay`` are AdamW's; ``seed`` and ``tensor_id`` key the Philox
    stream of stochastic rounding (``round_mode`` 1 = round to nearest, the
    Sec. 5.1 ablation).  ``act`` is "int8" (8-bit integer activation codes,
    exact integer forward) or "fp8" (E4M3 activations and weight image).
    ``optimizer`` is "adamw" or "adafactor" (``adafactor`` holds its other
    hyper-parameters as a dict for ``dqt.adafactor``); ``packed`` stores
    ternary codes 2 bits each.
    """

    def __init__(self, in_features, out_features, bits=1.58, lr=1e-3, betas=(0.9, 0.999),
                 eps=1e-8, weight_decay=0.0, seed=1234, tensor_id=0, init_std=0.02,
                 init_seed=0, round_mode=0, act="int8", optimizer="adamw", packed=False,
                 adafactor=None, device="cuda"):
        super().__init__()
        if in_features % 8 or out_features % 8:
            raise ValueError("in_features and out_features must be multiples of 8")
        if act not in ("int8", "fp8"):
            raise ValueError("act must be 'int8' or 'fp8'")
        if act == "fp8" and in_features % 16:
            raise ValueError("the E4M3 forward needs in_features a multiple of 16")
        self.act = act
        if optimizer not in ("adamw", "adafactor"):
            raise ValueError("optimizer must be 'adamw' or 'adafactor'")
        self.optimizer = optimizer
        self.packed = bool(packed)
        self.adafactor = dict(adafactor or {})
        self.in_features = in_features
        self.out_features = out_features
        g = dqt.grid(bits)
        self.grid_tuple = (g.qmin, g.qmax)
        # E4M3 weight image: the codes themselves up to 16 in magnitude (<= 5
        # bits), else the split image [N, 2K] of 16 (c >> 4) and c & 15
        self.w8_split = act == "fp8" and (g.qmin < -16 or g.qmax > 16)
        if self.w8_split and in_features % 128:
            raise ValueError("the split E4M3 forward (6- to 8-bit codes) needs in_features a "
                             "multiple of 128")
        if self.packed and (g.qmin, g.qmax) != (-1, 1):
            raise ValueError("packed storage holds ternary codes only")
        self.lr, self.betas, self.eps, self.weight_decay = lr, tuple(betas), eps, weight_decay
        self.round_mode = round_mode
        self.update_in_backward = True
        gen = torch.Generator(device="cpu")
        gen.manual_seed(int(init_seed))
        w0 = (torch.randn(out_features, in_features, generator=gen) * init_std).to(device)
        codes, s_w = dqt.dqt_absmean_init(w0, self.grid_tuple)
        del w0
        if self.packed:
            codes = dqt.dqt_pack_ternary(codes)
        self.register_buffer("codes", codes)
        if optimizer == "adamw":
            self.register_buffer("m", torch.zeros(out_features, in_features, device=device))
            self.register_buffer("v", torch.zeros(out_features, in_features, device=device))
        else:
            # Adafactor's factored second moment: row and column means
            self.register_buffer("R", torch.zeros(out_features, device=device))
            self.register_buffer("C", torch.zeros(in_features, device=device))
        # changed-code counter (Sec. 5.2 update frequency), accumulated
        self.register_buffer("changed", torch.zeros(1, dtype=torch.int64, device=device))
        self.s_w = float(s_w)
        self.step = 0
        self.seed = int(seed)
        self.tensor_id = int(tensor_id)
        # device-resident update constants (CUDA-graph replay), see prepare_step
        self.uc_dev = None
        # the codes' bf16 (and, with act="fp8", E4M3) operand images, kept
        # from step to step: the AdamW update on int8 codes rewrites them with
        # the codes it writes, after this step's dX has read them (one stream:
        # the update is ordered after dX), so no step converts the codes;
        # they are rebuilt when the codes' version counter says the codes
        # were changed from outside (copy_, load_state_dict)
        self._img = self._img8 = None
        self._img_version = self._img8_version = -1
        # anchor: a 0-element tensor that requires grad, so the layer's
        # backward (and with it the DQT update) runs even if x does not
        self._anchor = torch.nn.Parameter(torch.zeros(0, device=device), requires_grad=True)

    # host scalars of the DQT state travel in state_dict as extra state
    def get_extra_state(self):
        return {"s_w": self.s_w, "step": self.step, "seed": self.seed, "tensor_id": self.tensor_id}

    def set_extra_state(self, state):
        self.s_w = float(state["s_w"])
        self.step = int(state["step"])
        self.seed = int(state["seed"])
        self.tensor_id = int(state["tensor_id"])

    def forward(self, x):
        return _BitLinearFn.apply(x, self._anchor, self)

    def int8_codes(self):
        """The codes as an int8 [N, K] tensor (unpacked if stored packed)."""
        if not self.packed:
            return self.codes
        n = self.out_features * self.in_features
        return dqt.dqt_unpack_ternary(self.codes, n).view(self.out_features, self.in_features)

    def weight_bf16(self):
        shape = (self.out_features, self.in_features)
        if self.packed:
            return dqt.dqt_packed_to_bf16(self.codes, shape)
        return dqt.dqt_codes_to_bf16(self.codes)

    def weight_fp8(self):
        shape = (self.out_features, self.in_features)
        if self.packed:
            return dqt.dqt_packed_to_fp8(self.codes, shape)
        if self.w8_split:
            return dqt.dqt_codes_to_fp8_split(self.codes)
        return dqt.dqt_codes_to_fp8(self.codes, self.grid_tuple)

    def _images_kept(self):
        # the updates that write the images: AdamW on int8 codes
        return self.optimizer == "adamw" and not self.packed

    def image_bf16(self):
        """The bf16 image of the current codes (the forward's and dX's
        operand); kept from step to step where the update rewrites it."""
        if not self._images_kept():
            return self.weight_bf16()
        if self._img is None:
            self._img = torch.empty((self.out_features, self.in_features), dtype=torch.bfloat16,
                                    device=self.codes.device)
            self._img_version = -1
        if self._img_version != self.codes._version:
            dqt.dqt_codes_to_bf16(self.codes, self._img)
            self._img_version = self.codes._version
        return self._img

    def image_fp8(self):
        """The E4M3 image of the current codes (the FP8 forward's operand),
        kept like image_bf16."""
        if not self._images_kept():
            return self.weight_fp8()
        if self._img8 is None:
            self._img8 = torch.empty((self.out_features,
                                      self.in_features * (2 if self.w8_split else 1)),
                                     dtype=torch.uint8, device=self.codes.device)
            self._img8_version = -1
        if self._img8_version != self.codes._version:
            if self.w8_split:
                dqt.dqt_codes_to_fp8_split(self.codes, self._img8)
            else:
                dqt.dqt_codes_to_fp8(self.codes, self.grid_tuple, self._img8)
            self._img8_version = self.codes._version
        return self._img8

    def _next_images(self):
        # the kept images that are current: the update writes the images of
        # the codes it writes into them (an image not current stays stale and
        # is rebuilt when next used)
        v = self.codes._version
        img = self._img if self._img is not None and self._img_version == v else None
        img8 = self._img8 if self._img8 is not None and self._img8_version == v else None
        if img8 is not None and self.w8_split and self.uc_dev is not None:
            # with the constants in device memory the update cannot tell the
            # grid, and writes the plain E4M3 image only: the split one is
            # rebuilt from the new codes at the next forward
            img8 = None
            self._img8_version = -1
        return img, img8

    def _hyper(self, step):
        hp = dqt.adamw(lr=self.lr, beta1=self.betas[0], beta2=self.betas[1], eps=self.eps,
                       weight_decay=self.weight_decay, step=step)
        sr = dqt.sr_stream(seed=self.seed, tensor_id=self.tensor_id, round_mode=self.round_mode)
        return hp, sr

    def use_device_consts(self, dev_row):
        """Read the update constants from `dev_row` (a 16-byte aligned row of a device
        block) when the update kernel runs.  The step then advances in
        prepare_step(), not in backward, so that a captured training step
        replays with a new step each time (AdamW, int8 codes)."""
        if self.optimizer != "adamw" or self.packed:
            raise ValueError("device-resident update constants need AdamW on int8 codes")
        self.uc_dev = dev_row

    def prepare_step(self, host_row):
        """Advance the step and write its update constants into `host_row`."""
        self.step += 1
        hp, sr = self._hyper(self.step)
        dqt.dqt_update_consts(hp, sr, self.grid_tuple, self.s_w, out=host_row)

    def _dqt_update(self, dy2, xdq):
        if self.optimizer == "adafactor":
            self.step += 1
            hp = dqt.adafactor(lr=self.lr, weight_decay=self.weight_decay, step=self.step,
                               **self.adafactor)
            sr = dqt.sr_stream(seed=self.seed, tensor_id=self.tensor_id,
                               round_mode=self.round_mode)
            dqt.dqt_bitlinear_bwd_dw_adafactor(dy2, xdq, self.codes, self.s_w, self.R, self.C, hp,
                                               sr, self.grid_tuple, packed=self.packed,
                                               changed_out=self.changed)
            return
        if self.packed:
            self.step += 1
            hp, sr = self._hyper(self.step)
            dqt.dqt_bitlinear_bwd_dw_update_packed(dy2, xdq, self.codes, self.s_w, self.m, self.v,
                                                   hp, sr, changed_out=self.changed)
            return
        img, img8 = self._next_images()
        if self.uc_dev is not None:
            dqt.dqt_bitlinear_bwd_dw_update_dev(dy2, xdq, self.codes, self.m, self.v, self.uc_dev,
                                                changed_out=self.changed, W_img_next=img,
                                                W8_next=img8)
            return
        self.step += 1
        hp, sr = self._hyper(self.step)
        dqt.dqt_bitlinear_bwd_dw_update_img(dy2, xdq, self.codes, self.s_w, self.m, self.v, hp, sr,
                                            self.grid_tuple, changed_out=self.changed,
                                            W_img_next=img, W8_next=img8)

    def extra_repr(self):
        return "in_features=%d, out_features=%d, grid=%s, act=%s, optimizer=%s, packed=%s" % (
            self.in_features, self.out_features, self.grid_tuple, self.act, self.optimizer,
            self.packed)
