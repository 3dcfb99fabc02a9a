"""LLaMA-structured decoder whose linear layers are DQT BitLinear layers.

The paper trains LLaMA-2-structured models (Sec. 4.1) with every weight
matrix of the transformer blocks kept at n bits and updated by stochastic
rounding (Sec. 3.2, Eq. 5).  Here q, k, v, o, gate, up and down are
``DQTBitLinear`` layers running on this library's kernels (``act="fp8"``:
the FP8-environment forward of Sec. 4.3); the token
embedding, the RMSNorm gains and the output head stay in bf16 and are trained
by an ordinary optimiser (which weights the paper keeps in high precision is
not stated; this is the BitNet convention).  Causal attention
(``scaled_dot_product_attention``) is a PyTorch operation around the BitLinear
hot path; RMSNorm, the rotary position embedding, the SwiGLU gate and the
token cross-entropy run on this library's decoder-support kernels (one bf16
pass each way with fp32 arithmetic, no fp32 copies of q, k or the logits).

A training step is ``loss = model(ids, targets); loss.backward();
opt.step(); opt.zero_grad()``: each BitLinear applies its DQT update during
its own backward, the optimiser only sees the bf16 parameters
(``model.dense_parameters()``).  For CUDA-graph replay of whole steps,
``enable_graph_updates()`` moves the per-step update constants to device
memory (``prepare_step(slot)`` on the host, ``upload_update_consts(slot)``
stream-ordered before each replay).
"""

import torch
import torch.nn.functional as F
from torch.nn.attention import SDPBackend, sdpa_kernel

from . import dqt
from .bitlinear import DQTBitLinear

# Attention runs on PyTorch's FlashAttention kernels (memory-efficient
# attention where FlashAttention does not apply), never on cuDNN's fused
# attention: a CUDA-graph replay of this decoder raised an illegal memory
# access with the cuDNN backend selected, and a PyTorch default that changes
# between versions must not route back onto it.
_SDPA_BACKENDS = [SDPBackend.FLASH_ATTENTION, SDPBackend.EFFICIENT_ATTENTION]

__all__ = ["DecoderConfig", "DQTDecoder"]


class DecoderConfig:
    def __init__(self, layers=12, hidden=768, heads=12, ffn=2048, vocab=32000, bits=1.58,
                 lr=1e-3, seed=1234, rope_theta=10000.0, norm_eps=1e-6, act="int8",
                 optimizer="adamw", packed=False):
        self.layers, self.hidden, self.heads, self.ffn, self.vocab = layers, hidden, heads, ffn, vocab
        self.bits, self.lr, self.seed, self.act = bits, lr, seed, act
        self.optimizer, self.packed = optimizer, packed
        self.rope_theta, self.norm_eps = rope_theta, norm_eps


class RMSNorm(torch.nn.Module):
    def __init__(self, dim, eps, device):
        super().__init__()
        self.eps = eps
        self.weight = torch.nn.Parameter(torch.ones(dim, device=device, dtype=torch.bfloat16))

    def forward(self, x):
        D = x.shape[-1]
        if D % 8 == 0 and D <= 2048:
            return _RMSNorm.apply(x, self.weight, self.eps)
        # wider rows: PyTorch's fused RMSNorm (statistics in fp32)
        return F.rms_norm(x, (D,), self.weight, self.eps)


class _RMSNorm(torch.autograd.Function):
    """RMSNorm of bf16 rows (statistics and products in fp32) on the library's
    kernels: one pass forward; backward one pass for dx plus a fixed-order
    column reduction for the gain gradient."""

    @staticmethod
    def forward(ctx, x, w, eps):
        x2 = x.reshape(-1, x.shape[-1]).contiguous()
        y, rstd = dqt.dqt_rmsnorm_bf16(x2, w, eps)
        ctx.save_for_backward(x2, w, rstd)
        return y.view(x.shape)

    @staticmethod
    def backward(ctx, dy):
        x2, w, rstd = ctx.saved_tensors
        dx, dw = dqt.dqt_rmsnorm_bwd_bf16(x2, w, rstd, dy.reshape(x2.shape).contiguous())
        return dx.view(dy.shape), dw, None


class _Rope(torch.autograd.Function):
    """Rotary position embedding (LLaMA form: interleaved pairs (x[2i], x[2i+1])
    of each head times exp(i theta)) of x bf16 [B, S, H, D]; cos_sin fp32
    [S, D/2, 2].  The backward rotates the gradient by -theta (the transpose)."""

    @staticmethod
    def forward(ctx, x, cos_sin):
        ctx.save_for_backward(cos_sin)
        return dqt.dqt_rope_bf16(x.contiguous(), cos_sin)

    @staticmethod
    def backward(ctx, g):
        (cos_sin,) = ctx.saved_tensors
        return dqt.dqt_rope_bf16(g.contiguous(), cos_sin, inverse=True), None


class _SwiGLU(torch.autograd.Function):
    """h = silu(g) * u of two bf16 tensors of one shape, in one pass each way."""

    @staticmethod
    def forward(ctx, g, u):
        g, u = g.contiguous(), u.contiguous()
        ctx.save_for_backward(g, u)
        return dqt.dqt_swiglu_bf16(g, u)

    @staticmethod
    def backward(ctx, dh):
        g, u = ctx.saved_tensors
        return dqt.dqt_swiglu_bwd_bf16(g, u, dh.contiguous())


class _TokenCrossEntropy(torch.autograd.Function):
    """Mean token cross-entropy of bf16 logits [M, V] (log-sum-exp in fp32)
    over the rows whose target lies in [0, V); the gradient is written in bf16."""

    @staticmethod
    def forward(ctx, logits, targets):
        lse, row_loss = dqt.dqt_cross_entropy_fwd_bf16(logits, targets)
        n = ((targets >= 0) & (targets < logits.shape[1])).sum().to(torch.float32)
        ctx.save_for_backward(logits, targets, lse, n)
        return row_loss.sum() / n

    @staticmethod
    def backward(ctx, g):
        logits, targets, lse, n = ctx.saved_tensors
        scale = (g.to(torch.float32) / n).reshape(1)
        return dqt.dqt_cross_entropy_bwd_bf16(logits, targets, lse, scale), None


class Block(torch.nn.Module):
    def __init__(self, cfg, index, device):
        super().__init__()
        h, f = cfg.hidden, cfg.ffn
        self.heads = cfg.heads
        self.attn_norm = RMSNorm(h, cfg.norm_eps, device)
        self.mlp_norm = RMSNorm(h, cfg.norm_eps, device)

        def bl(k, n, j):
            tid = index * 8 + j  # distinct Philox stream and initial draw per weight
            return DQTBitLinear(k, n, bits=cfg.bits, lr=cfg.lr, seed=cfg.seed, tensor_id=tid,
                                init_seed=cfg.seed * 1000 + tid, act=cfg.act,
                                optimizer=cfg.optimizer, packed=cfg.packed, device=device)

        self.q, self.k, self.v, self.o = bl(h, h, 0), bl(h, h, 1), bl(h, h, 2), bl(h, h, 3)
        self.gate, self.up, self.down = bl(h, f, 4), bl(h, f, 5), bl(f, h, 6)

    def forward(self, x, cos_sin):
        B, S, Hd = x.shape
        nh = self.heads
        hd = Hd // nh
        a = self.attn_norm(x)
        # rotary embedding in the [B, S, H, D] layout the projections produce
        # (cos_sin: [S, D/2, 2]); attention reads head-major views of it, so
        # no layout copy is made in either direction
        q = _Rope.apply(self.q(a).view(B, S, nh, hd), cos_sin).transpose(1, 2)
        k = _Rope.apply(self.k(a).view(B, S, nh, hd), cos_sin).transpose(1, 2)
        v = self.v(a).view(B, S, nh, hd).transpose(1, 2)
        with sdpa_kernel(_SDPA_BACKENDS):
            o = F.scaled_dot_product_attention(q, k, v, is_causal=True)
        x = x + self.o(o.transpose(1, 2).reshape(B, S, Hd))
        m = self.mlp_norm(x)
        return x + self.down(_SwiGLU.apply(self.gate(m), self.up(m)))


class DQTDecoder(torch.nn.Module):
    def __init__(self, cfg, device="cuda"):
        super().__init__()
        self.cfg = cfg
        g = torch.Generator(device="cpu")
        g.manual_seed(cfg.seed)
        emb = torch.randn(cfg.vocab, cfg.hidden, generator=g) * 0.02
        head = torch.randn(cfg.vocab, cfg.hidden, generator=g) * 0.02
        self.embed = torch.nn.Parameter(emb.to(device=device, dtype=torch.bfloat16))
        self.blocks = torch.nn.ModuleList([Block(cfg, i, device) for i in range(cfg.layers)])
        self.norm = RMSNorm(cfg.hidden, cfg.norm_eps, device)
        self.head = torch.nn.Parameter(head.to(device=device, dtype=torch.bfloat16))
        hd = cfg.hidden // cfg.heads
        self.register_buffer("inv_freq", 1.0 / (cfg.rope_theta ** (torch.arange(0, hd, 2, device=device,
                                                                                  dtype=torch.float32) / hd)),
                             persistent=False)

    def bitlinear_layers(self):
        return [m for m in self.modules() if isinstance(m, DQTBitLinear)]

    # ---- CUDA-graph replay of whole training steps ----
    def enable_graph_updates(self):
        """Move the per-step update constants of every BitLinear to one device
        block (one row per layer, dqt_update_consts_size() bytes rounded up to a
        multiple of 64) fed from two pinned host blocks.  Per step:
        prepare_step(slot) fills host block `slot` on the host, then
        upload_update_consts(slot) copies it, stream-ordered, ahead of the
        step's kernels (e.g. right before replaying a captured step).  Alternate
        the slots so the host never rewrites a block a pending copy reads."""
        from . import dqt
        layers = self.bitlinear_layers()
        row = (dqt.lib().dqt_update_consts_size() + 63) // 64 * 64
        dev = layers[0].codes.device
        self._uc_host = torch.zeros((2, len(layers), row), dtype=torch.uint8).pin_memory()
        self._uc_dev = torch.zeros((len(layers), row), dtype=torch.uint8, device=dev)
        self._uc_copied = [None, None]
        for i, layer in enumerate(layers):
            layer.use_device_consts(self._uc_dev[i])

    def prepare_step(self, slot=0):
        ev = self._uc_copied[slot]
        if ev is not None:
            ev.synchronize()  # the copy that last read this host block is done
        for i, layer in enumerate(self.bitlinear_layers()):
            layer.prepare_step(self._uc_host[slot, i])

    def upload_update_consts(self, slot=0):
        self._uc_dev.copy_(self._uc_host[slot], non_blocking=True)
        ev = torch.cuda.Event()
        ev.record()
        self._uc_copied[slot] = ev

    def dense_parameters(self):
        """The bf16 parameters an ordinary optimiser trains (not the BitLinear codes)."""
        return [p for n, p in self.named_parameters() if not n.endswith("_anchor")]

    def forward(self, ids, targets=None):
        B, S = ids.shape
        x = F.embedding(ids, self.embed)
        t = torch.arange(S, device=ids.device, dtype=torch.float32)
        ang = torch.outer(t, self.inv_freq)
        cos_sin = torch.stack((torch.cos(ang), torch.sin(ang)), dim=-1)  # [S, D/2, 2]
        for blk in self.blocks:
            x = blk(x, cos_sin)
        x = self.norm(x)
        logits = x @ self.head.t()
        if targets is None:
            return logits
        return _TokenCrossEntropy.apply(logits.view(-1, logits.shape[-1]),
                                        targets.reshape(-1).to(torch.int64).contiguous())

    def bitlinear_flops_per_step(self, tokens):
        """Forward + dX + dW FLOPs of all BitLinear layers for `tokens` tokens."""
        return sum(6.0 * tokens * m.in_features * m.out_features for m in self.bitlinear_layers())
