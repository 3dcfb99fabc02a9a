"""Data-parallel DQT weight update across ranks (one process per GPU).

The paper trains its DQT models on 4 to 16 GPUs (Sec. 4.1, Hardware).  In
data parallelism every rank computes the forward, dX and the fp32 weight
gradient of its own micro-batch; the ranks then need one update of the
shared low-bit weight.  DQT keeps no high-precision master weight (Sec. 3.2),
so the exchange is:

1. reduce-scatter of the fp32 weight gradient over a flat partition of the
   weight: rank r receives the summed gradient of its shard [lo_r, hi_r);
2. the AdamW + stochastic-rounding update (Sec. 4.1, Eq. 1, Eq. 5) of that
   shard on that rank, ZeRO-1 style: a rank holds the AdamW moments of its
   shard only;
3. all-gather of the int8 codes: one byte per weight comes back, a quarter
   of what an fp32 master-weight all-gather moves.

Element e of the weight draws the Philox uniform of its global index e
(``dqt_sr_t.elem0`` = lo_r for the shard), so the codes after the exchange do
not depend on the number of ranks: N ranks give the codes of the one-rank
update of the summed gradient, bit for bit.

The gradient is summed over ranks (a mean loss is the caller's upstream
scaling).  The partition pads the weight to a multiple of ``world_size`` x
``align`` elements (``align`` 16: every shard starts 16-byte aligned for the
int8 codes and 64-byte aligned for the fp32 state); the padding is never
updated.
"""
import torch
import torch.distributed as dist


class ShardPlan:
    """Flat partition of a weight of `numel` elements over `world_size` ranks."""

    def __init__(self, numel, world_size, rank, align=16):
        if numel <= 0 or world_size <= 0 or not 0 <= rank < world_size or align % 4:
            raise ValueError("bad shard plan arguments")
        per = -(-numel // world_size)
        self.numel = numel
        self.world_size = world_size
        self.rank = rank
        self.shard = -(-per // align) * align
        self.padded = self.shard * world_size
        # a rank past the end of a small weight owns an empty shard
        self.lo, self.hi = self.bounds(rank)
        self.n_local = self.hi - self.lo

    def bounds(self, r):
        lo = r * self.shard
        return lo, max(lo, min(lo + self.shard, self.numel))


def _dqt_update(grad, W, s_w, m, v, hp, sr, grid, changed_out):
    from . import dqt
    return dqt.dqt_sr_update(grad, W, s_w, m, v, hp, sr, grid, changed_out=changed_out)


class DataParallelUpdater:
    """The exchange of one DQT weight tensor.

    Buffers (on the device of `codes`):
      grad_full   fp32 [padded]  the rank's local weight gradient; the GEMM
                                 writes its first `numel` entries
                                 (``grad_view()``), the padding stays 0
      grad_shard  fp32 [shard]   the reduce-scatter result
      m, v        fp32 [shard]   AdamW moments of this rank's shard (ZeRO-1)
      codes_shard int8 [shard]   this rank's authoritative codes
      codes_full  int8 [padded]  every rank's codes after the all-gather; its
                                 first `numel` entries are the weight

    `update_fn(grad, W, s_w, m, v, hp, sr, grid, changed_out)` applies the
    update to one flat shard; the default is the library's dqt_sr_update.
    """

    def __init__(self, codes, group=None, update_fn=None, align=16):
        self.group = group
        ws = dist.get_world_size(group)
        rk = dist.get_rank(group)
        self.shape = tuple(codes.shape)
        self.plan = ShardPlan(codes.numel(), ws, rk, align)
        p = self.plan
        dev = codes.device
        self.grad_full = torch.zeros(p.padded, dtype=torch.float32, device=dev)
        self.grad_shard = torch.zeros(p.shard, dtype=torch.float32, device=dev)
        self.m = torch.zeros(p.shard, dtype=torch.float32, device=dev)
        self.v = torch.zeros(p.shard, dtype=torch.float32, device=dev)
        self.codes_full = torch.zeros(p.padded, dtype=torch.int8, device=dev)
        self.codes_full[: p.numel].copy_(codes.reshape(-1))
        self.codes_shard = self.codes_full[p.lo: p.lo + p.shard].clone()
        self.update_fn = update_fn or _dqt_update

    def grad_view(self):
        """The rank's local gradient, shaped like the weight (GEMM output)."""
        return self.grad_full[: self.plan.numel].view(self.shape)

    def codes_view(self):
        """The gathered codes, shaped like the weight (GEMM operand)."""
        return self.codes_full[: self.plan.numel].view(self.shape)

    def load_moments(self, m_full, v_full):
        """Take this rank's shard of full moments (e.g. from a checkpoint)."""
        p = self.plan
        self.m.zero_()
        self.v.zero_()
        self.m[: p.n_local].copy_(m_full.reshape(-1)[p.lo: p.hi])
        self.v[: p.n_local].copy_(v_full.reshape(-1)[p.lo: p.hi])

    def step(self, s_w, hp, sr, grid, changed_out=None):
        """Reduce-scatter the gradient, update this rank's shard, all-gather the
        codes.  `sr` is the tensor's stream; its elem0 is set per shard here."""
        from . import dqt
        p = self.plan
        dist.reduce_scatter_tensor(self.grad_shard, self.grad_full, op=dist.ReduceOp.SUM,
                                   group=self.group)
        if p.n_local > 0:
            sr_shard = dqt.sr_stream(seed=sr.seed, tensor_id=sr.tensor_id,
                                     round_mode=sr.round_mode, elem0=sr.elem0 + p.lo)
            n = p.n_local
            self.update_fn(self.grad_shard[:n], self.codes_shard[:n], s_w, self.m[:n],
                           self.v[:n], hp, sr_shard, grid, changed_out)
        dist.all_gather_into_tensor(self.codes_full, self.codes_shard, group=self.group)
        return self.codes_view()
