"""The data-parallel exchange of the DQT update (paper_2412_04787_gb300/dp.py)
on CPU gloo ranks, with the oracle's update as the per-shard step.

Sec. 4.1 trains on 4-16 GPUs; in data parallelism the fp32 weight gradient is
reduce-scattered over a flat partition of the weight, each rank updates its
shard (holding only that shard's AdamW moments), and the int8 codes are
all-gathered.  Because every element draws the Philox uniform of its global
index, the gathered codes must equal the one-process update of the summed
gradient, bit for bit, for any number of ranks and any partition.  The
gradients here are integer multiples of 2^-30 below 2^-7 in magnitude, so
their sum is exact in fp32 in whatever order the collective adds them.
No GPU is used.
"""
import os
import socket

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import oracle
from paper_2412_04787_gb300 import dp, dqt, inputs

N, K = 37, 24  # 888 weights: shards of 448 / 304 elements, the last one short
STEPS = 3
LR, WD = 1e-2, 0.01


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _grad(rank, step):
    r = np.random.default_rng(1000 * step + rank)
    return (r.integers(-(1 << 23), 1 << 23, (N, K)) * 2.0 ** -30).astype(np.float32)


def _codes0(bits):
    qmin, qmax = oracle.grid(bits)
    c, s_w, _ = oracle.absmean_init(inputs.normal((N, K), 0.02, seed=5).numpy(), qmin, qmax)
    return c, float(s_w), (qmin, qmax)


def _oracle_update_fn(grad, W, s_w, m, v, hp, sr, grid, changed_out):
    """One flat shard through the oracle (the stand-in for dqt_sr_update)."""
    k = oracle.adamw_consts(hp.lr, hp.beta1, hp.beta2, hp.eps, hp.weight_decay, hp.step, s_w)
    c1, m1, v1, ch = oracle.update_shard(grad.numpy(), W.numpy(), m.numpy(), v.numpy(), k,
                                         grid[0], grid[1], sr.seed, hp.step, sr.tensor_id,
                                         sr.elem0, sr.round_mode)
    W.copy_(torch.from_numpy(c1))
    m.copy_(torch.from_numpy(m1))
    v.copy_(torch.from_numpy(v1))
    if changed_out is not None:
        changed_out += ch


def _worker(rank, world, port, bits, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        c0, s_w, grid = _codes0(bits)
        upd = dp.DataParallelUpdater(torch.from_numpy(c0), update_fn=_oracle_update_fn)
        p = upd.plan
        codes = []
        for step in range(1, STEPS + 1):
            upd.grad_view().copy_(torch.from_numpy(_grad(rank, step)))
            hp = dqt.adamw(lr=LR, weight_decay=WD, step=step)
            sr = dqt.sr_stream(seed=77, tensor_id=3)
            changed = torch.zeros(1, dtype=torch.int64)
            upd.step(s_w, hp, sr, grid, changed_out=changed)
            # every rank holds the whole, identical weight after the gather
            codes.append(upd.codes_view().numpy().copy())
        # the padding of the partition is never touched
        assert not upd.codes_full[p.numel:].any()
        out[rank] = (codes, upd.m[: p.n_local].numpy().copy(),
                     upd.v[: p.n_local].numpy().copy(), p.lo, p.hi, p.shard)
    finally:
        dist.barrier()
        dist.destroy_process_group()


def _reference(world, bits):
    c, s_w, (qmin, qmax) = _codes0(bits)
    m = np.zeros((N, K), np.float32)
    v = np.zeros((N, K), np.float32)
    codes = []
    for step in range(1, STEPS + 1):
        g = sum(_grad(r, step).astype(np.float64) for r in range(world)).astype(np.float32)
        k = oracle.adamw_consts(np.float32(LR), np.float32(0.9), np.float32(0.999),
                                np.float32(1e-8), np.float32(WD), step, s_w)
        c, m, v, _ = oracle.update(g, c, m, v, k, qmin, qmax, 77, step, 3)
        codes.append(c.copy())
    return codes, m.ravel(), v.ravel()


@pytest.mark.parametrize("world,bits", [(2, 1.58), (3, 8)])
def test_sharded_update_equals_unsharded(world, bits):
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, world, port, bits, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(180)
        assert p.exitcode == 0
    ref_codes, ref_m, ref_v = _reference(world, bits)
    for r in range(world):
        codes, m, v, lo, hi, shard = out[r]
        for step in range(STEPS):
            assert np.array_equal(codes[step], ref_codes[step]), (r, step)
        # ZeRO-1: rank r holds exactly the moments of its shard
        assert np.array_equal(m.view(np.uint32), ref_m[lo:hi].view(np.uint32))
        assert np.array_equal(v.view(np.uint32), ref_v[lo:hi].view(np.uint32))
        assert lo % 16 == 0 and shard % 16 == 0
    assert any((ref_codes[-1] != _codes0(bits)[0]).ravel())  # the codes did move


def test_shard_plan_covers_the_weight_once():
    for numel in (1, 15, 16, 888, 4099, 11_534_336):
        for world in (1, 2, 3, 8, 16):
            plans = [dp.ShardPlan(numel, world, r) for r in range(world)]
            covered = np.zeros(numel, np.int32)
            for p in plans:
                assert p.lo % 16 == 0 and p.shard % 16 == 0 and p.padded == world * p.shard
                covered[p.lo: p.hi] += 1
            assert (covered == 1).all()
            assert sum(p.n_local for p in plans) == numel


def test_exchange_bytes_per_weight():
    """What the exchange moves per weight and rank: the reduce-scatter sends
    (world-1)/world of the 4-byte gradient, the all-gather receives
    (world-1)/world of the 1-byte codes -- a quarter of an fp32 gather."""
    p = dp.ShardPlan(11_534_336, 8, 0)
    rs = (p.world_size - 1) * p.shard * 4
    ag = (p.world_size - 1) * p.shard * 1
    assert ag * 4 == rs
