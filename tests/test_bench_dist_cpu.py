"""Multi-rank host logic of bench.py on CPU: two gloo ranks agree on the
max-over-ranks time and the whole-job throughput, and only rank 0 of the
reference arm does work.  No GPU is used."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    ws, r, local = bench._dist()
    ms = 100.0 + 50.0 * rank  # rank 1 is the slow one
    mx = bench.max_over_ranks(ms, "cpu")
    val = bench.aggregate_tokens_per_s(ws, bench.T_TOK, 10, mx)
    out[rank] = (ws, r, local, mx, val)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_aggregation():
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, out)) for r in range(2)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(120)
        assert p.exitcode == 0
    for r in range(2):
        ws, rank, local, mx, val = out[r]
        assert (ws, rank, local) == (2, r, r)
        assert mx == 150.0  # max over ranks
        assert val == pytest.approx(2 * 8192 * 10 / 0.150)


def test_single_process_helpers():
    import bench
    assert bench.max_over_ranks(3.5, "cpu") == 3.5
    assert bench.aggregate_tokens_per_s(1, 8192, 20, 1000.0) == pytest.approx(8192 * 20)


def test_reference_arm_nonzero_rank_does_nothing(monkeypatch, capsys):
    import bench
    monkeypatch.setenv("RANK", "1")
    monkeypatch.setenv("WORLD_SIZE", "2")

    class A:
        steps, warmup = 1, 3
    bench.run_reference(A())
    assert capsys.readouterr().out == ""
