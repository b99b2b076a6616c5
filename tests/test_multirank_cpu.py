"""Multi-rank host logic on CPU (gloo, world size 2).

The eviction pass shards by unit with no data-path collective: every rank
processes its own cache and the benchmark's only collectives aggregate the
timing (max over ranks) and the processed tokens (sum). This runs that exact
code (bench.aggregate_ranks) in two gloo processes.
"""

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
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench

    t_ms = [2.0, 3.0][rank]
    tokens = [1000, 1000][rank]
    value, t_job, w = bench.aggregate_ranks(t_ms, tokens, dist, "cpu")
    out[rank] = (value, t_job, w)
    dist.barrier()
    dist.destroy_process_group()


def test_two_ranks_aggregate_max_time_and_total_tokens():
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
        value, t_job, w = out[r]
        assert w == 2 and t_job == 3.0
        assert value == pytest.approx(2000 / 3e-3)


def test_single_process_aggregate_is_identity():
    import bench

    value, t, w = bench.aggregate_ranks(4.0, 500, None)
    assert w == 1 and t == 4.0 and value == pytest.approx(500 / 4e-3)
