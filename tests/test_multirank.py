"""The multi-GPU path is replicas only (one stream per rank, no collective on the data
path): the host-side pieces -- distinct inputs per rank and the whole-job reduction of
bench.py (max timed region, summed tokens and calls) -- run here as two gloo ranks on CPU."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed, tokens, calls = 1.5 + rank, 15 * (10 + rank), 7 + 3 * rank
        out = bench.combine_ranks(elapsed, tokens, calls, dist, torch.device("cpu"))
        q.put((rank, out, bench.replica_first_frame(rank)))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_combine_like_the_bench():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    for rank, (elapsed, tokens, calls), first in res:
        assert elapsed == 2.5 and tokens == 15 * 21 and calls == 17       # max, sum, sum
    assert res[0][2] != res[1][2]                                         # each replica its own frames


def test_single_process_needs_no_collective():
    assert bench.combine_ranks(1.0, 30, 2) == (1.0, 30, 2)
