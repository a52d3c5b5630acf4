"""Host-side logic of bench.py: the max-over-ranks / sum-over-ranks timing
reduction on world_size 2 over gloo, and argument defaults."""
from __future__ import annotations

import os
import socket

import pytest
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, q):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        elapsed = [3.0, 5.0][rank]
        mx = bench.max_over_ranks(elapsed, world)
        tot = bench.sum_over_ranks(100.0 * (rank + 1), world)
        bench.barrier(world)
        q.put((rank, mx, tot))
    finally:
        dist.destroy_process_group()


def test_rank_reductions_gloo_world2():
    ctx = mp.get_context("spawn")
    q = ctx.Queue()
    port = _free_port()
    procs = [ctx.Process(target=_worker, args=(r, 2, port, q)) for r in range(2)]
    for p in procs:
        p.start()
    res = sorted(q.get(timeout=120) for _ in procs)
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    assert [r[1] for r in res] == [5.0, 5.0]      # the slowest rank sets the time
    assert [r[2] for r in res] == [300.0, 300.0]  # bytes of all ranks add up


def test_single_process_reductions_are_identity():
    assert bench.max_over_ranks(2.5, 1) == 2.5
    assert bench.sum_over_ranks(2.5, 1) == 2.5


def test_defaults():
    a = bench.parse_args([])
    assert a.gpus == 1 and a.impl == "ours" and a.warmup >= 3 and a.workload == bench.DEFAULT_WORKLOAD
