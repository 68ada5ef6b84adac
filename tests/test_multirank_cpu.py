"""The multi-GPU path of bench.py, exercised as two gloo ranks on CPU.

Lanes shard across ranks with no data-path collective: every rank replays its own
seeded population, and the job's step time is the maximum over ranks.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    import torch
    import torch.distributed as dist

    import bench
    import workloads as W

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        progs = W.random_exprs(n_programs=2, B=8, n_points=16, seed=bench.rank_seed(rank))
        ms = 10.0 + 5.0 * rank
        out[rank] = (bench.max_over_ranks(ms, torch.device("cpu")), progs[0].params.copy())
    finally:
        dist.destroy_process_group()


def test_two_ranks_shard_and_take_max():
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(2, port, out), nprocs=2, join=True)
        r0, r1 = out[0], out[1]
    assert r0[0] == r1[0] == 15.0          # the slowest rank's time
    assert not np.array_equal(r0[1], r1[1])  # distinct populations per rank
