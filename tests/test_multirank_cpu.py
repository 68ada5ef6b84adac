"""The multi-GPU path, exercised as gloo ranks on CPU.

One population of lanes splits into contiguous per-rank slices (section 6: candidates
share nothing, so the replay needs no exchange); every rank writes its own slice of
loss and gradient, and rank 0 gathers the slices on the host after the replay.  The
job's step time is the maximum over ranks.  No replay runs here: each rank fills its
slice with a known function of the global lane index, which is what a correct gather
must reassemble into the unsplit layout.
"""
import os
import socket

import numpy as np
import pytest
import torch.multiprocessing as mp

from paper_2607_03574_gb300.shard import lane_slice


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


@pytest.mark.parametrize("B", [0, 1, 7, 64, 4097, 65536])
@pytest.mark.parametrize("world", [1, 2, 3, 4, 8])
def test_slices_are_disjoint_balanced_and_cover(B, world):
    bounds = [lane_slice(B, world, r) for r in range(world)]
    assert bounds[0][0] == 0 and bounds[-1][1] == B
    for (a, b), (c, _) in zip(bounds, bounds[1:]):
        assert b == c                                    # contiguous, in rank order
    sizes = [b - a for a, b in bounds]
    assert min(sizes) >= 0 and max(sizes) - min(sizes) <= 1  # balanced
    assert sizes == sorted(sizes, reverse=True)         # the remainder goes to the first ranks
    owner = np.full(B, -1)
    for r, (a, b) in enumerate(bounds):
        assert (owner[a:b] == -1).all()
        owner[a:b] = r
    assert (owner >= 0).all()


def test_bad_partition_arguments_raise():
    for args in ((10, 0, 0), (10, 2, 2), (10, 2, -1), (-1, 2, 0)):
        with pytest.raises(ValueError):
            lane_slice(*args)


def _lane_values(lanes, P):
    """A stand-in for a replay's per-lane outputs: loss[b] = 0.5 b, grad[b, k] = b + k / 8."""
    lanes = np.asarray(lanes, dtype=np.float64)
    return 0.5 * lanes, lanes[:, None] + np.arange(P)[None, :] / 8.0


def _worker(rank, world, port, out, B, P):
    import torch
    import torch.distributed as dist

    import bench
    from paper_2607_03574_gb300.shard import gather_lanes

    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        lo, hi = lane_slice(B, world, rank)
        loss, grad = _lane_values(range(lo, hi), P)
        gl = gather_lanes(loss, B, world, rank)
        gg = gather_lanes(grad, B, world, rank)
        ms = 10.0 + 5.0 * rank
        out[rank] = (bench.max_over_ranks(ms, torch.device("cpu")), (lo, hi), gl, gg)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("B,P", [(4096, 3), (4097, 2), (5, 12)])
def test_two_ranks_write_their_slices_and_rank0_gathers(B, P):
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out, B, P), nprocs=world, join=True)
        res = [out[r] for r in range(world)]
    assert res[0][0] == res[1][0] == 15.0          # the slowest rank's time
    assert res[0][1] == (0, -(-B // 2)) and res[1][1] == (-(-B // 2), B)
    assert res[1][2] is None and res[1][3] is None  # only rank 0 holds the gathered population
    want_loss, want_grad = _lane_values(range(B), P)
    np.testing.assert_array_equal(res[0][2], want_loss)
    np.testing.assert_array_equal(res[0][3], want_grad)


def test_bench_population_slices_one_population():
    """bench.py's per-rank workload is the rank's slice of one population: the union of
    the slices over ranks is the unsplit population, and rank 0's slice at N ranks holds
    the same lanes as the N = 1 population's first lanes for the single-tape workloads."""
    import argparse

    import bench
    args = argparse.Namespace(config=4, lanes=64, programs=3, dtype="f64")
    whole, _, _ = bench.population(args, 4, world=1, rank=0, lanes_per_rank=128)
    parts = [bench.population(args, 4, world=2, rank=r, lanes_per_rank=64)[0] for r in range(2)]
    np.testing.assert_array_equal(np.concatenate([p[0].params for p in parts]), whole[0].params)
    assert parts[0][0].program == parts[1][0].program == whole[0].program
    one, _, _ = bench.population(args, 4, world=1, rank=0, lanes_per_rank=64)
    np.testing.assert_array_equal(parts[0][0].params, one[0].params)
    progs2 = [bench.population(args, 2, world=2, rank=r, lanes_per_rank=16)[0] for r in range(2)]
    assert len(progs2[0]) == len(progs2[1]) == 3
    for a, b in zip(*progs2):
        assert a.program == b.program and a.B == b.B == 16
        assert not np.array_equal(a.params, b.params)
