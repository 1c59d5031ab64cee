"""The multi-GPU path's host logic on CPU: the window partition, and the
max-over-ranks timing with two gloo ranks (127.0.0.1)."""
import os
import socket

import pytest
import torch
import torch.multiprocessing as mp

from paper_2506_08520_gb300 import shard


@pytest.mark.parametrize("n,world", [(0, 2), (1, 2), (7, 2), (14400, 4), (920, 8), (5, 3)])
def test_window_range_partitions_exactly(n, world):
    ranges = [shard.window_range(n, r, world) for r in range(world)]
    assert ranges[0][0] == 0 and ranges[-1][1] == n
    for (a0, a1), (b0, b1) in zip(ranges, ranges[1:]):
        assert a1 == b0  # contiguous, no overlap
    sizes = [b - a for a, b in ranges]
    assert max(sizes) - min(sizes) <= 1


def test_window_range_rejects_bad_ranks():
    with pytest.raises(ValueError):
        shard.window_range(10, 2, 2)
    with pytest.raises(ValueError):
        shard.window_range(10, 0, 0)


def test_aggregate_rate():
    assert shard.aggregate_rate(1000, 10, 2.0, 4) == pytest.approx(4 * 1000 * 10 / 2e-3)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    torch.distributed.init_process_group("gloo", rank=rank, world_size=world)
    try:
        t = shard.max_over_ranks(1.5 + rank)  # rank-dependent "elapsed ms"
        lo, hi = shard.window_range(1025, rank, world)
        sizes = torch.tensor([hi - lo], dtype=torch.int64)
        torch.distributed.all_reduce(sizes)  # the ranks cover every window once
        out[rank] = (t, int(sizes.item()))
    finally:
        torch.distributed.destroy_process_group()


def test_two_gloo_ranks_reduce_the_slowest_time():
    world, port = 2, _free_port()
    with mp.get_context("spawn").Manager() as m:
        out = m.dict()
        mp.start_processes(_rank, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        got = dict(out)
    assert got == {0: (2.5, 1025), 1: (2.5, 1025)}
    assert shard.max_over_ranks(3.0) == 3.0  # no process group: the value itself
