"""The benchmark's multi-rank aggregation with world size 2 over gloo on CPU.

Every rank runs an independent replica; the benchmark takes the maximum of
the per-rank times and reports the whole job's time per step as that maximum
divided by the number of ranks.
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


def _worker(rank, world, port, values, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        mx, per_job = bench.aggregate_over_ranks(values[rank], world, device="cpu")
        out[rank] = (mx, per_job)
    finally:
        dist.destroy_process_group()


def test_two_ranks_take_the_max_and_divide_by_the_ranks():
    world = 2
    values = [[0.070, 2.50, 0.75], [0.066, 2.61, 0.80]]
    with mp.Manager() as mgr:
        out = mgr.dict()
        mp.spawn(_worker, args=(world, _free_port(), values, out), nprocs=world, join=True)
        got = dict(out)
    for rank in range(world):
        mx, per_job = got[rank]
        assert mx == pytest.approx([0.070, 2.61, 0.80])
        assert per_job == pytest.approx([0.035, 1.305, 0.40])


def test_one_rank_is_unchanged():
    import bench
    mx, per_job = bench.aggregate_over_ranks([0.07, 2.6], 1)
    assert mx == pytest.approx([0.07, 2.6]) and per_job == pytest.approx([0.07, 2.6])
