"""Host logic of bench.py's multi-process mode, on CPU with gloo ranks.

Streams are independent replicas, one per GPU, so the only cross-rank step
is the max over ranks of the timed step and end-to-end times; the reported
value is the units all ranks processed over the slowest rank (weak scaling).
"""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, units, out):
    import bench
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        values, worst = bench.combine_ranks(times[rank], units, dist)
        out[rank] = (values, worst)
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_combine_ranks_takes_the_slowest_rank(world):
    times = [[2.0 + r, 5.0 - r] for r in range(world)]  # step ms, e2e ms per rank
    units = 20
    out = mp.Manager().dict()
    mp.start_processes(_rank_main, args=(world, _free_port(), times, units, out), nprocs=world, join=True,
                       start_method="spawn")
    slow_step = max(t[0] for t in times)
    slow_e2e = max(t[1] for t in times)
    for r in range(world):
        values, worst = out[r]
        assert worst == [slow_step, slow_e2e]
        assert values[0] == pytest.approx(units * world / (slow_step / 1e3))
        assert values[1] == pytest.approx(units * world / (slow_e2e / 1e3))


def test_combine_ranks_single_process():
    import bench
    values, worst = bench.combine_ranks([4.0, 8.0], 20)
    assert worst == [4.0, 8.0]
    assert values == [pytest.approx(5000.0), pytest.approx(2500.0)]


def test_dist_env_defaults(monkeypatch):
    import bench
    for k in ("WORLD_SIZE", "RANK", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench._dist_env() == (1, 0, 0)
    monkeypatch.setenv("WORLD_SIZE", "4")
    monkeypatch.setenv("RANK", "3")
    monkeypatch.setenv("LOCAL_RANK", "1")
    assert bench._dist_env() == (4, 3, 1)
