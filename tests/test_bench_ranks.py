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


def _shard_main(rank, world, port, out):
    import numpy as np
    import oracle
    from workloads import draw_factor_set, draw_inputs, rounded_factors
    dist.init_process_group("gloo", init_method=f"tcp://127.0.0.1:{port}", rank=rank, world_size=world)
    try:
        D, H, T, B, K = 12, 16, 4, 6, 8
        gates = rounded_factors([draw_factor_set(H, D + H, K, 10, 8800 + g) for g in range(4)], "bf16")
        x = draw_inputs(T, B, D, "uniform", 88)
        lo, hi = rank * B // world, (rank + 1) * B // world   # this rank's streams
        mine = oracle.run_lstm([gates], x[:, lo:hi], K, checkpoints=[3, K])
        parts = [None] * world
        dist.all_gather_object(parts, (lo, hi, mine["h"], mine["ckpt_h"]))
        if rank == 0:
            full = oracle.run_lstm([gates], x, K, checkpoints=[3, K])
            h = np.concatenate([p[2] for p in parts], axis=1)
            ck = np.concatenate([p[3] for p in parts], axis=2)
            out["ok"] = (np.allclose(h, full["h"], rtol=0, atol=1e-13) and
                         np.allclose(ck, full["ckpt_h"], rtol=0, atol=1e-13) and
                         [p[:2] for p in parts] == [(r * B // world, (r + 1) * B // world) for r in range(world)])
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_streams_split_across_ranks_concatenate_to_the_whole_batch(world):
    """Large-batch sharding: each rank runs its B/G streams with the same
    factors and no collective on the data path; concatenating the ranks'
    outputs along the stream axis gives the whole batch's outputs (streams
    are independent).  Checked on the oracle with gloo ranks."""
    out = mp.Manager().dict()
    mp.start_processes(_shard_main, args=(world, _free_port(), out), nprocs=world, join=True, start_method="spawn")
    assert out["ok"]
