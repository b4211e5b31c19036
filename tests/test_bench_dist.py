"""Multi-rank host logic of bench.py on CPU (gloo, world size 2): barriers,
the max over ranks of the timed region, and the whole-job aggregate."""
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


def _worker(rank, world, port, out_path):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    w, r, local = bench.dist_env()
    assert (w, r, local) == (world, rank, rank)
    bench.init_dist(w, "gloo")
    bench.barrier(w)
    # rank r pretends its timed region took (r + 1) seconds of 10 units each
    slowest = bench.max_over_ranks(float(rank + 1), w)
    rate = bench.aggregate_rate(10.0, w, slowest)
    bench.barrier(w)
    if rank == 0:
        with open(out_path, "w") as f:
            f.write(f"{slowest} {rate}")
    dist.destroy_process_group()


def test_two_rank_max_and_aggregate(tmp_path):
    out = tmp_path / "result.txt"
    mp.start_processes(_worker, args=(2, _free_port(), str(out)), nprocs=2, start_method="spawn",
                       join=True)
    slowest, rate = map(float, out.read_text().split())
    assert slowest == 2.0
    assert rate == pytest.approx(10.0 * 2 / 2.0)


def test_single_rank_needs_no_process_group():
    import bench
    assert not dist.is_initialized()
    assert bench.max_over_ranks(3.5, 1) == 3.5
    assert bench.aggregate_rate(6.0, 1, 2.0) == 3.0
