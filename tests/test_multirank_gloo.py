"""The multi-rank bookkeeping of bench.py on two CPU ranks (gloo).

Trees are independent, so ranks verify batches of their own; the only
exchange is the max-reduction of the timed region, and the reported value is
the whole job's rate.  The GPU part of a rank is not exercised here."""

import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench


def _free_port():
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, out_dir):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # each rank times a different amount of work; the slowest sets the job time
        local_ms = 10.0 + 5.0 * rank
        job_ms = bench.max_over_ranks(local_ms, world, torch.device("cpu"))
        rate = bench.whole_job_rate(128, world, 4, job_ms)
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{bench.rank_seed(3, rank)} {job_ms} {rate}\n")
    finally:
        dist.destroy_process_group()


def test_two_ranks_share_the_job_time_and_report_the_whole_job(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    rows = [open(tmp_path / f"rank{r}.txt").read().split() for r in range(world)]
    seeds = [int(r[0]) for r in rows]
    assert len(set(seeds)) == world                   # independent batches
    for _, job_ms, rate in rows:
        assert float(job_ms) == pytest.approx(15.0)   # max over ranks
        assert float(rate) == pytest.approx(128 * 2 * 4 / 0.015)


def test_single_rank_needs_no_process_group():
    assert bench.max_over_ranks(7.5, 1, None) == 7.5
    assert bench.whole_job_rate(64, 1, 10, 2.0) == pytest.approx(64 * 10 / 0.002)
    assert bench.rank_seed(5, 0) == 5
