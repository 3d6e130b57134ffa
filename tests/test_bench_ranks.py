"""The multi-rank host logic of bench.py (one process per GPU under
torchrun, replicas only: no collective on the data path) on CPU, with two
gloo ranks: per-rank inputs, the job's timed region as the maximum over the
ranks, the whole-job value, and a single reporting rank."""

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


def _rank_main(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world),
                      LOCAL_RANK=str(rank))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, local, w = bench.dist_env()
        local_ms = 10.0 + 5.0 * r           # rank 1 is the slower one
        job_ms = bench.job_region_ms(local_ms, w)
        out[r] = (r, local, w, bench.rank_seed(1234, r), job_ms, bench.job_value(w, 16, 64, job_ms / 200),
                  bench.reports(r))
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_aggregate_like_the_driver_expects():
    world, port = 2, _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_rank_main, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert sorted(res) == [0, 1]
    for r in (0, 1):
        rank, local, w, seed, job_ms, value, rep = res[r]
        assert (rank, local, w) == (r, r, 2)
        assert seed == 1234 + r                      # distinct inputs and Philox keys per rank
        assert job_ms == 15.0                        # the slowest rank's region, on every rank
        assert value == pytest.approx(2 * 16 * 64 / (15.0 / 200 * 1e-3))
        assert rep == (r == 0)                       # only rank 0 prints


def test_single_rank_needs_no_process_group():
    assert bench.job_region_ms(12.5, 1) == 12.5
    assert bench.job_value(1, 16, 64, 0.05) == pytest.approx(16 * 64 / 0.05e-3)
