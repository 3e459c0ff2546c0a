"""Host-side logic of the multi-process bench on CPU ranks (gloo, world size 2): each rank draws its own
sequences, the job time is the slowest rank's, and the throughput counts every rank's sequences. No GPU and no
data-path collective: the decode sequences are independent, so ranks only exchange their step times."""
import os
import socket

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

import bench
from paper_2609_03949_gb300 import datagen


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out: dict) -> None:
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        r, w, _ = bench.dist_env()
        assert (r, w) == (rank, world)
        # each rank's own sequences: a small workload of the bench's shape family, seeded per rank
        wl = datagen.make_workload(2, 4, 256, seed=bench.rank_seed(rank), n_planted=2, planted_hi=256 - 16,
                                   device="cpu")
        digest = float(wl.cache.float().sum())
        gathered = [None] * world
        dist.all_gather_object(gathered, digest)
        # step times differ per rank; the job's time is the slowest one
        local_ms = 1.0 + rank
        job_ms = bench.max_over_ranks(local_ms, dist, torch.device("cpu"))
        out[rank] = (gathered, job_ms, bench.job_throughput(2, world, job_ms))
    finally:
        dist.destroy_process_group()


def test_two_ranks_host_logic():
    world = 2
    port = _free_port()
    with mp.get_context("spawn").Manager() as mgr:    # no fork: the test process may already run threads
        out = mgr.dict()
        mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, start_method="spawn", join=True)
        res = dict(out)
    assert set(res) == {0, 1}
    digests = res[0][0]
    assert digests == res[1][0]
    assert digests[0] != digests[1], "ranks must draw different sequences"
    for rank in range(world):
        _, job_ms, value = res[rank]
        assert job_ms == pytest.approx(2.0)                   # max over ranks, seen identically by every rank
        assert value == pytest.approx(2 * world / (2.0e-3))   # all ranks' sequences over the slowest rank's time


def test_single_process_is_identity():
    assert bench.max_over_ranks(1.25, None, None) == 1.25
    assert bench.job_throughput(64, 1, 1.5) == pytest.approx(64 / 1.5e-3)
