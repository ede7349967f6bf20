"""The bench's N > 1 path on the CPU: two ranks in a `gloo` process group
(world size 2, rendezvous on 127.0.0.1) run the same aggregation the GPU ranks
run over NCCL.  The path has no data-path collective (replicas only): each
rank's timed totals are maximised over the ranks, and rank 0 turns the
slowest replica's time into whole-job queries/s."""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
sys.path.insert(0, ROOT)

import bench  # noqa: E402


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, totals, out):
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        dist.barrier()
        got = bench.slowest_replica(totals[rank], world, torch.device("cpu"))
        dist.barrier()
        out.put((rank, got))
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks_agree_on_the_slowest_replica():
    world, port = 2, _free_port()
    # Per rank: total of the timed steps and of the end-to-end calls (ms).
    totals = [[12.5, 30.0], [14.25, 28.0]]
    ctx = mp.get_context("spawn")
    out = ctx.Queue()
    procs = [ctx.Process(target=_rank_main, args=(r, world, port, totals, out))
             for r in range(world)]
    for p in procs:
        p.start()
    results = dict(out.get(timeout=120) for _ in range(world))
    for p in procs:
        p.join(timeout=60)
        assert p.exitcode == 0
    # Every rank sees the element-wise maximum over the ranks.
    for r in range(world):
        assert results[r] == [14.25, 30.0]
    # Rank 0's whole-job figure: all ranks' queries over the slowest time.
    assert bench.job_rate(256, 200, world, results[0][0]) == pytest.approx(
        256 * 200 * 2 / 14.25e-3)


def test_one_rank_is_the_identity():
    assert bench.slowest_replica([3.0, 4.5], 1, torch.device("cpu")) == [3.0, 4.5]
    assert bench.job_rate(1, 10, 1, 5.0) == pytest.approx(2000.0)
