"""The N > 1 path of bench.py (replicas, one rank per GPU, no exchange
step), run as two gloo ranks on the CPU: the job time is the slowest rank's,
every rank draws its own batch, and the throughput counts all ranks."""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str):
    import torch.distributed as dist
    sys.path.insert(0, ROOT)
    import bench
    os.environ["MASTER_ADDR"] = "127.0.0.1"
    os.environ["MASTER_PORT"] = str(port)
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        # rank r reports timings (1 + r, 10 - r): the job sees (world, 10)
        got = bench.max_over_ranks([1.0 + rank, 10.0 - rank])
        seed = bench.rank_input_seed(1234, rank)
        with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
            f.write(f"{got[0]} {got[1]} {seed}\n")
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks(tmp_path):
    import torch.multiprocessing as mp
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world, start_method="spawn")
    rows = [open(tmp_path / f"rank{r}.txt").read().split() for r in range(world)]
    for r, (a, b, seed) in enumerate(rows):
        assert float(a) == float(world) and float(b) == 10.0  # both ranks hold the maxima
    assert [int(seed) for (_, _, seed) in rows] == [1234, 1234 + 7919]  # distinct batches, rank 0 unchanged


def test_single_process_and_throughput():
    sys.path.insert(0, ROOT)
    import bench
    assert bench.max_over_ranks([3.0, 4.0]) == [3.0, 4.0]  # no process group: the values themselves
    # 2 ranks x 1.933 GOP per step in 28.3 us
    assert abs(bench.job_tops(2, 1.933e9, 0.0283) - 2 * 1.933e9 / 28.3e-6 / 1e12) < 1e-9
    assert bench.job_tops(1, 1e12, 1000.0) == 1.0
