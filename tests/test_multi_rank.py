"""The bench's N > 1 host path on CPU: two ranks over gloo on 127.0.0.1.

With --gpus N every rank runs its own replica (weak scaling, no data-path collective); the
ranks meet only at the barriers around the timed region and in the maximum of their times.
The reference arm runs on rank 0 alone; the other ranks return 0 without work.
"""
import os
import socket
import sys

import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port() -> int:
    with socket.socket(socket.AF_INET, socket.SOCK_STREAM) as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank: int, world: int, port: int, out_dir: str):
    os.environ.update({"RANK": str(rank), "WORLD_SIZE": str(world), "LOCAL_RANK": str(rank),
                       "MASTER_ADDR": "127.0.0.1", "MASTER_PORT": str(port),
                       "IQ_BENCH_GLOO": "1"})
    sys.path.insert(0, ROOT)
    import bench
    import torch.distributed as dist

    r, w, local = bench.dist_setup(world)
    assert (r, w, local) == (rank, world, rank)
    bench.barrier(w)
    # each rank's own time; every rank must see the slowest
    got = bench.max_over_ranks(10.0 + 7.5 * rank, w, "cpu")
    bench.barrier(w)
    # the reference arm: rank 0 alone runs the oracle; here only the others are called
    rc = bench.run_reference(None, rank, w) if rank != 0 else 0
    dist.destroy_process_group()
    with open(os.path.join(out_dir, f"rank{rank}.txt"), "w") as f:
        f.write(f"{got} {rc}\n")


def test_two_ranks_barrier_max_and_reference_arm(tmp_path):
    world = 2
    mp.start_processes(_rank_main, args=(world, _free_port(), str(tmp_path)), nprocs=world,
                       join=True, start_method="spawn")
    for rank in range(world):
        got, rc = open(tmp_path / f"rank{rank}.txt").read().split()
        assert float(got) == 10.0 + 7.5 * (world - 1)
        assert int(rc) == 0


def test_single_rank_needs_no_process_group(monkeypatch):
    sys.path.insert(0, ROOT)
    import bench
    for k in ("RANK", "WORLD_SIZE", "LOCAL_RANK"):
        monkeypatch.delenv(k, raising=False)
    assert bench.dist_setup(1) == (0, 1, 0)
    bench.barrier(1)
    assert bench.max_over_ranks(3.25, 1, "cpu") == 3.25
