"""The N>1 bench path on CPU: two gloo ranks reduce their timings with max (the job is as slow as
its slowest rank) and the whole-job throughput counts the bytes of every rank."""
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


def _worker(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    import bench
    assert bench.dist_env() == (world, rank, 0)
    total, dec, enc = bench.reduce_over_ranks(1.0 + rank, 0.5 + 0.25 * rank, 10.0 - rank, world, "cpu")
    gbs = bench.job_decode_gbs(world, 3, 1e9, dec)
    out[rank] = torch.tensor([total, dec, enc, gbs], dtype=torch.float64)
    dist.barrier()
    dist.destroy_process_group()


def test_two_rank_reduction_uses_max_and_sums_bytes():
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    os.environ["PYTHONPATH"] = root + os.pathsep + os.environ.get("PYTHONPATH", "")
    world = 2
    out = torch.zeros((world, 4), dtype=torch.float64).share_memory_()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, start_method="spawn")
    for rank in range(world):
        total, dec, enc, gbs = out[rank].tolist()
        assert total == 2.0 and dec == 0.75 and enc == 10.0
        assert gbs == pytest.approx(2 * 3 * 1e9 / 0.75 / 1e9)
