"""The bench's N > 1 host logic on CPU: two gloo ranks on 127.0.0.1.

With N GPUs the bench runs one independent replica of the workload per rank
(the scans shard over units with no exchange), takes the step time as the
maximum over ranks and counts every rank's tokens.  The reference arm runs on
rank 0 only; other ranks return without work.
"""
import os
import socket
import sys

import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _worker(rank, world, port, out):
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        import bench
        import workloads as W

        my_ms = [1.5, 4.0][rank]
        step_ms, value = bench.combine_ranks(my_ms, 1000, world, torch.device("cpu"))
        dist.barrier()
        args = bench.argparse.Namespace(steps=1, warmup=3, workload="c1")
        ref = bench.run_reference(args, W.workload("c1"), rank, world) if rank == 1 else None
        out[rank] = (step_ms, value, ref is None)
    finally:
        dist.destroy_process_group()


def test_two_rank_max_time_and_whole_job_value():
    world = 2
    mgr = mp.Manager()
    out = mgr.dict()
    mp.start_processes(_worker, args=(world, _free_port(), out), nprocs=world, join=True,
                       start_method="spawn")
    for rank in range(world):
        step_ms, value, ref_skipped = out[rank]
        assert step_ms == pytest.approx(4.0)
        assert value == pytest.approx(world * 1000 / 4.0e-3)
        assert ref_skipped
