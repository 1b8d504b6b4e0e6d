"""The multi-rank path of the benchmark on CPU: world size 2 over gloo.

Ranks run independent replicas (weak scaling); the only cross-rank steps are
the barrier around the timed region and the max over the ranks' times, from
which the whole-job throughput is formed.  Those run here as two spawned
processes with a gloo process group on 127.0.0.1.
"""
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


def _rank_main(rank, world, port, out_path):
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    bench.barrier(world)
    ms = 100.0 + 50.0 * rank          # rank 1 is the slower replica
    worst = bench.max_over_ranks(ms, world)
    value = bench.job_value(1000.0, world, worst)
    bench.barrier(world)
    with open(f"{out_path}.{rank}", "w") as f:
        f.write(f"{worst} {value}")
    dist.destroy_process_group()


@pytest.mark.timeout(120)
def test_two_rank_max_and_job_value(tmp_path):
    world, port = 2, _free_port()
    out = str(tmp_path / "r")
    mp.start_processes(_rank_main, args=(world, port, out), nprocs=world, start_method="spawn")
    for r in range(world):
        worst, value = map(float, open(f"{out}.{r}").read().split())
        assert worst == 150.0                       # both ranks agree on the slowest time
        assert value == pytest.approx(2 * 1000.0 / 0.150)   # all ranks' units over it


def test_single_rank_needs_no_process_group():
    import sys
    sys.path.insert(0, os.path.dirname(os.path.dirname(os.path.abspath(__file__))))
    import bench
    assert bench.max_over_ranks(42.0, 1) == 42.0
    assert bench.job_value(10.0, 1, 1000.0) == pytest.approx(10.0)
    bench.barrier(1)
