"""The multi-GPU mode of bench.py, on the CPU: N independent replicas (one per
rank, no data exchange), timed by the slowest rank, whole-job throughput =
N x the bytes one rank processes / that time.  Two gloo ranks stand in for two
GPUs; only the host-side aggregation (barrier, max over ranks, throughput)
runs, which is all the multi-rank path adds to the single-GPU step.
"""
import os
import socket
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank_main(rank, world, port, times, out_dir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank), WORLD_SIZE=str(world))
    sys.path.insert(0, ROOT)
    import torch.distributed as dist
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        bench.barrier(world)
        slowest = bench.max_over_ranks(times[rank], world)
        gbs = bench.job_throughput(1_000_000_000, 10, world, slowest)
        with open(os.path.join(out_dir, "rank%d.txt" % rank), "w") as f:
            f.write("%r %r\n" % (slowest, gbs))
    finally:
        dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_replica_aggregation_over_gloo_ranks(tmp_path, world):
    import torch.multiprocessing as mp
    times = [0.5 + 0.25 * r for r in range(world)][::-1]  # the slowest rank is rank 0
    mp.start_processes(_rank_main, args=(world, _free_port(), times, str(tmp_path)), nprocs=world,
                       start_method="spawn", join=True)
    got = [tuple(float(x) for x in open(tmp_path / ("rank%d.txt" % r)).read().split()) for r in range(world)]
    slowest = max(times)
    for s, gbs in got:  # every rank agrees on the slowest time and the job figure
        assert s == slowest
        assert gbs == pytest.approx(world * 1.0 * 10 / slowest)


def test_single_rank_needs_no_process_group():
    sys.path.insert(0, ROOT)
    import bench
    bench.barrier(1)
    assert bench.max_over_ranks(0.125, 1) == 0.125
    assert bench.job_throughput(2_000_000_000, 4, 1, 2.0) == pytest.approx(4.0)
