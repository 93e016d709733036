"""The multi-rank logic of bench.py on CPU: two gloo ranks, each with its own
batch, timings reduced by max, whole-job throughput counted over all ranks."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    port = s.getsockname()[1]
    s.close()
    return port


def _worker(rank, world, port, out):
    import bench
    import workloads
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    try:
        wl = workloads.WORKLOADS[workloads.SMALL]
        seed = bench.rank_seed(wl, rank)
        times = [1.0 + rank, 10.0 - rank]          # rank 1 is slower on the first, faster on the second
        mx = bench.max_over_ranks(times, world)
        out[rank] = (seed, mx)
        dist.barrier()
    finally:
        dist.destroy_process_group()


def test_two_gloo_ranks():
    world = 2
    port = _free_port()
    with mp.Manager() as m:
        out = m.dict()
        mp.spawn(_worker, args=(world, port, out), nprocs=world, join=True)
        res = dict(out)
    assert res[0][1] == res[1][1] == [2.0, 10.0]   # max over ranks, element-wise
    assert res[0][0] != res[1][0]                   # every rank draws its own batch


def test_job_throughput_counts_every_rank():
    import bench
    assert bench.job_throughput(10**9, 1, 1000.0) == pytest.approx(1.0)
    assert bench.job_throughput(10**9, 4, 1000.0) == pytest.approx(4.0)
    assert bench.max_over_ranks([3.0, 4.0], 1) == [3.0, 4.0]
