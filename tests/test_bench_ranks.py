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


def test_alu_view_and_paper_summary():
    import bench
    import workloads
    wl = workloads.WORKLOADS[bench.DEFAULT_WORKLOAD]
    updates = wl.B * 4 * wl.D * wl.N * wl.L
    v = bench.alu_view("full_scan", wl, 1.0)               # one millisecond
    assert v["bound"] == "alu" and v["achieved"] == pytest.approx(updates * 1e3)
    assert v["peak"] == pytest.approx(4 * 152 * 2.07e9 * 32 / 5)
    assert v["frac"] == pytest.approx(v["achieved"] / v["peak"])
    assert bench.alu_view("mean_scan", wl, 1.0)["peak"] == pytest.approx(32 * 152 * 2.07e9)
    assert bench.alu_view("cross_scan", wl, 1.0) is None
    ps = {"w": {"scan_only_full": {"us": 10.0, "gbs": 678.48}, "shape": {"B": 1}}}
    out = bench.paper_style_summary(ps, 6784.8)
    assert out["w"]["scan_only_full"]["frac_of_peak"] == pytest.approx(0.1)
    assert out["paper_a6000_base_512x3136"]["scan_only_full_ms"] == 5.86
    assert bench.paper_style_summary(None, 6784.8) is None
