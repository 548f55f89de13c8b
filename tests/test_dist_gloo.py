"""The multi-process (N > 1) path of bench.py on CPU: two gloo ranks, each
with its own query batches (replicas, no data-path collective), agree on the
job time through a max over ranks and report whole-job throughput."""
import os
import socket

import pytest

torch = pytest.importorskip("torch")
import torch.distributed as dist  # noqa: E402
import torch.multiprocessing as mp  # noqa: E402


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _rank(rank, world, port, out):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), RANK=str(rank),
                      WORLD_SIZE=str(world), LOCAL_RANK=str(rank))
    import bench
    dist.init_process_group("gloo", rank=rank, world_size=world)
    cpu = torch.device("cpu")
    w, r, l = bench.dist_env()
    assert (w, r, l) == (world, rank, rank)
    bench.barrier(dist, cpu)
    # each rank pretends its timed region took a different time
    my_ms = 100.0 + 50.0 * rank
    mx = bench.reduce_max(dist, my_ms, cpu)
    value = bench.whole_job_qps(world, 8, 1024, mx)
    bench.barrier(dist, cpu)
    out[rank] = (mx, value)
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2])
def test_two_gloo_ranks_take_the_slowest_time(world):
    import sys
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=120)
        assert p.exitcode == 0
    slowest = 100.0 + 50.0 * (world - 1)
    for r in range(world):
        mx, value = out[r]
        assert mx == slowest
        assert abs(value - world * 8 * 1024 / (slowest / 1000.0)) < 1e-6


def test_single_rank_is_identity():
    import bench
    assert bench.reduce_max(None, 12.5, None) == 12.5
    assert bench.whole_job_qps(1, 16, 1024, 1000.0) == 16 * 1024
