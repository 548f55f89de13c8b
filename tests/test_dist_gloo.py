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


# ------------------------------------------------------------ row shards

def _shard_rank(rank, world, port, out):
    """One shard of a row-sharded search on CPU: the oracle stands in for
    this process's GPU search over its rows; the product's host logic
    (shard bounds, id offsets, the gather and the count sum) runs over gloo."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    import numpy as np
    import oracle
    from paper_2607_22922_gb300 import shard, synth
    dist.init_process_group("gloo", rank=rank, world_size=world)
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=5003)
    ix = synth.pq_space_index(w)
    cond = synth.make_conditioning(ix)
    r0, r1 = shard.shard_bounds(w.N, world, rank, align=1024)
    res = {}
    for sel, k in ((0.01, 10), (0.5, 10), (0.002, 40)):
        qs = synth.make_queries(ix, sel, nq=12)
        li, ld, ln = oracle.search(ix.codes[r0:r1], [a[r0:r1] for a in ix.attrs], ix.codebook, qs.q,
                                   qs.preds, k, bank=cond.bank, W=cond.W, seeds=cond.seeds, wz=qs.wz)
        gi = shard.offset_ids(torch.from_numpy(li), r0)
        all_d, all_i, total = shard.gather_results(torch.from_numpy(ld), gi, torch.from_numpy(ln))
        res[(sel, k)] = (all_d.numpy(), all_i.numpy(), total.numpy())
    out[rank] = (r0, r1, res)
    dist.destroy_process_group()


@pytest.mark.parametrize("world", [2, 3])
def test_row_shards_merge_to_the_whole_search(world):
    """Each rank searches its rows, the per-shard top-k lists are gathered
    and merged by (dist, id): the result equals the search over all rows
    (ids, distances and pass counts), including queries whose pool holds
    fewer than k rows on some shard."""
    import sys
    import numpy as np
    root = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
    if root not in sys.path:
        sys.path.insert(0, root)
    import oracle
    from paper_2607_22922_gb300 import synth
    oracle.build()
    ctx = mp.get_context("spawn")
    mgr = ctx.Manager()
    out = mgr.dict()
    port = _free_port()
    procs = [ctx.Process(target=_shard_rank, args=(r, world, port, out)) for r in range(world)]
    for p in procs:
        p.start()
    for p in procs:
        p.join(timeout=180)
        assert p.exitcode == 0
    bounds = [out[r][:2] for r in range(world)]
    assert bounds[0][0] == 0 and bounds[-1][1] == 5003
    assert all(bounds[r][1] == bounds[r + 1][0] for r in range(world - 1))
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=5003)
    ix = synth.pq_space_index(w)
    cond = synth.make_conditioning(ix)
    for (sel, k), (all_d, all_i, total) in out[0][2].items():
        # every rank gathered the same lists
        for r in range(1, world):
            np.testing.assert_array_equal(out[r][2][(sel, k)][1], all_i)
        qs = synth.make_queries(ix, sel, nq=12)
        oi, od, on = oracle.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, k, bank=cond.bank,
                                   W=cond.W, seeds=cond.seeds, wz=qs.wz)
        np.testing.assert_array_equal(total, on)
        for i in range(12):
            cand_i = all_i[:, i, :].ravel()
            cand_d = all_d[:, i, :].ravel()
            keep = cand_i >= 0
            mi, md = oracle.topk(cand_d[keep], cand_i[keep], k)
            np.testing.assert_array_equal(mi, oi[i])
            np.testing.assert_array_equal(md[mi >= 0], od[i][oi[i] >= 0])


def test_shard_bounds_cover_the_rows_in_order():
    from paper_2607_22922_gb300 import shard
    for N in (1, 1023, 1024, 5003, 10**6 + 7):
        for world in (1, 2, 3, 8):
            b = [shard.shard_bounds(N, world, r) for r in range(world)]
            assert b[0][0] == 0 and b[-1][1] == N
            for r in range(world - 1):
                assert b[r][1] == b[r + 1][0]
                assert b[r][1] % 1024 == 0 or b[r][1] == N
    with pytest.raises(ValueError):
        shard.shard_bounds(10, 2, 2)
