"""Row shards on the GPU: ifvs_merge_topk (Select across shards) against
the oracle's top-k, and an index split into row shards — searched shard by
shard on one GPU, ids offset, the per-shard lists stacked as an all-gather
would stack them, then merged — against the oracle's search over all rows
and the unsharded index."""
import numpy as np
import pytest

from paper_2607_22922_gb300 import shard, synth
from parity_util import check_topk, close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ifvs():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs as mod
    return mod


def _lists(rng, G, nq, k, pad_frac, ties):
    """Per-shard sorted lists with disjoint ids, some padded, some tied."""
    d = np.full((G, nq, k), np.inf, np.float32)
    ids = np.full((G, nq, k), -1, np.int64)
    for g in range(G):
        for q in range(nq):
            nv = k if rng.random() > pad_frac else int(rng.integers(0, k))
            vals = rng.integers(0, 50, nv).astype(np.float32) * 0.25 if ties else \
                rng.random(nv).astype(np.float32) * 100
            rows = g * 10**9 + rng.choice(10**6, nv, replace=False)
            o = np.lexsort((rows, vals))
            d[g, q, :nv] = vals[o]
            ids[g, q, :nv] = rows[o]
    return d, ids


@pytest.mark.parametrize("G,k", [(1, 1), (2, 10), (3, 100), (8, 256), (16, 256), (64, 64)])
@pytest.mark.parametrize("ties", [False, True])
def test_merge_topk_matches_oracle(ifvs, orc, G, k, ties):
    rng = np.random.default_rng(G * 1000 + k + ties)
    nq = 37
    d, ids = _lists(rng, G, nq, k, 0.3, ties)
    oi, od = ifvs.ifvs_merge_topk(d, ids, k)
    for q in range(nq):
        keep = ids[:, q, :].ravel() >= 0
        ri, rd = orc.topk(d[:, q, :].ravel()[keep].astype(np.float64), ids[:, q, :].ravel()[keep], k)
        np.testing.assert_array_equal(oi[q], ri)
        np.testing.assert_array_equal(od[q][ri >= 0], rd[ri >= 0].astype(np.float32))
        assert np.isinf(od[q][ri < 0]).all()


def test_merge_topk_device_io_and_errors(ifvs):
    import torch
    rng = np.random.default_rng(3)
    d, ids = _lists(rng, 4, 50, 32, 0.2, True)
    hi, hd = ifvs.ifvs_merge_topk(d, ids, 32)
    dev = torch.device("cuda", 0)
    s = torch.cuda.Stream(dev)
    td, ti = torch.from_numpy(d).to(dev), torch.from_numpy(ids).to(dev)
    oi = torch.empty((50, 32), dtype=torch.int64, device=dev)
    od = torch.empty((50, 32), dtype=torch.float32, device=dev)
    ifvs.ifvs_merge_topk(td, ti, 32, dists_out=od, ids_out=oi, flags=ifvs.IFVS_F_DEVICE_IO,
                         stream=s.cuda_stream)
    s.synchronize()
    np.testing.assert_array_equal(oi.cpu().numpy(), hi)
    np.testing.assert_array_equal(od.cpu().numpy(), hd)
    with pytest.raises(ifvs.IfvsError) as e:
        ifvs.ifvs_merge_topk(np.zeros((17, 1, 256), np.float32), np.zeros((17, 1, 256), np.int64), 256)
    assert e.value.code == -5
    with pytest.raises(ValueError):
        ifvs.ifvs_merge_topk(d, ids[:, :, :16], 32)


@pytest.mark.parametrize("G", [2, 3])
def test_row_shards_equal_the_whole_index(ifvs, orc, oracle_index, G):
    import torch
    w = synth.scaled(synth.WORKLOADS["gmm100m-d128-m16"], N=300_007)
    ix = oracle_index(w).ix
    cond = synth.make_conditioning(ix)
    dev = torch.device("cuda", 0)
    whole = ifvs.Index(ix.codes, ix.attrs)
    whole.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    parts = []
    for r in range(G):
        r0, r1 = shard.shard_bounds(w.N, G, r)
        g = ifvs.Index(np.ascontiguousarray(ix.codes[r0:r1]), [np.ascontiguousarray(a[r0:r1]) for a in ix.attrs])
        g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
        parts.append((r0, g))
    for sel in (0.001, 0.1, 1.0):
        qs = synth.make_queries(ix, sel, nq=24)
        k = w.k
        all_d, all_i, total = [], [], 0
        for r0, g in parts:
            i, d, n = g.search(qs.q, qs.preds, k, wz=qs.wz)
            all_i.append(shard.offset_ids(i, r0))
            all_d.append(d)
            total = total + n
        mi, md = ifvs.ifvs_merge_topk(np.stack(all_d), np.stack(all_i), k)
        wi, wd, wn = whole.search(qs.q, qs.preds, k, wz=qs.wz)
        np.testing.assert_array_equal(total, wn)
        oi, od, on, st = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, k, bank=cond.bank,
                                    W=cond.W, seeds=cond.seeds, wz=qs.wz, want_stages=True)
        np.testing.assert_array_equal(total, on)
        for q in range(len(qs.q)):
            bm, _ = orc.filter_bitmap(ix.attrs, qs.preds[q:q + 1])
            passing = np.unpackbits(bm.view(np.uint8), bitorder="little")[:w.N].astype(bool)
            all_dist = orc.adc_all(st["lut"][q], ix.codes)
            check_topk(mi[q], md[q], oi[q], od[q], all_dist, passing)
            fin = np.isfinite(wd[q])
            assert close(md[q][fin], wd[q][fin]).all()
    whole.close()
    for _, g in parts:
        g.close()
