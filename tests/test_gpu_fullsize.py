"""Parity at the benchmark's full size: 10^8 PQ-coded rows, 1024-query
batches, k = 100, conditioning on, the launch configuration bench.py times.
The oracle recomputes sampled queries of every selectivity bin one by one
(it scans all 10^8 rows per query); the other queries are checked through
properties that hold at any size."""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import bitmap_rows, check_topk

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

SAMPLES = (0, 1023)   # queries of each batch recomputed by the oracle


@pytest.fixture(scope="module")
def full():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs
    w = synth.WORKLOADS["gmm100m-d128-m16"]
    ix = synth.make_index(w)
    cond = synth.make_conditioning(ix)
    g = ifvs.Index(ix.codes, ix.attrs)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    yield w, ix, cond, g
    g.close()


@pytest.mark.parametrize("sel", synth.WORKLOADS["gmm100m-d128-m16"].sels)
def test_full_size_batch(full, orc, sel):
    w, ix, cond, g = full
    qs = synth.make_queries(ix, sel, nq=w.batch)
    ids, d, npass = g.search(qs.q, qs.preds, w.k, wz=qs.wz)
    # properties for every query of the batch
    attr = ix.attrs[0]
    lo = qs.preds["c"][:, 0]["lo"]
    hi = qs.preds["c"][:, 0]["hi"]
    for i in range(w.batch):
        nv = min(w.k, int(npass[i]))
        assert (ids[i, :nv] >= 0).all() and (ids[i, nv:] == -1).all()
        a = attr[ids[i, :nv]]
        assert ((a >= lo[i]) & (a < hi[i])).all(), "a returned row fails its predicate"
        assert (np.diff(d[i, :nv].astype(np.float64)) >= 0).all()
        assert len(np.unique(ids[i, :nv])) == nv
    # exact pass counts for every query (the oracle's filter is a plain loop)
    for i in SAMPLES:
        _, n = orc.filter_bitmap(ix.attrs, qs.preds[i:i + 1])
        assert npass[i] == n
    # element by element for the sampled queries
    for i in SAMPLES:
        oi, od, on, st = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q[i:i + 1],
                                    qs.preds[i:i + 1], w.k, bank=cond.bank, W=cond.W,
                                    seeds=cond.seeds, wz=qs.wz[i:i + 1], want_stages=True)
        assert on[0] == npass[i]
        bm, _ = orc.filter_bitmap(ix.attrs, qs.preds[i:i + 1])
        passing = bitmap_rows(bm, w.N)
        all_d = orc.adc_all(st["lut"][0], ix.codes)
        check_topk(ids[i], d[i], oi[0], od[0], all_d, passing)
