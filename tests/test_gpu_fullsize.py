"""Parity at the workloads' stated sizes: sift1m-d128-m16 (10^6 rows),
gist1m-d960-m120 (10^6 x 120 subspaces), deep10m-d96-m12 (10^7 rows, two
columns, conjunctive predicates on the bitmap path) and gmm100m-d128-m16
(10^8 rows, k = 100), each built by its recipe with the oracle (mixture
vectors, Lloyd-trained codebook, float32 encoding of every row).  Every bin
runs one 1024-query batch with conditioning on, as bench.py does; 32
queries per bin, spread over the batch (the paired and unpaired queries of
the sorted-copy path among them), are recomputed by the oracle over all
rows and compared element by element, and every query of the batch is
checked through properties that hold at any size."""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import check_topk_sparse

pytestmark = [pytest.mark.gpu, pytest.mark.slow]

FULL = ["sift1m-d128-m16", "gist1m-d960-m120", "deep10m-d96-m12", "gmm100m-d128-m16"]
BATCH = 1024
SAMPLES = 32


def _passes(attrs, preds, ids):
    """Pass flags of rows ``ids`` [nq][k] (-1 ignored) for each query's
    predicate: every clause, every operator, int64 comparisons."""
    ok = ids >= 0
    safe = np.where(ok, ids, 0)
    for j in range(4):
        c = preds["c"][:, j]
        on = preds["n_clauses"] > j
        a = np.stack([attrs[col][safe[i]].astype(np.int64) for i, col in enumerate(c["col"])])
        lo, hi, op = c["lo"][:, None], c["hi"][:, None], c["op"][:, None]
        cond = np.select([op == 0, op == 1, op == 2, op == 3, op == 4, op == 5],
                         [a == lo, (a >= lo) & (a < hi), a >= lo, a < lo, a > lo, a <= lo], default=False)
        ok &= cond | ~on[:, None]
    return ok


@pytest.fixture(scope="module", params=FULL)
def full(request, oracle_index):
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs
    w = synth.WORKLOADS[request.param]
    oi = oracle_index(w)
    cond = synth.make_conditioning(oi.ix)
    g = ifvs.Index(oi.ix.codes, oi.ix.attrs, D=w.D, K=w.K)
    g.load_codebooks(oi.ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    yield w, oi, cond, g
    g.close()


def test_full_size_matches_oracle(full):
    w, oi, cond, g = full
    ix = oi.ix
    pick = np.unique(np.linspace(0, BATCH - 1, SAMPLES).astype(np.int64))
    ties = compared = 0
    for sel in w.sels:
        qs = synth.make_queries(ix, sel, nq=BATCH)
        ids, d, npass = g.search(qs.q, qs.preds, w.k, wz=qs.wz)
        # every query: valid prefix, padding, passing rows, ascending, unique
        ok = _passes(ix.attrs, qs.preds, ids)
        for i in range(BATCH):
            nv = min(w.k, int(npass[i]))
            assert (ids[i, :nv] >= 0).all() and (ids[i, nv:] == -1).all(), (sel, i)
            assert ok[i, :nv].all(), "query %d of the %g bin returned a failing row" % (i, sel)
            assert (np.diff(d[i, :nv].astype(np.float64)) >= 0).all()
            assert len(np.unique(ids[i, :nv])) == nv
        # pass counts of one-column ranges by binary search on the sorted column
        if not w.conjunctive:
            srt = np.sort(ix.attrs[0])
            c = qs.preds["c"][:, 0]
            cnt = np.searchsorted(srt, c["hi"], "left") - np.searchsorted(srt, c["lo"], "left")
            np.testing.assert_array_equal(npass, cnt)
        # the sampled queries element by element against the oracle
        res = oi.search(cond, qs.q[pick], qs.preds[pick], qs.wz[pick], w.k, check_ids=ids[pick])
        for j, i in enumerate(pick):
            r = res[j]
            assert npass[i] == r["npass"], (sel, i)
            ties += check_topk_sparse(ids[i], d[i], r["ids"], r["dists"], r["check_dist"], r["check_pass"])
            compared += int((r["ids"] >= 0).sum())
    # Every id that differs was checked to be tied with the k-th distance
    # within the tolerance, and the distances agree rank by rank: that is
    # the part of a top-k that is unique when distances tie.  Which of the
    # tied rows fill the last ranks is not: rows of one mixture component
    # often share all their codes (equal distances in exact arithmetic), the
    # float32 sum order of a row depends on its position, so the GPU breaks
    # such ties by the last ulp where the oracle (fp64) breaks them by id.
    # On deep10m (1024 components, 12 subspaces of 256 codewords) about one
    # id in ten at k = 10 is such a tie; the share is reported, not bounded.
    print("%s: %d of %d compared ids differ by a tie at the k-th distance" % (w.name, ties, compared))
