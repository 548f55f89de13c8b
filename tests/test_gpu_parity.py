"""CUDA path vs oracle, element by element, on seeded inputs of the five
workload shapes (reduced so that the oracle finishes in seconds, with ragged
tails), through the C ABI.  Each index follows its workload's recipe: the
stated mixture, a PQ codebook trained by the oracle's Lloyd iterations and
the oracle's float32 encoding of every row."""
import math

import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import REL, bitmap_rows, check_topk, close

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ifvs():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs as mod
    return mod


W = synth.WORKLOADS
CASES = {
    "gmm10k-d128-m16": (W["gmm10k-d128-m16"], 30),
    "sift200k-d128-m16": (synth.scaled(W["sift1m-d128-m16"], N=200_003), 16),
    "gist30k-d960-m120": (synth.scaled(W["gist1m-d960-m120"], N=30_011), 6),
    "deep300k-d96-m12": (synth.scaled(W["deep10m-d96-m12"], N=300_007), 12),
    "gmm500k-d128-m16-k100": (synth.scaled(W["gmm100m-d128-m16"], N=500_009), 8),
}


class Case:
    pass


@pytest.fixture(scope="module", params=list(CASES))
def case(request, ifvs, orc, oracle_index):
    w, nq = CASES[request.param]
    c = Case()
    c.name, c.w = request.param, w
    c.ix = oracle_index(w).ix
    c.cond = synth.make_conditioning(c.ix)
    c.g = ifvs.Index(c.ix.codes, c.ix.attrs)
    c.g.load_codebooks(c.ix.codebook, bank=c.cond.bank, W=c.cond.W, hash_seeds=c.cond.seeds)
    c.bins = []
    for s in w.sels:
        qs = synth.make_queries(c.ix, s, nq=nq)
        ids, d, npass, st = orc.search(c.ix.codes, c.ix.attrs, c.ix.codebook, qs.q, qs.preds, w.k,
                                       bank=c.cond.bank, W=c.cond.W, seeds=c.cond.seeds,
                                       wz=qs.wz, want_stages=True)
        c.bins.append((qs, ids, d, npass, st))
    yield c
    c.g.close()


def _passing(orc, ix, pred):
    bm, _ = orc.filter_bitmap(ix.attrs, pred)
    return bm, bitmap_rows(bm, ix.w.N)


def test_filter_bitmaps_bit_exact(case, orc):
    for qs, _, _, npass, _ in case.bins:
        bm, gn = case.g.filter(qs.preds)
        np.testing.assert_array_equal(gn, npass)
        for i in range(len(qs.preds)):
            ref, _ = orc.filter_bitmap(case.ix.attrs, qs.preds[i:i + 1])
            np.testing.assert_array_equal(bm[i], ref)


def test_conditioning_and_tables(case):
    w = case.w
    for qs, _, _, _, st in case.bins:
        g = case.g.condition(qs.q, qs.preds, wz=qs.wz, want_cifvs=True)
        np.testing.assert_array_equal(g["bank_idx"], st["bank_idx"][:, :w.h])
        assert close(g["alpha"], st["alpha"][:, :w.M * w.r], 1e-6).all()
        assert close(g["wf"], st["wf"], 1e-6).all()
        assert close(g["lut"], st["lut"], REL).all(), np.max(np.abs(g["lut"] - st["lut"]) / st["lut"])
        # C_iFVS of the first query against C_PQ + alpha . W from the oracle's alpha
        import oracle
        a = st["alpha"][0, :w.M * w.r].reshape(w.M, w.r)
        Cref = oracle.condition(case.ix.codebook, a, case.cond.W)
        np.testing.assert_allclose(g["C_ifvs"][0], Cref, rtol=1e-5, atol=1e-6 * np.abs(Cref).max())


def test_search_matches_oracle(case, orc):
    ties = compared = 0
    for qs, oi, od, npass, st in case.bins:
        ids, d, gn = case.g.search(qs.q, qs.preds, case.w.k, wz=qs.wz)
        np.testing.assert_array_equal(gn, npass)
        for i in range(len(qs.q)):
            _, passing = _passing(orc, case.ix, qs.preds[i:i + 1])
            all_d = orc.adc_all(st["lut"][i], case.ix.codes)
            ties += check_topk(ids[i], d[i], oi[i], od[i], all_d, passing)
            compared += int((oi[i] >= 0).sum())
    # every differing id is tied with the k-th distance within the tolerance
    # (rows that share their codes tie exactly; the float32 sum order depends
    # on the row's position); they must stay a small share of the ids
    assert ties <= max(2, compared // 20), (ties, compared)


def test_scan_alone_from_oracle_tables(case, orc):
    """Rank + Select given the oracle's tables (as fp32) and bitmaps."""
    qs, _, _, _, st = case.bins[-1]
    lut32 = st["lut"].astype(np.float32)
    bms = np.stack([orc.filter_bitmap(case.ix.attrs, qs.preds[i:i + 1])[0] for i in range(len(qs.q))])
    ids, d = case.g.scan_topk(lut32, bms, case.w.k)
    for i in range(len(qs.q)):
        all_d = orc.adc_all(lut32[i].astype(np.float64), case.ix.codes)
        passing = bitmap_rows(bms[i], case.w.N)
        sel = np.nonzero(passing)[0]
        oi, od = orc.topk(all_d[sel], sel, case.w.k)
        check_topk(ids[i], d[i], oi, od, all_d, passing)


def test_plain_pq_reduction(case, orc, ifvs):
    """IFVS_F_PLAIN_PQ and no w_z: alpha = 0, w_f = 1 (plain PQ ADC)."""
    qs = case.bins[0][0]
    oi, od, npass = orc.search(case.ix.codes, case.ix.attrs, case.ix.codebook, qs.q, qs.preds, case.w.k)
    ids, d, gn = case.g.search(qs.q, qs.preds, case.w.k, flags=ifvs.IFVS_F_PLAIN_PQ)
    np.testing.assert_array_equal(gn, npass)
    base = orc.condition(case.ix.codebook, None, None)
    ones = orc.filter_weights(None, case.w.D)
    for i in range(len(qs.q)):
        _, passing = _passing(orc, case.ix, qs.preds[i:i + 1])
        all_d = orc.adc_all(orc.lut(qs.q[i], base, ones), case.ix.codes)
        check_topk(ids[i], d[i], oi[i], od[i], all_d, passing)


# ------------------------------------------------------------ edge cases

def _small(ifvs, N, M=16, K=256, ds=2, seed=0, attrs=None, dup_rows=False, vectors=False):
    rng = np.random.default_rng(seed)
    codes = rng.integers(0, K, size=(N, M)).astype(np.uint8)
    if dup_rows:
        codes[1::2] = codes[0::2][: N // 2]          # exact ties: pairs of equal rows
    if attrs is None:
        attrs = [rng.integers(0, 100, N).astype(np.int32)]
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    X = rng.standard_normal((N, M * ds)).astype(np.float32) if vectors else None
    g = ifvs.Index(codes, attrs, vectors=X, D=M * ds, K=K)
    g.load_codebooks(Cpq)
    return g, codes, attrs, Cpq, X


def _queries(n, D, seed=1):
    return np.random.default_rng(seed).standard_normal((n, D)).astype(np.float32)


def _preds(n, lo, hi, col=0, op=synth.OP_RANGE):
    p = synth.empty_predicates(n)
    p["n_clauses"] = 1
    p["c"][:, 0]["col"] = col
    p["c"][:, 0]["op"] = op
    p["c"][:, 0]["lo"] = lo
    p["c"][:, 0]["hi"] = hi
    return p


def _check_plain(orc, g, codes, attrs, Cpq, q, preds, k, **kw):
    oi, od, npass = orc.search(codes, attrs, Cpq, q, preds, k)
    ids, d, gn = g.search(q, preds, k, **kw)
    np.testing.assert_array_equal(gn, npass)
    base = orc.condition(Cpq, None, None)
    ones = orc.filter_weights(None, q.shape[1])
    ties = 0
    for i in range(len(q)):
        passing = bitmap_rows(orc.filter_bitmap(attrs, preds[i:i + 1])[0], len(codes))
        all_d = orc.adc_all(orc.lut(q[i], base, ones), codes)
        ties += check_topk(ids[i], d[i], oi[i], od[i], all_d, passing)
    return ids, d, ties


@pytest.mark.parametrize("N", [1, 31, 33, 1023, 1025, 4097])
def test_ragged_sizes(ifvs, orc, N):
    g, codes, attrs, Cpq, _ = _small(ifvs, N, seed=N)
    q = _queries(5, 32)
    _check_plain(orc, g, codes, attrs, Cpq, q, _preds(5, [0, 10, 50, 0, 99], [100, 60, 51, 0, 100]), 10)


@pytest.mark.parametrize("M", [1, 4, 8, 12, 16, 24, 32, 120, 128])
def test_subspace_counts(ifvs, orc, M):
    g, codes, attrs, Cpq, _ = _small(ifvs, 3000, M=M, ds=1 if M > 64 else 2, seed=M)
    q = _queries(4, codes.shape[1] * Cpq.shape[2], seed=M)
    _check_plain(orc, g, codes, attrs, Cpq, q, _preds(4, [0, 20, 0, 5], [100, 40, 3, 95]), 10)


@pytest.mark.parametrize("K", [1, 16, 100, 256])
def test_codebook_sizes(ifvs, orc, K):
    g, codes, attrs, Cpq, _ = _small(ifvs, 5000, K=K, seed=K)
    q = _queries(3, 32, seed=K)
    _check_plain(orc, g, codes, attrs, Cpq, q, _preds(3, [0, 30, 0], [100, 70, 1]), 20)


@pytest.mark.parametrize("k", [1, 2, 31, 32, 33, 64, 65, 100, 128, 129, 256])
def test_k_values_and_padding(ifvs, orc, k):
    g, codes, attrs, Cpq, _ = _small(ifvs, 20000, seed=k)
    q = _queries(4, 32, seed=k)
    # second query passes exactly 1 row value band, third none, fourth all
    _check_plain(orc, g, codes, attrs, Cpq, q, _preds(4, [10, 7, 200, -5], [60, 8, 300, 1000]), k)


def test_exact_ties_go_to_the_smaller_id(ifvs, orc):
    g, codes, attrs, Cpq, _ = _small(ifvs, 8192, dup_rows=True, seed=3)
    q = _queries(6, 32, seed=3)
    ids, d, ties = _check_plain(orc, g, codes, attrs, Cpq, q, _preds(6, 0, 100), 50)
    assert ties == 0     # exact ties are decided by id on both sides


def test_predicate_forms(ifvs, orc):
    rng = np.random.default_rng(5)
    N = 7000
    date = rng.integers(0, 3650, N).astype(np.int32)
    cat = rng.integers(-50, 50, N).astype(np.int16)
    other = rng.integers(-2**31, 2**31, N, dtype=np.int64).astype(np.int32)
    g, codes, attrs, Cpq, _ = _small(ifvs, N, attrs=[date, cat, other], seed=5)
    p = synth.empty_predicates(8)
    p[1]["n_clauses"] = 2
    synth.set_clause(p[1], 0, 1, synth.OP_EQ, -3)
    synth.set_clause(p[1], 1, 0, synth.OP_RANGE, 100, 2000)
    p[2]["n_clauses"] = 1
    synth.set_clause(p[2], 0, 1, synth.OP_LT, 0)
    p[3]["n_clauses"] = 2
    synth.set_clause(p[3], 0, 0, synth.OP_GT, 1000)
    synth.set_clause(p[3], 1, 0, synth.OP_LE, 1010)
    p[4]["n_clauses"] = 4
    synth.set_clause(p[4], 0, 2, synth.OP_GE, 0)
    synth.set_clause(p[4], 1, 0, synth.OP_GE, 10)
    synth.set_clause(p[4], 2, 1, synth.OP_GT, -10)
    synth.set_clause(p[4], 3, 0, synth.OP_LT, 3000)
    p[5]["n_clauses"] = 2                                 # disjoint: nothing passes
    synth.set_clause(p[5], 0, 0, synth.OP_GE, 5)
    synth.set_clause(p[5], 1, 0, synth.OP_LT, 3)
    p[6]["n_clauses"] = 1                                 # outside the int16 range
    synth.set_clause(p[6], 0, 1, synth.OP_EQ, 40000)
    p[7]["n_clauses"] = 1
    synth.set_clause(p[7], 0, 2, synth.OP_RANGE, -2**40, 2**40)
    q = _queries(8, 32, seed=5)
    bm, gn = g.filter(p)
    for i in range(8):
        ref, n = orc.filter_bitmap(attrs, p[i:i + 1])
        np.testing.assert_array_equal(bm[i], ref)
        assert gn[i] == n
    _check_plain(orc, g, codes, attrs, Cpq, q, p, 16)


def test_sub_batches_and_determinism(ifvs, orc):
    g, codes, attrs, Cpq, _ = _small(ifvs, 30000, seed=8)
    q = _queries(37, 32, seed=8)
    preds = _preds(37, np.arange(37), np.arange(37) + 40)
    a = g.search(q, preds, 25)
    b = g.search(q, preds, 25, sub_batch=5)
    c = g.search(q, preds, 25)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    for x, y in zip(a, c):
        np.testing.assert_array_equal(x, y)


def test_device_io_matches_host_io(ifvs):
    torch = pytest.importorskip("torch")
    g, codes, attrs, Cpq, _ = _small(ifvs, 20000, seed=9)
    q = _queries(16, 32, seed=9)
    preds = _preds(16, np.arange(16) * 3, np.arange(16) * 3 + 50)
    ids, d, n = g.search(q, preds, 10)
    dev = torch.device("cuda:0")
    tq = torch.from_numpy(q).to(dev)
    tp = torch.from_numpy(preds.view(np.uint8).copy()).to(dev)
    ti = torch.empty((16, 10), dtype=torch.int64, device=dev)
    td = torch.empty((16, 10), dtype=torch.float32, device=dev)
    tn = torch.empty(16, dtype=torch.int64, device=dev)
    s = torch.cuda.current_stream()
    g.search(tq, tp, 10, ids=ti, dists=td, npass=tn, flags=ifvs.IFVS_F_DEVICE_IO,
             stream=s.cuda_stream)
    s.synchronize()
    np.testing.assert_array_equal(ti.cpu().numpy(), ids)
    np.testing.assert_array_equal(td.cpu().numpy(), d)
    np.testing.assert_array_equal(tn.cpu().numpy(), n)
    # device-resident index upload gives the same index
    g2 = ifvs.Index(torch.from_numpy(codes).to(dev), [torch.from_numpy(a).to(dev) for a in attrs],
                    D=32, device_io=True)
    g2.load_codebooks(Cpq)
    for x, y in zip(g2.search(q, preds, 10), (ids, d, n)):
        np.testing.assert_array_equal(x, y)


def test_rerank_matches_oracle(ifvs, orc):
    g, codes, attrs, Cpq, X = _small(ifvs, 12000, seed=11, vectors=True)
    q = _queries(6, 32, seed=11)
    preds = _preds(6, [0, 10, 20, 30, 40, 0], [100, 50, 60, 70, 80, 5])
    oi, od, _ = orc.search(codes, attrs, Cpq, q, preds, 60)
    # stand-alone rerank of the oracle's candidates
    ids, d = g.rerank(q, oi, 10)
    for i in range(6):
        ri, rd = orc.rerank(X, q[i], oi[i], 10)
        nv = int((ri >= 0).sum())
        ex = np.full(len(codes), np.inf)
        cand = oi[i][oi[i] >= 0]
        ex[cand] = ((X[cand].astype(np.float64) - q[i].astype(np.float64)) ** 2).sum(1)
        passing = np.zeros(len(codes), bool)
        passing[cand] = True
        check_topk(ids[i], d[i], ri, rd, ex, passing)
        assert nv == min(10, len(cand))
    # the whole path with rerank depth 60
    ids2, d2, _ = g.search(q, preds, 10, rerank=60)
    for i in range(6):
        ri, rd = orc.rerank(X, q[i], oi[i], 10)
        nv = int((ri >= 0).sum())
        assert close(d2[i][:nv], rd[:nv]).all()


def test_errors_are_reported(ifvs):
    g, codes, attrs, Cpq, _ = _small(ifvs, 1000, seed=12)
    q = _queries(2, 32)
    bad = _preds(2, 0, 10, col=3)
    with pytest.raises(ifvs.IfvsError) as e:
        g.search(q, bad, 10)
    assert e.value.code == ifvs.IFVS_ERR_ARG
    for k in (0, 257):
        with pytest.raises(ifvs.IfvsError):
            g.search(q, _preds(2, 0, 10), k)
    with pytest.raises(ifvs.IfvsError) as e:
        g.search(q, _preds(2, 0, 10), 10, rerank=20)     # no raw vectors loaded
    assert e.value.code == ifvs.IFVS_ERR_STATE
    h = ifvs.ifvs_load_index(codes, attrs, D=32)
    with pytest.raises(ifvs.IfvsError) as e:
        ifvs.ifvs_search_batch(h, q, _preds(2, 0, 10), 10)
    assert e.value.code == ifvs.IFVS_ERR_STATE
    ifvs.ifvs_free(h)
    bad_codes = codes.copy()
    bad_codes[5, 3] = 200
    with pytest.raises(ifvs.IfvsError):
        ifvs.Index(bad_codes, attrs, D=32, K=100)
    # the index still works after the errors
    ids, d, n = g.search(q, _preds(2, 0, 100), 5)
    assert (ids >= 0).all() and n[0] == 1000


def test_stage_timing_counts_launches(ifvs):
    g, codes, attrs, Cpq, _ = _small(ifvs, 50000, seed=13)
    q = _queries(8, 32)
    g.stage_times(reset=True)
    g.search(q, _preds(8, 0, 50), 10, flags=ifvs.IFVS_F_STAGE_TIMING)
    t = g.stage_times(reset=True)
    # one attribute column: every predicate takes the sorted copy, so no
    # filter pass and no bitmap scan run.  filter: the scan plan; scan: the
    # pairing of the sorted-copy queries, the two- and one-query kernels
    # (M = 16)
    expected = {"predicate": 1, "filter": 1, "condition": 1, "lut": 2, "scan": 3, "merge": 1}
    for s, n in expected.items():
        assert t[s][1] == n and t[s][0] > 0.0
    assert t["rerank"][1] == 0
