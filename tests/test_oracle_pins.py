"""Pins of the oracle against what the paper and the mathematics fix.

None of these re-types an oracle formula: each compares the oracle with a
value written by hand from the paper's definitions (tests/golden), a
published test vector, a closed form, an invariant, or a library routine
(numpy / scipy) computing the same quantity another way.
"""
import json
import math
import os

import numpy as np
import pytest
from scipy.spatial.distance import cdist

from paper_2607_22922_gb300 import synth


def _pred(col, op, lo, hi=0, more=()):
    p = synth.empty_predicates(1)
    p[0]["n_clauses"] = 1 + len(more)
    synth.set_clause(p[0], 0, col, op, lo, hi)
    for i, (c, o, l, h) in enumerate(more):
        synth.set_clause(p[0], i + 1, c, o, l, h)
    return p


# ------------------------------------------------------------ worked example

@pytest.fixture(scope="module")
def worked(golden_dir):
    with open(os.path.join(golden_dir, "worked_example.json")) as f:
        return json.load(f)


def test_worked_example_conditioning_and_lut(orc, worked):
    g = worked
    Cpq = np.array(g["C_pq"], np.float32)
    W = np.array(g["W"], np.float32)
    bank = np.array(g["bank"], np.float32)
    seeds = np.array(g["seeds"], np.uint64)
    q = np.array(g["q"], np.float32)
    p = _pred(**g["pred"])
    idx = orc.fingerprint(q, p, seeds, g["B"])
    assert list(idx) == [0]
    a = orc.alpha(bank, idx).reshape(g["M"], g["r"])
    Cf = orc.condition(Cpq, a, W)
    np.testing.assert_array_equal(Cf, np.array(g["expected"]["C_ifvs"], np.float64))
    wf = orc.filter_weights(None, g["D"])
    lut = orc.lut(q, Cf, wf)
    np.testing.assert_array_equal(lut, np.array(g["expected"]["lut"], np.float64))
    codes = np.array(g["codes"], np.uint8)
    np.testing.assert_array_equal(orc.adc_all(lut, codes), g["expected"]["dist_all"])
    assert orc.score(q, Cf, wf, codes[2]) == g["expected"]["score_row2"]


def test_worked_example_search(orc, worked):
    g = worked
    attr = np.array(g["attr"], np.int32)
    p = _pred(**g["pred"])
    bm, npass = orc.filter_bitmap([attr], p)
    assert int(bm[0]) == g["expected"]["bitmap_word"] and npass == g["expected"]["npass"]
    ids, d, npass = orc.search(np.array(g["codes"], np.uint8), [attr],
                               np.array(g["C_pq"], np.float32),
                               np.array(g["q"], np.float32)[None], p, 4,
                               bank=np.array(g["bank"], np.float32),
                               W=np.array(g["W"], np.float32),
                               seeds=np.array(g["seeds"], np.uint64))
    assert list(ids[0]) == g["expected"]["top4_ids"]
    exp = [float(x) for x in g["expected"]["top4_dists"]]
    assert list(d[0][:3]) == exp[:3] and math.isinf(d[0][3])
    assert npass[0] == 3


# ------------------------------------------------------------ hashing

@pytest.fixture(scope="module")
def fp_golden(golden_dir):
    with open(os.path.join(golden_dir, "fingerprint_key.json")) as f:
        return json.load(f)


def test_fnv1a64_published_vectors(orc, fp_golden):
    for s, h in fp_golden["fnv1a64_vectors"].items():
        if s == "citation":
            continue
        assert orc.fnv1a64(s.encode()) == int(h, 16)


def test_splitmix64_published_sequence(orc, fp_golden):
    gamma = 0x9E3779B97F4A7C15
    outs = fp_golden["splitmix64_seed0"]["outputs"]
    for i, h in enumerate(outs):
        assert orc.splitmix64_finalize((gamma * (i + 1)) % 2**64) == int(h, 16)


def test_fingerprint_key_bytes(orc, fp_golden):
    g = fp_golden
    p = _pred(g["pred"]["col"], g["pred"]["op"], g["pred"]["lo"], g["pred"]["hi"])
    key = orc.fingerprint_key(np.array(g["q"], np.float32), p)
    assert key.hex() == g["key_hex"]


def test_fingerprint_uniform_and_seed_dependent(orc):
    rng = np.random.default_rng(7)
    B, n = 64, 6400
    seeds = np.array([11, 22], np.uint64)
    counts = np.zeros((2, B))
    same = 0
    for i in range(n):
        q = rng.standard_normal(8).astype(np.float32)
        idx = orc.fingerprint(q, _pred(0, 1, i, i + 5), seeds, B)
        counts[0, idx[0]] += 1
        counts[1, idx[1]] += 1
        same += idx[0] == idx[1]
    # chi-square with 63 dof: mean 63, sd ~11.2; 130 is beyond 5 sd
    for c in counts:
        chi2 = ((c - n / B) ** 2 / (n / B)).sum()
        assert chi2 < 130
    assert same < 3 * n / B   # two seeds act as independent hashes


def test_fingerprint_depends_on_predicate_and_query(orc):
    seeds = np.array([1, 2, 3], np.uint64)
    q = np.arange(16, dtype=np.float32)
    a = orc.fingerprint(q, _pred(0, 1, 10, 20), seeds, 1 << 30)
    b = orc.fingerprint(q, _pred(0, 1, 10, 21), seeds, 1 << 30)
    q2 = q.copy()
    q2[3] = np.nextafter(q2[3], np.float32(100))
    c = orc.fingerprint(q2, _pred(0, 1, 10, 20), seeds, 1 << 30)
    assert (a != b).all() and (a != c).all()


# ------------------------------------------------------------ alpha, w_f

def test_alpha_closed_form_and_duplicates(orc):
    B, Mr = 50, 12
    bank = np.repeat(np.arange(B, dtype=np.float32)[:, None], Mr, axis=1)  # row b = b
    for idx in ([3, 17], [5, 5], [0, 49, 7]):
        a = orc.alpha(bank, np.array(idx, np.uint32))
        np.testing.assert_array_equal(a, np.full(Mr, float(sum(idx))))


def test_softplus_fixed_points(orc):
    assert abs(orc.softplus(synth.WZ_IDENTITY) - 1.0) < 1e-15
    assert orc.softplus(0.0) == math.log(2.0)
    for x in np.linspace(-30, 30, 121):
        assert abs(orc.softplus(x) - orc.softplus(-x) - x) <= 1e-12 * max(1.0, abs(x))
    for x in np.linspace(-20, 20, 81):
        ref = math.log1p(math.exp(x))
        assert abs(orc.softplus(x) - ref) <= 1e-15 * max(1.0, ref) * 4
    assert orc.softplus(800.0) == 800.0
    assert 0.0 < orc.softplus(-700.0) < 1e-300


def test_filter_weights_identity_is_exactly_one(orc):
    np.testing.assert_array_equal(orc.filter_weights(None, 24), np.ones(24))


# ------------------------------------------------------------ conditioning

@pytest.fixture(scope="module")
def small_cb():
    rng = np.random.default_rng(3)
    M, K, ds, r = 3, 5, 2, 4
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    W = rng.standard_normal((M, r, K, ds)).astype(np.float32)
    return Cpq, W


def test_condition_zero_alpha_is_base_codebook(orc, small_cb):
    Cpq, W = small_cb
    M, r = Cpq.shape[0], W.shape[1]
    np.testing.assert_array_equal(orc.condition(Cpq, np.zeros((M, r)), W), Cpq.astype(np.float64))
    np.testing.assert_array_equal(orc.condition(Cpq, None, None), Cpq.astype(np.float64))


def test_condition_one_hot_alpha_selects_direction(orc, small_cb):
    Cpq, W = small_cb
    M, r = Cpq.shape[0], W.shape[1]
    for m in range(M):
        for j in range(r):
            a = np.zeros((M, r))
            a[m, j] = 1.0
            d = orc.condition(Cpq, a, W) - Cpq.astype(np.float64)
            for mm in range(M):
                exp = W[m, j].astype(np.float64) if mm == m else np.zeros_like(d[mm])
                np.testing.assert_allclose(d[mm], exp, rtol=0, atol=1e-6)


def test_condition_linear_in_alpha(orc, small_cb):
    Cpq, W = small_cb
    M, r = Cpq.shape[0], W.shape[1]
    rng = np.random.default_rng(5)
    a1, a2 = rng.standard_normal((M, r)), rng.standard_normal((M, r))
    base = Cpq.astype(np.float64)
    lhs = orc.condition(Cpq, a1 + a2, W) - base
    rhs = (orc.condition(Cpq, a1, W) - base) + (orc.condition(Cpq, a2, W) - base)
    np.testing.assert_allclose(lhs, rhs, rtol=1e-12, atol=1e-12)


# ------------------------------------------------------------ LUT, ADC, score

@pytest.fixture(scope="module")
def rank_case(orc):
    rng = np.random.default_rng(11)
    M, K, ds, r = 4, 16, 3, 2
    D = M * ds
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    W = rng.standard_normal((M, r, K, ds)).astype(np.float32) * 0.1
    a = rng.standard_normal((M, r))
    Cf = orc.condition(Cpq, a, W)
    q = rng.standard_normal(D).astype(np.float32)
    wz = rng.standard_normal(D).astype(np.float32)
    wf = orc.filter_weights(wz)
    codes = rng.integers(0, K, size=(200, M)).astype(np.uint8)
    return dict(M=M, K=K, ds=ds, D=D, Cf=Cf, q=q, wf=wf, codes=codes, Cpq=Cpq)


def test_adc_equals_weighted_l2_to_reconstruction(orc, rank_case):
    c = rank_case
    lut = orc.lut(c["q"], c["Cf"], c["wf"])
    dist = orc.adc_all(lut, c["codes"])
    rec = c["Cf"][np.arange(c["M"])[None, :], c["codes"]].reshape(len(c["codes"]), c["D"])
    w = c["wf"]
    ref = ((c["q"].astype(np.float64)[None, :] - rec) ** 2 * w[None, :]).sum(axis=1)
    np.testing.assert_allclose(dist, ref, rtol=1e-12)
    # the unweighted, unconditioned case is the Pre_IndexFlatL2_PQ distance
    ones = orc.filter_weights(None, c["D"])
    base = orc.condition(c["Cpq"], None, None)
    lut0 = orc.lut(c["q"], base, ones)
    rec0 = base[np.arange(c["M"])[None, :], c["codes"]].reshape(len(c["codes"]), c["D"])
    ref0 = cdist(c["q"].astype(np.float64)[None], rec0, "sqeuclidean")[0]
    np.testing.assert_allclose(orc.adc_all(lut0, c["codes"]), ref0, rtol=1e-12)


def test_printed_score_is_constant_minus_distance(orc, rank_case):
    c = rank_case
    lut = orc.lut(c["q"], c["Cf"], c["wf"])
    const = float((c["wf"] * c["q"].astype(np.float64) ** 2).sum())
    scores, dists = [], []
    for row in c["codes"]:
        s = orc.score(c["q"], c["Cf"], c["wf"], row)
        d = orc.adc(lut, row)
        assert abs((const - d) - s) <= 1e-10 * max(1.0, abs(const))
        scores.append(s)
        dists.append(d)
    # descending score order == ascending distance order
    assert list(np.argsort(-np.array(scores), kind="stable")) == \
        list(np.argsort(np.array(dists), kind="stable"))


def test_constant_weights_scale_distance(orc, rank_case):
    c = rank_case
    wz = np.full(c["D"], 1.25, np.float32)
    wf = orc.filter_weights(wz)
    lut_w = orc.lut(c["q"], c["Cf"], wf)
    lut_1 = orc.lut(c["q"], c["Cf"], orc.filter_weights(None, c["D"]))
    sp = math.log1p(math.exp(1.25))
    np.testing.assert_allclose(orc.adc_all(lut_w, c["codes"]),
                               sp * orc.adc_all(lut_1, c["codes"]), rtol=1e-12)


# ------------------------------------------------------------ top-k

def test_topk_against_library_sort(orc):
    rng = np.random.default_rng(2)
    d = rng.integers(0, 20, 500).astype(np.float64)     # many exact ties
    ids = rng.permutation(10_000)[:500].astype(np.int64)
    for k in (1, 10, 100, 500):
        oi, od = orc.topk(d, ids, k)
        order = np.lexsort((ids, d))[:k]
        np.testing.assert_array_equal(oi, ids[order])
        np.testing.assert_array_equal(od, d[order])


def test_topk_pads_when_fewer_candidates(orc):
    oi, od = orc.topk(np.array([3.0, 1.0]), np.array([7, 9]), 4)
    assert list(oi) == [9, 7, -1, -1] and od[0] == 1.0 and math.isinf(od[2])
    oi, od = orc.topk(np.zeros(0), np.zeros(0, np.int64), 3)
    assert list(oi) == [-1, -1, -1]


# ------------------------------------------------------------ filter

def test_filter_range_on_permutation_counts_exactly(orc):
    N = 1000
    perm = np.random.default_rng(4).permutation(N).astype(np.int32)
    for lo, hi in ((0, N), (10, 11), (100, 357), (500, 400), (-5, 3)):
        _, n = orc.filter_bitmap([perm], _pred(0, synth.OP_RANGE, lo, hi))
        assert n == max(0, min(hi, N) - max(lo, 0))
    bm, n = orc.filter_bitmap([perm], _pred(0, synth.OP_EQ, 123))
    assert n == 1
    row = int(np.nonzero(perm == 123)[0][0])
    assert bm[row // 32] == (1 << (row % 32))


def test_filter_operators_agree_with_their_range_forms(orc):
    a = np.random.default_rng(8).integers(-50, 50, 777).astype(np.int32)
    for v in (-51, -3, 0, 17, 49, 50):
        ge, _ = orc.filter_bitmap([a], _pred(0, synth.OP_GE, v))
        gt, _ = orc.filter_bitmap([a], _pred(0, synth.OP_GT, v))
        lt, _ = orc.filter_bitmap([a], _pred(0, synth.OP_LT, v))
        le, _ = orc.filter_bitmap([a], _pred(0, synth.OP_LE, v))
        np.testing.assert_array_equal(gt, orc.filter_bitmap([a], _pred(0, synth.OP_GE, v + 1))[0])
        np.testing.assert_array_equal(le, orc.filter_bitmap([a], _pred(0, synth.OP_LT, v + 1))[0])
        full = np.uint32(0xFFFFFFFF)
        tail = (np.uint32(1) << np.uint32(777 % 32)) - np.uint32(1)
        comp = ge ^ lt
        np.testing.assert_array_equal(comp[:-1], np.full(len(comp) - 1, full))
        assert comp[-1] == tail


def test_filter_all_pass_empty_and_tail(orc):
    a = np.arange(70, dtype=np.int32)
    p = synth.empty_predicates(1)                      # no clause: all rows pass
    bm, n = orc.filter_bitmap([a], p)
    assert n == 70 and list(bm) == [0xFFFFFFFF, 0xFFFFFFFF, 0x3F]
    bm, n = orc.filter_bitmap([a], _pred(0, synth.OP_GE, 5, more=[(0, synth.OP_LT, 3, 0)]))
    assert n == 0 and not bm.any()


def test_filter_int16_column_and_conjunction(orc):
    cat = np.array([-3, 5, 5, 7, -3, 5], np.int16)
    date = np.array([1, 2, 3, 4, 5, 6], np.int32)
    _, n = orc.filter_bitmap([date, cat], _pred(1, synth.OP_EQ, 5))
    assert n == 3
    bm, n = orc.filter_bitmap([date, cat], _pred(1, synth.OP_EQ, 5, more=[(0, synth.OP_RANGE, 3, 7)]))
    assert n == 2 and bm[0] == 0b100100
    bm, n = orc.filter_bitmap([date, cat], _pred(1, synth.OP_LT, 0))
    assert n == 2 and bm[0] == 0b010001


def test_filter_rejects_bad_clause(orc):
    a = np.arange(4, dtype=np.int32)
    with pytest.raises(ValueError):
        orc.filter_bitmap([a], _pred(1, synth.OP_EQ, 0))
    with pytest.raises(ValueError):
        orc.filter_bitmap([a], _pred(0, 9, 0))


# ------------------------------------------------------------ whole path

def test_reduces_to_plain_pq_adc(orc):
    """alpha = 0, w_f = 1 (the paper's initial state) is plain PQ ADC, whose
    ranking equals exact L2 to the reconstructions (Pre_IndexFlatL2_PQ)."""
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=3000, nq=5)
    ix = synth.pq_space_index(w)
    qs = synth.make_queries(ix, 0.5)
    ids, d, npass = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, 10)
    rec = ix.codebook[np.arange(w.M)[None, :], ix.codes].reshape(w.N, w.D).astype(np.float64)
    for i in range(5):
        bm, n = orc.filter_bitmap(ix.attrs, qs.preds[i:i + 1])
        assert n == npass[i]
        passing = np.nonzero(np.unpackbits(bm.view(np.uint8), bitorder="little")[:w.N])[0]
        full = cdist(qs.q[i:i + 1].astype(np.float64), rec[passing], "sqeuclidean")[0]
        order = np.lexsort((passing, full))[:10]
        np.testing.assert_array_equal(ids[i], passing[order])
        np.testing.assert_allclose(d[i], full[order], rtol=1e-12)


def test_search_stage_outputs_consistent(orc):
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=500, nq=3)
    ix = synth.pq_space_index(w)
    cond = synth.make_conditioning(ix)
    qs = synth.make_queries(ix, 0.5)
    ids, d, npass, st = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, 7,
                                   bank=cond.bank, W=cond.W, seeds=cond.seeds, wz=qs.wz,
                                   want_stages=True)
    for i in range(3):
        idx = orc.fingerprint(qs.q[i], qs.preds[i:i + 1], cond.seeds, w.B)
        np.testing.assert_array_equal(st["bank_idx"][i], idx)
        np.testing.assert_array_equal(st["alpha"][i], orc.alpha(cond.bank, idx))
        dist = orc.adc_all(st["lut"][i], ix.codes)
        bm, _ = orc.filter_bitmap(ix.attrs, qs.preds[i:i + 1])
        passing = np.nonzero(np.unpackbits(bm.view(np.uint8), bitorder="little")[:w.N])[0]
        order = np.lexsort((passing, dist[passing]))[:7]
        np.testing.assert_array_equal(ids[i], passing[order])


def test_exact_ground_truth_and_rerank(orc):
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=2000, nq=3)
    ix = synth.pq_space_index(w)
    X = synth.raw_vectors(ix)
    qs = synth.make_queries(ix, 0.1)
    for i in range(3):
        bm, n = orc.filter_bitmap(ix.attrs, qs.preds[i:i + 1])
        passing = np.nonzero(np.unpackbits(bm.view(np.uint8), bitorder="little")[:w.N])[0]
        gi, gd = orc.exact_topk(X, qs.q[i], bm, 10)
        ref = cdist(qs.q[i:i + 1].astype(np.float64), X[passing].astype(np.float64),
                    "sqeuclidean")[0]
        order = np.lexsort((passing, ref))[:10]
        np.testing.assert_array_equal(gi[:min(10, n)], passing[order])
        ri, rd = orc.rerank(X, qs.q[i], np.concatenate([passing, [-1]]), 10)
        np.testing.assert_array_equal(ri, gi)
        assert orc.recall(gi, gi) == 1.0


def test_recall_values(orc):
    assert orc.recall(np.array([1, 2, 3, 4]), np.array([4, 9, 1, 8])) == 0.5
    assert orc.recall(np.array([1, -1, -1]), np.array([1, -1, -1])) == 1.0
    assert orc.recall(np.array([5, 6]), np.array([7, 8])) == 0.0
    # padded ground truth: only its valid ids count
    assert orc.recall(np.array([1, 2, 3]), np.array([1, -1, -1])) == 1.0
    assert orc.recall(np.array([7, 2, 3]), np.array([1, 2, -1])) == 0.5


# ------------------------------------------------------------ PQ construction

def test_kmeans_objective_non_increasing_and_encode_is_argmin(orc):
    rng = np.random.default_rng(9)
    X = rng.standard_normal((600, 8)).astype(np.float32)
    Cq, obj = orc.kmeans_pq(X, 2, 16, 8, 123)
    assert (np.diff(obj, axis=1) <= 1e-9 * obj[:, :-1]).all()
    codes = orc.pq_encode(X, Cq)
    for m in range(2):
        d = cdist(X[:, m * 4:(m + 1) * 4].astype(np.float64), Cq[m], "sqeuclidean")
        np.testing.assert_array_equal(codes[:, m], d.argmin(axis=1))
    rec = np.stack([orc.reconstruct(Cq, c) for c in codes[:5]])
    np.testing.assert_array_equal(rec[:, :4], Cq[0][codes[:5, 0]])


def test_encode_ties_go_to_the_smaller_codeword(orc):
    # codewords 1 and 3 coincide; points on them must take codeword 1
    Cq = np.zeros((1, 4, 2))
    Cq[0] = [[5.0, 5.0], [1.0, 2.0], [9.0, 9.0], [1.0, 2.0]]
    X = np.array([[1.0, 2.0], [1.25, 2.0], [9.0, 9.0]], np.float32)
    np.testing.assert_array_equal(orc.pq_encode(X, Cq)[:, 0], [1, 1, 2])


def test_exact_distance_closed_form(orc):
    X = np.array([[0, 0, 0], [1, 2, 2], [3, 0, 4]], np.float32)
    gi, gd = orc.exact_topk(X, np.zeros(3, np.float32), None, 3)
    assert list(gi) == [0, 1, 2] and list(gd) == [0.0, 9.0, 25.0]
    ri, rd = orc.rerank(X, np.zeros(3, np.float32), np.array([2, -1, 1]), 2)
    assert list(ri) == [1, 2] and list(rd) == [9.0, 25.0]


def test_kmeans_exact_when_codewords_cover_distinct_points(orc):
    rng = np.random.default_rng(10)
    distinct = rng.standard_normal((20, 4)).astype(np.float32)
    X = distinct[rng.integers(0, 20, 300)]
    Cq, obj = orc.kmeans_pq(X, 1, 32, 10, 5)
    assert obj[0, -1] == 0.0


def test_kmeans_one_codeword_is_the_mean(orc):
    """K = 1: whatever row seeds it, one Lloyd iteration moves the codeword
    to the mean of the subspace's rows, and every later assignment costs the
    total sum of squares about that mean (textbook closed forms)."""
    rng = np.random.default_rng(31)
    X = (3.0 + 2.0 * rng.standard_normal((257, 6))).astype(np.float32)
    for seed in (0, 7, 123):
        Cq, obj = orc.kmeans_pq(X, 3, 1, 4, seed)
        x = X.astype(np.float64)
        for m in range(3):
            sub = x[:, 2 * m:2 * m + 2]
            mean = sub.mean(axis=0)
            np.testing.assert_allclose(Cq[m, 0], mean, rtol=1e-13, atol=0)
            ss = ((sub - mean) ** 2).sum()
            np.testing.assert_allclose(obj[m, 1:], ss, rtol=1e-12)
            assert obj[m, 0] >= ss


def test_kmeans_two_separated_groups_converge_to_the_group_means(orc):
    """K = 2 on two groups far apart (spread 0.1, distance 100): from any
    seeded start, including both seeds in one group, Lloyd's iteration ends
    at the two group means, with the within-group sum of squares as its
    objective."""
    rng = np.random.default_rng(32)
    a = (0.1 * rng.standard_normal((60, 2))).astype(np.float32)
    b = (np.array([100.0, -50.0]) + 0.1 * rng.standard_normal((25, 2))).astype(np.float32)
    X = np.concatenate([a, b])[rng.permutation(85)]
    x = X.astype(np.float64)
    ga = x[np.abs(x[:, 0]) < 50]
    gb = x[np.abs(x[:, 0]) >= 50]
    want = np.stack([ga.mean(axis=0), gb.mean(axis=0)])
    ss = ((ga - ga.mean(axis=0)) ** 2).sum() + ((gb - gb.mean(axis=0)) ** 2).sum()
    for seed in range(12):
        Cq, obj = orc.kmeans_pq(X, 1, 2, 8, seed)
        got = Cq[0][np.argsort(Cq[0][:, 0])]
        np.testing.assert_allclose(got, want, rtol=1e-12, atol=1e-12)
        np.testing.assert_allclose(obj[0, -1], ss, rtol=1e-12)


def test_sdc_properties(orc):
    rng = np.random.default_rng(12)
    Cq = rng.standard_normal((3, 8, 2))
    a = np.array([1, 5, 7], np.uint8)
    b = np.array([2, 5, 0], np.uint8)
    assert orc.sdc(Cq, a, a) == 0.0
    assert orc.sdc(Cq, a, b) == orc.sdc(Cq, b, a)
    ra, rb = orc.reconstruct(Cq, a), orc.reconstruct(Cq, b)
    assert abs(orc.sdc(Cq, a, b) - cdist(ra[None], rb[None], "sqeuclidean")[0, 0]) < 1e-12


# ------------------------------------------------------------ float32 encoding, Lloyd step

def test_encode_f32_agrees_with_fp64_away_from_ties(orc):
    rng = np.random.default_rng(21)
    X = rng.standard_normal((800, 16)).astype(np.float32)
    Cq = rng.standard_normal((2, 64, 8)).astype(np.float32)
    c32, d32 = orc.pq_encode_f32(X, Cq)
    c64 = orc.pq_encode(X, Cq.astype(np.float64))
    for m in range(2):
        d = cdist(X[:, m * 8:(m + 1) * 8].astype(np.float64), Cq[m].astype(np.float64), "sqeuclidean")
        srt = np.sort(d, axis=1)
        clear = (srt[:, 1] - srt[:, 0]) > 1e-5 * srt[:, 1]
        np.testing.assert_array_equal(c32[clear, m], c64[clear, m])
        np.testing.assert_allclose(d32[:, m], srt[:, 0], rtol=2e-6)
    assert clear.mean() > 0.99


def test_encode_f32_rounds_every_operation(orc):
    """x = (2^-12, 1 + 2^-12) against the zero codeword: the squares are
    2^-24 and 1 + 2^-11 + 2^-24; rounding the second square to float32 (a
    tie, to even) gives 1 + 2^-11, and adding 2^-24 ties back to 1 + 2^-11.
    A fused multiply-add would give 1 + 2^-11 + 2^-23 instead."""
    X = np.array([[2.0 ** -12, 1.0 + 2.0 ** -12]], np.float32)
    Cq = np.zeros((1, 1, 2), np.float32)
    _, dmin = orc.pq_encode_f32(X, Cq)
    assert float(dmin[0, 0]) == 1.0 + 2.0 ** -11


def test_encode_f32_ties_to_smaller_codeword(orc):
    Cq = np.array([[[5, 5], [1, 2], [9, 9], [1, 2]]], np.float32)
    X = np.array([[1.0, 2.0], [1.25, 2.0], [9.0, 9.0]], np.float32)
    codes, dmin = orc.pq_encode_f32(X, Cq)
    assert list(codes[:, 0]) == [1, 1, 2] and list(dmin[:, 0]) == [0.0, 0.0625, 0.0]


def test_lloyd_step_is_the_member_mean(orc):
    rng = np.random.default_rng(22)
    X = rng.standard_normal((500, 8)).astype(np.float32)
    C0 = X[rng.choice(500, 16, replace=False)].reshape(16, 2, 4).transpose(1, 0, 2).copy()
    C1, codes, obj = orc.lloyd_step(X, C0)
    c_ref, d_ref = orc.pq_encode_f32(X, C0)
    np.testing.assert_array_equal(codes, c_ref)
    np.testing.assert_allclose(obj, d_ref.astype(np.float64).sum(axis=0), rtol=1e-12)
    for m in range(2):
        sub = X[:, m * 4:(m + 1) * 4].astype(np.float64)
        cnt = np.bincount(codes[:, m], minlength=16)
        for k in range(16):
            if cnt[k]:
                np.testing.assert_array_equal(C1[m, k], sub[codes[:, m] == k].mean(axis=0).astype(np.float32))


def test_lloyd_step_reseeds_empty_codeword_with_farthest_point(orc):
    X = np.array([[0.0], [1.0], [10.0], [10.5]], np.float32)
    C0 = np.array([[[0.0], [10.0], [1000.0]]], np.float32)   # codeword 2 gets nobody
    C1, codes, obj = orc.lloyd_step(X, C0)
    assert list(codes[:, 0]) == [0, 0, 1, 1]
    # means 0.5 and 10.25; the farthest point is row 1 or row 3 (distance
    # 1.0 vs 0.25): row 1 (x = 1.0) becomes codeword 2
    np.testing.assert_array_equal(C1[0, :, 0], [0.5, 10.25, 1.0])
    assert obj[0] == 0.0 + 1.0 + 0.0 + 0.25


def test_lloyd_steps_do_not_increase_the_objective(orc):
    rng = np.random.default_rng(23)
    X = (rng.standard_normal((600, 8)) + rng.integers(0, 4, (600, 1)) * 3).astype(np.float32)
    C = X[:12].reshape(12, 2, 4).transpose(1, 0, 2).copy()
    last = None
    for _ in range(6):
        C, _, obj = orc.lloyd_step(X, C)
        if last is not None:
            assert (obj <= last * (1 + 1e-6)).all()
        last = obj
