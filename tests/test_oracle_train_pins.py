"""Pins of the oracle's training step (§2 "Learning"): gradients against
central finite differences of the loss, closed forms of the loss, the
initial state, hard negatives against a brute force over the pool, and the
SGD update.  CPU only."""
import math

import numpy as np
import pytest
from scipy.spatial.distance import cdist


def _grid(a, step=2.0 ** -8):
    """float32 values on a coarse grid, so that +-2^-12 stays exact."""
    return (np.round(np.asarray(a, np.float64) / step) * step).astype(np.float32)


def tiny(orc, seed=0, N=300, M=4, K=8, ds=2, r=3, B=16, h=2, nq=3, bank_scale=0.5):
    rng = np.random.default_rng(seed)
    D = M * ds
    codes = rng.integers(0, K, size=(N, M), dtype=np.uint8)
    attr = rng.integers(0, 100, size=N, dtype=np.int32)
    C_pq = _grid(rng.standard_normal((M, K, ds)))
    bank = _grid(rng.standard_normal((B, M * r)) * bank_scale)
    W = _grid(rng.standard_normal((M, r, K, ds)) * 0.25)
    seeds = rng.integers(0, 2 ** 63, size=h, dtype=np.int64).astype(np.uint64)
    wz = _grid(rng.standard_normal(D) * 0.5 + 0.5)
    q = _grid(rng.standard_normal((nq, D)))
    preds = np.zeros(nq, orc.PREDICATE_DTYPE)
    for i in range(nq):
        preds[i]["n_clauses"] = 1
        lo = int(rng.integers(0, 50))
        preds[i]["c"][0] = (0, orc.RANGE, lo, lo + 40)
    return dict(codes=codes, cols=[attr], C_pq=C_pq, bank=bank, W=W, seeds=seeds, wz=wz,
                queries=q, preds=preds)


def _cand(t, P, V, seed=1):
    rng = np.random.default_rng(seed)
    nq = len(t["queries"])
    c = np.stack([rng.choice(len(t["codes"]), V, replace=False) for _ in range(nq)]).astype(np.int64)
    return c


def _loss(orc, t, cand, P, tau, lam, **over):
    a = dict(t, **over)
    return orc.train_loss(a["codes"], a["C_pq"], a["bank"], a["W"], a["seeds"], a["wz"],
                          a["queries"], a["preds"], cand, P, tau, lam, grads=False)


def test_gradients_match_central_differences(orc):
    t = tiny(orc)
    P, V, tau, lam = 2, 7, 0.7, 0.3
    cand = _cand(t, P, V)
    cand[0, 5] = -1                      # an absent negative
    cand[1, 1] = -1                      # an absent positive
    cand[2, :P] = -1                     # a query without positives: anchor only
    L, gb, gW, gz = orc.train_loss(t["codes"], t["C_pq"], t["bank"], t["W"], t["seeds"], t["wz"],
                                   t["queries"], t["preds"], cand, P, tau, lam)
    eps = 2.0 ** -12
    for name, g in (("bank", gb), ("W", gW), ("wz", gz)):
        base = t[name]
        flat = base.reshape(-1)
        scale = np.abs(g).max()
        assert scale > 0
        for e in range(flat.size):
            up, dn = flat.copy(), flat.copy()
            up[e] += np.float32(eps)
            dn[e] -= np.float32(eps)
            assert float(up[e]) - float(flat[e]) == eps and float(flat[e]) - float(dn[e]) == eps
            fd = (_loss(orc, t, cand, P, tau, lam, **{name: up.reshape(base.shape)}) -
                  _loss(orc, t, cand, P, tau, lam, **{name: dn.reshape(base.shape)})) / (2 * eps)
            assert abs(fd - g.reshape(-1)[e]) <= 1e-6 * scale + 1e-6 * abs(fd), (name, e, fd, g.reshape(-1)[e])


def test_equal_distances_give_log_one_plus_n(orc):
    """One positive and n negatives at the same distance (identical codes):
    each softmax share is 1/(n+1), so L = log(n + 1); bank = 0 gives Delta = 0."""
    t = tiny(orc, seed=2)
    t["bank"] = np.zeros_like(t["bank"])
    t["codes"][:8] = t["codes"][0]
    for n in range(0, 7):
        cand = np.tile(np.arange(1 + n, dtype=np.int64), (3, 1))
        for tau in (0.1, 1.0, 25.0):
            L = _loss(orc, t, cand, 1, tau, 0.7)
            assert abs(L - math.log(n + 1)) < 1e-12


def test_two_positives_average_and_far_negatives_vanish(orc):
    """Two positives at the same distance as n negatives: each term is
    log(n + 1), so their mean is too.  A negative far beyond the positive
    (distance gap 1, tau = 1e-3) leaves L = 0 to double precision; one
    closer by a gap g gives L = g / tau + log(1 + exp(-g / tau)) -> g / tau."""
    t = tiny(orc, seed=3)
    t["bank"] = np.zeros_like(t["bank"])
    t["codes"][:6] = t["codes"][0]
    cand = np.tile(np.arange(6, dtype=np.int64), (3, 1))
    assert abs(_loss(orc, t, cand, 2, 0.5, 0.0) - math.log(5)) < 1e-12
    # row 10: code 0 everywhere; row 11: code 1 everywhere; one codebook with
    # C[m][1] = C[m][0] + (1, 0): distance gap exactly 1 * w for every query
    t["codes"][10] = 0
    t["codes"][11] = 1
    t["C_pq"][:, 1] = t["C_pq"][:, 0]
    t["C_pq"][0, 1, 0] += np.float32(1.0)
    t["wz"][:] = np.float32(math.log(math.e - 1))      # w_f = 1 (to 1e-8)
    for qi in range(3):
        t["queries"][qi] = t["C_pq"][:, 0].reshape(-1)   # the query sits on codeword 0
    near = np.array([[10, 11]] * 3, np.int64)          # positive at 0, negative at ~1
    far = np.array([[11, 10]] * 3, np.int64)           # positive at ~1, negative at 0
    assert _loss(orc, t, near, 1, 1e-3, 0.0) < 1e-300
    Lf = _loss(orc, t, far, 1, 1e-3, 0.0)
    assert abs(Lf - 1e3) < 1e-4                        # 1/tau * gap, gap = w_f ~ 1 - 1e-8


def test_anchor_of_a_one_hot_alpha(orc):
    """No positives: L = lambda ||Delta||^2.  With alpha = a e_{m,j},
    Delta[m] = a W[m, j] and zero elsewhere, so L = lambda a^2 ||W[m,j]||^2."""
    t = tiny(orc, seed=4, nq=1)
    idx = orc.fingerprint(t["queries"][0], t["preds"][0], t["seeds"], len(t["bank"]))
    M, r = t["W"].shape[:2]
    cand = np.full((1, 3), -1, np.int64)
    for m, j, a in ((0, 0, 0.5), (2, 1, -1.25), (3, 2, 2.0)):
        bank = np.zeros_like(t["bank"])
        bank[idx[0], m * r + j] = np.float32(a)
        mult = 2.0 if idx[0] == idx[1] else 1.0
        expect = 0.3 * (mult * a) ** 2 * float(np.sum(t["W"][m, j].astype(np.float64) ** 2))
        L = _loss(orc, t, cand, 1, 1.0, 0.3, bank=bank)
        assert abs(L - expect) <= 1e-12 * expect


def test_initial_state(orc):
    """alpha = 0 (zero bank): the W gradient is exactly zero (dL/dW = alpha
    x dL/dDelta), the anchor vanishes, and only fetched bank rows move."""
    t = tiny(orc, seed=5)
    t["bank"] = np.zeros_like(t["bank"])
    t["wz"][:] = np.float32(math.log(math.e - 1))
    cand = _cand(t, 2, 6, seed=9)
    L, gb, gW, gz = orc.train_loss(t["codes"], t["C_pq"], t["bank"], t["W"], t["seeds"], t["wz"],
                                   t["queries"], t["preds"], cand, 2, 0.5, 10.0)
    assert (gW == 0).all()
    fetched = set()
    for qi in range(3):
        fetched.update(int(i) for i in orc.fingerprint(t["queries"][qi], t["preds"][qi],
                                                       t["seeds"], len(t["bank"])))
    moved = set(np.nonzero(np.abs(gb).sum(1))[0].tolist())
    assert moved and moved <= fetched
    assert np.abs(gz).sum() > 0
    L0 = _loss(orc, t, cand, 2, 0.5, 0.0)
    assert abs(L - L0) < 1e-15 * max(1.0, abs(L))     # anchor = 0


def _recon(C_pq, codes):
    M = codes.shape[1]
    return np.concatenate([C_pq[m][codes[:, m]] for m in range(M)], axis=1).astype(np.float64)


@pytest.mark.parametrize("n_neg", [1, 5, 40])
def test_negatives_are_the_best_non_positive_pool_rows(orc, n_neg):
    """At alpha = 0 and w_f = 1 the distance is the squared L2 to the
    reconstruction (scipy cdist); the negatives are the pool rows outside
    the positives in increasing distance, the first n_neg, -1 padded.  The
    float32 w_z = ln(e - 1) makes w_f = 1 - O(1e-8), which can reorder rows
    whose exact distances tie, so the distance sequence is compared and the
    ids are checked to be distinct non-positive pool rows."""
    t = tiny(orc, seed=6, N=400, K=4)
    t["bank"] = np.zeros_like(t["bank"])
    t["wz"][:] = np.float32(math.log(math.e - 1))
    t["C_pq"] = np.round(t["C_pq"] * 4).astype(np.float32)      # integer codebook: exact distances
    t["queries"] = np.round(t["queries"] * 4).astype(np.float32)
    t["preds"]["c"][2, 0]["hi"] = t["preds"]["c"][2, 0]["lo"] + 3   # a small pool
    rec = _recon(t["C_pq"], t["codes"])
    attr = t["cols"][0].astype(np.int64)
    rng = np.random.default_rng(7)
    P = 3
    pos = np.full((3, P), -1, np.int64)
    pools, dists = [], []
    for qi in range(3):
        c = t["preds"]["c"][qi, 0]
        pool = np.nonzero((attr >= c["lo"]) & (attr < c["hi"]))[0]
        d = cdist(t["queries"][qi:qi + 1].astype(np.float64), rec, "sqeuclidean")[0]
        order = pool[np.lexsort((pool, d[pool]))]
        k = min(P, len(order))
        pos[qi, :k] = rng.permutation(order[: 2 * P])[:k]
        pools.append(set(pool.tolist()))
        dists.append(d)
    neg = orc.mine_negatives(t["codes"], t["cols"], t["C_pq"], t["bank"], t["W"], t["seeds"],
                             t["wz"], t["queries"], t["preds"], pos, n_neg)
    for qi in range(3):
        rest = sorted(i for i in pools[qi] if i not in set(pos[qi].tolist()))
        exp_d = np.sort(dists[qi][rest])[:n_neg]
        got = [int(i) for i in neg[qi] if i >= 0]
        assert len(got) == len(exp_d) and all(i == -1 for i in neg[qi][len(got):])
        assert len(set(got)) == len(got)
        assert all(i in pools[qi] and i not in set(pos[qi].tolist()) for i in got)
        np.testing.assert_array_equal(dists[qi][got], exp_d)
    if n_neg == 40:
        assert (neg[2] == -1).any()                               # the small pool ran out


def test_sgd_step_is_the_gradient_step_and_descends(orc):
    t = tiny(orc, seed=8)
    P, n_neg, tau, lam, lr = 2, 6, 0.8, 0.05, 1e-3
    pos = np.stack([np.arange(P) + 7 * qi for qi in range(3)]).astype(np.int64)
    L, b2, W2, z2, neg = orc.train_step(t["codes"], t["cols"], t["C_pq"], t["bank"], t["W"],
                                        t["seeds"], t["wz"], t["queries"], t["preds"], pos,
                                        n_neg, tau, lam, lr)
    np.testing.assert_array_equal(neg, orc.mine_negatives(
        t["codes"], t["cols"], t["C_pq"], t["bank"], t["W"], t["seeds"], t["wz"], t["queries"],
        t["preds"], pos, n_neg))
    cand = np.concatenate([pos, neg], axis=1)
    L1, gb, gW, gz = orc.train_loss(t["codes"], t["C_pq"], t["bank"], t["W"], t["seeds"], t["wz"],
                                    t["queries"], t["preds"], cand, P, tau, lam)
    assert L == L1
    np.testing.assert_array_equal(b2, (t["bank"] - lr * gb).astype(np.float32))
    np.testing.assert_array_equal(W2, (t["W"] - lr * gW).astype(np.float32))
    np.testing.assert_array_equal(z2, (t["wz"] - lr * gz).astype(np.float32))
    L2 = _loss(orc, t, cand, P, tau, lam, bank=b2, W=W2, wz=z2)
    assert L2 < L
    # a step size of its own for w_z: 0 keeps it, bank and W move as before
    _, b3, W3, z3, _ = orc.train_step(t["codes"], t["cols"], t["C_pq"], t["bank"], t["W"],
                                      t["seeds"], t["wz"], t["queries"], t["preds"], pos,
                                      n_neg, tau, lam, lr, lr_wz=0.0)
    np.testing.assert_array_equal(z3, t["wz"])
    np.testing.assert_array_equal(b3, b2)
    np.testing.assert_array_equal(W3, W2)
