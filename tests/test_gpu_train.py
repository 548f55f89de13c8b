"""Training of the bank, W and w_f on the GPU (§2 "Learning") against the
oracle: the loss and every gradient for the same candidates, hard-negative
mining, a whole SGD step, the initial state, determinism, device I/O and the
argument errors.

Tolerances: the GPU sums float32 distance terms in fp64 (relative error of
a distance ~1e-7, so the softmax weights move by ~1e-7 x dist / tau ~ 3e-6
at dist ~ 250, tau = 8) and accumulates gradients in float32 over at most a
few thousand terms; each gradient array is compared element by element
against the fp64 oracle within 2e-4 of that array's largest magnitude, the
loss within 1e-6 relative."""
import math

import numpy as np
import pytest

from paper_2607_22922_gb300 import synth

pytestmark = pytest.mark.gpu

P, NNEG, TAU, LAM = 10, 32, 8.0, 0.01
GRAD_TOL = 2e-4


@pytest.fixture(scope="module")
def ifvs():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs as mod
    return mod


class Case:
    def __init__(self, orc, n=5000, nq=8, sel=0.1, zero_bank=False, salt=0, r=None):
        w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=n)
        if r is not None:
            w = synth.scaled(w, r=r)
        self.w = w
        self.ix = synth.pq_space_index(w)
        self.cond = synth.make_conditioning(self.ix)
        self.qs = synth.make_queries(self.ix, sel, nq=nq, salt=salt)
        self.X = synth.raw_vectors(self.ix)
        self.bank = np.zeros_like(self.cond.bank) if zero_bank else self.cond.bank.copy()
        self.W = self.cond.W.copy()
        self.wz = self.qs.wz[0].copy()
        # positives: the exact filtered top-P over the raw vectors (§3.1)
        self.pos = np.full((nq, P), -1, np.int64)
        for i in range(nq):
            bm, _ = orc.filter_bitmap(self.ix.attrs, self.qs.preds[i])
            self.pos[i], _ = orc.exact_topk(self.X, self.qs.q[i], bm, P)

    def index(self, ifvs):
        g = ifvs.Index(self.ix.codes, self.ix.attrs, D=self.w.D, K=self.w.K)
        g.load_codebooks(self.ix.codebook, bank=self.bank, W=self.W, hash_seeds=self.cond.seeds)
        return g

    def oracle_negatives(self, orc, n_neg=NNEG):
        return orc.mine_negatives(self.ix.codes, self.ix.attrs, self.ix.codebook, self.bank, self.W,
                                  self.cond.seeds, self.wz, self.qs.q, self.qs.preds, self.pos, n_neg)

    def oracle_loss(self, orc, cand, tau=TAU, lam=LAM):
        return orc.train_loss(self.ix.codes, self.ix.codebook, self.bank, self.W, self.cond.seeds,
                              self.wz, self.qs.q, self.qs.preds, cand, P, tau, lam)


def _close(g, o, tol=GRAD_TOL):
    scale = np.abs(o).max()
    err = np.abs(g.astype(np.float64) - o).max()
    assert err <= tol * scale, (err, scale)


@pytest.fixture(scope="module")
def case(orc):
    return Case(orc)


def test_gradients_match_the_oracle(ifvs, orc, case):
    cand = np.concatenate([case.pos, case.oracle_negatives(orc)], 1)
    cand[1, 3] = -1                       # an absent positive
    cand[2, P + 5] = -1                   # an absent negative
    cand[3, :P] = -1                      # no positives: anchor only
    L, gb, gW, gz = case.oracle_loss(orc, cand)
    g = case.index(ifvs)
    Lg, gbg, gWg, gzg = g.train_grad(case.qs.q, case.qs.preds, case.wz, cand, P, TAU, LAM)
    assert abs(Lg - L) <= 1e-6 * abs(L)
    _close(gbg, gb)
    _close(gWg, gW)
    _close(gzg, gz)
    # rows no query fetched stay exactly zero
    untouched = np.abs(gb).sum(1) == 0
    assert (gbg[untouched] == 0).all()


@pytest.mark.parametrize("tau,lam", [(0.5, 0.0), (2.0, 1.0), (64.0, 0.1)])
def test_gradients_across_temperatures(ifvs, orc, case, tau, lam):
    cand = np.concatenate([case.pos, case.oracle_negatives(orc)], 1)
    L, gb, gW, gz = case.oracle_loss(orc, cand, tau, lam)
    g = case.index(ifvs)
    Lg, gbg, gWg, gzg = g.train_grad(case.qs.q, case.qs.preds, case.wz, cand, P, tau, lam)
    assert abs(Lg - L) <= 1e-6 * abs(L)
    # at tau = 0.5 the weights are 2x more sensitive to distance rounding
    tol = GRAD_TOL * (4 if tau < 1 else 1)
    _close(gbg, gb, tol)
    _close(gWg, gW, tol)
    _close(gzg, gz, tol)


@pytest.mark.parametrize("r", [1, 12, 32])
def test_gradients_for_other_ranks(ifvs, orc, r):
    """r = 1 and r > 8 run the kernels' wide-accumulator variants."""
    c = Case(orc, n=3000, nq=6, salt=4, r=r)
    cand = np.concatenate([c.pos, c.oracle_negatives(orc)], 1)
    L, gb, gW, gz = c.oracle_loss(orc, cand)
    g = c.index(ifvs)
    Lg, gbg, gWg, gzg = g.train_grad(c.qs.q, c.qs.preds, c.wz, cand, P, TAU, LAM)
    assert abs(Lg - L) <= 1e-6 * abs(L)
    _close(gbg, gb)
    _close(gWg, gW)
    _close(gzg, gz)


def _oracle_pool_dists(orc, case, i, bank, W, wz):
    _, _, _, st = orc.search(case.ix.codes, case.ix.attrs, case.ix.codebook, case.qs.q[i:i + 1],
                             case.qs.preds[i:i + 1], 1, bank=bank, W=W, seeds=case.cond.seeds,
                             wz=wz[None, :], want_stages=True)
    return orc.adc_all(st["lut"][0], case.ix.codes)


def _check_negatives(orc, case, neg, bank, W, wz, n_neg=NNEG):
    """The GPU's negatives are distinct non-positive pool rows whose oracle
    distances are the n_neg smallest of the pool outside the positives
    (rows may differ only among distances within 2e-5 relative)."""
    for i in range(len(neg)):
        bm, _ = orc.filter_bitmap(case.ix.attrs, case.qs.preds[i])
        rows = np.nonzero(np.unpackbits(bm.view(np.uint8), bitorder="little")[:case.w.N])[0]
        pos = set(case.pos[i].tolist())
        rest = np.array([r for r in rows if r not in pos], np.int64)
        d = _oracle_pool_dists(orc, case, i, bank, W, wz)
        best = np.sort(d[rest])[:n_neg]
        got = [int(x) for x in neg[i] if x >= 0]
        assert len(got) == len(best) and len(set(got)) == len(got)
        assert all(x in set(rest.tolist()) for x in got)
        np.testing.assert_allclose(np.sort(d[got]), best, rtol=2e-5)


def test_mining_and_a_zero_step(ifvs, orc, case):
    """lr = 0: the step only mines and evaluates; the parameters stay put."""
    g = case.index(ifvs)
    wz = case.wz.copy()
    L, neg = g.train_step(case.qs.q, case.qs.preds, wz, case.pos, NNEG, TAU, LAM, 0.0)
    _check_negatives(orc, case, neg, case.bank, case.W, case.wz)
    Lo = case.oracle_loss(orc, np.concatenate([case.pos, neg], 1))[0]
    assert abs(L - Lo) <= 1e-6 * abs(Lo)
    b, W = g.conditioning()
    np.testing.assert_array_equal(b, case.bank)
    np.testing.assert_array_equal(W, case.W)
    np.testing.assert_array_equal(wz, case.wz)


def test_one_step_matches_the_oracle(ifvs, orc, case):
    lr = 0.05
    g = case.index(ifvs)
    wz = case.wz.copy()
    L, neg = g.train_step(case.qs.q, case.qs.preds, wz, case.pos, NNEG, TAU, LAM, lr)
    Lo, b2, W2, z2, neg_o = orc.train_step(case.ix.codes, case.ix.attrs, case.ix.codebook, case.bank,
                                           case.W, case.cond.seeds, case.wz, case.qs.q,
                                           case.qs.preds, case.pos, NNEG, TAU, LAM, lr)
    np.testing.assert_array_equal(neg, neg_o)      # no near-ties on this case
    assert abs(L - Lo) <= 1e-6 * abs(Lo)
    b, W = g.conditioning()
    _, gb, gW, gz = case.oracle_loss(orc, np.concatenate([case.pos, neg_o], 1))
    for new, ref, grad in ((b, b2, gb), (W, W2, gW), (wz, z2, gz)):
        bound = lr * GRAD_TOL * np.abs(grad).max() + np.spacing(np.abs(ref).astype(np.float32))
        assert (np.abs(new.astype(np.float64) - ref) <= bound).all()


def test_initial_state_moves_only_the_bank_and_w_z(ifvs, orc):
    """alpha = 0 (zero bank): dL/dW is exactly 0 (alpha x dL/dDelta and the
    anchor's A_m both vanish), so the first step leaves W unchanged."""
    c = Case(orc, zero_bank=True, salt=1)
    g = c.index(ifvs)
    cand = np.concatenate([c.pos, c.oracle_negatives(orc)], 1)
    _, gb, gW, gz = g.train_grad(c.qs.q, c.qs.preds, c.wz, cand, P, TAU, 1.0)
    assert (gW == 0).all() and np.abs(gb).max() > 0 and np.abs(gz).max() > 0
    wz = c.wz.copy()
    g.train_step(c.qs.q, c.qs.preds, wz, c.pos, NNEG, TAU, 1.0, 0.1)
    b, W = g.conditioning()
    np.testing.assert_array_equal(W, c.W)
    assert not np.array_equal(b, c.bank) and not np.array_equal(wz, c.wz)


def test_frozen_w_z_step_matches_the_oracle(ifvs, orc, case):
    """lr_wz = 0 keeps w_f where it is while the bank and W take their step."""
    lr = 0.5
    g = case.index(ifvs)
    wz = case.wz.copy()
    g.train_step(case.qs.q, case.qs.preds, wz, case.pos, NNEG, TAU, LAM, lr, lr_wz=0.0)
    _, b2, W2, z2, neg_o = orc.train_step(case.ix.codes, case.ix.attrs, case.ix.codebook, case.bank,
                                          case.W, case.cond.seeds, case.wz, case.qs.q,
                                          case.qs.preds, case.pos, NNEG, TAU, LAM, lr, lr_wz=0.0)
    np.testing.assert_array_equal(wz, case.wz)
    np.testing.assert_array_equal(z2, case.wz)
    b, W = g.conditioning()
    _, gb, gW, _ = case.oracle_loss(orc, np.concatenate([case.pos, neg_o], 1))
    for new, ref, grad in ((b, b2, gb), (W, W2, gW)):
        bound = lr * GRAD_TOL * np.abs(grad).max() + np.spacing(np.abs(ref).astype(np.float32))
        assert (np.abs(new.astype(np.float64) - ref) <= bound).all()


def test_training_raises_recall_on_its_batch(ifvs, orc):
    """Repeated steps on one mini-batch from the paper's initial state (zero
    bank, w_f = 1 held fixed), negatives re-mined each step: the loss falls
    and the search ranks more of the ground truth into the top P."""
    c = Case(orc, zero_bank=True, salt=2, nq=16)
    g = c.index(ifvs)
    wz = c.wz.copy()

    def recall():
        ids, _, _ = g.search(c.qs.q, c.qs.preds, P, wz=np.tile(wz, (len(c.qs.q), 1)))
        return np.mean([len(np.intersect1d(a[a >= 0], b)) / max(1, (a >= 0).sum())
                        for a, b in zip(c.pos, ids)])

    r0 = recall()
    losses = [g.train_step(c.qs.q, c.qs.preds, wz, c.pos, NNEG, TAU, 0.001, 5.0, lr_wz=0.0)[0]
              for _ in range(30)]
    r1 = recall()
    assert losses[-1] < 0.8 * losses[0], losses
    assert r1 > r0 + 0.05, (r0, r1)


def test_deterministic_and_device_io(ifvs, orc, case):
    import torch
    cand = np.concatenate([case.pos, case.oracle_negatives(orc)], 1)
    g = case.index(ifvs)
    a = g.train_grad(case.qs.q, case.qs.preds, case.wz, cand, P, TAU, LAM)
    b = g.train_grad(case.qs.q, case.qs.preds, case.wz, cand, P, TAU, LAM)
    assert a[0] == b[0]
    for x, y in zip(a[1:], b[1:]):
        np.testing.assert_array_equal(x, y)
    dev = torch.device("cuda", 0)
    t = lambda x: torch.from_numpy(np.ascontiguousarray(x)).to(dev)
    pv = t(case.qs.preds.view(np.uint8).copy())
    B, Mr = case.bank.shape
    gb = torch.empty((B, Mr), dtype=torch.float32, device=dev)
    gW = torch.empty(case.W.shape, dtype=torch.float32, device=dev)
    gz = torch.empty(case.wz.shape, dtype=torch.float32, device=dev)
    s = torch.cuda.Stream(device=dev)
    L, _, _, _ = ifvs.ifvs_train_grad(g.h, t(case.qs.q), pv, t(case.wz), t(cand), P, TAU, LAM, B, Mr,
                                      case.W.shape, flags=ifvs.IFVS_F_DEVICE_IO, stream=s.cuda_stream,
                                      g_bank=gb, g_W=gW, g_wz=gz)
    assert L == a[0]
    np.testing.assert_array_equal(gb.cpu().numpy(), a[1])
    np.testing.assert_array_equal(gW.cpu().numpy(), a[2])
    np.testing.assert_array_equal(gz.cpu().numpy(), a[3])


def test_small_pool_and_no_negatives(ifvs, orc):
    """A pool smaller than P + n_neg pads the negatives with -1; n_neg = 0
    leaves only the anchor (each positive's softmax is over itself)."""
    c = Case(orc, n=3000, nq=4, sel=0.01, salt=3)
    g = c.index(ifvs)
    wz = c.wz.copy()
    L, neg = g.train_step(c.qs.q, c.qs.preds, wz, c.pos, 64, TAU, LAM, 0.0)
    _check_negatives(orc, c, neg, c.bank, c.W, c.wz, n_neg=64)
    assert (neg == -1).any()
    cand0 = c.pos.copy()
    L0, _, _, _ = g.train_grad(c.qs.q, c.qs.preds, c.wz, cand0, P, TAU, LAM)
    Lo0 = c.oracle_loss(orc, cand0)[0]
    assert abs(L0 - Lo0) <= 1e-6 * abs(Lo0)


def test_argument_errors(ifvs, orc, case):
    g = case.index(ifvs)
    cand = np.concatenate([case.pos, case.oracle_negatives(orc)], 1)
    bad = [dict(tau=0.0, lam=LAM), dict(tau=-1.0, lam=LAM), dict(tau=TAU, lam=-1.0),
           dict(tau=math.inf, lam=LAM)]
    for kw in bad:
        with pytest.raises(ifvs.IfvsError) as e:
            g.train_grad(case.qs.q, case.qs.preds, case.wz, cand, P, kw["tau"], kw["lam"])
        assert e.value.code == ifvs.IFVS_ERR_ARG
    for bad_id in (case.w.N, -5):                                # ids outside -1..N-1
        c2 = cand.copy()
        c2[0, 0] = bad_id
        with pytest.raises(ifvs.IfvsError) as e:
            g.train_grad(case.qs.q, case.qs.preds, case.wz, c2, P, TAU, LAM)
        assert e.value.code == ifvs.IFVS_ERR_ARG and "candidate" in str(e.value)
    with pytest.raises(ifvs.IfvsError) as e:                     # more than one mini-batch
        big = np.tile(case.qs.q, (129, 1))
        g.train_grad(big, np.tile(case.qs.preds, 129), case.wz, np.tile(cand, (129, 1)), P, TAU, LAM)
    assert e.value.code == ifvs.IFVS_ERR_ARG
    with pytest.raises(ifvs.IfvsError) as e:                     # mining deeper than IFVS_MAX_K
        g.train_step(case.qs.q, case.qs.preds, case.wz.copy(), case.pos, 300, TAU, LAM, 0.1)
    assert e.value.code == ifvs.IFVS_ERR_ARG
    plain = ifvs.Index(case.ix.codes, case.ix.attrs, D=case.w.D, K=case.w.K)
    plain.load_codebooks(case.ix.codebook)
    tp = ifvs._train_params(TAU, LAM, 0.0, P, NNEG, 0, None)
    rc = ifvs.lib().ifvs_train_grad(plain.h, None, None, 1, None, None, ifvs.C.byref(tp), None,
                                    None, None, None)
    assert rc == ifvs.IFVS_ERR_STATE
