"""The sorted-copy scan (a one-column predicate's pool read as a position
range of the codes sorted by that column) against the bitmap path and the
oracle.

Forcing one path or the other (list_max_ppm = 1000000 / -1) must give the
same pass counts exactly; each path's ids and distances are checked against
the oracle with the tie rule of the other parity tests, and against each
other: the paths add a row's M table entries in different orders, so their
distances agree to float32 rounding (1e-5 relative) and ids may differ only
among distances tied to that precision."""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import check_topk

pytestmark = pytest.mark.gpu

ALWAYS, NEVER = 1000000, -1


@pytest.fixture(scope="module")
def ifvs():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs as mod
    return mod


def _index(ifvs, N, M=16, K=256, ds=2, seed=0, i16=True, device_io=False):
    rng = np.random.default_rng(seed)
    codes = rng.integers(0, K, size=(N, M)).astype(np.uint8)
    codes[1::3] = codes[0::3][: len(codes[1::3])]       # exact ties in distance
    attrs = [rng.integers(-500, 500, N).astype(np.int32)]
    if i16:
        attrs.append(rng.integers(-20, 20, N).astype(np.int16))
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    if device_io:
        import torch
        dev = torch.device("cuda", 0)
        g = ifvs.Index(torch.from_numpy(codes).to(dev), [torch.from_numpy(a).to(dev) for a in attrs],
                       D=M * ds, K=K, device_io=True)
    else:
        g = ifvs.Index(codes, attrs, D=M * ds, K=K)
    g.load_codebooks(Cpq)
    return g, codes, attrs, Cpq


def _preds():
    """One-column predicates of every operator and width, on both columns,
    plus empty, all-pass and two-column ones (the latter take the bitmap path)."""
    rows = []
    for lo, hi in ((0, 1), (-3, 2), (-500, -490), (100, 160), (-200, 300), (-500, 500),
                   (499, 500), (600, 700), (7, 7)):
        rows.append([(0, synth.OP_RANGE, lo, hi)])
    for op, v in ((synth.OP_EQ, 17), (synth.OP_GE, 480), (synth.OP_LT, -470), (synth.OP_GT, 490),
                  (synth.OP_LE, -495), (synth.OP_EQ, 10 ** 6)):
        rows.append([(0, op, v)])
    for op, v in ((synth.OP_EQ, 3), (synth.OP_GE, 19), (synth.OP_LT, -19), (synth.OP_EQ, -20)):
        rows.append([(1, op, v)])
    rows.append([(0, synth.OP_RANGE, -10, 10), (0, synth.OP_GE, -2)])      # one column, two clauses
    rows.append([(0, synth.OP_RANGE, -100, 100), (1, synth.OP_EQ, 5)])    # two columns
    rows.append([])                                                        # all pass
    p = synth.empty_predicates(len(rows))
    for i, cl in enumerate(rows):
        p[i]["n_clauses"] = len(cl)
        for j, c in enumerate(cl):
            synth.set_clause(p[i], j, *c)
    return p


def _queries(n, D, seed=5):
    return np.random.default_rng(seed).standard_normal((n, D)).astype(np.float32)


def _check_oracle(orc, codes, attrs, Cpq, q, preds, k, ids, dists, npass):
    oi, od, on = orc.search(codes, attrs, Cpq, q, preds, k)
    np.testing.assert_array_equal(npass, on)
    _, _, _, st = orc.search(codes, attrs, Cpq, q, preds, 1, want_stages=True)
    for i in range(len(q)):
        all_d = orc.adc_all(st["lut"][i], codes)
        bm, _ = orc.filter_bitmap(attrs, preds[i])
        passing = np.unpackbits(bm.view(np.uint8), bitorder="little")[: len(codes)].astype(bool)
        check_topk(ids[i], dists[i], oi[i], od[i], all_d, passing)


def _same_up_to_rounding(a, b, rel=1e-5):
    """Two searches' (ids, dists, npass): equal counts and padding, distances
    rank by rank within rel, ids equal except among distances tied to 2 rel
    with the k-th."""
    ia, da, na = a
    ib, db, nb = b
    np.testing.assert_array_equal(na, nb)
    np.testing.assert_array_equal(ia < 0, ib < 0)
    for x, y, dx, dy in zip(ia, ib, da, db):
        nv = int((x >= 0).sum())
        if nv == 0:
            continue
        assert np.all(np.abs(dx[:nv].astype(np.float64) - dy[:nv]) <= rel * np.maximum(dy[:nv], 1e-30))
        kth = float(dy[nv - 1])
        dist_of = dict(zip(x[:nv].tolist(), dx[:nv].tolist()))
        dist_of.update(zip(y[:nv].tolist(), dy[:nv].tolist()))
        for i in set(x[:nv].tolist()) ^ set(y[:nv].tolist()):
            assert abs(dist_of[i] - kth) <= 2 * rel * kth


@pytest.mark.parametrize("N,k", [(1, 1), (1000, 10), (33333, 100), (100000, 256)])
def test_list_path_and_bitmap_path(ifvs, orc, N, k):
    g, codes, attrs, Cpq = _index(ifvs, N)
    p = _preds()
    q = _queries(len(p), Cpq.shape[0] * Cpq.shape[2])
    a = g.search(q, p, k, list_max_ppm=ALWAYS)
    b = g.search(q, p, k, list_max_ppm=NEVER)
    d = g.search(q, p, k)                      # the default: the sorted-copy path
    for x, z in zip(a, d):
        np.testing.assert_array_equal(x, z)
    _same_up_to_rounding(a, b)
    if N <= 33333:
        _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)
        _check_oracle(orc, codes, attrs, Cpq, q, p, k, *b)


@pytest.mark.parametrize("M", [1, 8, 12, 24, 120])
def test_list_path_other_subspace_counts(ifvs, orc, M):
    g, codes, attrs, Cpq = _index(ifvs, 20000, M=M, K=64, ds=3, seed=M)
    p = _preds()
    q = _queries(len(p), M * 3, seed=M)
    a = g.search(q, p, 20, list_max_ppm=ALWAYS)
    b = g.search(q, p, 20, list_max_ppm=NEVER)
    for x, z in zip(a, g.search(q, p, 20)):    # the default, for every M: the sorted copy
        np.testing.assert_array_equal(x, z)
    _same_up_to_rounding(a, b)
    _check_oracle(orc, codes, attrs, Cpq, q, p, 20, *a)
    _check_oracle(orc, codes, attrs, Cpq, q, p, 20, *b)


@pytest.mark.parametrize("k", [10, 100])
def test_pairs_of_wide_predicates(ifvs, orc, k):
    """Queries whose ranges on one column overlap by 3/4 of the longer one
    share a CTA (M = 16); shifted or narrow ranges, an odd query out and a
    query on the other column run alone.  Results as the bitmap path and
    the oracle."""
    g, codes, attrs, Cpq = _index(ifvs, 70000, seed=11)
    rows = [(-500, 500), (-500, 500), (-450, 500), (-500, 480), (-300, 400), (-250, 420),
            (-400, 300), (100, 200), (-480, 499)]
    p = synth.empty_predicates(len(rows) + 2)
    for i, (lo, hi) in enumerate(rows):
        p[i]["n_clauses"] = 1
        synth.set_clause(p[i], 0, 0, synth.OP_RANGE, lo, hi)
    p[9]["n_clauses"] = 1
    synth.set_clause(p[9], 0, 1, synth.OP_GE, -20)          # column 1 ...
    p[10]["n_clauses"] = 1
    synth.set_clause(p[10], 0, 0, synth.OP_GE, -500)        # ... beside column 0: no pair
    q = _queries(len(p), 32, seed=11)
    a = g.search(q, p, k, list_max_ppm=ALWAYS, pair_min_rows=1)
    b = g.search(q, p, k, list_max_ppm=NEVER)
    _same_up_to_rounding(a, b)
    _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)
    for x, y in zip(a, g.search(q, p, k, pair_min_rows=-1)):   # no pairs: one query per CTA
        np.testing.assert_array_equal(x, y)


def test_threshold_splits_a_batch(ifvs, orc):
    """A threshold of 1 % sends the narrow predicates of a batch to the
    sorted copy and the wide ones to the bitmap; results as either path."""
    g, codes, attrs, Cpq = _index(ifvs, 40000, seed=9)
    p = _preds()
    q = _queries(len(p), 32, seed=9)
    mixed = g.search(q, p, 30, list_max_ppm=10000)
    _same_up_to_rounding(mixed, g.search(q, p, 30, list_max_ppm=NEVER))
    _check_oracle(orc, codes, attrs, Cpq, q, p, 30, *mixed)


def test_list_path_with_conditioning_sub_batches_and_device_index(ifvs, orc, oracle_index):
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=60000)
    ix = oracle_index(w).ix
    cond = synth.make_conditioning(ix)
    qs = synth.make_queries(ix, 0.01, nq=70)
    for dio in (False, True):
        if dio:
            import torch
            dev = torch.device("cuda", 0)
            g = ifvs.Index(torch.from_numpy(ix.codes).to(dev),
                           [torch.from_numpy(a).to(dev) for a in ix.attrs], D=w.D, K=w.K,
                           device_io=True)
        else:
            g = ifvs.Index(ix.codes, ix.attrs, D=w.D, K=w.K)
        g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
        a = g.search(qs.q, qs.preds, 10, wz=qs.wz, list_max_ppm=ALWAYS, sub_batch=32)
        b = g.search(qs.q, qs.preds, 10, wz=qs.wz, list_max_ppm=NEVER)
        _same_up_to_rounding(a, b)
        oi, od, on = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, 10,
                                bank=cond.bank, W=cond.W, seeds=cond.seeds, wz=qs.wz)
        np.testing.assert_array_equal(a[2], on)


def test_threshold_and_launch_counts(ifvs):
    g, codes, attrs, Cpq = _index(ifvs, 50000, seed=3)
    p = _preds()
    q = _queries(len(p), 32)
    g.stage_times(reset=True)
    g.search(q, p, 10, flags=ifvs.IFVS_F_STAGE_TIMING)
    t = g.stage_times(reset=True)
    # plan + filter; the bitmap scan, the pairing of the sorted-copy queries,
    # the two-query and the one-query sorted-copy scans, for every k
    assert t["filter"][1] == 2 and t["scan"][1] == 4
    g.search(q, p, 100, flags=ifvs.IFVS_F_STAGE_TIMING)
    t = g.stage_times(reset=True)
    assert t["scan"][1] == 4
    g.search(q, p, 200, flags=ifvs.IFVS_F_STAGE_TIMING)
    t = g.stage_times(reset=True)
    assert t["scan"][1] == 4
    g.search(q, p, 100, flags=ifvs.IFVS_F_STAGE_TIMING, pair_min_rows=-1)
    t = g.stage_times(reset=True)
    assert t["scan"][1] == 2
    g.search(q, p, 10, flags=ifvs.IFVS_F_STAGE_TIMING, list_max_ppm=NEVER)
    t = g.stage_times(reset=True)
    assert t["filter"][1] == 1 and t["scan"][1] == 1
    for bad in (-2, 1000001):
        with pytest.raises(ifvs.IfvsError) as e:
            g.search(q, p, 10, list_max_ppm=bad)
        assert e.value.code == ifvs.IFVS_ERR_ARG
    with pytest.raises(ifvs.IfvsError) as e:
        g.search(q, p, 10, pair_min_rows=-2)
    assert e.value.code == ifvs.IFVS_ERR_ARG


def _wide_pairs():
    """Consecutive pairs of one-column ranges that share a two-query CTA:
    equal, shifted (blocks of one query only at either end), nested."""
    rows = [(-500, 500), (-500, 500), (-450, 500), (-500, 480), (-500, 400), (-420, 500),
            (-480, 490), (-490, 480), (-500, 500), (-375, 500)]
    p = synth.empty_predicates(len(rows))
    for i, (lo, hi) in enumerate(rows):
        p[i]["n_clauses"] = 1
        synth.set_clause(p[i], 0, 0, synth.OP_RANGE, lo, hi)
    return p


def _one_by_one(g, q, p, k, **kw):
    out = [g.search(q[i:i + 1], p[i:i + 1], k, **kw) for i in range(len(q))]
    return tuple(np.concatenate([o[j] for o in out]) for j in range(3))


@pytest.mark.parametrize("case", ["normal", "one_wide_subspace", "constant", "tiny_range", "huge"])
@pytest.mark.parametrize("k", [100, 128])
def test_pair_kernel_equals_one_query_kernel(ifvs, orc, case, k):
    """The two-query kernel drops rows by a quantised lower bound and
    rescores the rest exactly in the one-query kernel's order, so a batch
    whose queries pair up (pairing forced at this size) must return, bit for
    bit, what each query returns alone and what the batch returns with no
    pairs (one query per CTA, the one-query kernel).  Table shapes: ordinary; one subspace 1000x wider
    than the others (a loose bound: most rows rescored); every codeword of a
    subspace equal (a zero range: the test is off, all distances tie); a
    range of a few ulps; entries near 1e35."""
    N = 70001
    g, codes, attrs, Cpq = _index(ifvs, N, seed=21)
    rng = np.random.default_rng(22)
    if case == "one_wide_subspace":
        Cpq[3] *= 1000.0
    elif case == "constant":
        Cpq[:] = Cpq[:, :1, :]
    elif case == "tiny_range":
        Cpq = (1.0 + 1e-6 * rng.standard_normal(Cpq.shape)).astype(np.float32)
    elif case == "huge":
        Cpq = (Cpq * 1e17).astype(np.float32)
    g.load_codebooks(Cpq)
    p = _wide_pairs()
    q = _queries(len(p), Cpq.shape[0] * Cpq.shape[2], seed=23)
    if case == "huge":
        q *= 1e17
    if case == "tiny_range":
        q[:] = 1.0
    q[9] = q[8]                                    # a pair of identical vectors
    g.stage_times(reset=True)
    a = g.search(q, p, k, flags=ifvs.IFVS_F_STAGE_TIMING, pair_min_rows=1)
    assert g.stage_times(reset=True)["scan"][1] == 4   # bitmap, pairing, two-query, one-query scans
    for b in (_one_by_one(g, q, p, k, pair_min_rows=1), g.search(q, p, k, pair_min_rows=-1)):
        for x, y in zip(a, b):
            np.testing.assert_array_equal(x, y)
    if case != "huge":
        _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)


def test_pair_kernel_with_conditioning(ifvs, orc, oracle_index):
    """Wide pairs through the conditioned path (bank, W, w_z): the same
    bit-for-bit agreement with single queries, and the oracle's top-k."""
    w = synth.scaled(synth.WORKLOADS["gmm10k-d128-m16"], N=50001)
    ix = oracle_index(w).ix
    cond = synth.make_conditioning(ix)
    qs = synth.make_queries(ix, 1.0, nq=12)
    g = ifvs.Index(ix.codes, ix.attrs, D=w.D, K=w.K)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    a = g.search(qs.q, qs.preds, 100, wz=qs.wz, pair_min_rows=1)
    b = g.search(qs.q, qs.preds, 100, wz=qs.wz, pair_min_rows=-1)
    for j in range(3):
        np.testing.assert_array_equal(a[j], b[j])
    oi, od, on, st = orc.search(ix.codes, ix.attrs, ix.codebook, qs.q, qs.preds, 100, bank=cond.bank,
                                W=cond.W, seeds=cond.seeds, wz=qs.wz, want_stages=True)
    np.testing.assert_array_equal(a[2], on)
    for i in range(12):
        all_d = orc.adc_all(st["lut"][i], ix.codes)
        check_topk(a[0][i], a[1][i], oi[i], od[i], all_d, np.ones(w.N, bool))


@pytest.mark.parametrize("k", [10, 100, 200])
def test_pairing_by_sorted_ranges(ifvs, orc, k):
    """Ranges pair with the query whose range starts next to theirs
    (queries sorted by column and range start, in segments of 2048; pairing
    forced at this size): a batch of 2300 random windows (1 %, 10 % and 50 %
    of the values, both columns) must give bit for bit the same per-query
    results in a permuted order (other pairs form), with no pairs, and query
    by query, and the oracle's top-k."""
    N = 30011
    g, codes, attrs, Cpq = _index(ifvs, N, seed=31)
    rng = np.random.default_rng(32)
    nq = 2300
    p = synth.empty_predicates(nq)
    for i in range(nq):
        p[i]["n_clauses"] = 1
        if i % 7 == 6:
            lo = int(rng.integers(-20, 10))
            synth.set_clause(p[i], 0, 1, synth.OP_RANGE, lo, lo + int(rng.integers(1, 12)))
        else:
            w = int(rng.choice([10, 100, 500]))
            lo = int(rng.integers(-500, 500 - w + 1))
            synth.set_clause(p[i], 0, 0, synth.OP_RANGE, lo, lo + w)
    q = _queries(nq, Cpq.shape[0] * Cpq.shape[2], seed=33)
    a = g.search(q, p, k, sub_batch=nq, pair_min_rows=1)
    perm = rng.permutation(nq)
    b = g.search(q[perm], p[perm], k, sub_batch=nq, pair_min_rows=1)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x[perm], y)
    for x, y in zip(a, g.search(q, p, k, sub_batch=nq, pair_min_rows=-1)):
        np.testing.assert_array_equal(x, y)
    c = _one_by_one(g, q[:24], p[:24], k)
    for x, y in zip(a, c):
        np.testing.assert_array_equal(x[:24], y)
    _check_oracle(orc, codes, attrs, Cpq, q[:64], p[:64], k, *(x[:64] for x in a))


@pytest.mark.parametrize("k", [1, 10, 100, 200])
def test_bulk_copied_tiles_equal_vector_loads(ifvs, orc, k):
    """The one-query sorted-copy kernel reads each round's code rows either
    by bulk copies (TMA) into shared memory, the default, or by per-lane
    vector loads (IFVS_F_PLAIN_LOADS).  The rows, their sum order and the
    top-k logic are the same, so the two must agree bit for bit: ranges cut
    anywhere inside a block, empty and all-pass ranges, a ragged last block,
    one and several queries per sub-batch; and both match the oracle."""
    N = 150_001
    g, codes, attrs, Cpq = _index(ifvs, N, seed=31)
    p = _preds()
    q = _queries(len(p), Cpq.shape[0] * Cpq.shape[2], seed=32)
    a = g.search(q, p, k, pair_min_rows=-1)
    for b in (g.search(q, p, k, pair_min_rows=-1, flags=ifvs.IFVS_F_PLAIN_LOADS),
              g.search(q, p, k, pair_min_rows=-1, sub_batch=3),
              _one_by_one(g, q, p, k, pair_min_rows=-1)):
        for x, y in zip(a, b):
            np.testing.assert_array_equal(x, y)
    _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)


def test_bulk_copy_wait_runs_out_and_reports_timeout(ifvs, monkeypatch):
    """Every wait of the scan for a bulk-copied tile is bounded.  With
    IFVS_TEST_STALL_COPIES=1 the barriers expect more bytes than the copies
    deliver, so each wait runs out: the search must return IFVS_ERR_TIMEOUT
    (no fault, no hang), and the next search on the same index, with the
    variable unset, must return the results of one that never timed out."""
    g, codes, attrs, Cpq = _index(ifvs, 20_000, seed=41, i16=False)
    p = synth.empty_predicates(2)
    for i, (lo, hi) in enumerate(((-100, 300), (-500, 500))):
        p[i]["n_clauses"] = 1
        synth.set_clause(p[i], 0, 0, synth.OP_RANGE, lo, hi)
    q = _queries(2, Cpq.shape[0] * Cpq.shape[2], seed=42)
    ref = g.search(q, p, 10, pair_min_rows=-1)
    monkeypatch.setenv("IFVS_TEST_STALL_COPIES", "1")
    with pytest.raises(ifvs.IfvsError) as e:
        g.search(q, p, 10, pair_min_rows=-1)
    assert e.value.code == ifvs.IFVS_ERR_TIMEOUT
    monkeypatch.delenv("IFVS_TEST_STALL_COPIES")
    again = g.search(q, p, 10, pair_min_rows=-1)
    for x, y in zip(ref, again):
        np.testing.assert_array_equal(x, y)


@pytest.mark.parametrize("k", [10, 100])
def test_composite_copies_for_two_column_predicates(ifvs, orc, k):
    """An index of two columns keeps, besides one sorted copy per column,
    both composite copies (rows by (column j, column 1 - j)).  A predicate
    that fixes one column to a value and bounds the other (Listing 1's
    `category = c AND date range`) reads one position range of the copy
    keyed by the fixed column; pass counts must equal the oracle's and the
    bitmap path's exactly, and top-k the oracle's with the tie rule.  Cases:
    either column fixed, one- and two-sided bounds, both fixed, values
    absent, empty intervals, the largest and smallest int32 values (the
    composite key's carry); predicates fixing neither column take the
    bitmap path in the same batch."""
    N = 100_003
    rng = np.random.default_rng(51)
    M, K, ds = 16, 256, 2
    codes = rng.integers(0, K, size=(N, M)).astype(np.uint8)
    a0 = rng.integers(-40, 40, N).astype(np.int32)
    a0[::997] = np.iinfo(np.int32).max
    a0[5::991] = np.iinfo(np.int32).min
    a1 = rng.integers(-300, 300, N).astype(np.int16)
    a1[7::1009] = np.iinfo(np.int16).max
    attrs = [a0, a1]
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    g = ifvs.Index(codes, attrs, D=M * ds, K=K)
    g.load_codebooks(Cpq)
    i32, i16 = np.iinfo(np.int32), np.iinfo(np.int16)
    rows = [
        [(0, synth.OP_EQ, 3), (1, synth.OP_RANGE, -50, 120)],
        [(1, synth.OP_EQ, -17), (0, synth.OP_RANGE, -10, 30)],
        [(0, synth.OP_EQ, -40), (1, synth.OP_GE, 200)],
        [(1, synth.OP_EQ, 0), (0, synth.OP_LT, 0)],
        [(0, synth.OP_EQ, 12), (1, synth.OP_EQ, 44)],
        [(0, synth.OP_EQ, 1000), (1, synth.OP_RANGE, -300, 300)],     # value absent
        [(0, synth.OP_EQ, 5), (1, synth.OP_RANGE, 10, 10)],           # empty interval
        [(0, synth.OP_EQ, int(i32.max)), (1, synth.OP_LE, int(i16.max))],
        [(0, synth.OP_EQ, int(i32.min)), (1, synth.OP_GE, int(i16.min))],
        [(1, synth.OP_EQ, int(i16.max)), (0, synth.OP_GE, int(i32.min))],
        # neither column fixed: bitmap path
        [(0, synth.OP_RANGE, -5, 5), (1, synth.OP_RANGE, 0, 50)],
        [(0, synth.OP_LE, 10), (1, synth.OP_RANGE, -300, 250)],
        [(1, synth.OP_GE, -200), (0, synth.OP_RANGE, -40, 30)],
        [(0, synth.OP_GE, int(i32.min)), (1, synth.OP_LT, 290)],
        [(0, synth.OP_RANGE, -40, 40), (1, synth.OP_GE, int(i16.min))],
        [(0, synth.OP_EQ, -1), (1, synth.OP_RANGE, -300, 300), (0, synth.OP_GE, -1)],
    ]
    p = synth.empty_predicates(len(rows))
    for i, cl in enumerate(rows):
        p[i]["n_clauses"] = len(cl)
        for j, c in enumerate(cl):
            synth.set_clause(p[i], j, *c)
    q = _queries(len(rows), M * ds, seed=52)
    a = g.search(q, p, k, list_max_ppm=ALWAYS)
    b = g.search(q, p, k, list_max_ppm=NEVER)
    np.testing.assert_array_equal(a[2], b[2])
    _same_up_to_rounding(a, b)
    _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)
    # one query at a time, and the batch with pairing forced
    for x, y in zip(a, _one_by_one(g, q, p, k)):
        np.testing.assert_array_equal(x, y)
    for x, y in zip(a, g.search(q, p, k, pair_min_rows=1)):
        np.testing.assert_array_equal(x, y)
    g.close()


@pytest.mark.parametrize("M,ds,k", [(16, 2, 100), (12, 2, 10), (12, 2, 100), (8, 2, 10)])
def test_bitmap_blocks_of_mixed_density(ifvs, orc, M, ds, k):
    """The bitmap scan takes a 1024-row block in lockstep (all lanes on the
    same column, failing rows masked) when at least 448 of its 1024 rows
    pass, and otherwise lets each lane walk its own passing rows.  Blocks
    here pass exactly a set number of rows (all, none, 447, 448 and 449,
    sparse), in an order that makes the warps cross from
    one mode to the other many times and refill their word rings; 640
    queries put every block of the 300-block column in a single chunk.
    Forced onto the bitmap path, every query must give the sorted-copy
    path's pass count exactly and its top-k up to rounding, and a sample of
    queries must match the oracle."""
    n_blk = 300
    N = n_blk * 1024 + 333
    rng = np.random.default_rng(61)
    K = 256
    codes = rng.integers(0, K, size=(N, M)).astype(np.uint8)
    # passing rows per block; the lockstep threshold is 448
    pattern = (1024, 0, 512, 102, 448, 447, 922, 1, 614, 0, 449, 307, 1024, 1024, 51, 717)
    a0 = rng.integers(100, 1000, N).astype(np.int32)          # fails every predicate below
    for b in range(n_blk + 1):
        r0, r1 = b * 1024, min(N, b * 1024 + 1024)
        n_pass = pattern[(b * 7) % len(pattern)] * (r1 - r0) // 1024
        rows = r0 + rng.choice(r1 - r0, size=n_pass, replace=False)
        a0[rows] = rng.integers(0, 100, n_pass)
    attrs = [a0]
    Cpq = rng.standard_normal((M, K, ds)).astype(np.float32)
    g = ifvs.Index(codes, attrs, D=M * ds, K=K)
    g.load_codebooks(Cpq)
    nq = 640
    widths = (100, 97, 90, 75, 50, 44, 10, 1)
    p = synth.empty_predicates(nq)
    for i in range(nq):
        p[i]["n_clauses"] = 1
        synth.set_clause(p[i], 0, 0, synth.OP_RANGE, 0, widths[i % len(widths)])
    q = _queries(nq, M * ds, seed=62)
    a = g.search(q, p, k, list_max_ppm=ALWAYS)
    b = g.search(q, p, k, list_max_ppm=NEVER)
    np.testing.assert_array_equal(a[2], b[2])
    _same_up_to_rounding(a, b)
    sample = np.arange(0, nq, 41)
    _check_oracle(orc, codes, attrs, Cpq, q[sample], p[sample], k, *(x[sample] for x in b))
    g.close()


@pytest.mark.parametrize("M,ds,k", [(8, 2, 10), (24, 1, 100), (120, 1, 10), (120, 1, 200), (5, 3, 30)])
def test_generic_m_bulk_tiles_equal_vector_loads(ifvs, orc, M, ds, k):
    """For M other than 12 and 16 the one-query kernel reads one row per lane
    and round from a bulk-copied tile of 32 rows (lists of 256 keys leave no
    room for it: the vector-load kernel runs).  Both add a row's entries in
    the same order, so results must agree bit for bit, and with the oracle."""
    N = 70_001
    g, codes, attrs, Cpq = _index(ifvs, N, M=M, ds=ds, seed=61 + M)
    p = _preds()
    q = _queries(len(p), M * ds, seed=62)
    a = g.search(q, p, k, pair_min_rows=-1)
    b = g.search(q, p, k, pair_min_rows=-1, flags=ifvs.IFVS_F_PLAIN_LOADS)
    for x, y in zip(a, b):
        np.testing.assert_array_equal(x, y)
    _check_oracle(orc, codes, attrs, Cpq, q, p, k, *a)
