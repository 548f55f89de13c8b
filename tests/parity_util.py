"""Comparison rules between the CUDA path and the oracle.

Floating point: the kernels compute in fp32, the oracle in fp64; distances
must agree within REL = 1e-5 relative (the bound the fp32 sums stay within:
at most (M + ds) float32 roundings of non-negative terms, below 8e-6 for the
largest M = 120 here, typically far less).

Ids: a top-k is a set chosen by comparing floats, so where two candidates'
oracle distances lie within the tolerance of the k-th distance either may be
returned.  Everything else must match exactly: the number of valid results,
the padding, every returned id's pass bit, the ascending order, and every id
away from the k-th boundary.
"""
import numpy as np

REL = 1e-5


def close(g, o, rel=REL):
    g = np.asarray(g, np.float64)
    o = np.asarray(o, np.float64)
    return np.abs(g - o) <= rel * np.abs(o)


def bitmap_rows(bm, N):
    return np.unpackbits(np.ascontiguousarray(bm).view(np.uint8), bitorder="little")[:N].astype(bool)


def check_topk(gi, gd, oi, od, all_dist, passing, rel=REL):
    """gi/gd: GPU ids (int64) and fp32 dists of one query; oi/od: oracle's;
    all_dist: oracle fp64 distance of every row; passing: bool mask of rows.
    Returns the number of ids that differ by a boundary tie."""
    k = len(oi)
    nv = int((oi >= 0).sum())
    assert int((gi >= 0).sum()) == nv, "valid count %d vs %d" % ((gi >= 0).sum(), nv)
    assert (gi[nv:] == -1).all() and np.isinf(gd[nv:]).all(), "padding"
    g = gi[:nv]
    assert len(np.unique(g)) == nv, "duplicate ids"
    assert passing[g].all(), "returned a row that fails the predicate"
    assert (np.diff(gd[:nv].astype(np.float64)) >= 0).all(), "not ascending"
    assert close(gd[:nv], all_dist[g], rel).all(), "distance of a returned id"
    assert close(gd[:nv], od[:nv], rel).all(), "distance at a rank"
    if nv == 0:
        return 0
    kth = od[nv - 1]
    diff = set(g.tolist()) ^ set(oi[:nv].tolist())
    for i in diff:
        d = all_dist[i]
        assert abs(d - kth) <= 2 * rel * kth, "id %d (dist %.9g) is not tied with the k-th %.9g" % (i, d, kth)
    return len(diff) // 2


def check_topk_sparse(gi, gd, oi, od, g_odist, g_pass, rel=REL):
    """check_topk for large N, without the distance of every row:
    g_odist / g_pass are the oracle's distance and pass flag of each id the
    GPU returned (NaN / False for -1).  Returns the number of ids that differ
    by a boundary tie."""
    k = len(oi)
    nv = int((oi >= 0).sum())
    assert int((gi >= 0).sum()) == nv, "valid count %d vs %d" % ((gi >= 0).sum(), nv)
    assert (gi[nv:] == -1).all() and np.isinf(gd[nv:]).all(), "padding"
    g = gi[:nv]
    assert len(np.unique(g)) == nv, "duplicate ids"
    assert np.asarray(g_pass[:nv]).all(), "returned a row that fails the predicate"
    assert (np.diff(gd[:nv].astype(np.float64)) >= 0).all(), "not ascending"
    assert close(gd[:nv], g_odist[:nv], rel).all(), "distance of a returned id"
    assert close(gd[:nv], od[:nv], rel).all(), "distance at a rank"
    if nv == 0:
        return 0
    kth = od[nv - 1]
    gset, oset = set(g.tolist()), set(oi[:nv].tolist())
    for j, i in enumerate(g.tolist()):
        if i not in oset:
            d = g_odist[j]
            assert abs(d - kth) <= 2 * rel * kth, "id %d (dist %.9g) is not tied with the k-th %.9g" % (i, d, kth)
    for j, i in enumerate(oi[:nv].tolist()):
        if i not in gset:
            d = od[j]
            assert abs(d - kth) <= 2 * rel * kth, "missed id %d (dist %.9g), k-th %.9g" % (i, d, kth)
    return len(gset ^ oset) // 2
