"""The benchmark's recall ground truth filters rows with its own torch
predicate mask; it must pass exactly the rows the oracle's filter passes."""
import os
import sys

import numpy as np

from paper_2607_22922_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def test_pass_mask_equals_the_oracle_filter(orc):
    import torch
    import bench
    rng = np.random.default_rng(21)
    N = 3000
    attrs = [rng.integers(-1000, 1000, N).astype(np.int32), rng.integers(-40, 40, N).astype(np.int16)]
    nq = 60
    p = synth.empty_predicates(nq)
    for i in range(nq):
        n = int(rng.integers(0, 5))
        p[i]["n_clauses"] = n
        for j in range(n):
            col = int(rng.integers(0, 2))
            op = int(rng.integers(0, 6))
            span = 1000 if col == 0 else 40
            lo = int(rng.integers(-span - 5, span + 5))
            hi = lo + int(rng.integers(-3, 300))
            synth.set_clause(p[i], j, col, op, lo, hi)
    cols = [torch.from_numpy(a.astype(np.int64)) for a in attrs]
    mask = bench._pass_mask(cols, p, torch.device("cpu")).numpy()
    for i in range(nq):
        bm, npass = orc.filter_bitmap(attrs, p[i])
        rows = np.unpackbits(bm.view(np.uint8), bitorder="little")[:N].astype(bool)
        np.testing.assert_array_equal(mask[i], rows)
        assert int(mask[i].sum()) == npass


def test_sorted_path_share_follows_the_path_rule():
    """The benchmark reports which queries the library scans from a sorted
    copy: a predicate no row can pass; one on no column or on one column; on
    an index of two columns, one that fixes a column to a single value
    (after intersecting its clauses and clipping to the column's type) and
    bounds the other; each but the first only while its pool holds at most
    list_rows rows.  Predicates on both columns that fix neither, and
    predicates on several columns of a three-column index, take the bitmap
    path."""
    import bench
    i32 = np.zeros(4, np.int32)
    i16 = np.zeros(4, np.int16)
    cases = [
        ([(0, synth.OP_RANGE, -5, 5)], True),
        ([(1, synth.OP_GE, 3), (1, synth.OP_LT, 9)], True),                   # one column, two clauses
        ([], True),                                                           # every row passes
        ([(1, synth.OP_EQ, 4), (0, synth.OP_RANGE, 0, 100)], True),
        ([(0, synth.OP_EQ, -7), (1, synth.OP_LE, 20)], True),
        ([(1, synth.OP_LE, 4), (0, synth.OP_RANGE, 0, 100)], False),          # neither fixed
        ([(0, synth.OP_RANGE, 8, 9), (1, synth.OP_GT, 0)], True),             # width-one range
        ([(0, synth.OP_GE, 3), (0, synth.OP_LE, 3), (1, synth.OP_LT, 0)], True),   # fixed by two clauses
        ([(1, synth.OP_GE, 32767), (0, synth.OP_GT, 1)], True),               # fixed by the int16 bound
        ([(1, synth.OP_GE, 32766), (0, synth.OP_GT, 1)], False),
        ([(0, synth.OP_LT, -(2 ** 31) + 1), (1, synth.OP_RANGE, 0, 9)], True),   # int32 minimum only
        ([(1, synth.OP_EQ, 40000), (0, synth.OP_GE, 0)], True),               # no int16 value: empty
        ([(0, synth.OP_RANGE, 5, 5), (1, synth.OP_GE, 0)], True),             # empty range
    ]
    p = synth.empty_predicates(len(cases))
    for i, (cl, _) in enumerate(cases):
        p[i]["n_clauses"] = len(cl)
        for j, c in enumerate(cl):
            synth.set_clause(p[i], j, *c)
    small = np.zeros(len(cases))
    big = np.full(len(cases), 10.0)
    want = np.array([w for _, w in cases])
    np.testing.assert_array_equal(bench.sorted_path(p, [i32, i16], small, 5), want)
    empty = np.array([i >= len(cases) - 2 for i in range(len(cases))])
    np.testing.assert_array_equal(bench.sorted_path(p, [i32, i16], big, 5), empty)
    # three columns: only predicates on fewer than two columns have a copy
    three = np.array([len({c[0] for c in cl}) < 2 for cl, _ in cases]) | empty
    np.testing.assert_array_equal(bench.sorted_path(p, [i32, i16, i32], small, 5), three)
