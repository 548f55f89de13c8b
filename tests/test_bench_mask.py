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
