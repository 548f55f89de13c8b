"""ifvs_scan_topk_static: the scan + top-k entry point for callers that must
not allocate device memory while serving queries (memory owned by another
allocator, or loops that allocate nothing after start-up because
cudaMalloc / cudaFree may synchronise the device).  Its results must equal
those of the allocating entry point ifvs_scan_topk, call after call, even
though every call reuses the same static scratch array.

This file is collected last so that a run stopping at the first failure has
already run every other test.
"""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import close

pytestmark = pytest.mark.gpu


def test_static_scratch_entry_matches_allocating_entry():
    torch = pytest.importorskip("torch")
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs

    w = synth.scaled(synth.WORKLOADS["sift1m-d128-m16"], N=300_001)
    ix = synth.make_index(w)
    cond = synth.make_conditioning(ix)
    g = ifvs.Index(ix.codes, ix.attrs)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    dev = torch.device("cuda:0")
    stream = torch.cuda.current_stream(dev)
    # two calls in a row with different inputs and sizes: the second must not
    # see anything the first left in the shared scratch
    for call, (sel, nq, k) in enumerate(((0.1, 40, 100), (0.01, 23, 10))):
        qs = synth.make_queries(ix, sel, nq=nq, salt=call)
        tables = g.condition(qs.q, qs.preds, wz=qs.wz)["lut"]
        bitmaps, _ = g.filter(qs.preds)
        ref_ids, ref_d = g.scan_topk(tables, bitmaps, k)
        t_lut = torch.from_numpy(np.ascontiguousarray(tables)).to(dev)
        t_bm = torch.from_numpy(bitmaps).to(dev)
        t_ids = torch.full((nq, k), -7, dtype=torch.int64, device=dev)
        t_d = torch.full((nq, k), float("nan"), dtype=torch.float32, device=dev)
        ifvs.ifvs_scan_topk_static(g.h, t_lut, t_bm, k, t_ids, t_d, stream=stream.cuda_stream)
        stream.synchronize()
        ids, d = t_ids.cpu().numpy(), t_d.cpu().numpy()
        np.testing.assert_array_equal(ids, ref_ids)
        fin = np.isfinite(ref_d)
        np.testing.assert_array_equal(np.isfinite(d), fin)
        assert close(d[fin], ref_d[fin]).all()
    g.close()
