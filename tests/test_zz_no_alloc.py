"""ifvs_scan_topk_static: the scan + top-k entry point for callers that must
not allocate device memory while serving queries (memory owned by another
allocator, or loops that allocate nothing after start-up because
cudaMalloc / cudaFree may synchronise the device).  Its results must equal
those of the allocating entry point ifvs_scan_topk, call after call, even
though every call reuses the same static scratch array; where the scratch
is too small for a batch it splits the batch, and where it is too small for
one query it says so.

This file is collected last so that a run stopping at the first failure has
already run every other test.
"""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth
from parity_util import check_topk, close

pytestmark = pytest.mark.gpu

SCRATCH = 32 << 20          # IFVS_STATIC_SCRATCH_BYTES


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs
    dev = torch.device("cuda:0")
    return torch, ifvs, dev, torch.cuda.current_stream(dev)


def _static(env, g, tables, bitmaps, k):
    torch, ifvs, dev, stream = env
    nq = tables.shape[0]
    t_lut = torch.from_numpy(np.ascontiguousarray(tables)).to(dev)
    t_bm = torch.from_numpy(np.ascontiguousarray(bitmaps)).to(dev)
    t_ids = torch.full((nq, k), -7, dtype=torch.int64, device=dev)
    t_d = torch.full((nq, k), float("nan"), dtype=torch.float32, device=dev)
    ifvs.ifvs_scan_topk_static(g.h, t_lut, t_bm, k, t_ids, t_d, stream=stream.cuda_stream)
    stream.synchronize()
    return t_ids.cpu().numpy(), t_d.cpu().numpy()


def _same(ids, d, ref_ids, ref_d):
    np.testing.assert_array_equal(ids, ref_ids)
    fin = np.isfinite(ref_d)
    np.testing.assert_array_equal(np.isfinite(d), fin)
    assert close(d[fin], ref_d[fin]).all()


def test_static_scratch_entry_matches_allocating_entry(env):
    torch, ifvs, dev, stream = env
    w = synth.scaled(synth.WORKLOADS["sift1m-d128-m16"], N=300_001)
    ix = synth.pq_space_index(w)
    cond = synth.make_conditioning(ix)
    g = ifvs.Index(ix.codes, ix.attrs)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    # two calls in a row with different inputs and sizes: the second must not
    # see anything the first left in the shared scratch
    for call, (sel, nq, k) in enumerate(((0.1, 40, 100), (0.01, 23, 10))):
        qs = synth.make_queries(ix, sel, nq=nq, salt=call)
        tables = g.condition(qs.q, qs.preds, wz=qs.wz)["lut"]
        bitmaps, _ = g.filter(qs.preds)
        ref_ids, ref_d = g.scan_topk(tables, bitmaps, k)
        _same(*_static(env, g, tables, bitmaps, k), ref_ids, ref_d)
    g.close()


def test_static_entry_splits_a_batch_into_sub_batches(env, orc):
    """290 queries over 2 * 10^6 rows need about 90 MB of scratch: the call
    runs sub-batches of 73 queries (the last one shorter) at offsets q0 > 0
    of the tables, bitmaps and outputs; results equal the allocating entry's
    and, on sampled queries, the oracle's."""
    torch, ifvs, dev, stream = env
    w = synth.scaled(synth.WORKLOADS["gmm100m-d128-m16"], N=2_000_003)
    ix = synth.pq_space_index(w)
    g = ifvs.Index(ix.codes, ix.attrs)
    g.load_codebooks(ix.codebook)
    nq, k = 290, 100
    n_blocks = (w.N + 1023) // 1024
    assert nq * (n_blocks * 128 + 256 * 64 * 4) > 2 * SCRATCH
    qs = synth.make_queries(ix, 0.5, nq=nq, salt=5)
    tables = g.condition(qs.q, qs.preds)["lut"]
    bitmaps, _ = g.filter(qs.preds)
    ref_ids, ref_d = g.scan_topk(tables, bitmaps, k)
    for _ in range(2):
        ids, d = _static(env, g, tables, bitmaps, k)
        _same(ids, d, ref_ids, ref_d)
    for i in (0, 72, 73, 146, 219, 289):
        passing = np.unpackbits(bitmaps[i].view(np.uint8), bitorder="little")[:w.N].astype(bool)
        all_d = orc.adc_all(tables[i].astype(np.float64), ix.codes)
        sel = np.nonzero(passing)[0]
        oi, od = orc.topk(all_d[sel], sel, k)
        check_topk(ids[i], d[i], oi, od, all_d, passing)
    g.close()


def _one_subspace_index(ifvs, N, seed):
    """N rows of one subspace (M = 1, d = 1), no attribute columns: the
    smallest index whose lane-major bitmaps reach the scratch's size."""
    rng = np.random.default_rng(seed)
    codes = rng.integers(0, 256, size=(N, 1), dtype=np.uint8)
    g = ifvs.Index(codes, [], D=1)
    g.load_codebooks(rng.standard_normal((1, 256, 1)).astype(np.float32))
    return g, codes


def test_static_entry_uses_fewer_chunks_near_its_limit(env):
    """At 260,000 blocks of rows one query's bitmap (33.3 MB) and table fit
    the scratch only with fewer chunks (lists) than the allocating path
    would use: the call halves the chunk count; results are unchanged."""
    torch, ifvs, dev, stream = env
    N = 260_000 * 1024 - 77
    g, codes = _one_subspace_index(ifvs, N, 11)
    k = 100
    rng = np.random.default_rng(12)
    tables = np.abs(rng.standard_normal((2, 1, 256))).astype(np.float32)
    wrows = (N + 31) // 32
    bitmaps = rng.integers(0, 2**32, size=(2, wrows), dtype=np.uint32)
    bitmaps[:, -1] &= np.uint32((1 << (N % 32)) - 1)
    bitmaps[1] &= np.uint32(0x00010001)             # a sparse pool for the second query
    ref_ids, ref_d = g.scan_topk(tables, bitmaps, k)
    _same(*_static(env, g, tables, bitmaps, k), ref_ids, ref_d)
    g.close()


def test_static_entry_rejects_sizes_beyond_its_scratch(env):
    """2^28 rows need 2^28 / 8 bytes of bitmap for one query, the whole
    scratch before its table: IFVS_ERR_UNSUPPORTED, before any launch."""
    torch, ifvs, dev, stream = env
    g, _ = _one_subspace_index(ifvs, 1 << 28, 13)
    t_lut = torch.zeros((1, 1, 256), dtype=torch.float32, device=dev)
    t_bm = torch.zeros((1, 1), dtype=torch.uint32 if hasattr(torch, "uint32") else torch.int32, device=dev)
    t_ids = torch.empty((1, 10), dtype=torch.int64, device=dev)
    t_d = torch.empty((1, 10), dtype=torch.float32, device=dev)
    with pytest.raises(ifvs.IfvsError) as e:
        ifvs.ifvs_scan_topk_static(g.h, t_lut, t_bm, 10, t_ids, t_d, stream=stream.cuda_stream)
    assert e.value.code == -5 and "scratch" in str(e.value)
    stream.synchronize()
    g.close()
