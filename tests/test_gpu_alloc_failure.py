"""Device allocation failures, injected on the host: with IFVS_FAIL_ALLOC=n
the library's n-th device allocation fails as if the GPU were out of
memory (nothing is allocated and no GPU fault occurs).  Every entry point
must then return IFVS_ERR_OOM, leak nothing, and leave the index (and the
process's CUDA context) usable: the same calls succeed afterwards with
unchanged results."""
import os

import numpy as np
import pytest

from paper_2607_22922_gb300 import synth

pytestmark = pytest.mark.gpu

OOM = -2


@pytest.fixture(scope="module")
def env():
    torch = pytest.importorskip("torch")
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs
    yield torch, ifvs
    os.environ.pop("IFVS_FAIL_ALLOC", None)


def _free_bytes(torch):
    torch.cuda.synchronize()
    return torch.cuda.mem_get_info(0)[0]


def test_failed_loads_return_oom_and_leak_nothing(env):
    torch, ifvs = env
    w = synth.scaled(synth.WORKLOADS["deep10m-d96-m12"], N=100_003)
    ix = synth.pq_space_index(w)
    X = synth.raw_vectors(ix)
    g0 = ifvs.Index(ix.codes, ix.attrs, vectors=X)     # warm the context
    g0.close()
    before = _free_bytes(torch)
    failed = 0
    for n in range(1, 64):
        os.environ["IFVS_FAIL_ALLOC"] = str(n)
        try:
            g = ifvs.Index(ix.codes, ix.attrs, vectors=X)
        except ifvs.IfvsError as e:
            assert e.code == OOM, str(e)
            failed += 1
            continue
        finally:
            os.environ.pop("IFVS_FAIL_ALLOC", None)
        g.close()
        break
    assert failed >= 4, "the load made only %d device allocations" % failed
    assert _free_bytes(torch) >= before - (64 << 20), "failed loads leaked device memory"


def test_failed_search_keeps_the_index_usable(env):
    torch, ifvs = env
    w = synth.scaled(synth.WORKLOADS["deep10m-d96-m12"], N=200_003)
    ix = synth.pq_space_index(w)
    cond = synth.make_conditioning(ix)
    g = ifvs.Index(ix.codes, ix.attrs)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    small = synth.make_queries(ix, 0.01, nq=8)
    big = synth.make_queries(ix, 0.1, nq=600, salt=1)
    ref_small = g.search(small.q, small.preds, w.k, wz=small.wz)
    # the larger batch needs larger workspaces: the first allocation fails
    os.environ["IFVS_FAIL_ALLOC"] = "1"
    try:
        with pytest.raises(ifvs.IfvsError) as e:
            g.search(big.q, big.preds, w.k, wz=big.wz)
        assert e.value.code == OOM
        # another string restarts the count ("01" is the first allocation too)
        os.environ["IFVS_FAIL_ALLOC"] = "01"
        with pytest.raises(ifvs.IfvsError) as e:
            ifvs.ifvs_pq_encode(np.zeros((1000, w.D), np.float32), ix.codebook)
        assert e.value.code == OOM
    finally:
        os.environ.pop("IFVS_FAIL_ALLOC", None)
    # afterwards: the same calls succeed, the small batch's results unchanged
    a = g.search(big.q, big.preds, w.k, wz=big.wz)
    b = g.search(small.q, small.preds, w.k, wz=small.wz)
    for x, y in zip(b, ref_small):
        np.testing.assert_array_equal(x, y)
    sub = g.search(big.q[:100], big.preds[:100], w.k, wz=big.wz[:100])
    for x, y in zip(sub, a):
        np.testing.assert_array_equal(x, y[:100])
    codes = ifvs.ifvs_pq_encode(np.zeros((1000, w.D), np.float32), ix.codebook)
    assert codes.shape == (1000, w.M)
    g.close()
