"""PQ construction on the GPU vs the oracle: the encoder decides in float32
with the oracle's fixed operation order, so codes and minimum distances are
compared bit for bit; a Lloyd iteration's new centroids (fp64 means rounded
to float32, summed in another order) within one float32 ulp."""
import numpy as np
import pytest

from paper_2607_22922_gb300 import synth

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def ifvs():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs as mod
    return mod


def _data(w, n, seed):
    w = synth.scaled(w, N=n)
    X = synth.mixture_vectors(w, synth.mixture_centres(w))
    rng = np.random.default_rng(seed)
    C0 = X[rng.choice(n, w.K, replace=False)].reshape(w.K, w.M, w.ds).transpose(1, 0, 2).copy()
    return X, C0


CASES = [("gmm10k-d128-m16", 20_011), ("sift1m-d128-m16", 30_007), ("deep10m-d96-m12", 12_345),
         ("gist1m-d960-m120", 3_001)]


@pytest.mark.parametrize("name,n", CASES)
def test_encode_bit_exact(ifvs, orc, name, n):
    X, C0 = _data(synth.WORKLOADS[name], n, 1)
    codes, dmin = ifvs.ifvs_pq_encode(X, C0, want_dmin=True)
    rc, rd = orc.pq_encode_f32(X, C0)
    np.testing.assert_array_equal(codes, rc)
    np.testing.assert_array_equal(dmin, rd)


def test_encode_ragged_and_small_codebooks(ifvs, orc):
    rng = np.random.default_rng(4)
    for n, M, K, ds in ((1, 1, 1, 1), (33, 3, 5, 3), (257, 4, 16, 2), (1000, 2, 256, 12)):
        X = rng.standard_normal((n, M * ds)).astype(np.float32)
        C = rng.standard_normal((M, K, ds)).astype(np.float32)
        C[:, -1] = C[:, 0]                       # duplicate codeword: ties go to 0
        codes, dmin = ifvs.ifvs_pq_encode(X, C, want_dmin=True)
        rc, rd = orc.pq_encode_f32(X, C)
        np.testing.assert_array_equal(codes, rc)
        np.testing.assert_array_equal(dmin, rd)


def _ulp_close(a, b):
    a = np.asarray(a, np.float32)
    b = np.asarray(b, np.float32)
    return np.abs(a.astype(np.float64) - b.astype(np.float64)) <= np.spacing(np.maximum(np.abs(a), np.abs(b)))


@pytest.mark.parametrize("name,n", CASES[:3])
def test_one_lloyd_step(ifvs, orc, name, n):
    X, C0 = _data(synth.WORKLOADS[name], n, 2)
    C1, obj = ifvs.ifvs_pq_train(X, C0, 1)
    R1, _, robj = orc.lloyd_step(X, C0)
    assert _ulp_close(C1, R1).all()
    np.testing.assert_allclose(obj[0], robj, rtol=1e-12)


def test_empty_codewords_take_the_farthest_points(ifvs, orc):
    rng = np.random.default_rng(5)
    X = rng.standard_normal((4000, 16)).astype(np.float32)
    C0 = rng.standard_normal((2, 64, 8)).astype(np.float32)
    C0[:, 40:] += 100.0                          # 24 codewords per subspace attract nobody
    C1, _ = ifvs.ifvs_pq_train(X, C0, 1)
    R1, codes, _ = orc.lloyd_step(X, C0)
    assert (np.bincount(codes[:, 0], minlength=64)[40:] == 0).all()
    assert _ulp_close(C1, R1).all()


def test_lloyd_iterations_track_the_oracle(ifvs, orc):
    X, C = _data(synth.WORKLOADS["gmm10k-d128-m16"], 8_000, 3)
    G, gobj = ifvs.ifvs_pq_train(X, C, 5)
    R = C
    for it in range(5):
        R, _, robj = orc.lloyd_step(X, R)
        np.testing.assert_allclose(gobj[it], robj, rtol=1e-9)
    assert (np.diff(gobj, axis=0) <= 1e-6 * gobj[:-1]).all()
    assert _ulp_close(G, R).mean() > 0.999


def test_device_io_on_a_caller_stream(ifvs, orc):
    import torch
    X, C0 = _data(synth.WORKLOADS["gmm10k-d128-m16"], 9_999, 6)
    dev = torch.device("cuda", 0)
    s = torch.cuda.Stream(device=dev)
    Xd, Cd = torch.from_numpy(X).to(dev), torch.from_numpy(C0).to(dev)
    codes = torch.empty((len(X), C0.shape[0]), dtype=torch.uint8, device=dev)
    dmin = torch.empty((len(X), C0.shape[0]), dtype=torch.float32, device=dev)
    torch.cuda.synchronize()
    ifvs.ifvs_pq_encode(Xd, Cd, codes=codes, dmin=dmin, flags=ifvs.IFVS_F_DEVICE_IO,
                        stream=s.cuda_stream)
    s.synchronize()
    rc, rd = orc.pq_encode_f32(X, C0)
    np.testing.assert_array_equal(codes.cpu().numpy(), rc)
    np.testing.assert_array_equal(dmin.cpu().numpy(), rd)
    C1 = torch.empty_like(Cd)
    obj = torch.empty((2, C0.shape[0]), dtype=torch.float64, device=dev)
    ifvs.ifvs_pq_train(Xd, Cd, 2, C_out=C1, objective=obj, flags=ifvs.IFVS_F_DEVICE_IO,
                       stream=s.cuda_stream)
    H1, hobj = ifvs.ifvs_pq_train(X, C0, 2)
    np.testing.assert_array_equal(C1.cpu().numpy(), H1)
    np.testing.assert_array_equal(obj.cpu().numpy(), hobj)


def test_device_io_without_a_stream_orders_after_default_stream_work(ifvs):
    """With device I/O and no stream, the call runs on a stream of the
    library's own that must wait for the caller's pending work on the legacy
    default stream: vectors computed there by torch right before the call
    (no synchronisation in between) are encoded as if the call had waited."""
    import torch
    dev = torch.device("cuda", 0)
    torch.cuda.synchronize()
    M, K, ds, n = 16, 256, 8, 1 << 21
    with torch.cuda.stream(torch.cuda.default_stream(dev)):
        g = torch.Generator(device=dev)
        g.manual_seed(11)
        C = torch.randn((M, K, ds), generator=g, device=dev)
        for rep in range(3):
            torch.cuda.synchronize()
            # long default-stream work that produces X, then the call at once
            X = torch.randn((n, M * ds), generator=g, device=dev)
            for _ in range(4):
                X = torch.tanh(X * 1.5) * 2.0
            codes = torch.empty((n, M), dtype=torch.uint8, device=dev)
            ifvs.ifvs_pq_encode(X, C, codes=codes, flags=ifvs.IFVS_F_DEVICE_IO, stream=None)
            torch.cuda.synchronize()
            again = torch.empty_like(codes)
            ifvs.ifvs_pq_encode(X, C, codes=again, flags=ifvs.IFVS_F_DEVICE_IO, stream=None)
            torch.cuda.synchronize()
            assert torch.equal(codes, again), "the encode read X before it was written (rep %d)" % rep
