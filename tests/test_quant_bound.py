"""Host-side checks of the lower bound that lets the two- and four-query
scans drop rows without changing their results (no GPU).

The kernel quantises a query's table to 11 bits,
q[m][c] = floor(min(2047, max(0, (L[m][c] - lo_m) * inv))) with
inv = 2047 / max_m(hi_m - lo_m), all in float32, sums a row's sixteen q
values exactly as integers (S), and drops the row when S exceeds
quant_bound(k-th distance).  Dropping is safe only if every row whose float32
distance d (sixteen rounded additions from 0, in the kernel's order) is at
most the k-th distance has S <= quant_bound(k-th distance).  Below, that
arithmetic is replayed in numpy float32 (IEEE single rounding, like the
kernel's __fsub_rn / __fmul_rn / __fdiv_rn) on adversarial tables, with the
tightest threshold for each row (its own distance), and the packed
two-query candidate test is checked against the plain comparison.

The four-query kernel quantises to 5 bits (QMAX = 31) and keeps a row's
sum in two 8-bit halves (the words of look-ups 0-7 and 8-15, each byte
at most 8 * 31), tests X = floor(lo / 4) + floor(hi / 4) per byte against
B = floor(T / 4), and packs four queries' tests into one subtract; the same
replay checks that no row within its threshold fails that test.
"""
import zlib

import numpy as np
import pytest

F = np.float32
QMAX = 2047
INT_MAX = 2**31 - 1


def quant_params(L, qmax=QMAX):
    """L [16][K] float32 >= 0 -> (lo [16], inv, sl) as the kernel computes them."""
    lo = L.min(axis=1)
    hi = L.max(axis=1)
    r = F(0)
    sl = F(0)
    with np.errstate(invalid="ignore", over="ignore"):
        for m in range(L.shape[0]):
            r = max(r, F(hi[m] - lo[m]))
            sl = F(sl + lo[m])
    with np.errstate(divide="ignore", over="ignore"):
        inv = F(F(qmax) / r) if r > 0 else F(np.inf)
    if not (bool(np.all(lo >= 0)) and r > 0 and np.isfinite(inv) and np.isfinite(sl)):
        inv = F(0)
    return lo, inv, sl


def quantise(L, lo, inv, qmax=QMAX):
    with np.errstate(over="ignore", invalid="ignore"):
        y = (L - lo[:, None]).astype(F) * inv
    y = np.nan_to_num(y.astype(F), nan=0.0)
    return np.floor(np.minimum(F(qmax), np.maximum(F(0), y))).astype(np.int64)


def quant_bound(thr, sl, inv, margin=2.0 ** -12):
    """Vectorised over float32 thresholds; the kernel's quant_bound (margin:
    the relative slack of each step, 2^-12 in the kernel)."""
    thr = np.asarray(thr, F)
    out = np.full(thr.shape, INT_MAX, np.int64)
    if inv == 0:
        return out
    with np.errstate(over="ignore", invalid="ignore"):
        a = (thr * F(1 + margin)).astype(F)
        b = F(sl * F(1 - margin))
        t = ((a - b).astype(F) * F(inv * F(1 + margin))).astype(F)
    finite = thr.view(np.uint32) < 0x7F800000
    ok = finite & (t < F(1e9))
    out[ok] = np.where(t[ok] < 0, -1, np.floor(t[ok])).astype(np.int64)
    return out


def rows_of(L, codes, rot, qmax=QMAX, halves=False):
    """float32 distances in the kernel's order (byte s is subspace
    (s + rot) mod 16) and the exact integer sums of the quantised entries
    (halves: the sums of look-ups 0-7 and 8-15 apart)."""
    lo, inv, sl = quant_params(L, qmax)
    Q = quantise(L, lo, inv, qmax)
    d = np.zeros(len(codes), F)
    S = np.zeros((2, len(codes)), np.int64)
    for s in range(16):
        m = (s + rot) % 16
        c = codes[:, s]
        with np.errstate(over="ignore"):
            d = (d + L[m, c]).astype(F)
        S[s // 8] += Q[m, c]
    if halves:
        return d, S, sl, inv
    return d, S.sum(axis=0), sl, inv


def quad_x(S2):
    """The four-query kernel's per-byte value: floor(lo / 4) + floor(hi / 4)."""
    return (S2[0] >> 2) + (S2[1] >> 2)


def quad_b(T):
    """Its per-byte bound: floor(T / 4) clamped to [-1, 127]."""
    T = np.asarray(T, np.int64)
    return np.where(T < 0, -1, np.minimum(T >> 2, 127))


def tables(kind, rng):
    K = 256
    base = rng.standard_normal((16, K, 8)).astype(F)
    q = rng.standard_normal((16, 1, 8)).astype(F)
    L = ((q - base) ** 2).sum(axis=2).astype(F)
    if kind == "wide_subspace":
        L[5] = (L[5] * F(1000)).astype(F)
    elif kind == "tiny_range":
        L = (F(1) + F(1e-6) * np.abs(rng.standard_normal((16, K)))).astype(F)
    elif kind == "huge":
        L = (L * F(1e35)).astype(F)
    elif kind == "tiny":
        L = (L * F(1e-30)).astype(F)
    elif kind == "few_values":
        L = rng.integers(0, 3, size=(16, K)).astype(F) * F(0.1)
    elif kind == "zero_range":
        L = np.repeat(L[:, :1], K, axis=1)
    elif kind == "ulp_spaced":
        v = np.nextafter(F(3), F(4)) + np.arange(K, dtype=F) * F(2.0 ** -22)
        L = np.stack([rng.permutation(v) for _ in range(16)]).astype(F)
    return L


@pytest.mark.parametrize("kind", ["gaussian", "wide_subspace", "tiny_range", "huge", "tiny",
                                  "few_values", "zero_range", "ulp_spaced"])
def test_no_row_within_the_threshold_is_dropped(kind):
    rng = np.random.default_rng(zlib.crc32(kind.encode()))
    L = tables(kind, rng)
    n = 60000
    codes = rng.integers(0, 256, size=(n, 16))
    for rot in (0, 7, 15):
        d, S, sl, inv = rows_of(L, codes, rot)
        # the tightest threshold that admits a row is its own distance
        assert np.all(S <= quant_bound(d, sl, inv)), kind
        # a threshold one ulp lower may drop it, never a higher one
        up = np.nextafter(d, F(np.inf))
        assert np.all(S <= quant_bound(up, sl, inv))


def test_the_bound_drops_most_rows_beyond_the_kth():
    """Not vacuous: at the 100th-smallest distance of 10^5 rows, the rows
    kept for exact rescoring are few."""
    rng = np.random.default_rng(5)
    L = tables("gaussian", rng)
    codes = rng.integers(0, 256, size=(100000, 16))
    d, S, sl, inv = rows_of(L, codes, 0)
    kth = np.sort(d)[99]
    kept = int((S <= quant_bound(np.array([kth], F), sl, inv)[0]).sum())
    assert 100 <= kept < 1000, kept


def test_degenerate_tables_switch_the_test_off():
    for L in (np.zeros((16, 256), F), np.full((16, 256), np.inf, F),
              np.where(np.arange(256) == 3, F(-1), F(1)).astype(F)[None].repeat(16, 0)):
        lo, inv, sl = quant_params(L)
        assert inv == 0
        assert quant_bound(np.array([F(1)]), sl, inv)[0] == INT_MAX
    # the list not yet full (key all ones) or an infinite k-th distance: every row
    _, inv, sl = quant_params(tables("gaussian", np.random.default_rng(1)))
    thr = np.array([0xFFFFFFFF, 0x7F800000], np.uint32).view(F)
    assert (quant_bound(thr, sl, inv) == INT_MAX).all()


def test_packed_candidate_test_equals_the_comparisons():
    """Both queries' bounds in one word (bound + 0x8000 per half, bound
    clamped to [-1, 0x7FFF]) minus both sums (each <= 16 * 2047) keep bit
    15 / bit 31 exactly where S_A <= T_A / S_B <= T_B: no borrow crosses."""
    rng = np.random.default_rng(7)
    smax = 16 * QMAX
    sA = np.concatenate([np.arange(0, smax + 1, 37), [0, 1, smax - 1, smax]])
    tA = np.concatenate([np.arange(-1, 0x7FFF + 1, 41), [-1, 0, smax - 1, smax, 0x7FFF]])
    SA, TA = np.meshgrid(sA, tA)
    SA, TA = SA.ravel().astype(np.int64), TA.ravel().astype(np.int64)
    SB = rng.integers(0, smax + 1, SA.size)
    TB = rng.integers(-1, 0x7FFF + 1, SA.size)
    tpk = ((TA + 0x8000) | ((TB + 0x8000) << 16)).astype(np.uint32)
    sq = (SA | (SB << 16)).astype(np.uint32)
    diff = (tpk - sq).astype(np.uint32)     # wraps like the kernel's 32-bit subtract
    np.testing.assert_array_equal((diff & 0x8000) != 0, SA <= TA)
    np.testing.assert_array_equal((diff & 0x80000000) != 0, SB <= TB)


def test_the_margins_are_needed():
    """Without the 2^-12 slack the same replay drops rows that are within
    their threshold (float32 rounding of the distance and of the
    quantisation), so the checks above can tell a sound bound from an
    unsound one."""
    dropped = 0
    for kind in ("tiny_range", "ulp_spaced"):
        rng = np.random.default_rng(zlib.crc32(kind.encode()))
        L = tables(kind, rng)
        codes = rng.integers(0, 256, size=(60000, 16))
        for rot in (0, 7, 15):
            d, S, sl, inv = rows_of(L, codes, rot)
            dropped += int((S > quant_bound(d, sl, inv, margin=0.0)).sum())
    assert dropped > 0


@pytest.mark.parametrize("kind", ["gaussian", "wide_subspace", "tiny_range", "huge", "tiny",
                                  "few_values", "zero_range", "ulp_spaced"])
def test_four_query_test_drops_no_row_within_the_threshold(kind):
    rng = np.random.default_rng(zlib.crc32(kind.encode()) + 1)
    L = tables(kind, rng)
    codes = rng.integers(0, 256, size=(60000, 16))
    for rot in (0, 7, 15):
        d, S2, sl, inv = rows_of(L, codes, rot, qmax=31, halves=True)
        assert S2.max() <= 8 * 31                 # each 8-bit half without carry
        X = quad_x(S2)
        assert X.max() <= 124                     # bit 7 of each byte stays free
        for thr in (d, np.nextafter(d, F(np.inf))):
            assert np.all(X <= quad_b(quant_bound(thr, sl, inv))), kind


def test_four_query_test_is_not_vacuous():
    """At the 100th-smallest distance of 10^5 Gaussian rows the 5-bit test
    keeps a small share of the rows for exact rescoring."""
    rng = np.random.default_rng(9)
    L = tables("gaussian", rng)
    codes = rng.integers(0, 256, size=(100000, 16))
    d, S2, sl, inv = rows_of(L, codes, 0, qmax=31, halves=True)
    kth = np.sort(d)[99]
    kept = int((quad_x(S2) <= quad_b(quant_bound(np.array([kth], F), sl, inv))[0]).sum())
    assert 100 <= kept < 20000, kept


def test_packed_four_query_test_equals_the_comparisons():
    """Four bounds in one word (B + 0x80 per byte, B in [-1, 127]) minus
    four per-byte values X (each <= 124) keep bit 7 of byte j exactly where
    X_j <= B_j: no borrow crosses the bytes."""
    rng = np.random.default_rng(11)
    n = 200000
    X = rng.integers(0, 125, (4, n))
    B = rng.integers(-1, 128, (4, n))
    X[:, :1000] = 124
    B[:, 1000:2000] = -1
    B[:, 2000:3000] = X[:, 2000:3000]
    B[:, 3000:4000] = X[:, 3000:4000] - 1
    bpk = np.zeros(n, np.uint64)
    xpk = np.zeros(n, np.uint64)
    for j in range(4):
        bpk |= ((B[j] + 0x80) & 0xFF).astype(np.uint64) << np.uint64(8 * j)
        xpk |= X[j].astype(np.uint64) << np.uint64(8 * j)
    diff = (bpk.astype(np.uint32) - xpk.astype(np.uint32)).astype(np.uint32)
    for j in range(4):
        np.testing.assert_array_equal((diff >> (8 * j + 7)) & 1 == 1, X[j] <= B[j])


def test_packed_halves_sum_like_the_bytes():
    """The kernel adds whole 32-bit words: four 5-bit entries per word, eight
    words per half, so each byte of the half's sum is the sum of its
    query's entries (no carry), and ((lo >> 2) & 0x3F3F3F3F) + ((hi >> 2) &
    0x3F3F3F3F) is X byte by byte."""
    rng = np.random.default_rng(13)
    q = rng.integers(0, 32, (200000, 16, 4))
    q[:1000] = 31
    words = (q[..., 0] | (q[..., 1] << 8) | (q[..., 2] << 16) | (q[..., 3] << 24)).astype(np.uint64)
    lo = (words[:, :8].sum(axis=1) & 0xFFFFFFFF).astype(np.uint32)
    hi = (words[:, 8:].sum(axis=1) & 0xFFFFFFFF).astype(np.uint32)
    x = (((lo >> 2) & 0x3F3F3F3F) + ((hi >> 2) & 0x3F3F3F3F)).astype(np.uint32)
    for j in range(4):
        S2 = np.stack([q[:, :8, j].sum(axis=1), q[:, 8:, j].sum(axis=1)])
        np.testing.assert_array_equal((x >> (8 * j)) & 0xFF, quad_x(S2))
