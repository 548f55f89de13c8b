"""Host-side checks of the lower bound that lets the two-query scan drop rows
without changing its results (no GPU).

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
"""
import zlib

import numpy as np
import pytest

F = np.float32
QMAX = 2047
INT_MAX = 2**31 - 1


def quant_params(L):
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
        inv = F(F(QMAX) / r) if r > 0 else F(np.inf)
    if not (bool(np.all(lo >= 0)) and r > 0 and np.isfinite(inv) and np.isfinite(sl)):
        inv = F(0)
    return lo, inv, sl


def quantise(L, lo, inv):
    with np.errstate(over="ignore", invalid="ignore"):
        y = (L - lo[:, None]).astype(F) * inv
    y = np.nan_to_num(y.astype(F), nan=0.0)
    return np.floor(np.minimum(F(QMAX), np.maximum(F(0), y))).astype(np.int64)


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


def rows_of(L, codes, rot):
    """float32 distances in the kernel's order (byte s is subspace
    (s + rot) mod 16) and the exact integer sums of the quantised entries."""
    lo, inv, sl = quant_params(L)
    Q = quantise(L, lo, inv)
    d = np.zeros(len(codes), F)
    S = np.zeros(len(codes), np.int64)
    for s in range(16):
        m = (s + rot) % 16
        c = codes[:, s]
        with np.errstate(over="ignore"):
            d = (d + L[m, c]).astype(F)
        S += Q[m, c]
    return d, S, sl, inv


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
