"""Seeded synthetic workloads for the iFVS query path (inputs only).

This module draws the inputs of the query path and nothing else: raw
vectors from the stated mixtures, the rows and start codewords of the PQ
training sample, attribute columns, queries with predicates at a target
selectivity, the conditioning parameters (memory bank, W, hash seeds) and
per-query w_z.  It holds none of the method's arithmetic: no k-means, no
encoding, no distances, no look-up tables, no filtering, no top-k.

The paper measures on SIFT1M / SIFT10M with a 16 x 8 PQ (§3.1, §3.2) and
trained conditioning weights; neither the datasets nor the weights exist
here, so every workload is drawn from a seeded mixture with the stated
shapes.  A workload index is built in the paper's order (§1, PQ
background): raw vectors x = post(centre[c] + sigma * n) with c uniform over
the mixture's components and n standard normal; a PQ codebook trained by
Lloyd iterations per subspace on the first ``pq_sample`` rows, started from
K distinct sample rows; every row encoded as the argmin codeword per
subspace.  The two PQ steps are not done here: the test suite runs them
with the oracle (``oracle.pq_index``), the benchmark with the library's
own PQ kernels; ``Index`` holds the result.

``pq_space_index`` is a second, cheaper generator for shape and edge-case
tests (any M, K, N, including N < K): codes drawn directly in PQ space
around prototype codes.  No workload measurement uses it.
"""
from __future__ import annotations

import dataclasses
import math

import numpy as np

# Predicate records: n_clauses int32, reserved int32, 4 x {col int32, op
# int32, lo int64, hi int64} — 104 bytes, the layout of the C interface.
CLAUSE_DTYPE = np.dtype([("col", "<i4"), ("op", "<i4"), ("lo", "<i8"), ("hi", "<i8")])
PREDICATE_DTYPE = np.dtype([("n_clauses", "<i4"), ("reserved", "<i4"), ("c", CLAUSE_DTYPE, (4,))])
OP_EQ, OP_RANGE, OP_GE, OP_LT, OP_GT, OP_LE = 0, 1, 2, 3, 4, 5

# w_z at which softplus(w_z) = 1 (the paper's initial state w_f = 1).
WZ_IDENTITY = math.log(math.e - 1.0)


@dataclasses.dataclass(frozen=True)
class AttrSpec:
    kind: str          # "uniform" | "cluster10" | "zipf"
    lo: int
    hi: int            # exclusive upper bound of the value range
    dtype: str = "int32"
    zipf_s: float = 1.1


@dataclasses.dataclass(frozen=True)
class Workload:
    name: str
    N: int
    D: int
    M: int
    K: int
    clusters: int
    kind: str                  # "gauss" | "sift" | "gist" | "deep"
    attrs: tuple
    nq: int
    k: int
    sels: tuple
    batch: int = 0             # queries per search call (0 = all)
    conjunctive: bool = False  # category = c AND date range
    rho: float = 0.5           # pq_space_index only: probability that a row leaves its prototype code
    B: int = 4096              # memory-bank rows
    h: int = 2                 # hash functions
    r: int = 8                 # adjustment rank
    seed: int = 0x1F5
    pq_sample: int = 65_536    # rows of the PQ training sample (the first rows)
    pq_iters: int = 25         # Lloyd iterations of the PQ training

    @property
    def ds(self) -> int:
        return self.D // self.M

    @property
    def sigma(self) -> float:
        """Per-coordinate standard deviation of a component around its
        centre, before post-processing (0.3 is stated for the Gaussian
        mixture; the other kinds take a comparable spread in their units)."""
        return SIGMA[self.kind]


SIGMA = {"gauss": 0.3, "sift": 12.0, "gist": 0.01, "deep": 0.03}

WORKLOADS = {
    "gmm10k-d128-m16": Workload(
        "gmm10k-d128-m16", 10_000, 128, 16, 256, 32, "gauss",
        (AttrSpec("uniform", 0, 1000),), 100, 10, (0.01, 0.1, 0.5), seed=0x1F5),
    "sift1m-d128-m16": Workload(
        "sift1m-d128-m16", 1_000_000, 128, 16, 256, 256, "sift",
        (AttrSpec("uniform", 0, 3650),), 10_000, 10, (0.001, 0.01, 0.1, 0.5, 1.0),
        seed=0x1F6),
    "gist1m-d960-m120": Workload(
        "gist1m-d960-m120", 1_000_000, 960, 120, 256, 512, "gist",
        (AttrSpec("cluster10", 0, 5120),), 1_000, 10, (0.01, 0.1, 0.5), seed=0x1F7),
    "deep10m-d96-m12": Workload(
        "deep10m-d96-m12", 10_000_000, 96, 12, 256, 1024, "deep",
        (AttrSpec("uniform", 0, 3650), AttrSpec("zipf", 0, 100, "int16")), 10_000, 10,
        (0.0001, 0.001, 0.01, 0.1, 0.5), conjunctive=True, seed=0x1F8),
    "gmm100m-d128-m16": Workload(
        "gmm100m-d128-m16", 100_000_000, 128, 16, 256, 4096, "gauss",
        (AttrSpec("uniform", 0, 1_000_000),), 10_000, 100, (0.001, 0.01, 0.1, 1.0),
        batch=1024, seed=0x1F9),
}


def scaled(w: Workload, N: int | None = None, nq: int | None = None, **kw) -> Workload:
    """The same recipe at a smaller size (parity cases the oracle finishes)."""
    d = dict(kw)
    if N is not None:
        d["N"] = N
    if nq is not None:
        d["nq"] = nq
    return dataclasses.replace(w, **d)


# ---------------------------------------------------------------- mixtures

# Rows are drawn in blocks of BLOCK rows, each from its own seeded stream,
# so that any row range can be drawn (in parallel, or on the device) without
# drawing the rows before it.
BLOCK = 1 << 16


def mixture_centres(w: Workload) -> np.ndarray:
    """[clusters][D] float32 component centres, by kind: Gaussian N(0, 1);
    SIFT-like non-negative values N(30, 25) clipped to [0, 255]; GIST-like
    |N(0, 1)| scaled to unit norm; Deep-like N(0, 1) scaled to unit norm."""
    rng = np.random.default_rng([w.seed, 10])
    if w.kind == "gauss":
        c = rng.standard_normal((w.clusters, w.D))
    elif w.kind == "sift":
        c = np.clip(rng.normal(30.0, 25.0, (w.clusters, w.D)), 0.0, 255.0)
    elif w.kind == "gist":
        c = np.abs(rng.standard_normal((w.clusters, w.D)))
        c /= np.linalg.norm(c, axis=1, keepdims=True)
    elif w.kind == "deep":
        c = rng.standard_normal((w.clusters, w.D))
        c /= np.linalg.norm(c, axis=1, keepdims=True)
    else:
        raise ValueError(w.kind)
    return c.astype(np.float32)


def mixture_clusters(w: Workload, start: int = 0, stop: int | None = None) -> np.ndarray:
    """[stop - start] int32: the mixture component of each row (uniform)."""
    stop = w.N if stop is None else stop
    out = np.empty(stop - start, dtype=np.int32)
    for b0 in range(start - start % BLOCK, stop, BLOCK):
        rng = np.random.default_rng([w.seed, 11, b0 // BLOCK])
        cl = rng.integers(0, w.clusters, size=BLOCK, dtype=np.int32)
        a, b = max(b0, start), min(b0 + BLOCK, stop)
        out[a - start:b - start] = cl[a - b0:b - b0]
    return out


def post_process(kind: str, x: np.ndarray) -> np.ndarray:
    """The kind's value domain: SIFT-like rounded to integers and clipped to
    [0, 255]; GIST-like made non-negative and scaled to unit norm; Deep-like
    scaled to unit norm; Gaussian unchanged."""
    if kind == "sift":
        return np.clip(np.rint(x), 0.0, 255.0).astype(np.float32)
    if kind == "gist":
        x = np.abs(x)
        return (x / np.maximum(np.linalg.norm(x, axis=-1, keepdims=True), 1e-12)).astype(np.float32)
    if kind == "deep":
        return (x / np.maximum(np.linalg.norm(x, axis=-1, keepdims=True), 1e-12)).astype(np.float32)
    return x.astype(np.float32)


def mixture_vectors(w: Workload, centres: np.ndarray, start: int = 0,
                    stop: int | None = None) -> np.ndarray:
    """[stop - start][D] float32 raw vectors of rows [start, stop):
    post(centre[cluster] + sigma * n), n ~ N(0, I), drawn per BLOCK rows."""
    stop = w.N if stop is None else stop
    out = np.empty((stop - start, w.D), dtype=np.float32)
    for b0 in range(start - start % BLOCK, stop, BLOCK):
        a, b = max(b0, start), min(b0 + BLOCK, stop)
        cl = mixture_clusters(w, a, b)
        rng = np.random.default_rng([w.seed, 12, b0 // BLOCK])
        n = rng.standard_normal((BLOCK, w.D), dtype=np.float32)[a - b0:b - b0]
        out[a - start:b - start] = post_process(w.kind, centres[cl] + np.float32(w.sigma) * n)
    return out


def mixture_vectors_torch(w: Workload, centres_t, start: int, stop: int, device):
    """Raw vectors of rows [start, stop) drawn on a torch device, for
    datasets too large for the host: the same recipe as ``mixture_vectors``
    (same components per row) with torch's generator for the noise, seeded
    per 2^22-row block; rows must lie in one such block.  Not the same
    numbers as ``mixture_vectors``: an index is built from one of the two."""
    import torch
    block = 1 << 22
    if start // block != (stop - 1) // block:
        raise ValueError("rows must lie in one 2^22-row block")
    cl = torch.from_numpy(mixture_clusters(w, start, stop).astype(np.int64)).to(device)
    gen = torch.Generator(device=device)
    gen.manual_seed(int(w.seed) * 1_000_003 + 7 + start // block)
    noise = torch.randn((block, w.D), generator=gen, device=device, dtype=torch.float32)
    off = start % block
    x = centres_t[cl] + float(w.sigma) * noise[off:off + (stop - start)]
    if w.kind == "sift":
        x = torch.clamp(torch.round(x), 0.0, 255.0)
    elif w.kind == "gist":
        x = x.abs()
        x = x / x.norm(dim=1, keepdim=True).clamp_min(1e-12)
    elif w.kind == "deep":
        x = x / x.norm(dim=1, keepdim=True).clamp_min(1e-12)
    return x


def pq_sample_rows(w: Workload) -> int:
    """Rows of the PQ training sample: the first min(N, pq_sample) rows (the
    rows are independent draws, so these are a uniform sample)."""
    return min(w.N, w.pq_sample)


def pq_start_rows(w: Workload, n_sample: int) -> np.ndarray:
    """K distinct rows of the training sample whose sub-vectors are the
    start codewords of every subspace (seeded; n_sample >= K)."""
    if n_sample < w.K:
        raise ValueError("the PQ training sample needs at least K = %d rows" % w.K)
    return np.random.default_rng([w.seed, 13]).choice(n_sample, size=w.K, replace=False)


def pq_start_codebook(w: Workload, sample: np.ndarray) -> np.ndarray:
    """[M][K][ds] float32 start codewords: subspace m of codeword j is
    dimensions [m ds, (m+1) ds) of sample row pq_start_rows[j]."""
    rows = sample[pq_start_rows(w, sample.shape[0])]
    return np.ascontiguousarray(rows.reshape(w.K, w.M, w.ds).transpose(1, 0, 2), dtype=np.float32)


def attributes(w: Workload, cluster: np.ndarray) -> list:
    """The attribute columns: uniform int32, cluster-correlated int32
    (cluster * 10 + U[0, 10)), Zipf(1.1) int16 category."""
    attrs = []
    for ai, spec in enumerate(w.attrs):
        arng = np.random.default_rng([w.seed, 2, ai])
        if spec.kind == "uniform":
            a = arng.integers(spec.lo, spec.hi, size=w.N, dtype=np.int64)
        elif spec.kind == "cluster10":
            a = cluster.astype(np.int64) * 10 + arng.integers(0, 10, size=w.N)
        elif spec.kind == "zipf":
            p = zipf_probs(spec.hi - spec.lo, spec.zipf_s)
            a = spec.lo + arng.choice(len(p), size=w.N, p=p)
        else:
            raise ValueError(spec.kind)
        attrs.append(a.astype(np.int16 if spec.dtype == "int16" else np.int32))
    return attrs


def zipf_probs(n: int, s: float) -> np.ndarray:
    """P(value v) ∝ (v + 1)^-s for v in [0, n) (value 0 is the most common)."""
    p = 1.0 / np.arange(1, n + 1, dtype=np.float64) ** s
    return p / p.sum()


# ------------------------------------------------------------------ index

@dataclasses.dataclass
class Index:
    w: Workload
    codebook: np.ndarray        # [M][K][ds] float32
    codes: np.ndarray           # [N][M] uint8
    attrs: list                 # list of int32 / int16 arrays of length N
    cluster: np.ndarray         # [N] int32 mixture component of each row
    centres: np.ndarray         # [clusters][D] float32
    source: str                 # "mixture" (numpy rows), "mixture-torch" (device rows), "pq_space"
    prototypes: np.ndarray | None = None   # pq_space only: [clusters][M] uint8
    noise_sigma: float = 0.0               # pq_space only: residual noise


def mixture_index(w: Workload, codebook: np.ndarray, codes: np.ndarray,
                  source: str = "mixture") -> Index:
    """An Index of the mixture recipe from a trained codebook and the codes
    of every row (built by the caller: the oracle in tests, the library's PQ
    kernels in the benchmark)."""
    cluster = mixture_clusters(w)
    return Index(w, np.ascontiguousarray(codebook, np.float32), codes, attributes(w, cluster),
                 cluster, mixture_centres(w), source)


def pq_space_index(w: Workload, chunk: int = 4_000_000) -> Index:
    """Shape and edge-case generator: codewords drawn around mixture centres,
    every component has a prototype code, a row keeps each prototype code
    with probability 1 - rho and otherwise takes a uniform codeword; the
    row's raw vector is its reconstruction plus residual noise."""
    rng = np.random.default_rng(w.seed)
    centres = mixture_centres(w)
    jitter, noise = w.sigma, 0.5 * w.sigma
    owner = rng.integers(0, w.clusters, size=(w.M, w.K))
    cb = np.empty((w.M, w.K, w.ds), dtype=np.float32)
    for m in range(w.M):
        sub = centres[owner[m], m * w.ds:(m + 1) * w.ds]
        cb[m] = sub + jitter * rng.standard_normal(sub.shape)
    if w.kind == "sift":
        cb = np.clip(cb, 0.0, 255.0)
    elif w.kind == "gist":
        cb = np.abs(cb)
    prototypes = rng.integers(0, w.K, size=(w.clusters, w.M), dtype=np.uint8)

    codes = np.empty((w.N, w.M), dtype=np.uint8)
    cluster = np.empty(w.N, dtype=np.int32)
    keep_thresh = int(round((1.0 - w.rho) * 256))
    for s in range(0, w.N, chunk):
        e = min(w.N, s + chunk)
        crng = np.random.default_rng([w.seed, 1, s])
        cl = crng.integers(0, w.clusters, size=e - s, dtype=np.int32)
        keep = crng.integers(0, 256, size=(e - s, w.M), dtype=np.uint16) < keep_thresh
        rnd = crng.integers(0, w.K, size=(e - s, w.M), dtype=np.uint8)
        codes[s:e] = np.where(keep, prototypes[cl], rnd)
        cluster[s:e] = cl
    return Index(w, cb, codes, attributes(w, cluster), cluster, centres, "pq_space",
                 prototypes, noise)


def raw_vectors(ix: Index, start: int = 0, stop: int | None = None) -> np.ndarray:
    """Raw vectors of rows [start, stop) of a host-drawn index."""
    w = ix.w
    stop = w.N if stop is None else stop
    if ix.source == "mixture":
        return mixture_vectors(w, ix.centres, start, stop)
    if ix.source != "pq_space":
        raise ValueError("the rows of a %s index are drawn on the device" % ix.source)
    out = np.empty((stop - start, w.D), dtype=np.float32)
    block = BLOCK
    for s in range(start - start % block, stop, block):
        e = s + block
        rng = np.random.default_rng([w.seed, 3, s])
        noise = rng.standard_normal((block, w.D)).astype(np.float32) * ix.noise_sigma
        a, b = max(s, start), min(e, stop)
        if a >= b:
            continue
        codes = ix.codes[a:b]
        rec = ix.codebook[np.arange(w.M)[None, :], codes]          # [n][M][ds] gather
        x = rec.reshape(b - a, w.D) + noise[a - s:b - s]
        out[a - start:b - start] = post_process(w.kind, x)
    return out


# ---------------------------------------------------------------- queries

@dataclasses.dataclass
class Queries:
    q: np.ndarray          # [nq][D] float32
    preds: np.ndarray      # [nq] PREDICATE_DTYPE
    wz: np.ndarray         # [nq][D] float32
    sel: float             # target selectivity of the bin


def empty_predicates(n: int) -> np.ndarray:
    return np.zeros(n, dtype=PREDICATE_DTYPE)


def set_clause(pred, i, col, op, lo, hi=0):
    pred["c"][i]["col"] = col
    pred["c"][i]["op"] = op
    pred["c"][i]["lo"] = lo
    pred["c"][i]["hi"] = hi


def make_queries(ix: Index, sel: float, nq: int | None = None, salt: int = 0,
                 wz_sigma: float = 0.2) -> Queries:
    """Queries drawn from the index's mixture (a uniform component, its
    centre plus sigma * N(0, I), post-processed like the rows), each with a
    predicate whose target selectivity is ``sel``, plus per-query w_z
    around the identity."""
    w = ix.w
    nq = w.nq if nq is None else nq
    rng = np.random.default_rng([w.seed, 4, int(round(sel * 1e6)), salt])
    cl = rng.integers(0, w.clusters, size=nq)
    q = post_process(w.kind, ix.centres[cl] + np.float32(w.sigma) *
                     rng.standard_normal((nq, w.D), dtype=np.float32))

    preds = empty_predicates(nq)
    if w.conjunctive:
        date, cat = w.attrs[0], w.attrs[1]
        p = zipf_probs(cat.hi - cat.lo, cat.zipf_s)
        cum = np.cumsum(p)
        span = date.hi - date.lo
        for i in range(nq):
            if sel <= p[0]:
                ok = np.nonzero(p >= sel)[0]
                c = int(ok[rng.integers(0, len(ok))])
                width = int(min(span, max(1, round(sel / p[c] * span))))
                lo = date.lo + int(rng.integers(0, span - width + 1))
                preds[i]["n_clauses"] = 2
                set_clause(preds[i], 0, 1, OP_EQ, cat.lo + c)
                set_clause(preds[i], 1, 0, OP_RANGE, lo, lo + width)
            else:
                c = int(np.searchsorted(cum, sel))
                c = min(c, len(p) - 1)
                width = int(min(span, max(1, round(sel / cum[c] * span))))
                lo = date.lo + int(rng.integers(0, span - width + 1))
                preds[i]["n_clauses"] = 2
                set_clause(preds[i], 0, 1, OP_LE, cat.lo + c)
                set_clause(preds[i], 1, 0, OP_RANGE, lo, lo + width)
    else:
        a = w.attrs[0]
        span = a.hi - a.lo
        width = int(min(span, max(1, round(sel * span))))
        los = a.lo + rng.integers(0, span - width + 1, size=nq)
        preds["n_clauses"] = 1
        preds["c"][:, 0]["col"] = 0
        preds["c"][:, 0]["op"] = OP_RANGE
        preds["c"][:, 0]["lo"] = los
        preds["c"][:, 0]["hi"] = los + width
    wz = (WZ_IDENTITY + wz_sigma * rng.standard_normal((nq, w.D))).astype(np.float32)
    return Queries(q.astype(np.float32), preds, wz, sel)


# ------------------------------------------------------------ conditioning

@dataclasses.dataclass
class Conditioning:
    bank: np.ndarray       # [B][M*r] float32
    W: np.ndarray          # [M][r][K][ds] float32
    seeds: np.ndarray      # [h] uint64


def make_conditioning(ix: Index, scale: float = 0.05) -> Conditioning:
    """Stand-in values for the trained memory bank and W (the paper's trained
    weights are not available): bank ~ N(0, 1/h) so alpha ~ N(0, 1); W ~
    N(0, (scale * codeword spread of the subspace)^2)."""
    w = ix.w
    rng = np.random.default_rng([w.seed, 5])
    bank = (rng.standard_normal((w.B, w.M * w.r)) / math.sqrt(w.h)).astype(np.float32)
    spread = ix.codebook.reshape(w.M, -1).std(axis=1).astype(np.float64)
    W = rng.standard_normal((w.M, w.r, w.K, w.ds)) * (scale * spread)[:, None, None, None]
    seeds = rng.integers(0, 2**63, size=w.h, dtype=np.int64).astype(np.uint64)
    seeds ^= np.uint64(0x9E3779B97F4A7C15)
    return Conditioning(bank, W.astype(np.float32), seeds)
