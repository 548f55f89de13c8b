"""iFVS oracle — TEST INFRASTRUCTURE ONLY.

A thin ctypes wrapper over ``oracle/liboracle.so`` (plain C, fp64; see
``oracle.h`` for the paper map, the readings taken and the parity status of
each function).  Only the test suite, ``__graft_entry__.smoke()`` and the
CPU-baseline leg of ``bench.py`` may import this package.  It shares nothing
with the GPU library: predicates arrive as numpy structured arrays whose
layout this module defines for itself.
"""
from __future__ import annotations

import ctypes as C
import os
import subprocess

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SO = os.path.join(_HERE, "liboracle.so")
_SRC = os.path.join(_HERE, "oracle.c")
_HDR = os.path.join(_HERE, "oracle.h")

# One clause: col int32, op int32, lo int64, hi int64 (24 bytes); a predicate
# holds n_clauses (int32), a reserved int32 and four clauses (104 bytes).
CLAUSE_DTYPE = np.dtype([("col", "<i4"), ("op", "<i4"), ("lo", "<i8"), ("hi", "<i8")])
PREDICATE_DTYPE = np.dtype([("n_clauses", "<i4"), ("reserved", "<i4"), ("c", CLAUSE_DTYPE, (4,))])
assert CLAUSE_DTYPE.itemsize == 24 and PREDICATE_DTYPE.itemsize == 104

EQ, RANGE, GE, LT, GT, LE = 0, 1, 2, 3, 4, 5
I32, I16 = 0, 1


def build(force: bool = False) -> str:
    """Compile liboracle.so with gcc (portable flags, no FMA contraction)."""
    stale = (not os.path.exists(_SO)) or any(
        os.path.getmtime(p) > os.path.getmtime(_SO) for p in (_SRC, _HDR))
    if force or stale:
        tmp = _SO + ".tmp.%d" % os.getpid()
        cmd = ["gcc", "-std=c99", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
               "-fno-fast-math", "-Wall", "-o", tmp, _SRC, "-lm"]
        subprocess.check_call(cmd, cwd=_HERE)
        os.replace(tmp, _SO)
    return _SO


_lib = None


def lib():
    global _lib
    if _lib is None:
        # IFVS_ORACLE_SO points the wrapper at another build of oracle.c (the
        # mutation test loads copies with planted mistakes this way)
        so = os.environ.get("IFVS_ORACLE_SO")
        if not so:
            build()
            so = _SO
        L = C.CDLL(so)
        P, I32_, I64, U64, D = C.c_void_p, C.c_int32, C.c_int64, C.c_uint64, C.c_double
        sig = {
            "orc_row_passes": (C.c_int, [P, P, I32_, I64, P]),
            "orc_filter": (C.c_int, [P, P, I32_, I64, P, P, P]),
            "orc_fnv1a64": (U64, [P, I64]),
            "orc_splitmix64_finalize": (U64, [U64]),
            "orc_fingerprint_key": (I64, [P, I32_, P, P]),
            "orc_fingerprint": (None, [P, I32_, P, P, I32_, I64, P]),
            "orc_alpha": (None, [P, I64, I32_, P, I32_, P]),
            "orc_softplus": (D, [D]),
            "orc_filter_weights": (None, [P, I32_, P]),
            "orc_condition": (None, [P, P, P, I32_, I32_, I32_, I32_, P]),
            "orc_lut": (None, [P, P, P, I32_, I32_, I32_, P]),
            "orc_adc": (D, [P, P, I32_, I32_]),
            "orc_score": (D, [P, P, P, P, I32_, I32_, I32_]),
            "orc_topk": (None, [P, P, I64, I32_, P, P]),
            "orc_search": (C.c_int, [P, I64, I32_, I32_, I32_, P, P, I32_, P, P, I64, I32_,
                                     I32_, P, P, P, P, P, I64, I32_, P, P, P, P, P, P, P]),
            "orc_adc_all": (None, [P, P, I64, I32_, I32_, P]),
            "orc_exact_topk": (None, [P, I64, I32_, P, P, I32_, P, P]),
            "orc_rerank": (None, [P, I64, I32_, P, P, I32_, I32_, P, P]),
            "orc_recall": (D, [P, P, I32_]),
            "orc_kmeans_pq": (C.c_int, [P, I64, I32_, I32_, I32_, I32_, U64, P, P]),
            "orc_pq_encode": (None, [P, I64, I32_, I32_, I32_, P, P]),
            "orc_reconstruct": (None, [P, P, I32_, I32_, I32_, P]),
            "orc_sdc": (D, [P, P, P, I32_, I32_, I32_]),
            "orc_pq_encode_f32": (None, [P, I64, I32_, I32_, I32_, P, P, P]),
            "orc_lloyd_step": (None, [P, I64, I32_, I32_, I32_, P, P, P, P]),
            "orc_train_loss": (D, [P, I32_, I32_, I32_, P, P, I64, I32_, I32_, P, P, P, P, P,
                                   I64, P, I32_, I32_, D, D, P, P, P]),
            "orc_mine_negatives": (C.c_int, [P, I64, I32_, I32_, I32_, P, P, I32_, P, P, I64,
                                             I32_, I32_, P, P, P, P, P, I64, P, I32_, I32_, P]),
            "orc_train_step": (C.c_int, [P, I64, I32_, I32_, I32_, P, P, I32_, P, P, I64, I32_,
                                         I32_, P, P, P, P, P, I64, P, I32_, I32_, D, D, D, D, P,
                                         P, P, P, P]),
        }
        for name, (res, args) in sig.items():
            f = getattr(L, name)
            f.restype = res
            f.argtypes = args
        _lib = L
    return _lib


# ---------------------------------------------------------------- helpers

def _p(a):
    return None if a is None else a.ctypes.data_as(C.c_void_p)


def _c(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


def _preds(p):
    p = np.ascontiguousarray(p)
    if p.dtype.itemsize != PREDICATE_DTYPE.itemsize:
        raise ValueError("predicate records must be 104 bytes")
    return p.view(PREDICATE_DTYPE)


class _Cols:
    """Keeps attribute columns alive and exposes the void** / int32* pair."""

    def __init__(self, cols):
        self.arrays, types = [], []
        for a in cols:
            a = np.ascontiguousarray(a)
            if a.dtype == np.int32:
                types.append(I32)
            elif a.dtype == np.int16:
                types.append(I16)
            else:
                raise TypeError("attribute columns must be int32 or int16")
            self.arrays.append(a)
        self.ptrs = (C.c_void_p * max(1, len(cols)))(*[a.ctypes.data for a in self.arrays])
        self.types = np.array(types if types else [0], dtype=np.int32)
        self.n = len(cols)


# ---------------------------------------------------------------- API

def filter_bitmap(cols, pred):
    cs = _Cols(cols)
    N = len(cs.arrays[0]) if cs.n else 0
    bm = np.zeros(max(1, (N + 31) // 32), dtype=np.uint32)
    npass = C.c_int64(0)
    pr = _preds(np.asarray(pred).reshape(1))
    rc = lib().orc_filter(cs.ptrs, _p(cs.types), cs.n, N, _p(pr), _p(bm), C.byref(npass))
    if rc != 0:
        raise ValueError("invalid predicate")
    return bm[: (N + 31) // 32], int(npass.value)


def row_passes(cols, row, pred):
    cs = _Cols(cols)
    pr = _preds(np.asarray(pred).reshape(1))
    return lib().orc_row_passes(cs.ptrs, _p(cs.types), cs.n, int(row), _p(pr))


def fnv1a64(data: bytes) -> int:
    buf = np.frombuffer(data, dtype=np.uint8) if len(data) else np.zeros(1, np.uint8)
    return int(lib().orc_fnv1a64(_p(buf), len(data)))


def splitmix64_finalize(z: int) -> int:
    return int(lib().orc_splitmix64_finalize(C.c_uint64(z & (2**64 - 1))))


def fingerprint_key(q, pred) -> bytes:
    q = _c(q, np.float32)
    out = np.zeros(4 * q.size + 4 + 96, dtype=np.uint8)
    n = lib().orc_fingerprint_key(_p(q), q.size, _p(_preds(np.asarray(pred).reshape(1))), _p(out))
    return out[:n].tobytes()


def fingerprint(q, pred, seeds, B):
    q = _c(q, np.float32)
    seeds = _c(seeds, np.uint64)
    idx = np.zeros(len(seeds), dtype=np.uint32)
    lib().orc_fingerprint(_p(q), q.size, _p(_preds(np.asarray(pred).reshape(1))), _p(seeds),
                          len(seeds), int(B), _p(idx))
    return idx


def alpha(bank, idx):
    bank = _c(bank, np.float32)
    idx = _c(idx, np.uint32)
    out = np.zeros(bank.shape[1], dtype=np.float64)
    lib().orc_alpha(_p(bank), bank.shape[0], bank.shape[1], _p(idx), len(idx), _p(out))
    return out


def softplus(x: float) -> float:
    return float(lib().orc_softplus(float(x)))


def filter_weights(wz, D=None):
    if wz is None:
        out = np.zeros(D, dtype=np.float64)
        lib().orc_filter_weights(None, D, _p(out))
        return out
    wz = _c(wz, np.float32)
    out = np.zeros(wz.size, dtype=np.float64)
    lib().orc_filter_weights(_p(wz), wz.size, _p(out))
    return out


def condition(C_pq, alpha_mr, W):
    """C_pq [M][K][ds] f32; alpha [M][r] (or None); W [M][r][K][ds] f32 (or None)."""
    C_pq = _c(C_pq, np.float32)
    M, K, ds = C_pq.shape
    r = 0 if W is None else W.shape[1]
    a = _c(alpha_mr, np.float64)
    W = _c(W, np.float32)
    out = np.zeros((M, K, ds), dtype=np.float64)
    lib().orc_condition(_p(C_pq), _p(a), _p(W), M, K, ds, r, _p(out))
    return out


def lut(q, Cf, wf):
    q = _c(q, np.float32)
    Cf = _c(Cf, np.float64)
    wf = _c(wf, np.float64)
    M, K, ds = Cf.shape
    out = np.zeros((M, K), dtype=np.float64)
    lib().orc_lut(_p(q), _p(Cf), _p(wf), M, K, ds, _p(out))
    return out


def adc(lut_mk, code_row):
    lut_mk = _c(lut_mk, np.float64)
    code_row = _c(code_row, np.uint8)
    M, K = lut_mk.shape
    return float(lib().orc_adc(_p(lut_mk), _p(code_row), M, K))


def adc_all(lut_mk, codes):
    lut_mk = _c(lut_mk, np.float64)
    codes = _c(codes, np.uint8)
    M, K = lut_mk.shape
    out = np.zeros(codes.shape[0], dtype=np.float64)
    lib().orc_adc_all(_p(lut_mk), _p(codes), codes.shape[0], M, K, _p(out))
    return out


def score(q, Cf, wf, code_row):
    q = _c(q, np.float32)
    Cf = _c(Cf, np.float64)
    wf = _c(wf, np.float64)
    code_row = _c(code_row, np.uint8)
    M, K, ds = Cf.shape
    return float(lib().orc_score(_p(q), _p(Cf), _p(wf), _p(code_row), M, K, ds))


def topk(dist, ids, k):
    dist = _c(dist, np.float64)
    ids = _c(ids, np.int64)
    oi = np.zeros(k, dtype=np.int64)
    od = np.zeros(k, dtype=np.float64)
    lib().orc_topk(_p(dist), _p(ids), len(dist), k, _p(oi), _p(od))
    return oi, od


def search(codes, cols, C_pq, queries, preds, k, bank=None, W=None, seeds=None, wz=None,
           want_stages=False):
    """The whole query path of §2 for every query (fp64).

    Returns (ids [nq,k] int64, dists [nq,k] f64, npass [nq]) and, when
    ``want_stages``, a dict with bank_idx, alpha, wf and lut per query."""
    codes = _c(codes, np.uint8)
    N, M = codes.shape
    C_pq = _c(C_pq, np.float32)
    _, K, ds = C_pq.shape
    D = M * ds
    queries = _c(queries, np.float32).reshape(-1, D)
    nq = queries.shape[0]
    preds = _preds(preds)
    cs = _Cols(cols)
    bank = _c(bank, np.float32)
    W = _c(W, np.float32)
    seeds = _c(seeds, np.uint64)
    wz = None if wz is None else _c(wz, np.float32).reshape(nq, D)
    B = 0 if bank is None else bank.shape[0]
    h = 0 if seeds is None else len(seeds)
    r = 0 if W is None else W.shape[1]
    ids = np.zeros((nq, k), dtype=np.int64)
    dists = np.zeros((nq, k), dtype=np.float64)
    npass = np.zeros(nq, dtype=np.int64)
    st = None
    if want_stages:
        st = dict(bank_idx=np.zeros((nq, max(h, 1)), np.uint32),
                  alpha=np.zeros((nq, M * max(r, 1)), np.float64),
                  wf=np.zeros((nq, D), np.float64),
                  lut=np.zeros((nq, M, K), np.float64))
    rc = lib().orc_search(
        _p(codes), N, M, K, ds, cs.ptrs, _p(cs.types), cs.n, _p(C_pq), _p(bank), B, h, r,
        _p(W), _p(seeds), _p(queries), _p(preds), _p(wz), nq, k, _p(ids), _p(dists),
        _p(npass), _p(st["bank_idx"]) if st else None, _p(st["alpha"]) if st else None,
        _p(st["wf"]) if st else None, _p(st["lut"]) if st else None)
    if rc != 0:
        raise ValueError("invalid predicate")
    if want_stages:
        return ids, dists, npass, st
    return ids, dists, npass


def exact_topk(X, q, bitmap, k):
    X = _c(X, np.float32)
    q = _c(q, np.float32)
    bitmap = _c(bitmap, np.uint32)
    oi = np.zeros(k, dtype=np.int64)
    od = np.zeros(k, dtype=np.float64)
    lib().orc_exact_topk(_p(X), X.shape[0], X.shape[1], _p(q), _p(bitmap), k, _p(oi), _p(od))
    return oi, od


def rerank(X, q, cand, k):
    X = _c(X, np.float32)
    q = _c(q, np.float32)
    cand = _c(cand, np.int64)
    oi = np.zeros(k, dtype=np.int64)
    od = np.zeros(k, dtype=np.float64)
    lib().orc_rerank(_p(X), X.shape[0], X.shape[1], _p(q), _p(cand), len(cand), k, _p(oi),
                     _p(od))
    return oi, od


def recall(ids, gt):
    ids = _c(ids, np.int64)
    gt = _c(gt, np.int64)
    return float(lib().orc_recall(_p(ids), _p(gt), len(gt)))


def kmeans_pq(X, M, K, iters, seed):
    X = _c(X, np.float32)
    n, D = X.shape
    ds = D // M
    Cout = np.zeros((M, K, ds), dtype=np.float64)
    obj = np.zeros((M, iters), dtype=np.float64)
    rc = lib().orc_kmeans_pq(_p(X), n, D, M, K, iters, C.c_uint64(seed), _p(Cout), _p(obj))
    if rc != 0:
        raise ValueError("kmeans_pq: need D % M == 0 and n >= K")
    return Cout, obj


def pq_encode(X, Cpq):
    X = _c(X, np.float32)
    Cpq = _c(Cpq, np.float64)
    M, K, ds = Cpq.shape
    out = np.zeros((X.shape[0], M), dtype=np.uint8)
    lib().orc_pq_encode(_p(X), X.shape[0], X.shape[1], M, K, _p(Cpq), _p(out))
    return out


def reconstruct(Cf, code_row):
    Cf = _c(Cf, np.float64)
    code_row = _c(code_row, np.uint8)
    M, K, ds = Cf.shape
    out = np.zeros(M * ds, dtype=np.float64)
    lib().orc_reconstruct(_p(Cf), _p(code_row), M, K, ds, _p(out))
    return out


def sdc(Cf, cq, cv):
    Cf = _c(Cf, np.float64)
    M, K, ds = Cf.shape
    return float(lib().orc_sdc(_p(Cf), _p(_c(cq, np.uint8)), _p(_c(cv, np.uint8)), M, K, ds))


def pq_encode_f32(X, Cpq):
    """Argmin encoding decided in float32 (fixed order, no fused multiply-add)."""
    X = _c(X, np.float32)
    Cpq = _c(Cpq, np.float32)
    M, K, ds = Cpq.shape
    codes = np.zeros((X.shape[0], M), dtype=np.uint8)
    dmin = np.zeros((X.shape[0], M), dtype=np.float32)
    lib().orc_pq_encode_f32(_p(X), X.shape[0], X.shape[1], M, K, _p(Cpq), _p(codes), _p(dmin))
    return codes, dmin


def lloyd_step(X, C_in):
    """One Lloyd iteration per subspace from float32 centroids."""
    X = _c(X, np.float32)
    C_in = _c(C_in, np.float32)
    M, K, ds = C_in.shape
    C_out = np.zeros_like(C_in)
    codes = np.zeros((X.shape[0], M), dtype=np.uint8)
    obj = np.zeros(M, dtype=np.float64)
    lib().orc_lloyd_step(_p(X), X.shape[0], X.shape[1], M, K, _p(C_in), _p(C_out), _p(codes),
                         _p(obj))
    return C_out, codes, obj


# ---------------------------------------------------------------- learning (§2 "Learning")

def _train_common(codes, C_pq, bank, W, seeds, wz, queries, preds):
    codes = _c(codes, np.uint8)
    C_pq = _c(C_pq, np.float32)
    M = codes.shape[1]
    _, K, ds = C_pq.shape
    D = M * ds
    queries = _c(queries, np.float32).reshape(-1, D)
    return (codes, C_pq, _c(bank, np.float32), _c(W, np.float32), _c(seeds, np.uint64),
            _c(wz, np.float32).reshape(D), queries, _preds(preds), M, K, ds, D)


def train_loss(codes, C_pq, bank, W, seeds, wz, queries, preds, cand, P, tau, lam,
               grads=True):
    """Loss of the queries with candidate lists cand [nq][V] (positives first,
    P of them; -1 = absent) and one shared w_z [D]; with ``grads`` also
    dL/dbank [B][M r], dL/dW [M][r][K][ds], dL/dw_z [D] (fp64)."""
    codes, C_pq, bank, W, seeds, wz, queries, preds, M, K, ds, D = _train_common(
        codes, C_pq, bank, W, seeds, wz, queries, preds)
    cand = _c(cand, np.int64)
    nq, V = cand.shape
    B, Mr = bank.shape
    r = W.shape[1]
    gb = np.zeros((B, Mr)) if grads else None
    gW = np.zeros(W.shape) if grads else None
    gz = np.zeros(D) if grads else None
    L = lib().orc_train_loss(_p(codes), M, K, ds, _p(C_pq), _p(bank), B, len(seeds), r, _p(W),
                             _p(seeds), _p(wz), _p(queries), _p(preds), nq, _p(cand), P, V,
                             float(tau), float(lam), _p(gb), _p(gW), _p(gz))
    return (L, gb, gW, gz) if grads else L


def mine_negatives(codes, cols, C_pq, bank, W, seeds, wz, queries, preds, pos, n_neg):
    """Per query the n_neg best non-positive rows of the pool (-1 padded)."""
    codes, C_pq, bank, W, seeds, wz, queries, preds, M, K, ds, D = _train_common(
        codes, C_pq, bank, W, seeds, wz, queries, preds)
    pos = _c(pos, np.int64)
    nq, P = pos.shape
    cs = _Cols(cols)
    neg = np.zeros((nq, n_neg), np.int64)
    rc = lib().orc_mine_negatives(_p(codes), codes.shape[0], M, K, ds, cs.ptrs, _p(cs.types),
                                  cs.n, _p(C_pq), _p(bank), bank.shape[0], len(seeds),
                                  W.shape[1], _p(W), _p(seeds), _p(wz), _p(queries), _p(preds),
                                  nq, _p(pos), P, n_neg, _p(neg))
    if rc != 0:
        raise ValueError("invalid predicate")
    return neg


def train_step(codes, cols, C_pq, bank, W, seeds, wz, queries, preds, pos, n_neg, tau, lam, lr,
               lr_wz=None):
    """Mining, loss, gradient and one SGD step (step lr for bank and W, lr_wz
    for w_z, default lr); returns (loss, bank', W', w_z', negatives)."""
    lr_wz = lr if lr_wz is None else lr_wz
    codes, C_pq, bank, W, seeds, wz, queries, preds, M, K, ds, D = _train_common(
        codes, C_pq, bank, W, seeds, wz, queries, preds)
    pos = _c(pos, np.int64)
    nq, P = pos.shape
    cs = _Cols(cols)
    b2, W2, z2 = np.empty_like(bank), np.empty_like(W), np.empty_like(wz)
    neg = np.zeros((nq, n_neg), np.int64)
    loss = np.zeros(1)
    rc = lib().orc_train_step(_p(codes), codes.shape[0], M, K, ds, cs.ptrs, _p(cs.types), cs.n,
                              _p(C_pq), _p(bank), bank.shape[0], len(seeds), W.shape[1], _p(W),
                              _p(seeds), _p(wz), _p(queries), _p(preds), nq, _p(pos), P, n_neg,
                              float(tau), float(lam), float(lr), float(lr_wz), _p(b2), _p(W2),
                              _p(z2), _p(neg), _p(loss))
    if rc != 0:
        raise ValueError("invalid predicate")
    return float(loss[0]), b2, W2, z2, neg
