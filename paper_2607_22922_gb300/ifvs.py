"""Python binding of the C ABI in include/ifvs.h (argument marshalling only).

Every function here has the name of the C entry point it calls and passes
plain pointers and sizes: numpy arrays for host memory, or CUDA tensors
(anything with ``data_ptr()``) together with ``IFVS_F_DEVICE_IO`` for device
memory.  No computation of the query path happens in Python: if
``libifvs.so`` is missing the import fails.
"""
from __future__ import annotations

import ctypes as C
import os

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libifvs.so")

(IFVS_OK, IFVS_ERR_ARG, IFVS_ERR_OOM, IFVS_ERR_CUDA, IFVS_ERR_STATE, IFVS_ERR_UNSUPPORTED,
 IFVS_ERR_TIMEOUT) = 0, -1, -2, -3, -4, -5, -6
IFVS_OP_EQ, IFVS_OP_RANGE, IFVS_OP_GE, IFVS_OP_LT, IFVS_OP_GT, IFVS_OP_LE = 0, 1, 2, 3, 4, 5
IFVS_ATTR_I32, IFVS_ATTR_I16 = 0, 1
IFVS_F_DEVICE_IO, IFVS_F_STAGE_TIMING, IFVS_F_PLAIN_PQ, IFVS_F_PLAIN_LOADS = 0x1, 0x2, 0x4, 0x8
IFVS_MAX_K, IFVS_MAX_M, IFVS_MAX_ATTRS, IFVS_N_STAGES = 256, 128, 4, 9
STAGES = ("predicate", "filter", "condition", "lut", "scan", "merge", "rerank", "layout", "train")

# ifvs_predicate: 104 bytes (n_clauses, reserved, 4 x {col, op, lo, hi})
CLAUSE_DTYPE = np.dtype([("col", "<i4"), ("op", "<i4"), ("lo", "<i8"), ("hi", "<i8")])
PREDICATE_DTYPE = np.dtype([("n_clauses", "<i4"), ("reserved", "<i4"), ("c", CLAUSE_DTYPE, (4,))])


class IfvsError(RuntimeError):
    def __init__(self, code, msg):
        super().__init__("ifvs error %d: %s" % (code, msg))
        self.code = code


class SearchParams(C.Structure):
    _fields_ = [("flags", C.c_uint32), ("rerank", C.c_int32), ("sub_batch", C.c_int32),
                ("chunk_blocks", C.c_int32), ("list_max_ppm", C.c_int32), ("pair_min_rows", C.c_int32),
                ("stream", C.c_void_p)]


class TrainParams(C.Structure):
    _fields_ = [("tau", C.c_float), ("lam", C.c_float), ("lr", C.c_float), ("lr_wz", C.c_float),
                ("n_pos", C.c_int32), ("n_neg", C.c_int32), ("flags", C.c_uint32),
                ("stream", C.c_void_p)]


def _load():
    if not os.path.exists(LIB_PATH):
        raise ImportError("libifvs.so is not built (%s); run `python -c \"import __graft_entry__ "
                          "as g; g.build()\"` or `python -m paper_2607_22922_gb300.build`" % LIB_PATH)
    L = C.CDLL(LIB_PATH)
    P, I32, I64, U32 = C.c_void_p, C.c_int32, C.c_int64, C.c_uint32
    sig = {
        "ifvs_load_index": (C.c_int, [P, I32, P, I64, I32, I32, P, P, I32, P, I32, U32]),
        "ifvs_load_codebooks": (C.c_int, [P, P, I32, P, I64, I32, I32, P, P]),
        "ifvs_search_batch": (C.c_int, [P, P, P, I64, I32, P, P, P, P, P]),
        "ifvs_filter": (C.c_int, [P, P, I64, P, P, P]),
        "ifvs_condition": (C.c_int, [P, P, P, I64, P, P, P, P, P, P, P]),
        "ifvs_scan_topk": (C.c_int, [P, P, P, I64, I32, P, P, P]),
        "ifvs_rerank": (C.c_int, [P, P, P, I64, I32, I32, P, P, P]),
        "ifvs_scan_topk_static": (C.c_int, [P, P, P, I64, I32, P, P, P]),
        "ifvs_pq_encode": (C.c_int, [I32, P, I64, I32, I32, I32, P, P, P, U32, P]),
        "ifvs_merge_topk": (C.c_int, [I32, P, P, I64, I32, I32, P, P, U32, P]),
        "ifvs_pq_train": (C.c_int, [I32, P, I64, I32, I32, I32, I32, P, P, P, U32, P]),
        "ifvs_train_grad": (C.c_int, [P, P, P, I64, P, P, P, P, P, P, P]),
        "ifvs_train_step": (C.c_int, [P, P, P, I64, P, P, P, P, P]),
        "ifvs_get_conditioning": (C.c_int, [P, P, P, U32]),
        "ifvs_stage_times": (C.c_int, [P, P, P, I32]),
        "ifvs_canonical_predicate": (C.c_int, [P, P, I32, P, P, P]),
        "ifvs_index_info": (C.c_int, [P, P]),
        "ifvs_free": (None, [P]),
        "ifvs_last_error": (C.c_char_p, []),
        "ifvs_version": (C.c_char_p, []),
    }
    for name, (res, args) in sig.items():
        f = getattr(L, name)
        f.restype = res
        f.argtypes = args
    return L


_lib = _load()


def lib():
    return _lib


def ifvs_last_error() -> str:
    return _lib.ifvs_last_error().decode()


def ifvs_version() -> str:
    return _lib.ifvs_version().decode()


def _check(rc):
    if rc != IFVS_OK:
        raise IfvsError(rc, ifvs_last_error())


def _ptr(a):
    """Address of a numpy array or a tensor (None -> NULL)."""
    if a is None:
        return None
    if isinstance(a, np.ndarray):
        if not a.flags.c_contiguous:
            raise ValueError("arrays must be C-contiguous")
        return a.ctypes.data
    if hasattr(a, "data_ptr"):
        if hasattr(a, "is_contiguous") and not a.is_contiguous():
            raise ValueError("tensors must be contiguous")
        return a.data_ptr()
    raise TypeError("expected a numpy array or a tensor, got %r" % type(a))


def _params(flags=0, rerank=0, sub_batch=0, stream=None, chunk_blocks=0, list_max_ppm=0, pair_min_rows=0):
    p = SearchParams()
    p.flags = flags
    p.rerank = rerank
    p.sub_batch = sub_batch
    p.chunk_blocks = chunk_blocks
    p.list_max_ppm = list_max_ppm
    p.pair_min_rows = pair_min_rows
    p.stream = stream
    return p


def _host(a, dtype):
    return None if a is None else np.ascontiguousarray(a, dtype=dtype)


# ------------------------------------------------------------ entry points

def ifvs_load_index(codes, attrs, vectors=None, D=0, device=0, K=256, device_io=False):
    """codes [N][M] uint8; attrs: list of int32 / int16 columns of length N."""
    N, M = int(codes.shape[0]), int(codes.shape[1])
    if not device_io:
        codes = _host(codes, np.uint8)
        attrs = [np.ascontiguousarray(a) for a in attrs]
        vectors = _host(vectors, np.float32)
    types = []
    for a in attrs:
        dt = str(a.dtype).replace("torch.", "")
        if dt == "int32":
            types.append(IFVS_ATTR_I32)
        elif dt == "int16":
            types.append(IFVS_ATTR_I16)
        else:
            raise TypeError("attribute columns must be int32 or int16")
    ptrs = (C.c_void_p * max(1, len(attrs)))(*[_ptr(a) for a in attrs])
    ty = np.array(types if types else [0], dtype=np.int32)
    if vectors is not None and not D:
        D = int(vectors.shape[1])
    h = C.c_void_p()
    _check(_lib.ifvs_load_index(C.byref(h), device, _ptr(codes), N, M, K, ptrs, _ptr(ty),
                                len(attrs), _ptr(vectors), D,
                                IFVS_F_DEVICE_IO if device_io else 0))
    return h


def ifvs_load_codebooks(ix, C_pq, bank=None, h=0, r=0, W=None, hash_seeds=None):
    info = ifvs_index_info(ix)
    C_pq = _host(C_pq, np.float32)
    M, K, ds = C_pq.shape
    if (M, K) != (info["M"], info["K"]):
        raise ValueError("C_pq is %s; the index has M = %d, K = %d" % (C_pq.shape, info["M"], info["K"]))
    bank = _host(bank, np.float32)
    W = _host(W, np.float32)
    seeds = _host(hash_seeds, np.uint64)
    B = 0 if bank is None else bank.shape[0]
    if bank is not None:
        if W is None or seeds is None:
            raise ValueError("W and hash_seeds are required with a bank")
        h = len(seeds)
        r = W.shape[1]
        if W.shape != (M, r, K, ds) or bank.ndim != 2 or bank.shape[1] != M * r:
            raise ValueError("bank %s / W %s do not match M = %d, K = %d, ds = %d"
                             % (bank.shape, W.shape, M, K, ds))
    _check(_lib.ifvs_load_codebooks(ix, _ptr(C_pq), ds, _ptr(bank), B, h, r, _ptr(W), _ptr(seeds)))


def ifvs_search_batch(ix, queries, preds, k, wz=None, ids=None, dists=None, npass=None,
                      flags=0, rerank=0, sub_batch=0, stream=None, chunk_blocks=0, list_max_ppm=0,
                      pair_min_rows=0):
    """Host mode (default): numpy in, numpy out.  With IFVS_F_DEVICE_IO in
    ``flags`` every array (inputs and preallocated outputs) is a device tensor."""
    nq = int(queries.shape[0])
    dio = bool(flags & IFVS_F_DEVICE_IO)
    if not dio:
        queries = _host(queries, np.float32)
        preds = np.ascontiguousarray(preds)
        if preds.dtype.itemsize != 104:
            raise ValueError("predicates must be 104-byte records")
        wz = _host(wz, np.float32)
        if ids is None:
            ids = np.empty((nq, k), np.int64)
        if dists is None:
            dists = np.empty((nq, k), np.float32)
        if npass is None:
            npass = np.empty(nq, np.int64)
    p = _params(flags, rerank, sub_batch, stream, chunk_blocks, list_max_ppm, pair_min_rows)
    _check(_lib.ifvs_search_batch(ix, _ptr(queries), _ptr(preds), nq, k, _ptr(wz), C.byref(p),
                                  _ptr(ids), _ptr(dists), _ptr(npass)))
    return ids, dists, npass


def ifvs_filter(ix, preds, N, flags=0, sub_batch=0):
    preds = np.ascontiguousarray(preds)
    nq = len(preds)
    bm = np.empty((nq, (N + 31) // 32), np.uint32)
    npass = np.empty(nq, np.int64)
    p = _params(flags, 0, sub_batch)
    _check(_lib.ifvs_filter(ix, _ptr(preds), nq, C.byref(p), _ptr(bm), _ptr(npass)))
    return bm, npass


def ifvs_condition(ix, queries, preds, wz=None, M=None, K=256, ds=None, h=0, r=0, flags=0,
                   want_cifvs=False):
    queries = _host(queries, np.float32)
    preds = np.ascontiguousarray(preds)
    wz = _host(wz, np.float32)
    nq, D = queries.shape
    bank_idx = np.empty((nq, max(h, 1)), np.uint32)
    alpha = np.empty((nq, max(M * r, 1)), np.float32)
    wf = np.empty((nq, D), np.float32)
    lut = np.empty((nq, M, K), np.float32)
    cif = np.empty((nq, M, K, ds), np.float32) if want_cifvs else None
    p = _params(flags)
    _check(_lib.ifvs_condition(ix, _ptr(queries), _ptr(preds), nq, _ptr(wz), C.byref(p),
                               _ptr(bank_idx), _ptr(alpha), _ptr(wf), _ptr(cif), _ptr(lut)))
    return dict(bank_idx=bank_idx[:, :h], alpha=alpha[:, :M * r], wf=wf, lut=lut, C_ifvs=cif)


def ifvs_scan_topk(ix, lut, bitmaps, k, flags=0, sub_batch=0):
    lut = _host(lut, np.float32)
    bitmaps = _host(bitmaps, np.uint32)
    nq = lut.shape[0]
    ids = np.empty((nq, k), np.int64)
    dists = np.empty((nq, k), np.float32)
    p = _params(flags, 0, sub_batch)
    _check(_lib.ifvs_scan_topk(ix, _ptr(lut), _ptr(bitmaps), nq, k, C.byref(p), _ptr(ids),
                               _ptr(dists)))
    return ids, dists


def ifvs_scan_topk_static(ix, lut, bitmaps, k, ids, dists, stream=None):
    """Device tensors only (lut [nq][M][K] float32, bitmaps [nq][ceil(N/32)]
    uint32, ids [nq][k] int64, dists [nq][k] float32); enqueues on ``stream``
    and returns without synchronising.  Uses no device allocation."""
    nq = int(lut.shape[0])
    _check(_lib.ifvs_scan_topk_static(ix, _ptr(lut), _ptr(bitmaps), nq, k, stream, _ptr(ids),
                                      _ptr(dists)))
    return ids, dists


def ifvs_merge_topk(dists, ids, k=None, device=0, dists_out=None, ids_out=None, flags=0, stream=None):
    """Select across row shards: dists [G][nq][k] float32 and ids [G][nq][k]
    int64 (global row ids, -1 = padding) -> the k smallest by (dist, id) per
    query, [nq][k] each.  Host mode (default): numpy in, numpy out; with
    IFVS_F_DEVICE_IO every array is a device tensor (outputs preallocated)."""
    dio = bool(flags & IFVS_F_DEVICE_IO)
    G, nq, kk = (int(v) for v in dists.shape)
    k = kk if k is None else k
    if k != kk or tuple(ids.shape) != (G, nq, kk):
        raise ValueError("dists and ids must both be [G][nq][k]")
    if not dio:
        dists = _host(dists, np.float32)
        ids = _host(ids, np.int64)
        dists_out = np.empty((nq, k), np.float32)
        ids_out = np.empty((nq, k), np.int64)
    elif dists_out is None or ids_out is None:
        raise ValueError("device I/O needs preallocated outputs")
    _check(_lib.ifvs_merge_topk(device, _ptr(dists), _ptr(ids), nq, G, k, _ptr(dists_out), _ptr(ids_out),
                                flags, stream))
    return ids_out, dists_out


def ifvs_pq_encode(X, C_pq, device=0, want_dmin=False, codes=None, dmin=None, flags=0,
                   stream=None):
    """Host mode (default): numpy in, codes [n][M] uint8 (and dmin [n][M]
    float32) out.  With IFVS_F_DEVICE_IO in ``flags``, X, C_pq, ``codes``
    (and ``dmin``, if wanted) are preallocated device tensors; with a stream
    the call only enqueues the kernel."""
    dio = bool(flags & IFVS_F_DEVICE_IO)
    if not dio:
        X = _host(X, np.float32)
        C_pq = _host(C_pq, np.float32)
    n, D = int(X.shape[0]), int(X.shape[1])
    M, K, ds = (int(v) for v in C_pq.shape)
    if not dio:
        codes = np.empty((n, M), np.uint8)
        dmin = np.empty((n, M), np.float32) if want_dmin else None
    elif codes is None:
        raise ValueError("device I/O needs a preallocated codes tensor")
    _check(_lib.ifvs_pq_encode(device, _ptr(X), n, D, M, K, _ptr(C_pq), _ptr(codes), _ptr(dmin),
                               flags, stream))
    return (codes, dmin) if (want_dmin or dmin is not None) else codes


def ifvs_pq_train(X, C_init, iters, device=0, C_out=None, objective=None, flags=0, stream=None):
    """Lloyd iterations from C_init [M][K][ds]; returns (C_out, objective
    [iters][M]).  With IFVS_F_DEVICE_IO, X, C_init, ``C_out`` and ``objective``
    (or None) are device tensors."""
    dio = bool(flags & IFVS_F_DEVICE_IO)
    if not dio:
        X = _host(X, np.float32)
        C_init = _host(C_init, np.float32)
    n, D = int(X.shape[0]), int(X.shape[1])
    M, K, ds = (int(v) for v in C_init.shape)
    if not dio:
        C_out = np.empty_like(C_init)
        objective = np.empty((max(iters, 1), M), np.float64)
    elif C_out is None:
        raise ValueError("device I/O needs a preallocated C_out tensor")
    _check(_lib.ifvs_pq_train(device, _ptr(X), n, D, M, K, iters, _ptr(C_init), _ptr(C_out),
                              _ptr(objective), flags, stream))
    return C_out, (objective[:iters] if objective is not None else None)


def _train_params(tau, lam, lr, n_pos, n_neg, flags, stream, lr_wz=None):
    tp = TrainParams()
    tp.tau, tp.lam, tp.lr = float(tau), float(lam), float(lr)
    tp.lr_wz = float(lr if lr_wz is None else lr_wz)
    tp.n_pos, tp.n_neg = int(n_pos), int(n_neg)
    tp.flags = flags
    tp.stream = stream
    return tp


def ifvs_train_grad(ix, queries, preds, wz, cand, n_pos, tau, lam, B, Mr, W_shape, flags=0,
                    stream=None, g_bank=None, g_W=None, g_wz=None):
    """Loss and gradients (dL/dbank [B][Mr], dL/dW, dL/dw_z) of one mini-batch
    for given candidates cand [nq][n_pos + n_neg] (positives first)."""
    dio = bool(flags & IFVS_F_DEVICE_IO)
    nq, V = int(cand.shape[0]), int(cand.shape[1])
    if not dio:
        queries = _host(queries, np.float32)
        preds = np.ascontiguousarray(preds)
        wz = _host(wz, np.float32)
        cand = _host(cand, np.int64)
        g_bank = np.empty((B, Mr), np.float32)
        g_W = np.empty(W_shape, np.float32)
        g_wz = np.empty(wz.shape[-1], np.float32)
    tp = _train_params(tau, lam, 0.0, n_pos, V - n_pos, flags, stream)
    loss = C.c_double(0.0)
    _check(_lib.ifvs_train_grad(ix, _ptr(queries), _ptr(preds), nq, _ptr(wz), _ptr(cand),
                                C.byref(tp), _ptr(g_bank), _ptr(g_W), _ptr(g_wz), C.byref(loss)))
    return loss.value, g_bank, g_W, g_wz


def ifvs_train_step(ix, queries, preds, wz, positives, n_neg, tau, lam, lr, flags=0, stream=None,
                    negatives=None, lr_wz=None):
    """One SGD step (step lr for the bank and W, lr_wz for w_z, default lr);
    updates the index's bank and W and ``wz`` in place.  Returns (loss,
    negatives [nq][n_neg])."""
    dio = bool(flags & IFVS_F_DEVICE_IO)
    nq, P = int(positives.shape[0]), int(positives.shape[1])
    if not dio:
        queries = _host(queries, np.float32)
        preds = np.ascontiguousarray(preds)
        positives = _host(positives, np.int64)
        if not (isinstance(wz, np.ndarray) and wz.dtype == np.float32 and wz.flags.c_contiguous):
            raise ValueError("wz must be a C-contiguous float32 array (updated in place)")
        negatives = np.empty((nq, n_neg), np.int64)
    tp = _train_params(tau, lam, lr, P, n_neg, flags, stream, lr_wz)
    loss = C.c_double(0.0)
    _check(_lib.ifvs_train_step(ix, _ptr(queries), _ptr(preds), nq, _ptr(wz), _ptr(positives),
                                C.byref(tp), _ptr(negatives), C.byref(loss)))
    return loss.value, negatives


def ifvs_get_conditioning(ix, B, Mr, W_shape):
    bank = np.empty((B, Mr), np.float32)
    W = np.empty(W_shape, np.float32)
    _check(_lib.ifvs_get_conditioning(ix, _ptr(bank), _ptr(W), 0))
    return bank, W


def ifvs_rerank(ix, queries, cand, k, flags=0):
    queries = _host(queries, np.float32)
    cand = _host(cand, np.int64)
    nq, R = cand.shape
    ids = np.empty((nq, k), np.int64)
    dists = np.empty((nq, k), np.float32)
    p = _params(flags)
    _check(_lib.ifvs_rerank(ix, _ptr(queries), _ptr(cand), nq, R, k, C.byref(p), _ptr(ids),
                            _ptr(dists)))
    return ids, dists


def ifvs_stage_times(ix, reset=False):
    ms = np.zeros(IFVS_N_STAGES, np.float64)
    n = np.zeros(IFVS_N_STAGES, np.int64)
    _check(_lib.ifvs_stage_times(ix, _ptr(ms), _ptr(n), 1 if reset else 0))
    return {s: (float(ms[i]), int(n[i])) for i, s in enumerate(STAGES)}


def ifvs_canonical_predicate(pred, attr_types):
    pred = np.ascontiguousarray(np.asarray(pred).reshape(1))
    ty = np.ascontiguousarray(attr_types, dtype=np.int32)
    n = len(ty)
    lo = np.zeros(max(n, 1), np.int32)
    wm1 = np.zeros(max(n, 1), np.uint32)
    empty = C.c_int32(0)
    _check(_lib.ifvs_canonical_predicate(_ptr(pred), _ptr(ty), n, _ptr(lo), _ptr(wm1),
                                         C.byref(empty)))
    return lo[:n], wm1[:n], bool(empty.value)


def ifvs_index_info(ix):
    out = np.zeros(8, np.int64)
    _check(_lib.ifvs_index_info(ix, _ptr(out)))
    keys = ("N", "M", "K", "D", "ds", "n_attrs", "has_codebooks", "device_bytes")
    return {k: int(v) for k, v in zip(keys, out)}


def ifvs_free(ix):
    _lib.ifvs_free(ix)


class Index:
    """Owns an ifvs_index handle (freed on close / garbage collection)."""

    def __init__(self, codes, attrs, vectors=None, D=0, device=0, K=256, device_io=False):
        self.h = ifvs_load_index(codes, attrs, vectors, D, device, K, device_io)
        self.N, self.M = int(codes.shape[0]), int(codes.shape[1])
        self.K = K
        self._bank_shape = self._W_shape = None

    def load_codebooks(self, C_pq, bank=None, W=None, hash_seeds=None):
        ifvs_load_codebooks(self.h, C_pq, bank=bank, W=W, hash_seeds=hash_seeds)
        self.ds = int(np.asarray(C_pq).shape[2])
        self.r = 0 if W is None else int(np.asarray(W).shape[1])
        self.hh = 0 if hash_seeds is None else len(hash_seeds)
        if bank is not None:
            self._bank_shape = (int(bank.shape[0]), self.M * self.r)
            self._W_shape = (self.M, self.r, self.K, self.ds)
        else:
            self._bank_shape = self._W_shape = None
        return self

    def search(self, queries, preds, k, wz=None, **kw):
        return ifvs_search_batch(self.h, queries, preds, k, wz=wz, **kw)

    def filter(self, preds, **kw):
        return ifvs_filter(self.h, preds, self.N, **kw)

    def condition(self, queries, preds, wz=None, **kw):
        return ifvs_condition(self.h, queries, preds, wz, M=self.M, K=self.K, ds=self.ds,
                              h=self.hh, r=self.r, **kw)

    def scan_topk(self, lut, bitmaps, k, **kw):
        return ifvs_scan_topk(self.h, lut, bitmaps, k, **kw)

    def rerank(self, queries, cand, k, **kw):
        return ifvs_rerank(self.h, queries, cand, k, **kw)

    def _cond_shapes(self):
        if self._bank_shape is None:
            raise IfvsError(IFVS_ERR_STATE, "no memory bank loaded")
        return self._bank_shape, self._W_shape

    def train_grad(self, queries, preds, wz, cand, n_pos, tau, lam, **kw):
        (B, Mr), Ws = self._cond_shapes()
        return ifvs_train_grad(self.h, queries, preds, wz, cand, n_pos, tau, lam, B, Mr, Ws, **kw)

    def train_step(self, queries, preds, wz, positives, n_neg, tau, lam, lr, **kw):
        return ifvs_train_step(self.h, queries, preds, wz, positives, n_neg, tau, lam, lr, **kw)

    def conditioning(self):
        (B, Mr), Ws = self._cond_shapes()
        return ifvs_get_conditioning(self.h, B, Mr, Ws)

    def stage_times(self, reset=False):
        return ifvs_stage_times(self.h, reset)

    def info(self):
        return ifvs_index_info(self.h)

    def close(self):
        if getattr(self, "h", None):
            ifvs_free(self.h)
            self.h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass
