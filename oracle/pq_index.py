"""Workload indexes built with the oracle — TEST INFRASTRUCTURE ONLY.

Only the test suite and ``__graft_entry__.smoke()`` use this module.  It
builds a workload's PQ index in the order of the paper's PQ background (§1):
raw vectors drawn by ``synth`` from the stated mixture, a codebook trained by
the oracle's Lloyd iterations (``orc_lloyd_step``: float32 argmin
assignment, fp64 member means, farthest-row reseeding of empty codewords)
per subspace on the training sample, and every row encoded by the oracle's
float32 argmin encoder (``orc_pq_encode_f32``).  Nothing here comes from the
CUDA library.

Full-size workloads take minutes of CPU, so the work is spread over a
``spawn`` process pool (safe after CUDA is initialised in the parent; a
script that uses it must be a file, not standard input):
subspaces for the training, row ranges for the encoding, queries for the
searches.  Codes and attribute columns go through memory-mapped files in a
private temporary directory, which ``OracleIndex.close`` removes.
"""
from __future__ import annotations

import concurrent.futures as cf
import multiprocessing as mp
import os
import shutil
import tempfile

import numpy as np

from paper_2607_22922_gb300 import synth

ENCODE_ROWS = 1 << 18      # rows per encoding task (a multiple of synth.BLOCK)


def _workers(n_tasks: int, workers: int | None) -> int:
    w = workers if workers else (os.cpu_count() or 1)
    return max(1, min(w, n_tasks))


def _pool(n: int):
    # a worker that dies makes the executor raise (a Pool would restart it
    # and wait forever)
    return cf.ProcessPoolExecutor(max_workers=n, mp_context=mp.get_context("spawn"))


# ------------------------------------------------------------ training

def _lloyd_task(args):
    """Lloyd iterations for a group of subspaces (each is independent)."""
    import oracle
    sample, C0, iters = args
    C = C0
    objective = []
    for _ in range(iters):
        C, _, obj = oracle.lloyd_step(sample, C)
        objective.append(obj)
    return C, np.array(objective).reshape(iters, -1)


def train_codebook(w: synth.Workload, sample: np.ndarray, iters: int | None = None,
                   workers: int | None = None):
    """[M][K][ds] float32 codebook and the objective [iters][M] of each
    iteration, from synth's start codewords.  Subspaces run in parallel; a
    subspace's result does not depend on the others, so this equals one
    ``lloyd_step`` call over all M subspaces per iteration."""
    iters = w.pq_iters if iters is None else iters
    C0 = synth.pq_start_codebook(w, sample)
    n = _workers(w.M, workers)
    groups = [g for g in np.array_split(np.arange(w.M), n) if len(g)]
    tasks = []
    for g in groups:
        cols = np.concatenate([np.arange(m * w.ds, (m + 1) * w.ds) for m in g])
        tasks.append((np.ascontiguousarray(sample[:, cols]), np.ascontiguousarray(C0[g]), iters))
    if n == 1:
        res = [_lloyd_task(t) for t in tasks]
    else:
        with _pool(n) as pool:
            res = list(pool.map(_lloyd_task, tasks))
    C = np.concatenate([r[0] for r in res], axis=0)
    obj = np.concatenate([r[1] for r in res], axis=1)
    return C, obj


# ------------------------------------------------------------ encoding

def _encode_task(args):
    import oracle
    w, centres, C, a, b, path = args
    X = synth.mixture_vectors(w, centres, a, b)
    codes, _ = oracle.pq_encode_f32(X, C)
    out = np.load(path, mmap_mode="r+")
    out[a:b] = codes
    out.flush()
    return b - a


class OracleIndex:
    """A workload index built by the oracle (``ix``: a ``synth.Index``) and
    the memory-mapped copies of its codes and attributes for worker
    processes."""

    def __init__(self, w: synth.Workload, workers: int | None = None, iters: int | None = None):
        self.dir = tempfile.mkdtemp(prefix="ifvs_oracle_ix_")
        try:
            self._build(w, workers, iters)
        except BaseException:
            self.close()
            raise

    def _build(self, w, workers, iters):
        centres = synth.mixture_centres(w)
        sample = synth.mixture_vectors(w, centres, 0, synth.pq_sample_rows(w))
        C, self.objective = train_codebook(w, sample, iters, workers)
        self.paths = {"codes": os.path.join(self.dir, "codes.npy")}
        np.lib.format.open_memmap(self.paths["codes"], mode="w+", dtype=np.uint8,
                                  shape=(w.N, w.M)).flush()
        tasks = [(w, centres, C, a, min(w.N, a + ENCODE_ROWS), self.paths["codes"])
                 for a in range(0, w.N, ENCODE_ROWS)]
        n = _workers(len(tasks), workers)
        if n == 1:
            for t in tasks:
                _encode_task(t)
        else:
            with _pool(n) as pool:
                list(pool.map(_encode_task, tasks))
        codes = np.array(np.load(self.paths["codes"], mmap_mode="r"))
        self.ix = synth.mixture_index(w, C, codes)
        self.paths["attrs"] = []
        for i, a in enumerate(self.ix.attrs):
            p = os.path.join(self.dir, "attr%d.npy" % i)
            np.save(p, a)
            self.paths["attrs"].append(p)
        self.paths["codebook"] = os.path.join(self.dir, "codebook.npy")
        np.save(self.paths["codebook"], self.ix.codebook)

    def close(self):
        if self.dir:
            shutil.rmtree(self.dir, ignore_errors=True)
            self.dir = None

    def __del__(self):
        self.close()

    # -------------------------------------------------------- searches

    def search(self, cond, queries, preds, wz, k, check_ids=None, workers=None):
        """The oracle's whole path (§2) for each query, over every row, in
        worker processes.  Returns per query a dict: ids, dists, npass, lut
        and, when ``check_ids`` [nq][k'] is given, ``check_dist`` (the
        oracle's distance of each of those rows, NaN for -1) and
        ``check_pass`` (whether each passes the query's predicate)."""
        nq = len(queries)
        tasks = []
        for i in range(nq):
            tasks.append((self.paths, cond.bank, cond.W, cond.seeds, queries[i:i + 1], preds[i:i + 1],
                          None if wz is None else wz[i:i + 1], k,
                          None if check_ids is None else np.asarray(check_ids[i])))
        n = _workers(nq, workers)
        if n == 1:
            return [_search_task(t) for t in tasks]
        with _pool(n) as pool:
            return list(pool.map(_search_task, tasks))


def _search_task(args):
    import oracle
    paths, bank, W, seeds, q, pred, wz, k, check = args
    codes = np.load(paths["codes"], mmap_mode="r")
    attrs = [np.load(p, mmap_mode="r") for p in paths["attrs"]]
    cb = np.load(paths["codebook"])
    codes_a = np.asarray(codes)
    attrs_a = [np.asarray(a) for a in attrs]
    ids, d, npass, st = oracle.search(codes_a, attrs_a, cb, q, pred, k, bank=bank, W=W, seeds=seeds,
                                      wz=wz, want_stages=True)
    out = {"ids": ids[0], "dists": d[0], "npass": int(npass[0]), "lut": st["lut"][0]}
    if check is not None:
        cd = np.full(len(check), np.nan)
        cp = np.zeros(len(check), dtype=bool)
        for j, r in enumerate(check):
            if r >= 0:
                cd[j] = oracle.adc(st["lut"][0], codes_a[r])
                cp[j] = oracle.row_passes(attrs_a, int(r), pred[0])
        out["check_dist"] = cd
        out["check_pass"] = cp
    return out
