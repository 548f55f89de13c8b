#!/usr/bin/env python3
"""Benchmark of the iFVS query path: QPS at recall@k per selectivity bin.

Workload: gmm100m-d128-m16 — 10^8 PQ-coded rows (M = 16 subspaces x 8
dimensions, K = 256, uint8 codes, 1.6 GB), one int32 attribute uniform in
[0, 10^6), queries in batches of 1024 with range predicates at 0.1 %, 1 %,
10 % and 100 % selectivity, k = 100, conditioned codebooks (memory bank
B = 4096, h = 2, r = 8) and per-query w_z.  A step is one batch of 1024
queries through the whole path (filter, fingerprint, alpha, w_f, Delta,
C_iFVS, tables, scan, top-k merge); steps cycle through the four bins.

Printed (rank 0): one JSON line with the value (queries per second over
all ranks, inputs resident on the device), e2e (the same through the C ABI
with pinned host buffers), per-bin QPS and recall@k, the scan kernel's
roofline figures, clocks sampled during the timed region, and the oracle
timed on host cores as a reported CPU baseline.

``--impl reference`` times the oracle instead (the plain C CPU program of
the method), on a bounded sample of the same workload.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import statistics
import subprocess
import sys
import time

_T0 = time.time()


def phase(msg):
    """Progress of the run on stderr (seconds since start); stdout carries
    only the JSON line."""
    sys.stderr.write("[bench %7.1f s] %s\n" % (time.time() - _T0, msg))
    sys.stderr.flush()

import numpy as np

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

WORKLOAD = "gmm100m-d128-m16"
LIST_DEFAULT_PPM = 1000000   # the library's default sorted-copy threshold (always)
PAIR_DEFAULT_ROWS = 1 << 22  # the library's default span from which ranges pair
TRAIN_WORKLOAD = "sift1m-d128-m16"
CPU_SAMPLE_ROWS = 10_000_000


def parse():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=16)
    ap.add_argument("--warmup", type=int, default=4)
    ap.add_argument("--impl", default="ifvs", choices=["ifvs", "reference"])
    ap.add_argument("--workload", default=None,
                    help="default: %s (search, pq), %s (train)" % (WORKLOAD, TRAIN_WORKLOAD))
    ap.add_argument("--rows", type=int, default=0, help="override N (smaller runs)")
    ap.add_argument("--sels", default="", help="override the selectivity bins, comma-separated fractions")
    ap.add_argument("--recall-queries", type=int, default=64, help="per bin; 0 = skip")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--chunk-blocks", type=int, default=0, help="scan chunk size in 1024-row blocks (0 = auto)")
    ap.add_argument("--rerank", type=int, default=0,
                    help="exact float32 rerank of the R best ADC candidates (loads the raw vectors; 0 = off)")
    ap.add_argument("--list-max-ppm", type=int, default=0,
                    help="sorted-copy scan for one-column pools up to this many rows per million "
                         "(0 = library default: always, -1 = never)")
    ap.add_argument("--pair-min-rows", type=int, default=0,
                    help="two-query CTAs for overlapping one-column ranges spanning at least this many "
                         "rows (0 = library default, -1 = never)")
    ap.add_argument("--plain-loads", action="store_true",
                    help="one-query sorted-copy CTAs read code rows by vector loads, not bulk copies")
    ap.add_argument("--out", default="", help="also write the JSON line to this file")
    ap.add_argument("--mode", default="search", choices=["search", "pq", "train"],
                    help="search: the query path; pq: PQ encoding + Lloyd training of the index; "
                         "train: SGD steps on the bank, W and w_z")
    ap.add_argument("--train-neg", type=int, default=32, help="hard negatives per query (--mode train)")
    ap.add_argument("--train-tau", type=float, default=8.0, help="softmax temperature (--mode train)")
    ap.add_argument("--train-lambda", type=float, default=0.001, help="anchor weight (--mode train)")
    ap.add_argument("--train-lr", type=float, default=5.0, help="SGD step for bank and W (--mode train)")
    ap.add_argument("--train-lr-wz", type=float, default=0.0,
                    help="SGD step for w_z (--mode train; 0 keeps the initial w_f = 1)")
    ap.add_argument("--pq-rows", type=int, default=1 << 24, help="rows encoded per step (--mode pq)")
    ap.add_argument("--pq-train-rows", type=int, default=1 << 20, help="Lloyd sample rows (--mode pq)")
    ap.add_argument("--pq-iters", type=int, default=25, help="Lloyd iterations (--mode pq)")
    return ap.parse_args()


def workload(args):
    from paper_2607_22922_gb300 import synth
    name = args.workload or (TRAIN_WORKLOAD if args.mode == "train" else WORKLOAD)
    w = synth.WORKLOADS[name]
    if args.rows:
        w = synth.scaled(w, N=args.rows)
    if args.sels:
        w = synth.scaled(w, sels=tuple(float(x) for x in args.sels.split(",")))
    if w.batch <= 0:
        # workloads whose recipe names no batch size run 1024-query steps
        w = synth.scaled(w, batch=min(w.nq, 1024))
    return w


def dist_env():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return world, rank, local


def dist_init(world, device):
    if world <= 1:
        return None
    import torch
    import torch.distributed as dist
    backend = "nccl" if torch.cuda.is_available() else "gloo"
    kw = {"device_id": device} if backend == "nccl" else {}
    try:
        dist.init_process_group(backend=backend, **kw)
    except TypeError:
        dist.init_process_group(backend=backend)
    return dist


def reduce_max(dist, x, device):
    """Max of a float over ranks (identity for one rank)."""
    if dist is None:
        return x
    import torch
    t = torch.tensor([float(x)], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def whole_job_qps(world, steps, batch, max_ms):
    """Queries per second of the whole job: every rank ran `steps` batches of
    `batch` queries; the job took the slowest rank's time."""
    return world * steps * batch / (max_ms / 1000.0)


def barrier(dist, device=None):
    if dist is not None:
        if device is not None and dist.get_backend() == "nccl":
            dist.barrier(device_ids=[device.index])
        else:
            dist.barrier()


class Clocks:
    """nvidia-smi sampling of SM clocks and throttle reasons (every 200 ms)."""
    FIELDS = ("index,clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, gpu_id=None):
        self.proc = None
        self.gpu_id = gpu_id

    def start(self):
        cmd = ["nvidia-smi", "--query-gpu=" + self.FIELDS, "--format=csv,noheader,nounits",
               "-lms", "200"]
        if self.gpu_id:
            cmd[1:1] = ["-i", str(self.gpu_id)]
        try:
            self.proc = subprocess.Popen(cmd, stdout=subprocess.PIPE, stderr=subprocess.DEVNULL,
                                         text=True)
        except OSError:
            self.proc = None

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.25)
        self.proc.terminate()
        try:
            out, _ = self.proc.communicate(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
            out, _ = self.proc.communicate()
        mhz, mx, reasons = [], [], set()
        names = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")
        for line in out.strip().splitlines():
            f = [x.strip() for x in line.split(",")]
            if len(f) < 9:
                continue
            try:
                mhz.append(float(f[1]))
                mx.append(float(f[2]))
            except ValueError:
                continue
            for n, v in zip(names, f[5:9]):
                if v.lower().startswith("active"):
                    reasons.add(n)
        if not mhz:
            return None
        return {"sm_mhz": statistics.median(mhz), "sm_max_mhz": max(mx),
                "samples": len(mhz), "reasons": sorted(reasons)}


def measured_peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            d = json.load(f)
        return float(d["hbm_gbs"]), "measured"
    return 6800.0, "fallback"


SCAN_SOURCES = ("scan_common.cuh", "scan.cu", "scan_list.cu", "scan_pair.cu")


def sources_sha256(sources):
    """sha256 over the given csrc files, in order."""
    h = hashlib.sha256()
    for src in sources:
        with open(os.path.join(ROOT, "paper_2607_22922_gb300", "csrc", src), "rb") as f:
            h.update(f.read())
    return h.hexdigest()


def traffic_summary(summary, sources):
    """A committed ncu summary (profiles/), valid only while the kernels'
    source files are unchanged (their sha256 is recorded in it); None
    otherwise."""
    p = os.path.join(ROOT, "profiles", summary)
    if not os.path.exists(p):
        return None
    with open(p) as f:
        d = json.load(f)
    if d.get("sources") != list(sources) or d.get("sources_sha256") != sources_sha256(sources):
        return None
    return d


def kernel_traffic(summary, sources):
    """DRAM bytes per launch from a committed ncu summary (or None)."""
    d = traffic_summary(summary, sources)
    return None if d is None else d.get("dram_bytes_per_launch")


def scan_dram(workload_name, hbm_peak):
    """DRAM traffic of the scan stage per bin from the committed ncu summary
    of this workload (bytes per batch and GB/s over the kernel time under
    ncu, as a fraction of the measured HBM peak), or None."""
    d = traffic_summary("scan_traffic.json", SCAN_SOURCES)
    if d is None or d.get("workload_name") != workload_name:
        return None
    out = {"bytes_per_batch": d.get("dram_bytes_per_launch"), "source": "profiles/scan_traffic.json",
           "how": d.get("how"), "bins": {}}
    for sel, gb in d.get("per_bin_dram_GB", {}).items():
        ms = d.get("per_bin_duration_ms_under_ncu", {}).get(sel)
        gbs = gb / (ms / 1000.0) if ms else None
        out["bins"][sel] = {"dram_GB": gb, "ms_under_ncu": ms, "GBps": gbs,
                            "frac_of_hbm": gbs / hbm_peak if gbs and hbm_peak else None}
    return out


# ------------------------------------------------------------ index

def build_index_gpu(w, device, ifvs, local):
    """The workload's index built on the device with the library's PQ
    kernels, in the paper's order (§1): raw vectors drawn from the stated
    mixture block by block on the device (never on the host), a codebook
    trained by ``w.pq_iters`` Lloyd iterations (ifvs_pq_train) on the first
    ``w.pq_sample`` rows from synth's start codewords, and every row encoded
    (ifvs_pq_encode).  Returns the synth.Index (host codes) and the seconds
    spent."""
    import torch
    from paper_2607_22922_gb300 import synth
    t0 = time.time()
    dio = ifvs.IFVS_F_DEVICE_IO
    # every step (torch's draws and the library's calls) runs on one stream
    # of its own, so each library call reads inputs that are already written
    st = torch.cuda.Stream(device=device)
    with torch.cuda.stream(st):
        return _build_index_gpu(w, device, ifvs, local, st, dio, t0)


def _build_index_gpu(w, device, ifvs, local, st, dio, t0):
    import torch
    from paper_2607_22922_gb300 import synth
    sptr = st.cuda_stream
    ct = torch.from_numpy(synth.mixture_centres(w)).to(device)
    n_s = synth.pq_sample_rows(w)
    block = 1 << 22
    sample = torch.cat([synth.mixture_vectors_torch(w, ct, a, min(n_s, a + block), device)
                        for a in range(0, n_s, block)])
    C0 = torch.from_numpy(synth.pq_start_codebook(w, sample.cpu().numpy())).to(device)
    C = torch.empty_like(C0)
    ifvs.ifvs_pq_train(sample, C0, w.pq_iters, device=local, C_out=C, objective=None, flags=dio, stream=sptr)
    del sample
    codes = torch.empty((w.N, w.M), dtype=torch.uint8, device=device)
    for a in range(0, w.N, block):
        b = min(w.N, a + block)
        x = synth.mixture_vectors_torch(w, ct, a, b, device)
        ifvs.ifvs_pq_encode(x, C, device=local, codes=codes[a:b], flags=dio, stream=sptr)
    st.synchronize()
    ix = synth.mixture_index(w, C.cpu().numpy(), codes.cpu().numpy(), source="mixture-torch")
    del codes, ct
    torch.cuda.empty_cache()
    return ix, time.time() - t0


def device_vectors(w, ix, a, b, device, centres_t=None):
    """Raw vectors of rows [a, b) of a device-built index (one 2^22 block)."""
    import torch
    from paper_2607_22922_gb300 import synth
    ct = centres_t if centres_t is not None else torch.from_numpy(ix.centres).to(device)
    return synth.mixture_vectors_torch(w, ct, a, b, device)


# ------------------------------------------------------------ CPU baseline

def cpu_baseline(w, ix, cond, batches, max_seconds=30.0):
    """The oracle as it stands, single-threaded, on one query per bin over the
    first CPU_SAMPLE_ROWS rows; per-query time scaled by N / rows."""
    import oracle
    rows = min(CPU_SAMPLE_ROWS, w.N)
    codes = ix.codes[:rows]
    attrs = [a[:rows] for a in ix.attrs]
    t_total, nq = 0.0, 0
    for qs in batches:
        t0 = time.perf_counter()
        oracle.search(codes, attrs, ix.codebook, qs.q[:1], qs.preds[:1], w.k, bank=cond.bank,
                      W=cond.W, seeds=cond.seeds, wz=qs.wz[:1])
        t_total += (time.perf_counter() - t0) * (w.N / rows)
        nq += 1
        if t_total > max_seconds * (w.N / rows):
            break
    return {"value": nq / t_total, "unit": "queries/s", "cores": 1, "kind": "oracle",
            "sample": "1 query per selectivity bin (%d bins) over the first %d of %d rows, "
                      "time scaled by N/rows" % (nq, rows, w.N)}


def _oracle_worker(args):
    """One oracle query in a worker process (memory-mapped sample arrays)."""
    import oracle
    paths, k, qi = args
    codes = np.load(paths["codes"], mmap_mode="r")
    attrs = [np.load(p, mmap_mode="r") for p in paths["attrs"]]
    arr = {n: np.load(paths[n]) for n in ("codebook", "bank", "W", "seeds", "q", "preds", "wz")}
    t0 = time.perf_counter()
    oracle.search(np.asarray(codes), [np.asarray(a) for a in attrs], arr["codebook"], arr["q"][qi:qi + 1],
                  arr["preds"][qi:qi + 1], k, bank=arr["bank"], W=arr["W"], seeds=arr["seeds"],
                  wz=arr["wz"][qi:qi + 1])
    return time.perf_counter() - t0


def cpu_baseline_parallel(w, ix, cond, batches, queries_per_core=2):
    """The same oracle on every host core: a spawn process pool (the GPU is
    in use in this process) runs one query per task over memory-mapped
    copies of the first CPU_SAMPLE_ROWS rows; throughput = queries / wall
    time, scaled by N / rows."""
    import multiprocessing as mp
    import shutil
    import tempfile
    import oracle
    oracle.build()
    cores = os.cpu_count() or 1
    rows = min(CPU_SAMPLE_ROWS, w.N)
    d = tempfile.mkdtemp(prefix="ifvs_cpu_")
    try:
        paths = {"codes": os.path.join(d, "codes.npy"), "attrs": []}
        np.save(paths["codes"], ix.codes[:rows])
        for i, a in enumerate(ix.attrs):
            pa = os.path.join(d, "attr%d.npy" % i)
            np.save(pa, a[:rows])
            paths["attrs"].append(pa)
        nq = cores * queries_per_core
        pick = [(b, j) for j in range(nq) for b in range(len(batches))][:nq]
        q = np.stack([batches[b].q[j % len(batches[b].q)] for b, j in pick])
        pr = np.stack([batches[b].preds[j % len(batches[b].q)] for b, j in pick])
        wz = np.stack([batches[b].wz[j % len(batches[b].q)] for b, j in pick])
        for n, v in (("codebook", ix.codebook), ("bank", cond.bank), ("W", cond.W), ("seeds", cond.seeds),
                     ("q", q), ("preds", pr), ("wz", wz)):
            paths[n] = os.path.join(d, n + ".npy")
            np.save(paths[n], v)
        with mp.get_context("spawn").Pool(cores) as pool:
            pool.map(_oracle_worker, [(paths, w.k, 0)] * cores)          # warm: load the library
            t0 = time.perf_counter()
            pool.map(_oracle_worker, [(paths, w.k, i) for i in range(nq)])
            wall = time.perf_counter() - t0
    finally:
        shutil.rmtree(d, ignore_errors=True)
    return {"value": nq / (wall * (w.N / rows)), "unit": "queries/s", "cores": cores, "kind": "oracle",
            "sample": "%d queries cycling through the bins, %d worker processes, over the first %d of %d "
                      "rows; wall time scaled by N/rows" % (nq, cores, rows, w.N)}


# ------------------------------------------------------------ recall

def _pass_mask(attr_blocks, preds, device):
    """[nq][n] pass mask of the predicates (every clause, every operator, in
    int64) on one block of the attribute columns; measurement code for the
    recall ground truth."""
    import torch
    nq = len(preds)
    n = attr_blocks[0].shape[0]
    stack = torch.stack(attr_blocks)                          # [n_attrs][n]
    ok = torch.ones((nq, n), dtype=torch.bool, device=device)
    nc = torch.from_numpy(preds["n_clauses"].astype(np.int64)).to(device)
    for j in range(4):
        cl = preds["c"][:, j]
        col = torch.from_numpy(np.clip(cl["col"], 0, len(attr_blocks) - 1).astype(np.int64)).to(device)
        op = torch.from_numpy(cl["op"].astype(np.int64)).to(device)[:, None]
        lo = torch.from_numpy(cl["lo"].astype(np.int64)).to(device)[:, None]
        hi = torch.from_numpy(cl["hi"].astype(np.int64)).to(device)[:, None]
        a = stack[col]                                        # [nq][n]
        cond = torch.where(op == 0, a == lo,
               torch.where(op == 1, (a >= lo) & (a < hi),
               torch.where(op == 2, a >= lo,
               torch.where(op == 3, a < lo,
               torch.where(op == 4, a > lo, a <= lo)))))
        ok &= cond | (nc[:, None] <= j)
    return ok


def exact_topk_gpu(w, ix, q, preds, k, device):
    """Exact filtered top-k (§3.1) over the raw vectors (drawn on the device
    block by block) in fp64 with torch: ids [nq][k] (-1 padded), outside any
    timed region."""
    import torch
    from paper_2607_22922_gb300 import synth
    block = 1 << 22
    ct = torch.from_numpy(ix.centres).to(device)
    qs_all = torch.from_numpy(np.ascontiguousarray(q)).to(device).double()
    nq = qs_all.shape[0]
    best_d = torch.full((nq, k), float("inf"), dtype=torch.float64, device=device)
    best_i = torch.full((nq, k), -1, dtype=torch.int64, device=device)
    qn = (qs_all * qs_all).sum(1, keepdim=True)
    for s in range(0, w.N, block):
        e = min(w.N, s + block)
        x = device_vectors(w, ix, s, e, device, ct).double()
        d = qn + (x * x).sum(1)[None, :] - 2.0 * qs_all @ x.T
        cols = [torch.from_numpy(a[s:e].astype(np.int64)).to(device) for a in ix.attrs]
        ok = _pass_mask(cols, preds, device)
        d = torch.where(ok, d, torch.full_like(d, float("inf")))
        kk = min(k, e - s)
        dv, di = torch.topk(d, kk, dim=1, largest=False)
        di = di + s
        cd = torch.cat([best_d, dv], 1)
        ci = torch.cat([best_i, di], 1)
        o = torch.argsort(cd, dim=1, stable=True)[:, :k]
        best_d = torch.gather(cd, 1, o)
        best_i = torch.gather(ci, 1, o)
        best_i = torch.where(torch.isinf(best_d), torch.full_like(best_i, -1), best_i)
    return best_i.cpu().numpy()


def recall_vs(gt, ids):
    r = []
    for g, i in zip(gt, ids):
        valid = g[g >= 0]
        if len(valid):
            r.append(len(np.intersect1d(valid, i)) / len(valid))
    return float(np.mean(r)) if r else None


def recall_at_k(w, ix, batches, ids_by_bin, nsample, device):
    """recall@k of the returned ids against the exact filtered top-k (§3.1)
    over the raw vectors, for the first ``nsample`` queries of each bin."""
    q = np.concatenate([b.q[:nsample] for b in batches])
    preds = np.concatenate([b.preds[:nsample] for b in batches])
    gt = exact_topk_gpu(w, ix, q, preds, w.k, device)
    out = {}
    for b, (qs, ids) in enumerate(zip(batches, ids_by_bin)):
        out[qs.sel] = recall_vs(gt[b * nsample:(b + 1) * nsample], ids[:nsample])
    return out


def sorted_path(preds, attrs, npass, list_rows):
    """Queries the library scans from a sorted copy, by its rule: a predicate
    no row can pass; a predicate on no column or on one column whose pool
    holds at most list_rows rows; on an index of two columns, one that fixes
    a column to a single value and bounds the other, pool size likewise.
    Clause intervals are intersected per column and clipped to the column's
    type, as the library canonicalises them."""
    ends = {0: lambda c: (c["lo"], c["lo"]), 1: lambda c: (c["lo"], c["hi"] - 1),
            2: lambda c: (c["lo"], None), 3: lambda c: (None, c["lo"] - 1),
            4: lambda c: (c["lo"] + 1, None), 5: lambda c: (None, c["lo"])}
    out = np.zeros(len(preds), bool)
    for i, p in enumerate(preds):
        iv = {}
        for c in p["c"][:int(p["n_clauses"])]:
            col = int(c["col"])
            info = np.iinfo(attrs[col].dtype)
            lo, hi = ends[int(c["op"])](c)
            lo = info.min if lo is None else max(int(lo), info.min)
            hi = info.max if hi is None else min(int(hi), info.max)
            a, b = iv.get(col, (info.min, info.max))
            iv[col] = (max(a, lo), min(b, hi))
        small = npass[i] <= list_rows
        if any(a > b for a, b in iv.values()):
            out[i] = True
        elif len(iv) == 0:
            out[i] = len(attrs) > 0 and small
        elif len(iv) == 1:
            out[i] = small
        elif len(iv) == 2 and len(attrs) == 2:
            out[i] = small and any(a == b for a, b in iv.values())
    return out


def scan_lookups(w, qs, sorted_vals, on_list, npass, pair_rows, seg=2048):
    """Shared-memory look-ups the scan stage executes for one batch, by the
    library's pairing rule for one-column ranges of the sorted copy (M = 16;
    sort by (column, range start, query) per 2048-query segment; neighbours
    2j, 2j+1 pair when 3/4 of the longer range is common and the two span at
    least pair_rows): a pair costs the union of its ranges x M (one load
    serves both queries), any other query its pool x M."""
    n = len(qs.q)
    a = np.zeros(n, np.int64)
    b = np.zeros(n, np.int64)
    col = np.zeros(n, np.int64)
    c0 = qs.preds["c"][:, 0]
    col[on_list] = c0["col"][on_list]
    for cc in np.unique(col[on_list]):
        sel = on_list & (col == cc)
        v = sorted_vals[cc]
        # bounds clipped to the column's type, so that the search does not
        # convert the whole column to int64
        info = np.iinfo(v.dtype)
        a[sel] = np.searchsorted(v, np.clip(c0["lo"][sel], info.min, info.max).astype(v.dtype), "left")
        hi = c0["hi"][sel]
        bb = np.searchsorted(v, np.clip(hi, info.min, info.max).astype(v.dtype), "left")
        b[sel] = np.where(hi > info.max, len(v), bb)
    paired = np.zeros(n, bool)
    union = 0.0

    def pair_ok(x, y):
        lx, ly = b[x] - a[x], b[y] - a[y]
        if col[x] != col[y] or lx <= 0 or ly <= 0:
            return False
        common = min(b[x], b[y]) - max(a[x], a[y])
        span = max(b[x], b[y]) - min(a[x], a[y])
        return 4 * common >= 3 * max(lx, ly) and span >= pair_rows

    if w.M == 16 and pair_rows >= 0:
        for s0 in range(0, n, seg):
            idx = [i for i in range(s0, min(n, s0 + seg)) if on_list[i]]
            idx.sort(key=lambda i: (col[i], a[i], i))
            for j in range(0, len(idx) - 1, 2):
                x, y = idx[j], idx[j + 1]
                if pair_ok(x, y):
                    paired[x] = paired[y] = True
                    union += max(b[x], b[y]) - min(a[x], a[y])
    single = float(npass[~paired].sum())
    return {"lookups": (single + union) * w.M, "paired_share": float(paired.mean())}


# ------------------------------------------------------------ arms

def run_ifvs(args):
    import torch
    world, rank, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("no CUDA device: the benchmark needs a GPU")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    dist = dist_init(world, device)
    from paper_2607_22922_gb300 import build, synth
    if rank == 0 or world == 1:
        build.build()
    barrier(dist, device)
    build.build()
    from paper_2607_22922_gb300 import ifvs

    w = workload(args)
    t0 = time.time()
    ix, t_pq = build_index_gpu(w, device, ifvs, local)
    phase("index built (%.1f s)" % t_pq)
    cond = synth.make_conditioning(ix)
    batches = [synth.make_queries(ix, s, nq=w.batch, salt=rank) for s in w.sels]
    t_gen = time.time() - t0
    t_load0 = time.time()
    if args.rerank > 0:
        # the raw vectors, drawn on the device block by block, go into the
        # index for the exact rerank (device I/O load: nothing on the host)
        ct = torch.from_numpy(ix.centres).to(device)
        vecs = torch.empty((w.N, w.D), dtype=torch.float32, device=device)
        for s0 in range(0, w.N, 1 << 22):
            s1 = min(w.N, s0 + (1 << 22))
            vecs[s0:s1] = device_vectors(w, ix, s0, s1, device, ct)
        g = ifvs.Index(torch.from_numpy(ix.codes).to(device),
                       [torch.from_numpy(a).to(device) for a in ix.attrs], vectors=vecs, D=w.D,
                       device=local, K=w.K, device_io=True)
        del vecs, ct
        torch.cuda.empty_cache()
    else:
        g = ifvs.Index(ix.codes, ix.attrs, device=local)
    g.load_codebooks(ix.codebook, bank=cond.bank, W=cond.W, hash_seeds=cond.seeds)
    t_load = time.time() - t_load0
    phase("index loaded")

    stream = torch.cuda.Stream(device=device)
    sptr = stream.cuda_stream
    nb = len(batches)
    dev_in, dev_out = [], []
    for qs in batches:
        dev_in.append((torch.from_numpy(qs.q).to(device),
                       torch.from_numpy(qs.preds.view(np.uint8).copy()).to(device),
                       torch.from_numpy(qs.wz).to(device)))
        n = len(qs.q)
        dev_out.append((torch.empty((n, w.k), dtype=torch.int64, device=device),
                        torch.empty((n, w.k), dtype=torch.float32, device=device),
                        torch.empty(n, dtype=torch.int64, device=device)))
    torch.cuda.synchronize()
    flags = ifvs.IFVS_F_DEVICE_IO | ifvs.IFVS_F_STAGE_TIMING | (ifvs.IFVS_F_PLAIN_LOADS if args.plain_loads else 0)

    def step(i):
        b = i % nb
        q, p, wz = dev_in[b]
        oi, od, on = dev_out[b]
        ifvs.ifvs_search_batch(g.h, q, p, w.k, wz=wz, ids=oi, dists=od, npass=on,
                               flags=flags, stream=sptr, chunk_blocks=args.chunk_blocks,
                               list_max_ppm=args.list_max_ppm, rerank=args.rerank,
                               pair_min_rows=args.pair_min_rows)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    g.stage_times(reset=True)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    gpu_uuid = None
    try:
        gpu_uuid = torch.cuda.get_device_properties(device).uuid
        gpu_uuid = "GPU-" + str(gpu_uuid) if gpu_uuid is not None else None
    except Exception:
        gpu_uuid = None
    clocks = Clocks(gpu_uuid)
    barrier(dist, device)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    with torch.cuda.stream(stream):
        ev[0].record(stream)
        for i in range(args.steps):
            step(args.warmup + i)
            ev[i + 1].record(stream)
    torch.cuda.synchronize()
    barrier(dist, device)
    clk = clocks.stop()
    step_ms = [ev[i].elapsed_time(ev[i + 1]) for i in range(args.steps)]
    total_ms = ev[0].elapsed_time(ev[-1])
    max_ms = reduce_max(dist, total_ms, device)
    stages = g.stage_times(reset=True)
    launches = sum(v[1] for v in stages.values())

    # per-bin figures and the scan-stage roofline
    per_bin = {}
    n_blocks = (w.N + 1023) // 1024
    ppm = args.list_max_ppm if args.list_max_ppm != 0 else LIST_DEFAULT_PPM
    list_rows = -1 if ppm < 0 else w.N * ppm // 1000000
    pair_rows = args.pair_min_rows if args.pair_min_rows != 0 else PAIR_DEFAULT_ROWS
    lookups_total = code_bytes_total = 0.0
    sorted_vals = [np.sort(a) for a in ix.attrs]
    for b, qs in enumerate(batches):
        ms_b = [step_ms[i] for i in range(args.steps) if (args.warmup + i) % nb == b]
        npass = dev_out[b][2].cpu().numpy().astype(np.float64)
        nsteps_b = len(ms_b)
        on_list = sorted_path(qs.preds, ix.attrs, npass, list_rows)
        lk = scan_lookups(w, qs, sorted_vals, on_list, npass, pair_rows)
        lookups_total += nsteps_b * lk["lookups"]
        code_bytes_total += nsteps_b * float(npass.sum()) * w.M
        per_bin[str(qs.sel)] = {
            "qps": (len(qs.q) * nsteps_b) / (sum(ms_b) / 1000.0) if ms_b else None,
            "ms_per_batch": float(np.mean(ms_b)) if ms_b else None,
            "mean_selectivity": float(npass.mean() / w.N),
            "sorted_path_share": float(on_list.mean()),
            "paired_share": lk["paired_share"]}
    # The scan stage (per batch: k_pair_items, k_scan_list_pair, k_scan_list
    # and k_scan, one launch of each) is the unit.  Its binding resource is
    # the shared-memory look-up rate: one conflict-free 32-lane load per SM
    # per cycle.  Executed look-ups per batch: passing positions x M for a
    # query scanned alone, and for a pair of queries the positions of the
    # union of their ranges x M (one load serves both).  Code bytes (every
    # query's pool once) are reported beside it: DRAM carries far less,
    # because the CTAs of a batch share the codes through L2.
    scan_ms, _ = stages["scan"]
    nbatch = args.steps
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    mhz = (clk or {}).get("sm_mhz") or (clk or {}).get("sm_max_mhz") or 2070.0
    peak = sms * 32 * mhz * 1e6
    achieved = (lookups_total / nbatch) / (scan_ms / nbatch / 1000.0) if scan_ms > 0 else None
    hbm_peak, peak_kind = measured_peaks()
    dram = scan_dram(w.name, hbm_peak)
    roofline = {"kernel": "scan stage (k_pair_items + k_scan_list_pair + k_scan_list_bulk; k_scan_list and"
                          " k_scan where a query takes them)",
                "bound": "smem", "achieved": achieved, "peak": peak, "unit": "look-ups/s",
                "frac": achieved / peak if achieved else None,
                "traffic": dram["bytes_per_batch"] if dram else None,
                "peak_kind": "derived: %d SMs x 32 lanes x %.0f MHz (median SM clock under load; one "
                             "conflict-free 32-lane shared load per SM per cycle)" % (sms, mhz),
                "launch_unit": "one batch of the scan stage (its four kernels)",
                "avg_launch_ms": scan_ms / nbatch,
                "lookups_per_launch": lookups_total / nbatch,
                "code_bytes_per_launch": code_bytes_total / nbatch,
                "code_bytes_per_s": (code_bytes_total / nbatch) / (scan_ms / nbatch / 1000.0) if scan_ms > 0 else None,
                "dram": dram, "hbm_peak_gbs": hbm_peak, "hbm_peak_kind": peak_kind}
    share = {k: v[0] for k, v in stages.items()}

    phase("timed steps done")
    # end to end through the C ABI with pinned host buffers
    e2e = None
    if not args.no_e2e:
        host_in, host_out = [], []
        for qs in batches:
            n = len(qs.q)
            hq = torch.from_numpy(qs.q).pin_memory()
            hp = torch.from_numpy(qs.preds.view(np.uint8).copy()).pin_memory()
            hw = torch.from_numpy(qs.wz).pin_memory()
            host_in.append((hq.numpy(), hp.numpy().view(synth.PREDICATE_DTYPE), hw.numpy(), (hq, hp, hw)))
            ho = (torch.empty((n, w.k), dtype=torch.int64).pin_memory(),
                  torch.empty((n, w.k), dtype=torch.float32).pin_memory(),
                  torch.empty(n, dtype=torch.int64).pin_memory())
            host_out.append((ho[0].numpy(), ho[1].numpy(), ho[2].numpy(), ho))

        def hstep(i):
            b = i % nb
            q, p, wz, _ = host_in[b]
            oi, od, on, _ = host_out[b]
            ifvs.ifvs_search_batch(g.h, q, p, w.k, wz=wz, ids=oi, dists=od, npass=on, stream=sptr,
                                   chunk_blocks=args.chunk_blocks, list_max_ppm=args.list_max_ppm,
                                   rerank=args.rerank, pair_min_rows=args.pair_min_rows,
                                   flags=ifvs.IFVS_F_PLAIN_LOADS if args.plain_loads else 0)

        for i in range(args.warmup):
            hstep(i)
        barrier(dist, device)
        torch.cuda.synchronize()
        t0 = time.perf_counter()
        for i in range(args.steps):
            hstep(args.warmup + i)
        torch.cuda.synchronize()
        e_ms = (time.perf_counter() - t0) * 1000.0
        barrier(dist, device)
        e_ms = reduce_max(dist, e_ms, device)
        nq_b = w.batch
        e2e = {"value": whole_job_qps(world, args.steps, nq_b, e_ms), "unit": "queries/s",
               "h2d_bytes_per_step": nq_b * (w.D * 4 * 2 + 104),
               "d2h_bytes_per_step": nq_b * (w.k * 12 + 8)}

    phase("e2e done")
    # recall@k (outside the timed regions)
    recall = None
    if args.recall_queries > 0 and rank == 0:
        ids_by_bin = [dev_out[b][0].cpu().numpy()[:args.recall_queries] for b in range(nb)]
        recall = recall_at_k(w, ix, batches, ids_by_bin, args.recall_queries, device)
        for s, r in recall.items():
            per_bin[str(s)]["recall@%d" % w.k] = r

    phase("recall done")
    cpu = cpu_par = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        cpu = cpu_baseline(w, ix, cond, batches)
        cpu_par = cpu_baseline_parallel(w, ix, cond, batches)

    phase("cpu baselines done")
    value = whole_job_qps(world, args.steps, w.batch, max_ms)
    line = {
        "metric": "QPS at recall@%d per selectivity bin (code-scan HBM GB/s vs peak)" % w.k,
        "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": max_ms / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f32 (uint8 codes)",
        "data": "synthetic (seeded Gaussian-mixture PQ index; paper datasets and trained weights absent)",
        "config": {"workload": w.name, "N": w.N, "D": w.D, "M": w.M, "K": w.K, "k": w.k,
                   "rerank": args.rerank,
                   "batch": w.batch, "bins": list(w.sels), "B": w.B, "h": w.h, "r": w.r,
                   "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2 (%.1f GB codes + %.1f GB attributes)"
                         % (w.N * w.M / 1e9, w.N * 4 / 1e9)},
        "bins": per_bin, "roofline": roofline, "stage_ms": share, "gpu_launches": launches,
        "clocks": clk, "e2e": e2e, "cpu_baseline": cpu, "cpu_baseline_parallel": cpu_par,
        "setup_s": round(t_gen, 1), "index_build_s": round(t_pq, 1), "index_load_s": round(t_load, 1),
    }
    if rank == 0:
        s = json.dumps(line)
        print(s, flush=True)
        if args.out:
            with open(args.out, "w") as f:
                f.write(s + "\n")
    g.close()
    if dist is not None:
        dist.destroy_process_group()


def run_pq(args):
    """PQ construction (the offline step before the query path): a step
    encodes one slice of raw vectors against the workload's codebook with
    one kernel; Lloyd training on a sample is timed beside it."""
    import torch
    world, rank, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("no CUDA device: the benchmark needs a GPU")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    dist = dist_init(world, device)
    from paper_2607_22922_gb300 import build, synth
    if rank == 0 or world == 1:
        build.build()
    barrier(dist, device)
    build.build()
    from paper_2607_22922_gb300 import ifvs

    w = workload(args)
    rows = min(args.pq_rows, w.N)
    t0 = time.time()
    # raw vectors of the workload's mixture (drawn on the device) and the
    # codebook the workload's recipe trains on its first pq_sample rows
    ct = torch.from_numpy(synth.mixture_centres(w)).to(device)
    block = 1 << 22
    X = torch.empty((rows, w.D), dtype=torch.float32, device=device)
    for s0 in range(0, rows, block):
        s1 = min(rows, s0 + block)
        X[s0:s1] = synth.mixture_vectors_torch(w, ct, s0, s1, device)
    codes = torch.empty((rows, w.M), dtype=torch.uint8, device=device)
    stream = torch.cuda.Stream(device=device)
    sptr = stream.cuda_stream
    dio = ifvs.IFVS_F_DEVICE_IO
    n_s = min(synth.pq_sample_rows(w), rows)
    cb = torch.empty((w.M, w.K, w.ds), dtype=torch.float32, device=device)
    ifvs.ifvs_pq_train(X[:n_s], torch.from_numpy(synth.pq_start_codebook(w, X[:n_s].cpu().numpy())).to(device),
                       w.pq_iters, device=local, C_out=cb, objective=None, flags=dio,
                       stream=torch.cuda.current_stream(device).cuda_stream)
    torch.cuda.synchronize()
    codebook_host = cb.cpu().numpy()
    t_gen = time.time() - t0

    def step():
        ifvs.ifvs_pq_encode(X, cb, device=local, codes=codes, flags=dio, stream=sptr)

    with torch.cuda.stream(stream):
        for _ in range(args.warmup):
            step()
    torch.cuda.synchronize()
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(args.steps + 1)]
    clocks = Clocks()
    barrier(dist, device)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    with torch.cuda.stream(stream):
        ev[0].record(stream)
        for i in range(args.steps):
            step()
            ev[i + 1].record(stream)
    torch.cuda.synchronize()
    barrier(dist, device)
    clk = clocks.stop()
    total_ms = ev[0].elapsed_time(ev[-1])
    max_ms = reduce_max(dist, total_ms, device)
    launch_ms = total_ms / args.steps

    # roofline: three rounded float32 operations (sub, mul, add) per row,
    # codeword and dimension; the FP32 pipes of 152 SMs x 128 lanes at the
    # SM clock (one operation per lane per cycle)
    props = torch.cuda.get_device_properties(device)
    sms = props.multi_processor_count
    mhz = (clk or {}).get("sm_max_mhz") or 2070.0
    ops = 3.0 * rows * w.K * w.D
    achieved = ops / (launch_ms / 1000.0) / 1e12
    peak = sms * 128 * mhz * 1e6 / 1e12
    roofline = {"kernel": "k_pq_assign", "bound": "alu", "achieved": achieved, "peak": peak,
                "unit": "TFLOP/s", "frac": achieved / peak,
                "traffic": kernel_traffic("pq_encode_traffic.json", ("pq.cu",)),
                "peak_kind": "derived: %d SMs x 128 FP32 lanes x %.0f MHz (max SM clock)" % (sms, mhz),
                "avg_launch_ms": launch_ms, "algorithmic_flop_per_launch": ops,
                "algorithmic_bytes_per_launch": rows * (w.D * 4 + w.M)}

    # Lloyd training on a sample (device I/O, 25 iterations by default)
    n_tr = min(args.pq_train_rows, rows)
    rng = np.random.default_rng(7)
    pick = torch.from_numpy(np.sort(rng.choice(n_tr, w.K, replace=False))).to(device)
    C0 = X[:n_tr][pick].reshape(w.K, w.M, w.ds).permute(1, 0, 2).contiguous()
    C1 = torch.empty_like(C0)
    obj = torch.empty((args.pq_iters, w.M), dtype=torch.float64, device=device)
    ifvs.ifvs_pq_train(X[:n_tr], C0, 1, device=local, C_out=C1, objective=obj[:1], flags=dio,
                       stream=sptr)
    torch.cuda.synchronize()
    t1 = time.perf_counter()
    ifvs.ifvs_pq_train(X[:n_tr], C0, args.pq_iters, device=local, C_out=C1, objective=obj,
                       flags=dio, stream=sptr)
    torch.cuda.synchronize()
    tr_s = time.perf_counter() - t1
    o = obj.sum(1).cpu().numpy()
    lloyd = {"rows": n_tr, "iters": args.pq_iters, "seconds": tr_s,
             "ms_per_iter": tr_s * 1000.0 / max(1, args.pq_iters),
             "objective_first": float(o[0]), "objective_last": float(o[-1]),
             "objective_non_increasing": bool((np.diff(o) <= 1e-9 * np.abs(o[:-1])).all())}

    # end to end: host vectors (pinned) in, host codes out, through the C ABI
    e2e = None
    if not args.no_e2e:
        hX = X.cpu().pin_memory()
        hXn = hX.numpy()
        ifvs.ifvs_pq_encode(hXn, codebook_host, device=local)
        barrier(dist, device)
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        for _ in range(args.steps):
            ifvs.ifvs_pq_encode(hXn, codebook_host, device=local)
        e_ms = (time.perf_counter() - t1) * 1000.0
        barrier(dist, device)
        e_ms = reduce_max(dist, e_ms, device)
        e2e = {"value": world * args.steps * rows / (e_ms / 1000.0), "unit": "rows/s",
               "h2d_bytes_per_step": rows * w.D * 4 + w.M * w.K * w.ds * 4,
               "d2h_bytes_per_step": rows * w.M}
        del hX

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        sample = 20_000
        Xs = X[:sample].cpu().numpy()
        t1 = time.perf_counter()
        done = 0
        while time.perf_counter() - t1 < 10.0:
            oracle.pq_encode_f32(Xs, codebook_host)
            done += sample
        sec = time.perf_counter() - t1
        cpu = {"value": done / sec, "unit": "rows/s", "cores": 1, "kind": "oracle",
               "sample": "float32 encode of the first %d rows, repeated for >= 10 s" % sample}

    line = {
        "metric": "PQ encode throughput (rows/s)", "value": world * args.steps * rows / (max_ms / 1000.0),
        "unit": "rows/s", "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": max_ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32", "data": "synthetic (seeded Gaussian-mixture vectors)",
        "config": {"workload": "%s raw vectors, PQ encode in %d-row slices" % (w.name, rows),
                   "rows_per_step": rows, "D": w.D, "M": w.M, "K": w.K,
                   "parallelism": "replicas" if world > 1 else "single",
                   "l2": "inputs larger than L2 (%.1f GB per step)" % (rows * w.D * 4 / 1e9)},
        "roofline": roofline, "lloyd": lloyd, "gpu_launches": args.steps, "clocks": clk,
        "e2e": e2e, "cpu_baseline": cpu, "setup_s": round(t_gen, 1),
    }
    if rank == 0:
        s = json.dumps(line)
        print(s, flush=True)
        if args.out:
            with open(args.out, "w") as f:
                f.write(s + "\n")
    if dist is not None:
        dist.destroy_process_group()


def run_train(args):
    """Training of the bank, W and w_z (§2 "Learning"): each step is one
    mini-batch of queries through ifvs_train_step (mining with the query
    path, loss, gradient, SGD); steps cycle through the selectivity bins.
    Positives are the exact filtered top-k over the raw vectors, computed
    outside the timed region; the parameters start from the paper's initial
    state (zero bank, w_f = 1)."""
    import torch
    world, rank, local = dist_env()
    if not torch.cuda.is_available():
        raise SystemExit("no CUDA device: the benchmark needs a GPU")
    device = torch.device("cuda", local)
    torch.cuda.set_device(device)
    dist = dist_init(world, device)
    from paper_2607_22922_gb300 import build, synth
    if rank == 0 or world == 1:
        build.build()
    barrier(dist, device)
    build.build()
    from paper_2607_22922_gb300 import ifvs

    w = workload(args)
    P, n_neg = w.k, args.train_neg
    t0 = time.time()
    ix, _ = build_index_gpu(w, device, ifvs, local)
    cond = synth.make_conditioning(ix)
    batches = [synth.make_queries(ix, s, nq=w.batch, salt=rank) for s in w.sels]
    gts = [exact_topk_gpu(w, ix, b.q, b.preds, P, device) for b in batches]
    t_gen = time.time() - t0
    bank0 = np.zeros_like(cond.bank)
    wz0 = np.full(w.D, math.log(math.e - 1.0), np.float32)
    g = ifvs.Index(ix.codes, ix.attrs, D=w.D, K=w.K, device=local)
    g.load_codebooks(ix.codebook, bank=bank0, W=cond.W, hash_seeds=cond.seeds)

    def recall_now(wz_host):
        ids = []
        for b in batches:
            i, _, _ = g.search(b.q, b.preds, P, wz=np.tile(wz_host, (len(b.q), 1)))
            ids.append(i)
        return [recall_vs(gt, i) for gt, i in zip(gts, ids)]

    rec0 = recall_now(wz0)
    stream = torch.cuda.Stream(device=device)
    sptr = stream.cuda_stream
    nb = len(batches)
    dev_in = [(torch.from_numpy(b.q).to(device),
               torch.from_numpy(b.preds.view(np.uint8).copy()).to(device),
               torch.from_numpy(gt).to(device)) for b, gt in zip(batches, gts)]
    wz = torch.from_numpy(wz0.copy()).to(device)
    neg = torch.empty((w.batch, n_neg), dtype=torch.int64, device=device)
    flags = ifvs.IFVS_F_DEVICE_IO | ifvs.IFVS_F_STAGE_TIMING
    losses = []

    def step(i):
        q, p, pos = dev_in[i % nb]
        L, _ = ifvs.ifvs_train_step(g.h, q, p, wz, pos, n_neg, args.train_tau, args.train_lambda,
                                    args.train_lr, flags=flags, stream=sptr, negatives=neg,
                                    lr_wz=args.train_lr_wz)
        losses.append(L)

    for i in range(args.warmup):
        step(i)
    torch.cuda.synchronize()
    g.stage_times(reset=True)
    ev = [torch.cuda.Event(enable_timing=True) for _ in range(2)]
    clocks = Clocks()
    barrier(dist, device)
    torch.cuda.synchronize()
    clocks.start()
    time.sleep(0.3)
    with torch.cuda.stream(stream):
        ev[0].record(stream)
        for i in range(args.steps):
            step(args.warmup + i)
        ev[1].record(stream)
    torch.cuda.synchronize()
    barrier(dist, device)
    clk = clocks.stop()
    total_ms = ev[0].elapsed_time(ev[1])
    max_ms = reduce_max(dist, total_ms, device)
    stages = g.stage_times(reset=True)
    launches = sum(v[1] for v in stages.values())
    rec1 = recall_now(wz.cpu().numpy())

    # end to end through the C ABI with host arrays (queries, predicates,
    # positives and w_z in; w_z, negatives and the loss out)
    e2e = None
    if not args.no_e2e:
        wzh = wz.cpu().numpy().copy()

        def hstep(i):
            b = batches[i % nb]
            ifvs.ifvs_train_step(g.h, b.q, b.preds, wzh, gts[i % nb], n_neg, args.train_tau,
                                 args.train_lambda, args.train_lr, stream=sptr,
                                 lr_wz=args.train_lr_wz)

        for i in range(args.warmup):
            hstep(i)
        barrier(dist, device)
        torch.cuda.synchronize()
        t1 = time.perf_counter()
        for i in range(args.steps):
            hstep(args.warmup + i)
        torch.cuda.synchronize()
        e_ms = reduce_max(dist, (time.perf_counter() - t1) * 1000.0, device)
        e2e = {"value": whole_job_qps(world, args.steps, w.batch, e_ms), "unit": "queries/s",
               "h2d_bytes_per_step": w.batch * (w.D * 4 + 104 + P * 8) + w.D * 4,
               "d2h_bytes_per_step": w.batch * n_neg * 8 + w.D * 4 + w.batch * 8}

    cpu = None
    if rank == 0 and world == 1 and not args.no_cpu_baseline:
        import oracle
        oracle.build()
        b = batches[2 % nb]
        nsamp = 4
        t1 = time.perf_counter()
        oracle.train_step(ix.codes, ix.attrs, ix.codebook, bank0, cond.W, cond.seeds, wz0,
                          b.q[:nsamp], b.preds[:nsamp], gts[2 % nb][:nsamp], n_neg,
                          args.train_tau, args.train_lambda, args.train_lr, args.train_lr_wz)
        sec = time.perf_counter() - t1
        cpu = {"value": nsamp / sec, "unit": "queries/s", "cores": 1, "kind": "oracle",
               "sample": "one training step on %d queries of the %g bin (full N)" % (nsamp, b.sel)}

    # roofline of the dominant kernel, the mining scan: with the codes in L2
    # its bound is the shared-memory look-up rate (one conflict-free 32-lane
    # load per SM per cycle); look-ups per launch = passing rows x M
    srt = np.sort(ix.attrs[0].astype(np.int64))
    npass = [np.searchsorted(srt, b.preds["c"][:, 0]["hi"], "left") -
             np.searchsorted(srt, b.preds["c"][:, 0]["lo"], "left") for b in batches]
    lookups = sum(float(npass[(args.warmup + i) % nb].sum()) * w.M for i in range(args.steps))
    scan_ms, scan_n = stages["scan"]
    sms = torch.cuda.get_device_properties(device).multi_processor_count
    mhz = (clk or {}).get("sm_max_mhz") or 2070.0
    peak = sms * 32 * mhz * 1e6
    achieved = (lookups / scan_n) / (scan_ms / scan_n / 1000.0) if scan_n else None
    roofline = {"kernel": "k_scan (mining)", "bound": "smem", "achieved": achieved, "peak": peak,
                "unit": "look-ups/s", "frac": achieved / peak if achieved else None, "traffic": None,
                "peak_kind": "derived: %d SMs x 32 lanes x %.0f MHz (one conflict-free shared load "
                             "per SM per cycle)" % (sms, mhz),
                "avg_launch_ms": scan_ms / scan_n if scan_n else None,
                "lookups_per_launch": lookups / scan_n if scan_n else None}
    train_ms = stages["train"][0]
    line = {
        "metric": "training throughput (queries per second through ifvs_train_step)",
        "value": whole_job_qps(world, args.steps, w.batch, max_ms), "unit": "queries/s",
        "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
        "ms_per_step": max_ms / args.steps, "higher_is_better": True, "scaling": "weak",
        "vs_baseline": None, "dtype": "f32 (fp64 distance sums and softmax)",
        "data": "synthetic (seeded Gaussian-mixture PQ index; paper datasets absent)",
        "config": {"workload": "%s, SGD on bank/W/w_z, %d-query mini-batches" % (w.name, w.batch),
                   "N": w.N, "D": w.D, "M": w.M, "K": w.K, "B": w.B, "h": w.h, "r": w.r,
                   "n_pos": P, "n_neg": n_neg, "tau": args.train_tau, "lambda": args.train_lambda,
                   "lr": args.train_lr, "lr_wz": args.train_lr_wz, "bins": list(w.sels),
                   "parallelism": "replicas" if world > 1 else "single",
                   "l2": "codes (%.0f MB) fit in L2" % (w.N * w.M / 1e6)},
        "roofline": roofline, "stage_ms": {k: v[0] for k, v in stages.items()},
        "train_share": train_ms / sum(v[0] for v in stages.values()),
        "gpu_launches": launches, "clocks": clk, "e2e": e2e, "cpu_baseline": cpu,
        "loss_first": losses[0], "loss_last": losses[-1],
        "recall@%d_before" % P: rec0, "recall@%d_after" % P: rec1, "setup_s": round(t_gen, 1),
    }
    if rank == 0:
        s = json.dumps(line)
        print(s, flush=True)
        if args.out:
            with open(args.out, "w") as f:
                f.write(s + "\n")
    g.close()
    if dist is not None:
        dist.destroy_process_group()


def run_reference(args):
    """The oracle as it stands on the host cores, over every row of the
    workload: each step runs one query per worker process (one worker per
    core, a spawn pool), the queries cycling through the bins.  The index is
    built by the oracle too (oracle.pq_index: the workload's mixture, Lloyd
    training on its first pq_sample rows, float32 encoding of every row),
    outside the timed region; no GPU is used."""
    world, rank, _ = dist_env()
    if rank != 0:
        return
    import concurrent.futures as cf
    import multiprocessing as mp
    from paper_2607_22922_gb300 import synth
    import oracle
    from oracle import pq_index
    oracle.build()
    w = workload(args)
    cores = os.cpu_count() or 1
    t0 = time.time()
    oix = pq_index.OracleIndex(w, workers=cores)
    t_build = time.time() - t0
    ix = oix.ix
    cond = synth.make_conditioning(ix)
    nb = len(w.sels)
    per_bin = max(1, -(-(args.steps + args.warmup) * cores // nb))
    batches = [synth.make_queries(ix, s, nq=min(per_bin, max(w.batch, 1)), salt=rank) for s in w.sels]

    def tasks(i):
        out = []
        for c in range(cores):
            j = i * cores + c
            qs = batches[j % nb]
            r = (j // nb) % len(qs.q)
            out.append((oix.paths, cond.bank, cond.W, cond.seeds, qs.q[r:r + 1], qs.preds[r:r + 1],
                        qs.wz[r:r + 1], w.k, None))
        return out

    try:
        with cf.ProcessPoolExecutor(max_workers=cores, mp_context=mp.get_context("spawn")) as pool:
            for i in range(args.warmup):
                list(pool.map(pq_index._search_task, tasks(i)))
            t0 = time.perf_counter()
            for i in range(args.steps):
                list(pool.map(pq_index._search_task, tasks(args.warmup + i)))
            sec = time.perf_counter() - t0
    finally:
        oix.close()
    value = args.steps * cores / sec
    sample = ("%d queries per step (one per worker process, %d processes) cycling through the %d bins, "
              "each over all %d rows; index built by the oracle in %.0f s before timing"
              % (cores, cores, nb, w.N, t_build))
    line = {
        "impl": "reference",
        "metric": "QPS at recall@%d per selectivity bin (code-scan HBM GB/s vs peak)" % w.k,
        "value": value, "unit": "queries/s", "n_gpus": world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": sec * 1000.0 / args.steps,
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
        "data": "synthetic", "config": {"workload": w.name, "N": w.N, "k": w.k,
                                        "batch": cores, "bins": list(w.sels)},
        "cpu_baseline": {"value": value, "unit": "queries/s", "cores": cores, "kind": "oracle",
                         "sample": sample},
        "e2e": {"value": value, "unit": "queries/s", "h2d_bytes_per_step": 0,
                "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    args = parse()
    if args.impl == "reference":
        run_reference(args)
    elif args.mode == "pq":
        run_pq(args)
    elif args.mode == "train":
        run_train(args)
    else:
        run_ifvs(args)


if __name__ == "__main__":
    main()
