"""Builds ``libifvs.so`` (the CUDA library behind include/ifvs.h) in-tree.

Each ``csrc/*.cu`` file is compiled for sm_103a only, in parallel, then
linked into a shared library next to this file.  ``python -m
paper_2607_22922_gb300.build [-v]`` rebuilds it; ``-v`` prints ptxas
resource usage (registers, spills, shared memory).
"""
from __future__ import annotations

import concurrent.futures as cf
import fcntl
import os
import shutil
import subprocess
import sys

HERE = os.path.dirname(os.path.abspath(__file__))
ROOT = os.path.dirname(HERE)
CSRC = os.path.join(HERE, "csrc")
INCLUDE = os.path.join(ROOT, "include")
OBJDIR = os.path.join(HERE, "_build")
SO = os.path.join(HERE, "libifvs.so")
ARCH = ["-gencode", "arch=compute_103a,code=sm_103a"]


def nvcc() -> str:
    cand = [os.environ.get("NVCC"), shutil.which("nvcc"), "/usr/local/cuda/bin/nvcc"]
    for c in cand:
        if c and os.path.exists(c):
            return c
    raise RuntimeError("nvcc not found: the CUDA toolkit is required to build libifvs.so")


def sources():
    return sorted(os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith(".cu"))


def _deps():
    hdrs = [os.path.join(CSRC, f) for f in os.listdir(CSRC) if f.endswith((".cuh", ".h"))]
    hdrs.append(os.path.join(INCLUDE, "ifvs.h"))
    return hdrs


def _stale(target, deps):
    if not os.path.exists(target):
        return True
    t = os.path.getmtime(target)
    return any(os.path.getmtime(d) > t for d in deps)


def build(force: bool = False, verbose: bool = False) -> str:
    """Compiles stale objects and relinks; concurrent callers (test workers)
    serialise on a lock file so that none links a half-written object."""
    os.makedirs(OBJDIR, exist_ok=True)
    with open(os.path.join(OBJDIR, ".lock"), "w") as lk:
        fcntl.flock(lk, fcntl.LOCK_EX)
        try:
            return _build_locked(force, verbose)
        finally:
            fcntl.flock(lk, fcntl.LOCK_UN)


def _build_locked(force: bool, verbose: bool) -> str:
    exe = nvcc()
    common = ARCH + ["-O3", "-lineinfo", "-std=c++17", "-Xcompiler", "-fPIC",
                     "-I", INCLUDE, "-I", CSRC]
    if verbose:
        common += ["-Xptxas", "-v"]
    hdrs = _deps()
    jobs = []
    for src in sources():
        name = os.path.basename(src)
        obj = os.path.join(OBJDIR, name[:-3] + ".o")
        if force or verbose or _stale(obj, [src] + hdrs + [os.path.abspath(__file__)]):
            jobs.append(([exe] + common + ["-c", src, "-o", obj + ".tmp"], obj))
    objs = [os.path.join(OBJDIR, os.path.basename(s)[:-3] + ".o") for s in sources()]

    def run(job):
        cmd, obj = job
        p = subprocess.run(cmd, capture_output=True, text=True)
        if p.returncode == 0:
            os.replace(obj + ".tmp", obj)
        return cmd, p

    if jobs:
        with cf.ThreadPoolExecutor(max_workers=min(len(jobs), os.cpu_count() or 4)) as ex:
            for cmd, p in ex.map(run, jobs):
                if verbose or p.returncode != 0:
                    sys.stderr.write(p.stdout + p.stderr)
                if p.returncode != 0:
                    raise RuntimeError("nvcc failed: " + " ".join(cmd[-3:]))
    if force or jobs or _stale(SO, objs):
        tmp = SO + ".tmp.%d" % os.getpid()
        cmd = [exe] + ARCH + ["-shared", "-o", tmp] + objs + ["-lcudart"]
        p = subprocess.run(cmd, capture_output=True, text=True)
        if p.returncode != 0:
            sys.stderr.write(p.stdout + p.stderr)
            raise RuntimeError("link of libifvs.so failed")
        os.replace(tmp, SO)
    return SO


if __name__ == "__main__":
    build(force="-f" in sys.argv, verbose="-v" in sys.argv)
    print(SO)
