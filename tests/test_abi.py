"""The C-ABI library without a GPU: it loads, exports every symbol that
include/*.h declares, and its host-side logic (predicate canonicalisation,
argument checks, error reporting) behaves as documented."""
import ctypes
import glob
import os
import re

import numpy as np
import pytest

from paper_2607_22922_gb300 import synth

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    from paper_2607_22922_gb300 import build
    build.build()
    from paper_2607_22922_gb300 import ifvs
    return ifvs


def declared_symbols():
    names = set()
    for h in glob.glob(os.path.join(ROOT, "include", "*.h")):
        text = open(h).read()
        text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
        for m in re.finditer(r"^[A-Za-z_][\w \t\*]*?\b(ifvs_\w+)\s*\(", text, flags=re.M):
            names.add(m.group(1))
    return names


def test_exports_every_declared_symbol(lib):
    names = declared_symbols()
    assert {"ifvs_load_index", "ifvs_load_codebooks", "ifvs_search_batch"} <= names
    so = ctypes.CDLL(lib.LIB_PATH)
    missing = [n for n in sorted(names) if not hasattr(so, n)]
    assert not missing, missing


def test_version_and_error_string(lib):
    assert "sm_103a" in lib.ifvs_version()
    rc = lib.lib().ifvs_search_batch(None, None, None, 1, 10, None, None, None, None, None)
    assert rc == lib.IFVS_ERR_ARG
    assert "NULL" in lib.ifvs_last_error()


def test_predicate_records_match_the_abi(lib):
    assert lib.PREDICATE_DTYPE.itemsize == 104 == synth.PREDICATE_DTYPE.itemsize


def test_parameter_structs_match_the_header(lib, tmp_path):
    """sizeof / offsetof of the header's structs, compiled by gcc, against
    the binding's ctypes layouts."""
    import subprocess
    structs = {"ifvs_search_params": (lib.SearchParams,
                                      ["flags", "rerank", "sub_batch", "chunk_blocks",
                                       "list_max_ppm", "pair_min_rows", "stream"]),
               "ifvs_train_params": (lib.TrainParams,
                                     ["tau", "lambda", "lr", "lr_wz", "n_pos", "n_neg", "flags",
                                      "stream"])}
    lines = ['#include <stdio.h>', '#include <stddef.h>', '#include "ifvs.h"', "int main(void) {"]
    for name, (_, fields) in structs.items():
        lines.append('printf("%%zu\\n", sizeof(%s));' % name)
        for f in fields:
            lines.append('printf("%%zu\\n", offsetof(%s, %s));' % (name, f))
    lines += ['printf("%zu\\n", sizeof(ifvs_predicate));', "return 0; }"]
    src = tmp_path / "layout.c"
    src.write_text("\n".join(lines))
    exe = tmp_path / "layout"
    inc = os.path.join(os.path.dirname(os.path.dirname(os.path.abspath(__file__))), "include")
    subprocess.check_call(["gcc", "-std=c99", "-I", inc, "-o", str(exe), str(src)])
    got = [int(x) for x in subprocess.check_output([str(exe)], text=True).split()]
    want = []
    for name, (cls, fields) in structs.items():
        want.append(ctypes.sizeof(cls))
        names = [f[0] for f in cls._fields_]
        for f in fields:
            want.append(getattr(cls, "lam" if f == "lambda" else f).offset)
        assert len(names) == len(fields)
    want.append(lib.PREDICATE_DTYPE.itemsize)
    assert got == want


def _pred(*clauses):
    p = synth.empty_predicates(1)
    p[0]["n_clauses"] = len(clauses)
    for i, c in enumerate(clauses):
        synth.set_clause(p[0], i, *c)
    return p


def _eval_canonical(lo, wm1, empty, cols):
    """Apply the canonical intervals the way the filter kernel does:
    row passes iff (uint32)(a_c - lo_c) <= wm1_c for every column."""
    n = len(cols[0])
    if empty:
        return np.zeros(n, bool)
    ok = np.ones(n, bool)
    for c, a in enumerate(cols):
        off = (a.astype(np.int64) - int(lo[c])) & 0xFFFFFFFF
        ok &= off <= int(wm1[c])
    return ok


@pytest.mark.parametrize("seed", range(6))
def test_canonical_intervals_agree_with_oracle_filter(lib, orc, seed):
    rng = np.random.default_rng(seed)
    n = 3000
    a32 = rng.integers(-2**31, 2**31, n, dtype=np.int64).astype(np.int32)
    a32[:10] = [-2**31, 2**31 - 1, 0, -1, 1, 5, 6, 7, -2**31 + 1, 2**31 - 2]
    a16 = rng.integers(-2**15, 2**15, n).astype(np.int16)
    a16[:4] = [-32768, 32767, 0, -1]
    small = rng.integers(-20, 20, n).astype(np.int32)
    cols = [a32, a16, small]
    types = [lib.IFVS_ATTR_I32, lib.IFVS_ATTR_I16, lib.IFVS_ATTR_I32]
    edge = [-2**63, -2**31 - 1, -2**31, -32769, -32768, -5, -1, 0, 1, 6, 32767, 32768,
            2**31 - 1, 2**31, 2**63 - 1]
    for trial in range(60):
        nc = int(rng.integers(0, 5))
        clauses = []
        for _ in range(nc):
            col = int(rng.integers(0, 3))
            op = int(rng.integers(0, 6))
            lo = int(rng.choice(edge)) if rng.random() < 0.4 else int(rng.integers(-40, 40))
            hi = int(rng.choice(edge)) if rng.random() < 0.4 else int(rng.integers(-40, 40))
            clauses.append((col, op, lo, hi))
        p = _pred(*clauses)
        lo, wm1, empty = lib.ifvs_canonical_predicate(p, types)
        mine = _eval_canonical(lo, wm1, empty, cols)
        bm, npass = orc.filter_bitmap(cols, p)
        ref = np.unpackbits(bm.view(np.uint8), bitorder="little")[:n].astype(bool)
        np.testing.assert_array_equal(mine, ref, err_msg=str(clauses))
        assert npass == int(mine.sum())


def test_canonical_rejects_malformed(lib):
    types = [lib.IFVS_ATTR_I32]
    with pytest.raises(lib.IfvsError):
        lib.ifvs_canonical_predicate(_pred((1, synth.OP_EQ, 0, 0)), types)
    with pytest.raises(lib.IfvsError):
        lib.ifvs_canonical_predicate(_pred((0, 17, 0, 0)), types)
    p = _pred((0, synth.OP_EQ, 0, 0))
    p[0]["n_clauses"] = 5
    with pytest.raises(lib.IfvsError):
        lib.ifvs_canonical_predicate(p, types)
    p = _pred((0, synth.OP_EQ, 0, 0))
    p[0]["reserved"] = 1
    with pytest.raises(lib.IfvsError):
        lib.ifvs_canonical_predicate(p, types)


def test_load_index_argument_checks(lib):
    codes = np.zeros((10, 16), np.uint8)
    a = np.zeros(10, np.int32)
    bad = [
        dict(codes=np.zeros((10, 200), np.uint8), attrs=[a]),      # M > 128
        dict(codes=codes, attrs=[np.zeros(10, np.float32)]),       # attribute type
    ]
    for kw in bad:
        with pytest.raises((lib.IfvsError, TypeError)):
            lib.ifvs_load_index(**kw)
    with pytest.raises(lib.IfvsError) as e:
        lib.ifvs_load_index(codes, [a], D=100)                     # D % M != 0
    assert e.value.code == lib.IFVS_ERR_ARG


@pytest.mark.skipif(os.path.exists("/dev/nvidia0"), reason="only meaningful without a GPU")
def test_no_device_is_reported_not_faked(lib):
    with pytest.raises(lib.IfvsError) as e:
        lib.ifvs_load_index(np.zeros((10, 16), np.uint8), [np.zeros(10, np.int32)])
    assert e.value.code == lib.IFVS_ERR_CUDA
