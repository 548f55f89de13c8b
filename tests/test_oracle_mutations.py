"""The pins must catch plausible mistakes in the oracle.

Each case plants one mistake in a copy of oracle/oracle.c (a dropped term, a
wrong sign, index or bound, a transposed operand, a changed constant, a
reversed tie rule), builds it, and runs tests/test_oracle_pins.py against
it (and tests/test_oracle_train_pins.py): at least one pin must fail.  Nothing here touches the GPU path.
"""
import os
import shutil
import subprocess
import sys

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "oracle.c")

MUTATIONS = {
    "range upper bound inclusive": ("case ORC_RANGE: ok = (c->lo <= a && a < c->hi);",
                                    "case ORC_RANGE: ok = (c->lo <= a && a <= c->hi);"),
    "bitmap bit order": ("bitmap[i / 32] |= (uint32_t)1u << (i % 32);",
                         "bitmap[i / 32] |= (uint32_t)1u << (31 - i % 32);"),
    "GT as GE": ("case ORC_GT: ok = (a > c->lo);", "case ORC_GT: ok = (a >= c->lo);"),
    "FNV prime": ("hsh *= 1099511628211ull;", "hsh *= 1099511628213ull;"),
    "splitmix shift": ("z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;",
                       "z = (z ^ (z >> 26)) * 0x94d049bb133111ebull;"),
    "key drops hi": ("put_le(out + n + 16, (uint64_t)p->c[i].hi, 8);",
                     "put_le(out + n + 16, (uint64_t)p->c[i].lo, 8);"),
    "alpha keeps one row": ("for (int32_t i = 0; i < h; ++i)\n        for (int32_t t = 0; t < Mr; ++t) alpha[t] +=",
                            "for (int32_t i = 0; i < 1; ++i)\n        for (int32_t t = 0; t < Mr; ++t) alpha[t] +="),
    "softplus drops x": ("if (x > 0) return x + log1p(exp(-x));", "if (x > 0) return log1p(exp(-x));"),
    "W transposed (m, j)": ("delta += alpha[m * r + j] *\n                                 (double)W[(((int64_t)m * r + j) * K + k) * ds + t];",
                            "delta += alpha[j * M + m] *\n                                 (double)W[(((int64_t)m * r + j) * K + k) * ds + t];"),
    "C_PQ minus Delta": ("C[((int64_t)m * K + k) * ds + t] = (double)C_pq[((int64_t)m * K + k) * ds + t] + delta;",
                         "C[((int64_t)m * K + k) * ds + t] = (double)C_pq[((int64_t)m * K + k) * ds + t] - delta;"),
    "LUT drops w_f": ("s += wf[m * ds + t] * diff * diff;", "s += diff * diff;"),
    "LUT abs instead of square": ("s += wf[m * ds + t] * diff * diff;", "s += wf[m * ds + t] * fabs(diff);"),
    "ADC skips last subspace": ("for (int32_t m = 0; m < M; ++m) s += lut[(int64_t)m * K + code_row[m]];",
                                "for (int32_t m = 0; m + 1 < M; ++m) s += lut[(int64_t)m * K + code_row[m]];"),
    "score factor 2 dropped": ("s += 2.0 * w * (double)q[m * ds + t] * c - w * c * c;",
                               "s += w * (double)q[m * ds + t] * c - w * c * c;"),
    "ties to the larger id": ("if (x->id < y->id) return -1;\n    if (x->id > y->id) return 1;",
                              "if (x->id < y->id) return 1;\n    if (x->id > y->id) return -1;"),
    "padding distance 0": ("out_dist[j] = INFINITY;", "out_dist[j] = 0.0;"),
    "search reads the wrong bit": ("if (bitmap[i / 32] >> (i % 32) & 1u) {\n                dist[n] = orc_adc",
                                   "if (bitmap[i / 32] >> ((i + 1) % 32) & 1u) {\n                dist[n] = orc_adc"),
    "exact distance not squared": ("& 1u)) continue;\n        double s = 0.0;\n        for (int32_t d = 0; d < D; ++d) {\n            double diff = (double)q[d] - (double)X[i * D + d];\n            s += diff * diff;",
                                   "& 1u)) continue;\n        double s = 0.0;\n        for (int32_t d = 0; d < D; ++d) {\n            double diff = (double)q[d] - (double)X[i * D + d];\n            s += fabs(diff);"),
    "rerank distance not squared": ("if (i < 0 || i >= N) continue;\n        double s = 0.0;\n        for (int32_t d = 0; d < D; ++d) {\n            double diff = (double)q[d] - (double)X[i * D + d];\n            s += diff * diff;",
                                    "if (i < 0 || i >= N) continue;\n        double s = 0.0;\n        for (int32_t d = 0; d < D; ++d) {\n            double diff = (double)q[d] - (double)X[i * D + d];\n            s += fabs(diff);"),
    "k-means update reads subspace 0": ("sum[(int64_t)assign[i] * ds + t] += (double)X[i * D + m * ds + t];",
                                        "sum[(int64_t)assign[i] * ds + t] += (double)X[i * D + t];"),
    "k-means assigns the farthest codeword": ("double d = sq_dist_sub(x, C + (int64_t)c * ds, ds);\n                    if (d < bd) {",
                                              "double d = sq_dist_sub(x, C + (int64_t)c * ds, ds);\n                    if (d > bd) {"),
    "k-means mean off by one": ("C[(int64_t)c * ds + t] = sum[(int64_t)c * ds + t] / (double)cnt[c];",
                                "C[(int64_t)c * ds + t] = sum[(int64_t)c * ds + t] / (double)(cnt[c] + 1);"),
    "encode ties to the larger codeword": ("            if (d < bd) {\n                    bd = d;\n                    best = c;\n                }\n            }\n            codes[i * M + m] = (uint8_t)best;\n        }\n}",
                                           "            if (d <= bd) {\n                    bd = d;\n                    best = c;\n                }\n            }\n            codes[i * M + m] = (uint8_t)best;\n        }\n}"),
    "SDC wrong codeword": ("double diff = C[((int64_t)m * K + cq[m]) * ds + t] - C[((int64_t)m * K + cv[m]) * ds + t];",
                           "double diff = C[((int64_t)m * K + cq[m]) * ds + t] - C[((int64_t)m * K + cq[m]) * ds + t];"),
    "recall counts invalid ids": ("if (gt[j] < 0) continue;", "if (gt[j] < -1) continue;"),
    "f32 encode fused multiply-add": ("float sq = diff * diff;\n        s = s + sq;", "s = fmaf(diff, diff, s);"),
    "f32 encode ties to the larger": ("                if (d < bd) {\n                    bd = d;\n                    best = c;\n                }\n            }\n            codes[i * M + m] = (uint8_t)best;\n            if (dmin)",
                                      "                if (d <= bd) {\n                    bd = d;\n                    best = c;\n                }\n            }\n            codes[i * M + m] = (uint8_t)best;\n            if (dmin)"),
    "Lloyd keeps the old centroid": ("Co[(int64_t)c * ds + t] = cnt[c] > 0 ? (float)(sum[(int64_t)c * ds + t] / (double)cnt[c])",
                                     "Co[(int64_t)c * ds + t] = cnt[c] > 0 ? Ci[(int64_t)c * ds + t]"),
    "Lloyd reseeds with the nearest point": ("if (dmin[i * M + m] > dmin[far * M + m]) far = i;", "if (dmin[i * M + m] < dmin[far * M + m]) far = i;"),
    "train: negatives pushed the wrong way": ("if (cq[n] >= 0) gam[n] -= exp(-(dist[n] - dmin) / tau) / Z / tau;",
                                              "if (cq[n] >= 0) gam[n] += exp(-(dist[n] - dmin) / tau) / Z / tau;"),
    "train: anchor gradient halved": ("const double gD = gC[e] + 2.0 * lambda * delta[e];",
                                      "const double gD = gC[e] + lambda * delta[e];"),
    "train: w_z gradient without the sigmoid": ("g_wz[d] += gw[d] * sigmoid((double)wz[d]) / (double)nq;",
                                                "g_wz[d] += gw[d] / (double)nq;"),
    "train: positives summed, not averaged": ("lpos /= npos;",
                                              "lpos /= 1;"),
    "train: mining keeps positives": ("if (!is_pos) neg[qi * n_neg + got++] = id;",
                                      "neg[qi * n_neg + got++] = id;"),
    "train: W gradient without alpha": ("g_W[w] += alpha[m * r + j] * gD / (double)nq;",
                                        "g_W[w] += gD / (double)nq;"),
    "train: codeword gradient sign": ("gC[e] += gam[v] * (-2.0 * wf[m * ds + t] * diff);",
                                      "gC[e] += gam[v] * (2.0 * wf[m * ds + t] * diff);"),
    "train: bank gradient to the first fetch only": ("for (int32_t i = 0; i < h; ++i)\n            for (int32_t e = 0; e < Mr; ++e) g_bank",
                                                     "for (int32_t i = 0; i < 1; ++i)\n            for (int32_t e = 0; e < Mr; ++e) g_bank"),
    "train: w_z stepped with the bank's step size": ("wz_out[d] = (float)((double)wz[d] - lr_wz * gz[d]);",
                                                     "wz_out[d] = (float)((double)wz[d] - lr * gz[d]);"),
    "train: SGD ascends": ("bank_out[e] = (float)((double)bank[e] - lr * gb[e]);",
                           "bank_out[e] = (float)((double)bank[e] + lr * gb[e]);"),
}


@pytest.fixture(scope="module")
def source():
    with open(SRC) as f:
        return f.read()


@pytest.mark.parametrize("name", sorted(MUTATIONS))
def test_pins_catch_mutation(name, source, tmp_path):
    old, new = MUTATIONS[name]
    assert source.count(old) == 1, "mutation anchor not found exactly once: " + name
    mutated = source.replace(old, new)
    d = tmp_path / "o"
    d.mkdir()
    (d / "oracle.c").write_text(mutated)
    shutil.copy(os.path.join(ROOT, "oracle", "oracle.h"), d / "oracle.h")
    so = str(d / "liboracle_mut.so")
    subprocess.check_call(["gcc", "-std=c99", "-O2", "-fPIC", "-shared", "-ffp-contract=off",
                           "-o", so, str(d / "oracle.c"), "-lm"])
    env = dict(os.environ, IFVS_ORACLE_SO=so)
    p = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(ROOT, "tests", "test_oracle_pins.py"),
                        os.path.join(ROOT, "tests", "test_oracle_train_pins.py")],
                       cwd=ROOT, env=env, capture_output=True, text=True, timeout=600)
    assert p.returncode != 0, "no pin caught the mutation '%s'" % name
