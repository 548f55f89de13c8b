/*
 * iFVS oracle — TEST INFRASTRUCTURE ONLY (see oracle.h for the paper map and
 * the readings taken).  Plain C99, fp64, no blocking, no fusion: every
 * function follows one definition of the paper and is meant to be checked
 * against it by eye.  Compiled with -ffp-contract=off so that x86 and Arm
 * give the same bits.
 */
#include "oracle.h"

#include <math.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------ */
/* Filter: §2 stage 1 ("the relational predicate f is evaluated over each
 * vector node's relational attributes"), predicate form of Listing 1:
 * a conjunction of comparisons on attribute columns.                  */

static int64_t attr_value(const void* const* cols, const int32_t* types, int32_t col,
                          int64_t row) {
    if (types[col] == ORC_I16) return (int64_t)((const int16_t*)cols[col])[row];
    return (int64_t)((const int32_t*)cols[col])[row];
}

int orc_row_passes(const void* const* cols, const int32_t* types, int32_t n_attrs,
                   int64_t row, const orc_predicate* p) {
    if (p->n_clauses < 0 || p->n_clauses > 4) return -1;
    int pass = 1;
    for (int32_t i = 0; i < p->n_clauses; ++i) {
        const orc_clause* c = &p->c[i];
        if (c->col < 0 || c->col >= n_attrs) return -1;
        if (types[c->col] != ORC_I32 && types[c->col] != ORC_I16) return -1;
        int64_t a = attr_value(cols, types, c->col, row);
        int ok;
        switch (c->op) {
            case ORC_EQ: ok = (a == c->lo); break;
            case ORC_RANGE: ok = (c->lo <= a && a < c->hi); break;
            case ORC_GE: ok = (a >= c->lo); break;
            case ORC_LT: ok = (a < c->lo); break;
            case ORC_GT: ok = (a > c->lo); break;
            case ORC_LE: ok = (a <= c->lo); break;
            default: return -1;
        }
        pass = pass && ok;
    }
    return pass;
}

int orc_filter(const void* const* cols, const int32_t* types, int32_t n_attrs,
               int64_t N, const orc_predicate* p, uint32_t* bitmap, int64_t* npass) {
    int64_t words = (N + 31) / 32;
    for (int64_t w = 0; w < words; ++w) bitmap[w] = 0;
    int64_t count = 0;
    for (int64_t i = 0; i < N; ++i) {
        int r = orc_row_passes(cols, types, n_attrs, i, p);
        if (r < 0) return -1;
        if (r) {
            bitmap[i / 32] |= (uint32_t)1u << (i % 32);
            ++count;
        }
    }
    if (npass) *npass = count;
    return 0;
}

/* ------------------------------------------------------------------ */
/* Fingerprint: §2 says <q,f> is hashed by h independent hash functions into
 * a bank of B rows but names no function.  Reading: FNV-1a-64 (Fowler, Noll,
 * Vo; offset basis 14695981039346656037, prime 1099511628211) over the key
 * bytes, then hash i = SplitMix64 finalizer (Steele, Lea, Flood 2014) of
 * (base XOR seed_i), reduced modulo B.                                */

uint64_t orc_fnv1a64(const uint8_t* bytes, int64_t n) {
    uint64_t hsh = 14695981039346656037ull;
    for (int64_t i = 0; i < n; ++i) {
        hsh ^= (uint64_t)bytes[i];
        hsh *= 1099511628211ull;
    }
    return hsh;
}

uint64_t orc_splitmix64_finalize(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

static void put_le(uint8_t* out, uint64_t v, int nbytes) {
    for (int b = 0; b < nbytes; ++b) out[b] = (uint8_t)(v >> (8 * b));
}

int64_t orc_fingerprint_key(const float* q, int32_t D, const orc_predicate* p, uint8_t* out) {
    int64_t n = 0;
    for (int32_t d = 0; d < D; ++d) {
        uint32_t bits;
        memcpy(&bits, &q[d], 4);
        put_le(out + n, bits, 4);
        n += 4;
    }
    int32_t nc = p->n_clauses;
    put_le(out + n, (uint32_t)nc, 4);
    n += 4;
    for (int32_t i = 0; i < nc && i < 4; ++i) {
        put_le(out + n, (uint32_t)p->c[i].col, 4);
        put_le(out + n + 4, (uint32_t)p->c[i].op, 4);
        put_le(out + n + 8, (uint64_t)p->c[i].lo, 8);
        put_le(out + n + 16, (uint64_t)p->c[i].hi, 8);
        n += 24;
    }
    return n;
}

void orc_fingerprint(const float* q, int32_t D, const orc_predicate* p,
                     const uint64_t* seeds, int32_t h, int64_t B, uint32_t* idx) {
    uint8_t* key = (uint8_t*)malloc((size_t)(4 * D + 4 + 24 * 4));
    int64_t n = orc_fingerprint_key(q, D, p, key);
    uint64_t base = orc_fnv1a64(key, n);
    free(key);
    for (int32_t i = 0; i < h; ++i)
        idx[i] = (uint32_t)(orc_splitmix64_finalize(base ^ seeds[i]) % (uint64_t)B);
}

/* ------------------------------------------------------------------ */
/* Conditioning: §2.  alpha = sum of the h fetched bank rows (viewed as
 * M x r);  w_f = softplus(w_z);  Delta = alpha . W;  C_iFVS = C_PQ + Delta. */

void orc_alpha(const float* bank, int64_t B, int32_t Mr, const uint32_t* idx, int32_t h,
               double* alpha) {
    (void)B;
    for (int32_t t = 0; t < Mr; ++t) alpha[t] = 0.0;
    for (int32_t i = 0; i < h; ++i)
        for (int32_t t = 0; t < Mr; ++t) alpha[t] += (double)bank[(int64_t)idx[i] * Mr + t];
}

double orc_softplus(double x) {
    /* log(1 + e^x), written so that neither branch overflows. */
    if (x > 0) return x + log1p(exp(-x));
    return log1p(exp(x));
}

void orc_filter_weights(const float* wz, int32_t D, double* wf) {
    for (int32_t d = 0; d < D; ++d) wf[d] = wz ? orc_softplus((double)wz[d]) : 1.0;
}

void orc_condition(const float* C_pq, const double* alpha, const float* W,
                   int32_t M, int32_t K, int32_t ds, int32_t r, double* C) {
    for (int32_t m = 0; m < M; ++m)
        for (int32_t k = 0; k < K; ++k)
            for (int32_t t = 0; t < ds; ++t) {
                double delta = 0.0;
                if (alpha && W)
                    for (int32_t j = 0; j < r; ++j)
                        delta += alpha[m * r + j] *
                                 (double)W[(((int64_t)m * r + j) * K + k) * ds + t];
                C[((int64_t)m * K + k) * ds + t] = (double)C_pq[((int64_t)m * K + k) * ds + t] + delta;
            }
}

/* Rank: §2 stage 2.  The printed score is
 *   score(v) = sum_m sum_d [ 2 w_{m,d} q_{m,d} C[m,code_v[m]]_d - w_{m,d} C[m,code_v[m]]_d^2 ]
 * = sum_{m,d} w q^2 - sum_{m,d} w (q - C)^2.
 * The first term is fixed per query, so ranking by score (descending) is
 * ranking by dist = sum_m LUT[m][code_v[m]] (ascending) with the weighted
 * ADC table below. */
void orc_lut(const float* q, const double* C, const double* wf,
             int32_t M, int32_t K, int32_t ds, double* lut) {
    for (int32_t m = 0; m < M; ++m)
        for (int32_t k = 0; k < K; ++k) {
            double s = 0.0;
            for (int32_t t = 0; t < ds; ++t) {
                double diff = (double)q[m * ds + t] - C[((int64_t)m * K + k) * ds + t];
                s += wf[m * ds + t] * diff * diff;
            }
            lut[(int64_t)m * K + k] = s;
        }
}

double orc_adc(const double* lut, const uint8_t* code_row, int32_t M, int32_t K) {
    double s = 0.0;
    for (int32_t m = 0; m < M; ++m) s += lut[(int64_t)m * K + code_row[m]];
    return s;
}

double orc_score(const float* q, const double* C, const double* wf, const uint8_t* code_row,
                 int32_t M, int32_t K, int32_t ds) {
    double s = 0.0;
    for (int32_t m = 0; m < M; ++m)
        for (int32_t t = 0; t < ds; ++t) {
            double c = C[((int64_t)m * K + code_row[m]) * ds + t];
            double w = wf[m * ds + t];
            s += 2.0 * w * (double)q[m * ds + t] * c - w * c * c;
        }
    return s;
}

/* ------------------------------------------------------------------ */
/* Select: §2 stage 3.  A full sort of the candidates by (dist, id), then
 * the first k. */

typedef struct { double d; int64_t id; } pair_t;

static int pair_cmp(const void* a, const void* b) {
    const pair_t* x = (const pair_t*)a;
    const pair_t* y = (const pair_t*)b;
    if (x->d < y->d) return -1;
    if (x->d > y->d) return 1;
    if (x->id < y->id) return -1;
    if (x->id > y->id) return 1;
    return 0;
}

void orc_topk(const double* dist, const int64_t* ids, int64_t n, int32_t k,
              int64_t* out_ids, double* out_dist) {
    pair_t* v = (pair_t*)malloc(sizeof(pair_t) * (size_t)(n > 0 ? n : 1));
    for (int64_t i = 0; i < n; ++i) {
        v[i].d = dist[i];
        v[i].id = ids[i];
    }
    qsort(v, (size_t)n, sizeof(pair_t), pair_cmp);
    for (int32_t j = 0; j < k; ++j) {
        if (j < n) {
            out_ids[j] = v[j].id;
            out_dist[j] = v[j].d;
        } else {
            out_ids[j] = -1;
            out_dist[j] = INFINITY;
        }
    }
    free(v);
}

/* ------------------------------------------------------------------ */
/* The whole query path of §2, one query after another. */

int orc_search(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
               const void* const* cols, const int32_t* types, int32_t n_attrs,
               const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
               const float* W, const uint64_t* seeds,
               const float* queries, const orc_predicate* preds, const float* wz, int64_t nq,
               int32_t k, int64_t* out_ids, double* out_dist, int64_t* npass,
               uint32_t* bank_idx, double* alpha_out, double* wf_out, double* lut_out) {
    int32_t D = M * ds;
    int64_t words = (N + 31) / 32;
    uint32_t* bitmap = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)(words > 0 ? words : 1));
    uint32_t* idx = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)(h > 0 ? h : 1));
    double* alpha = (double*)malloc(sizeof(double) * (size_t)(M * (r > 0 ? r : 1)));
    double* wf = (double*)malloc(sizeof(double) * (size_t)D);
    double* C = (double*)malloc(sizeof(double) * (size_t)M * K * ds);
    double* lut = (double*)malloc(sizeof(double) * (size_t)M * K);
    double* dist = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    int64_t* ids = (int64_t*)malloc(sizeof(int64_t) * (size_t)(N > 0 ? N : 1));
    int rc = 0;
    for (int64_t qi = 0; qi < nq; ++qi) {
        const float* q = queries + qi * D;
        const orc_predicate* p = &preds[qi];
        int64_t np = 0;
        if (orc_filter(cols, types, n_attrs, N, p, bitmap, &np) != 0) {
            rc = -1;
            break;
        }
        if (npass) npass[qi] = np;
        int conditioned = (bank != NULL && W != NULL && h > 0 && r > 0);
        if (conditioned) {
            orc_fingerprint(q, D, p, seeds, h, B, idx);
            orc_alpha(bank, B, M * r, idx, h, alpha);
            if (bank_idx)
                for (int32_t i = 0; i < h; ++i) bank_idx[qi * h + i] = idx[i];
            if (alpha_out)
                for (int32_t t = 0; t < M * r; ++t) alpha_out[qi * M * r + t] = alpha[t];
        }
        orc_filter_weights(wz ? wz + qi * D : NULL, D, wf);
        if (wf_out)
            for (int32_t d = 0; d < D; ++d) wf_out[qi * D + d] = wf[d];
        orc_condition(C_pq, conditioned ? alpha : NULL, conditioned ? W : NULL, M, K, ds, r, C);
        orc_lut(q, C, wf, M, K, ds, lut);
        if (lut_out)
            for (int64_t t = 0; t < (int64_t)M * K; ++t) lut_out[qi * M * K + t] = lut[t];
        int64_t n = 0;
        for (int64_t i = 0; i < N; ++i)
            if (bitmap[i / 32] >> (i % 32) & 1u) {
                dist[n] = orc_adc(lut, codes + i * M, M, K);
                ids[n] = i;
                ++n;
            }
        orc_topk(dist, ids, n, k, out_ids + qi * k, out_dist + qi * k);
    }
    free(bitmap);
    free(idx);
    free(alpha);
    free(wf);
    free(C);
    free(lut);
    free(dist);
    free(ids);
    return rc;
}

void orc_adc_all(const double* lut, const uint8_t* codes, int64_t N, int32_t M, int32_t K,
                 double* out) {
    for (int64_t i = 0; i < N; ++i) out[i] = orc_adc(lut, codes + i * M, M, K);
}

/* ------------------------------------------------------------------ */
/* Exact ground truth (§3.1) and exact rerank (the Pre_IndexFlatL2 baseline
 * of §3.2 restricted to candidates). */

void orc_exact_topk(const float* X, int64_t N, int32_t D, const float* q,
                    const uint32_t* bitmap, int32_t k, int64_t* out_ids, double* out_dist) {
    double* dist = (double*)malloc(sizeof(double) * (size_t)(N > 0 ? N : 1));
    int64_t* ids = (int64_t*)malloc(sizeof(int64_t) * (size_t)(N > 0 ? N : 1));
    int64_t n = 0;
    for (int64_t i = 0; i < N; ++i) {
        if (bitmap && !(bitmap[i / 32] >> (i % 32) & 1u)) continue;
        double s = 0.0;
        for (int32_t d = 0; d < D; ++d) {
            double diff = (double)q[d] - (double)X[i * D + d];
            s += diff * diff;
        }
        dist[n] = s;
        ids[n] = i;
        ++n;
    }
    orc_topk(dist, ids, n, k, out_ids, out_dist);
    free(dist);
    free(ids);
}

void orc_rerank(const float* X, int64_t N, int32_t D, const float* q, const int64_t* cand,
                int32_t R, int32_t k, int64_t* out_ids, double* out_dist) {
    double* dist = (double*)malloc(sizeof(double) * (size_t)(R > 0 ? R : 1));
    int64_t* ids = (int64_t*)malloc(sizeof(int64_t) * (size_t)(R > 0 ? R : 1));
    int64_t n = 0;
    for (int32_t j = 0; j < R; ++j) {
        int64_t i = cand[j];
        if (i < 0 || i >= N) continue;
        double s = 0.0;
        for (int32_t d = 0; d < D; ++d) {
            double diff = (double)q[d] - (double)X[i * D + d];
            s += diff * diff;
        }
        dist[n] = s;
        ids[n] = i;
        ++n;
    }
    orc_topk(dist, ids, n, k, out_ids, out_dist);
    free(dist);
    free(ids);
}

double orc_recall(const int64_t* ids, const int64_t* gt, int32_t k) {
    int32_t valid = 0, hit = 0;
    for (int32_t j = 0; j < k; ++j) {
        if (gt[j] < 0) continue;
        ++valid;
        for (int32_t u = 0; u < k; ++u)
            if (ids[u] == gt[j]) {
                ++hit;
                break;
            }
    }
    return valid ? (double)hit / (double)valid : 1.0;
}

/* ------------------------------------------------------------------ */
/* PQ construction.  Subspace m holds dimensions [m ds, (m+1) ds). */

static uint64_t sm64_next(uint64_t* state) {
    *state += 0x9e3779b97f4a7c15ull;
    return orc_splitmix64_finalize(*state);
}

static double sq_dist_sub(const float* x, const double* c, int32_t ds) {
    double s = 0.0;
    for (int32_t t = 0; t < ds; ++t) {
        double diff = (double)x[t] - c[t];
        s += diff * diff;
    }
    return s;
}

int orc_kmeans_pq(const float* X, int64_t n, int32_t D, int32_t M, int32_t K, int32_t iters,
                  uint64_t seed, double* C_out, double* objective_per_iter) {
    if (M <= 0 || D % M != 0 || n < K || K <= 0) return -1;
    int32_t ds = D / M;
    int64_t* perm = (int64_t*)malloc(sizeof(int64_t) * (size_t)n);
    int32_t* assign = (int32_t*)malloc(sizeof(int32_t) * (size_t)n);
    double* dmin = (double*)malloc(sizeof(double) * (size_t)n);
    double* sum = (double*)malloc(sizeof(double) * (size_t)K * ds);
    int64_t* cnt = (int64_t*)malloc(sizeof(int64_t) * (size_t)K);
    for (int32_t m = 0; m < M; ++m) {
        double* C = C_out + (int64_t)m * K * ds;
        /* K distinct rows: the first K of a seeded Fisher-Yates shuffle. */
        uint64_t st = seed ^ ((uint64_t)m * 0x9e3779b97f4a7c15ull);
        for (int64_t i = 0; i < n; ++i) perm[i] = i;
        for (int32_t j = 0; j < K; ++j) {
            int64_t pick = j + (int64_t)(sm64_next(&st) % (uint64_t)(n - j));
            int64_t tmp = perm[j];
            perm[j] = perm[pick];
            perm[pick] = tmp;
            for (int32_t t = 0; t < ds; ++t)
                C[(int64_t)j * ds + t] = (double)X[perm[j] * D + m * ds + t];
        }
        for (int32_t it = 0; it < iters; ++it) {
            /* assignment: nearest centroid, ties to the smallest index */
            double obj = 0.0;
            for (int64_t i = 0; i < n; ++i) {
                const float* x = X + i * D + m * ds;
                int32_t best = 0;
                double bd = sq_dist_sub(x, C, ds);
                for (int32_t c = 1; c < K; ++c) {
                    double d = sq_dist_sub(x, C + (int64_t)c * ds, ds);
                    if (d < bd) {
                        bd = d;
                        best = c;
                    }
                }
                assign[i] = best;
                dmin[i] = bd;
                obj += bd;
            }
            if (objective_per_iter) objective_per_iter[(int64_t)m * iters + it] = obj;
            /* update: mean of the members; an empty cluster takes the point
             * farthest from its centroid (ties to the smallest row). */
            for (int64_t t = 0; t < (int64_t)K * ds; ++t) sum[t] = 0.0;
            for (int32_t c = 0; c < K; ++c) cnt[c] = 0;
            for (int64_t i = 0; i < n; ++i) {
                cnt[assign[i]]++;
                for (int32_t t = 0; t < ds; ++t)
                    sum[(int64_t)assign[i] * ds + t] += (double)X[i * D + m * ds + t];
            }
            for (int32_t c = 0; c < K; ++c)
                if (cnt[c] > 0)
                    for (int32_t t = 0; t < ds; ++t)
                        C[(int64_t)c * ds + t] = sum[(int64_t)c * ds + t] / (double)cnt[c];
            for (int32_t c = 0; c < K; ++c)
                if (cnt[c] == 0) {
                    int64_t far = 0;
                    for (int64_t i = 1; i < n; ++i)
                        if (dmin[i] > dmin[far]) far = i;
                    for (int32_t t = 0; t < ds; ++t)
                        C[(int64_t)c * ds + t] = (double)X[far * D + m * ds + t];
                    dmin[far] = 0.0;
                }
        }
    }
    free(perm);
    free(assign);
    free(dmin);
    free(sum);
    free(cnt);
    return 0;
}

void orc_pq_encode(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                   const double* C, uint8_t* codes) {
    int32_t ds = D / M;
    for (int64_t i = 0; i < n; ++i)
        for (int32_t m = 0; m < M; ++m) {
            const float* x = X + i * D + m * ds;
            const double* Cm = C + (int64_t)m * K * ds;
            int32_t best = 0;
            double bd = sq_dist_sub(x, Cm, ds);
            for (int32_t c = 1; c < K; ++c) {
                double d = sq_dist_sub(x, Cm + (int64_t)c * ds, ds);
                if (d < bd) {
                    bd = d;
                    best = c;
                }
            }
            codes[i * M + m] = (uint8_t)best;
        }
}

void orc_reconstruct(const double* C, const uint8_t* code_row, int32_t M, int32_t K,
                     int32_t ds, double* x) {
    for (int32_t m = 0; m < M; ++m)
        for (int32_t t = 0; t < ds; ++t) x[m * ds + t] = C[((int64_t)m * K + code_row[m]) * ds + t];
}

double orc_sdc(const double* C, const uint8_t* cq, const uint8_t* cv, int32_t M, int32_t K,
               int32_t ds) {
    double s = 0.0;
    for (int32_t m = 0; m < M; ++m)
        for (int32_t t = 0; t < ds; ++t) {
            double diff = C[((int64_t)m * K + cq[m]) * ds + t] - C[((int64_t)m * K + cv[m]) * ds + t];
            s += diff * diff;
        }
    return s;
}

/* ------------------------------------------------------------------ */
/* Encoding and Lloyd iterations decided in float32 (see oracle.h).  With
 * -ffp-contract=off each expression below is one float32 rounding. */

static float sq_dist_sub_f32(const float* x, const float* c, int32_t ds) {
    float s = 0.0f;
    for (int32_t t = 0; t < ds; ++t) {
        float diff = x[t] - c[t];
        float sq = diff * diff;
        s = s + sq;
    }
    return s;
}

void orc_pq_encode_f32(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                       const float* C, uint8_t* codes, float* dmin) {
    int32_t ds = D / M;
    for (int64_t i = 0; i < n; ++i)
        for (int32_t m = 0; m < M; ++m) {
            const float* x = X + i * D + m * ds;
            const float* Cm = C + (int64_t)m * K * ds;
            int32_t best = 0;
            float bd = sq_dist_sub_f32(x, Cm, ds);
            for (int32_t c = 1; c < K; ++c) {
                float d = sq_dist_sub_f32(x, Cm + (int64_t)c * ds, ds);
                if (d < bd) {
                    bd = d;
                    best = c;
                }
            }
            codes[i * M + m] = (uint8_t)best;
            if (dmin) dmin[i * M + m] = bd;
        }
}

void orc_lloyd_step(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                    const float* C_in, float* C_out, uint8_t* codes, double* objective) {
    int32_t ds = D / M;
    float* dmin = (float*)malloc(sizeof(float) * (size_t)(n > 0 ? n : 1) * M);
    double* sum = (double*)malloc(sizeof(double) * (size_t)K * ds);
    int64_t* cnt = (int64_t*)malloc(sizeof(int64_t) * (size_t)K);
    orc_pq_encode_f32(X, n, D, M, K, C_in, codes, dmin);
    for (int32_t m = 0; m < M; ++m) {
        double obj = 0.0;
        for (int64_t t = 0; t < (int64_t)K * ds; ++t) sum[t] = 0.0;
        for (int32_t c = 0; c < K; ++c) cnt[c] = 0;
        for (int64_t i = 0; i < n; ++i) {
            int32_t c = codes[i * M + m];
            cnt[c]++;
            obj += (double)dmin[i * M + m];
            for (int32_t t = 0; t < ds; ++t) sum[(int64_t)c * ds + t] += (double)X[i * D + m * ds + t];
        }
        if (objective) objective[m] = obj;
        float* Co = C_out + (int64_t)m * K * ds;
        const float* Ci = C_in + (int64_t)m * K * ds;
        for (int32_t c = 0; c < K; ++c)
            for (int32_t t = 0; t < ds; ++t)
                Co[(int64_t)c * ds + t] = cnt[c] > 0 ? (float)(sum[(int64_t)c * ds + t] / (double)cnt[c])
                                                     : Ci[(int64_t)c * ds + t];
        for (int32_t c = 0; c < K; ++c)
            if (cnt[c] == 0 && n > 0) {
                int64_t far = 0;
                for (int64_t i = 1; i < n; ++i)
                    if (dmin[i * M + m] > dmin[far * M + m]) far = i;
                for (int32_t t = 0; t < ds; ++t) Co[(int64_t)c * ds + t] = X[far * D + m * ds + t];
                dmin[far * M + m] = 0.0f;
            }
    }
    free(dmin);
    free(sum);
    free(cnt);
}

/* ------------------------------------------------------------------ */
/* Learning C_iFVS and w_f: §2 "Learning".  The paper fixes the initial
 * state (alpha = 0, i.e. a zero bank, and w_f = 1), the positives (the
 * query's ground-truth rows), the hard negatives (the highest-scoring rows of
 * the pool that are not ground truth, under the current parameters), an
 * anchor term that keeps C_iFVS close to C_PQ, and which parameters move
 * (bank, W, w_f; C_PQ and the codes stay fixed).  Readings for what it
 * leaves open:
 *   score = -dist (the printed score minus sum w q^2, a per-query constant
 *   that no softmax sees);
 *   per positive g of a query, softmax cross-entropy of g against the
 *   query's negatives N at temperature tau,
 *     l_g = dist_g / tau + log( exp(-dist_g / tau) + sum_{n in N} exp(-dist_n / tau) ),
 *   averaged over the query's positives, plus lambda * ||Delta||^2 summed
 *   over all M K ds entries (= ||C_iFVS - C_PQ||^2);
 *   L = the mean of that over the queries;
 *   w_f = softplus(w_z) with one learned w_z [D] for all queries (the
 *   predicate Transformer that would give w_z per predicate is not given);
 *   optimiser: plain SGD, theta <- theta - lr * dL/dtheta, with a step size
 *   of its own for w_z (a jointly learned w_z can shrink every weight toward
 *   0: at a fixed temperature that lowers the loss whenever positives trail
 *   hard negatives, whatever it does to the ranking). */

static double sigmoid(double x) {
    if (x >= 0) return 1.0 / (1.0 + exp(-x));
    double e = exp(x);
    return e / (1.0 + e);
}

double orc_train_loss(const uint8_t* codes, int32_t M, int32_t K, int32_t ds,
                      const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                      const float* W, const uint64_t* seeds, const float* wz,
                      const float* queries, const orc_predicate* preds, int64_t nq,
                      const int64_t* cand, int32_t P, int32_t V, double tau, double lambda,
                      double* g_bank, double* g_W, double* g_wz) {
    const int32_t D = M * ds, Mr = M * r;
    const int64_t nC = (int64_t)M * K * ds, nW = (int64_t)M * r * K * ds;
    uint32_t* idx = (uint32_t*)malloc(sizeof(uint32_t) * (size_t)h);
    double* alpha = (double*)malloc(sizeof(double) * (size_t)Mr);
    double* wf = (double*)malloc(sizeof(double) * (size_t)D);
    double* C = (double*)malloc(sizeof(double) * (size_t)nC);
    double* delta = (double*)malloc(sizeof(double) * (size_t)nC);
    double* lut = (double*)malloc(sizeof(double) * (size_t)M * K);
    double* dist = (double*)malloc(sizeof(double) * (size_t)(V > 0 ? V : 1));
    double* gam = (double*)malloc(sizeof(double) * (size_t)(V > 0 ? V : 1));
    double* gC = (double*)malloc(sizeof(double) * (size_t)nC);
    double* gw = (double*)malloc(sizeof(double) * (size_t)D);
    double* galpha = (double*)malloc(sizeof(double) * (size_t)Mr);
    const int grads = (g_bank != NULL && g_W != NULL && g_wz != NULL);
    if (grads) {
        for (int64_t e = 0; e < B * Mr; ++e) g_bank[e] = 0.0;
        for (int64_t e = 0; e < nW; ++e) g_W[e] = 0.0;
        for (int32_t d = 0; d < D; ++d) g_wz[d] = 0.0;
    }
    orc_filter_weights(wz, D, wf);
    double L = 0.0;
    for (int64_t qi = 0; qi < nq; ++qi) {
        const float* q = queries + qi * D;
        const int64_t* cq = cand + qi * V;
        orc_fingerprint(q, D, &preds[qi], seeds, h, B, idx);
        orc_alpha(bank, B, Mr, idx, h, alpha);
        /* Delta[m][k][t] = sum_j alpha[m][j] W[m][j][k][t]; C = C_PQ + Delta */
        for (int32_t m = 0; m < M; ++m)
            for (int32_t k = 0; k < K; ++k)
                for (int32_t t = 0; t < ds; ++t) {
                    double s = 0.0;
                    for (int32_t j = 0; j < r; ++j)
                        s += alpha[m * r + j] * (double)W[(((int64_t)m * r + j) * K + k) * ds + t];
                    delta[((int64_t)m * K + k) * ds + t] = s;
                }
        orc_condition(C_pq, alpha, W, M, K, ds, r, C);
        orc_lut(q, C, wf, M, K, ds, lut);
        for (int32_t v = 0; v < V; ++v) {
            dist[v] = cq[v] >= 0 ? orc_adc(lut, codes + cq[v] * M, M, K) : 0.0;
            gam[v] = 0.0;
        }
        /* positive term: softmax cross-entropy of each positive against N */
        int32_t npos = 0;
        double lpos = 0.0;
        for (int32_t g = 0; g < P; ++g) {
            if (cq[g] < 0) continue;
            ++npos;
            double dmin = dist[g];
            for (int32_t n = P; n < V; ++n)
                if (cq[n] >= 0 && dist[n] < dmin) dmin = dist[n];
            double Z = exp(-(dist[g] - dmin) / tau);
            for (int32_t n = P; n < V; ++n)
                if (cq[n] >= 0) Z += exp(-(dist[n] - dmin) / tau);
            lpos += dist[g] / tau - dmin / tau + log(Z);
            /* d l_g / d dist_g = (1 - p_g) / tau;  d l_g / d dist_n = -p_n / tau */
            gam[g] += (1.0 - exp(-(dist[g] - dmin) / tau) / Z) / tau;
            for (int32_t n = P; n < V; ++n)
                if (cq[n] >= 0) gam[n] -= exp(-(dist[n] - dmin) / tau) / Z / tau;
        }
        if (npos > 0) {
            lpos /= npos;
            for (int32_t v = 0; v < V; ++v) gam[v] /= npos;
        }
        double anchor = 0.0;
        for (int64_t e = 0; e < nC; ++e) anchor += delta[e] * delta[e];
        L += (lpos + lambda * anchor) / (double)nq;
        if (!grads) continue;
        /* dL_q/dC at the candidates' codewords and dL_q/dw_f */
        for (int64_t e = 0; e < nC; ++e) gC[e] = 0.0;
        for (int32_t d = 0; d < D; ++d) gw[d] = 0.0;
        for (int32_t v = 0; v < V; ++v) {
            if (cq[v] < 0) continue;
            const uint8_t* code = codes + cq[v] * M;
            for (int32_t m = 0; m < M; ++m)
                for (int32_t t = 0; t < ds; ++t) {
                    const int64_t e = ((int64_t)m * K + code[m]) * ds + t;
                    const double diff = (double)q[m * ds + t] - C[e];
                    gC[e] += gam[v] * (-2.0 * wf[m * ds + t] * diff);
                    gw[m * ds + t] += gam[v] * diff * diff;
                }
        }
        /* dL_q/dDelta = dL_q/dC + 2 lambda Delta; chain rule through Delta = alpha . W */
        for (int32_t e = 0; e < Mr; ++e) galpha[e] = 0.0;
        for (int32_t m = 0; m < M; ++m)
            for (int32_t k = 0; k < K; ++k)
                for (int32_t t = 0; t < ds; ++t) {
                    const int64_t e = ((int64_t)m * K + k) * ds + t;
                    const double gD = gC[e] + 2.0 * lambda * delta[e];
                    for (int32_t j = 0; j < r; ++j) {
                        const int64_t w = (((int64_t)m * r + j) * K + k) * ds + t;
                        galpha[m * r + j] += gD * (double)W[w];
                        g_W[w] += alpha[m * r + j] * gD / (double)nq;
                    }
                }
        /* alpha = sum of the fetched bank rows: each fetch receives dL/dalpha */
        for (int32_t i = 0; i < h; ++i)
            for (int32_t e = 0; e < Mr; ++e) g_bank[(int64_t)idx[i] * Mr + e] += galpha[e] / (double)nq;
        /* w_f = softplus(w_z): dw_f/dw_z = sigmoid(w_z) */
        for (int32_t d = 0; d < D; ++d) g_wz[d] += gw[d] * sigmoid((double)wz[d]) / (double)nq;
    }
    free(idx);
    free(alpha);
    free(wf);
    free(C);
    free(delta);
    free(lut);
    free(dist);
    free(gam);
    free(gC);
    free(gw);
    free(galpha);
    return L;
}

int orc_mine_negatives(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
                       const void* const* cols, const int32_t* types, int32_t n_attrs,
                       const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                       const float* W, const uint64_t* seeds, const float* wz,
                       const float* queries, const orc_predicate* preds, int64_t nq,
                       const int64_t* pos, int32_t P, int32_t n_neg, int64_t* neg) {
    const int32_t D = M * ds, kk = P + n_neg;
    float* wzq = (float*)calloc((size_t)(nq > 0 ? nq : 1) * D, sizeof(float));
    int64_t* ids = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nq > 0 ? nq : 1) * (kk > 0 ? kk : 1));
    double* dd = (double*)malloc(sizeof(double) * (size_t)(nq > 0 ? nq : 1) * (kk > 0 ? kk : 1));
    for (int64_t qi = 0; qi < nq; ++qi)
        for (int32_t d = 0; d < D; ++d) wzq[qi * D + d] = wz[d];
    int rc = orc_search(codes, N, M, K, ds, cols, types, n_attrs, C_pq, bank, B, h, r, W, seeds,
                        queries, preds, wzq, nq, kk, ids, dd, NULL, NULL, NULL, NULL, NULL);
    /* the best n_neg of the pool that are not positives: at most P of the
     * top P + n_neg can be positives, so the rest of that list suffices */
    for (int64_t qi = 0; qi < nq && rc == 0; ++qi) {
        int32_t got = 0;
        for (int32_t j = 0; j < kk && got < n_neg; ++j) {
            const int64_t id = ids[qi * kk + j];
            if (id < 0) break;
            int is_pos = 0;
            for (int32_t g = 0; g < P; ++g)
                if (pos[qi * P + g] == id) is_pos = 1;
            if (!is_pos) neg[qi * n_neg + got++] = id;
        }
        for (; got < n_neg; ++got) neg[qi * n_neg + got] = -1;
    }
    free(wzq);
    free(ids);
    free(dd);
    return rc;
}

int orc_train_step(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
                   const void* const* cols, const int32_t* types, int32_t n_attrs,
                   const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                   const float* W, const uint64_t* seeds, const float* wz,
                   const float* queries, const orc_predicate* preds, int64_t nq,
                   const int64_t* pos, int32_t P, int32_t n_neg, double tau, double lambda,
                   double lr, double lr_wz, float* bank_out, float* W_out, float* wz_out,
                   int64_t* neg, double* loss) {
    const int32_t D = M * ds, V = P + n_neg;
    const int64_t nB = B * M * r, nW = (int64_t)M * r * K * ds;
    int64_t* cand = (int64_t*)malloc(sizeof(int64_t) * (size_t)(nq > 0 ? nq : 1) * (V > 0 ? V : 1));
    double* gb = (double*)malloc(sizeof(double) * (size_t)nB);
    double* gW = (double*)malloc(sizeof(double) * (size_t)nW);
    double* gz = (double*)malloc(sizeof(double) * (size_t)D);
    int rc = orc_mine_negatives(codes, N, M, K, ds, cols, types, n_attrs, C_pq, bank, B, h, r, W,
                                seeds, wz, queries, preds, nq, pos, P, n_neg, neg);
    if (rc == 0) {
        for (int64_t qi = 0; qi < nq; ++qi) {
            for (int32_t g = 0; g < P; ++g) cand[qi * V + g] = pos[qi * P + g];
            for (int32_t n = 0; n < n_neg; ++n) cand[qi * V + P + n] = neg[qi * n_neg + n];
        }
        *loss = orc_train_loss(codes, M, K, ds, C_pq, bank, B, h, r, W, seeds, wz, queries, preds,
                               nq, cand, P, V, tau, lambda, gb, gW, gz);
        for (int64_t e = 0; e < nB; ++e) bank_out[e] = (float)((double)bank[e] - lr * gb[e]);
        for (int64_t e = 0; e < nW; ++e) W_out[e] = (float)((double)W[e] - lr * gW[e]);
        for (int32_t d = 0; d < D; ++d) wz_out[d] = (float)((double)wz[d] - lr_wz * gz[d]);
    }
    free(cand);
    free(gb);
    free(gW);
    free(gz);
    return rc;
}
