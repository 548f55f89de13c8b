/*
 * iFVS oracle — TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct CPU restatement of the query-time method
 * of iFVS (instance-optimised filtered vector search, arXiv 2607.22922) in
 * fp64.  Only the test suite, the smoke check and the CPU-baseline leg of the
 * benchmark may load this library.  The GPU library shares no code, header,
 * table or helper with it; the two meet only through the seeded input
 * generator, which holds none of the method's arithmetic.
 *
 * Paper map (sections of the paper; its equations are unnumbered):
 *   Listing 1 (§1)        the filtered-vector-search query form
 *   §2, first paragraph   fingerprint of <q,f> into h rows of the memory
 *                         bank; alpha = sum of the fetched rows; w_z
 *   §2, display equations Delta = alpha . W,  w_f = softplus(w_z),
 *                         C_iFVS = C_PQ + Delta
 *   §2, stage 1 Filter    predicate over every row's attributes -> pool P
 *   §2, stage 2 Rank      score(v) = sum_m sum_d [2 w q C - w C^2]
 *   §2, stage 3 Select    top-k by score
 *   §2, "Learning"        alpha = 0, w_f = 1 reduces to plain PQ; the
 *                         training of bank, W and w_f (positives, mined
 *                         hard negatives, anchor to C_PQ)
 *   §3.1                  exact filtered ground truth over passing rows
 *   §3.2 B1               Pre_IndexFlatL2 / Pre_IndexFlatL2_PQ /
 *                         Pre_IndexPQ_ADC / Pre_IndexPQ_SDC
 *   §1 (PQ background)    M subspaces, K codewords each, uint8 codes
 *
 * Readings taken where the paper is silent or ambiguous:
 *   - hash: FNV-1a-64 over the canonical key bytes, then the SplitMix64
 *     output finalizer of (base XOR seed_i), modulo B;
 *   - Delta is the contraction of alpha[m][:] with W[m][:][k][t] over r;
 *   - w_f enters only the score, not C_iFVS;
 *   - the Rank score is turned into the weighted ADC distance
 *     dist = sum w (q - C)^2 = sum w q^2 - score, ranked ascending; ties in
 *     distance go to the smaller row id;
 *   - w_z absent means the paper's initial state w_f = 1 exactly.
 *
 * Parity status: every function here is pinned by tests/test_oracle_*.py.
 * orc_kmeans_pq's centroids after many iterations have no closed form from
 * a general seeded start; they are pinned where one exists (one codeword:
 * the mean; two well-separated groups: the group means; as many codewords
 * as distinct points: zero error), and its objective is pinned to be
 * non-increasing.
 */
#ifndef IFVS_ORACLE_H
#define IFVS_ORACLE_H
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Predicate layout used by the oracle (its own definition). */
typedef struct { int32_t col; int32_t op; int64_t lo; int64_t hi; } orc_clause;
typedef struct { int32_t n_clauses; int32_t reserved; orc_clause c[4]; } orc_predicate;

/* EQ: a == lo;  RANGE: lo <= a < hi;  GE: a >= lo;  LT: a < lo;
 * GT: a > lo;  LE: a <= lo.  All comparisons in int64. */
enum { ORC_EQ = 0, ORC_RANGE = 1, ORC_GE = 2, ORC_LT = 3, ORC_GT = 4, ORC_LE = 5 };
enum { ORC_I32 = 0, ORC_I16 = 1 };

/* Filter (§2 stage 1, Listing 1).  Returns 1 / 0 for pass / fail, -1 for an
 * invalid clause (column or operator out of range, n_clauses outside 0..4). */
int orc_row_passes(const void* const* cols, const int32_t* types, int32_t n_attrs,
                   int64_t row, const orc_predicate* p);
/* Bitmap of N rows, bit i of word i/32 (LSB first) = row i passes. */
int orc_filter(const void* const* cols, const int32_t* types, int32_t n_attrs,
               int64_t N, const orc_predicate* p, uint32_t* bitmap, int64_t* npass);

/* Fingerprint (§2): published hash definitions. */
uint64_t orc_fnv1a64(const uint8_t* bytes, int64_t n);
uint64_t orc_splitmix64_finalize(uint64_t z);
/* Canonical key bytes of <q, f>; returns the byte count written to `out`
 * (capacity must be >= 4*D + 4 + 24*4). */
int64_t orc_fingerprint_key(const float* q, int32_t D, const orc_predicate* p, uint8_t* out);
void orc_fingerprint(const float* q, int32_t D, const orc_predicate* p,
                     const uint64_t* seeds, int32_t h, int64_t B, uint32_t* idx);

/* alpha (§2): sum of the h fetched bank rows, each of length M*r. */
void orc_alpha(const float* bank, int64_t B, int32_t Mr, const uint32_t* idx, int32_t h,
               double* alpha);
/* softplus and w_f (§2).  wz == NULL means w_f = 1 exactly. */
double orc_softplus(double x);
void orc_filter_weights(const float* wz, int32_t D, double* wf);
/* C_iFVS = C_PQ + alpha . W (§2).  alpha or W NULL means Delta = 0.
 * C_pq [M][K][ds] fp32, alpha [M][r], W [M][r][K][ds] fp32 -> C [M][K][ds]. */
void orc_condition(const float* C_pq, const double* alpha, const float* W,
                   int32_t M, int32_t K, int32_t ds, int32_t r, double* C);
/* Weighted ADC table: lut[m][k] = sum_t wf[m ds + t] (q[m ds + t] - C[m][k][t])^2. */
void orc_lut(const float* q, const double* C, const double* wf,
             int32_t M, int32_t K, int32_t ds, double* lut);
double orc_adc(const double* lut, const uint8_t* code_row, int32_t M, int32_t K);
/* The Rank stage's score exactly as printed in §2 (for the identity pin). */
double orc_score(const float* q, const double* C, const double* wf, const uint8_t* code_row,
                 int32_t M, int32_t K, int32_t ds);

/* Select (§2 stage 3): the k smallest (dist, id) among `n` candidates.
 * Pads with id -1, dist +inf. */
void orc_topk(const double* dist, const int64_t* ids, int64_t n, int32_t k,
              int64_t* out_ids, double* out_dist);

/* Whole query path for nq queries.  Per query: filter, fingerprint, alpha,
 * w_f, C_iFVS, LUT, ADC over every passing row, top-k.
 * Optional outputs (NULL to skip): npass [nq], bank_idx [nq][h], alpha
 * [nq][M r], wf [nq][D], lut [nq][M][K]. */
int orc_search(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
               const void* const* cols, const int32_t* types, int32_t n_attrs,
               const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
               const float* W, const uint64_t* seeds,
               const float* queries, const orc_predicate* preds, const float* wz, int64_t nq,
               int32_t k, int64_t* out_ids, double* out_dist, int64_t* npass,
               uint32_t* bank_idx, double* alpha, double* wf, double* lut);

/* ADC of every row of `codes` against one LUT (fp64), no filter. */
void orc_adc_all(const double* lut, const uint8_t* codes, int64_t N, int32_t M, int32_t K,
                 double* out);

/* Exact filtered ground truth (§3.1; baseline Pre_IndexFlatL2 of §3.2):
 * unweighted L2 on the raw vectors over the passing rows, top-k. */
void orc_exact_topk(const float* X, int64_t N, int32_t D, const float* q,
                    const uint32_t* bitmap, int32_t k, int64_t* out_ids, double* out_dist);
/* Exact rerank of candidate ids (id -1 skipped): exact L2, top-k. */
void orc_rerank(const float* X, int64_t N, int32_t D, const float* q, const int64_t* cand,
                int32_t R, int32_t k, int64_t* out_ids, double* out_dist);
/* recall@k = |a ∩ gt| / (number of valid gt ids). */
double orc_recall(const int64_t* ids, const int64_t* gt, int32_t k);

/* PQ construction (§1 background; §3.2 uses 16 x 8).  Lloyd k-means per
 * subspace, `iters` iterations from K distinct seeded sample rows; an empty
 * cluster takes the point farthest from its centroid.  Then encoding by
 * argmin (ties -> smallest codeword). */
int orc_kmeans_pq(const float* X, int64_t n, int32_t D, int32_t M, int32_t K, int32_t iters,
                  uint64_t seed, double* C_out, double* objective_per_iter);
void orc_pq_encode(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                   const double* C, uint8_t* codes);
void orc_reconstruct(const double* C, const uint8_t* code_row, int32_t M, int32_t K,
                     int32_t ds, double* x);

/* The same encoding decided in float32, the precision of the GPU encoder:
 * per codeword, s = 0; for t ascending: s = s + (x_t - c_t) * (x_t - c_t),
 * each operation rounded to float32 (no fused multiply-add); argmin, ties to
 * the smallest codeword.  dmin (optional, [n][M]) receives the minimum. */
void orc_pq_encode_f32(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                       const float* C, uint8_t* codes, float* dmin);
/* One Lloyd iteration per subspace from float32 centroids C_in: assignment by
 * orc_pq_encode_f32; each non-empty cluster's new centroid is the fp64 mean
 * of its members rounded to float32; then every empty cluster, in increasing
 * order, takes the member point farthest from its centroid (largest float32
 * distance, ties to the smallest row), whose distance is then set to 0.
 * objective [M] (optional) = sum of the float32 minimum distances (fp64). */
void orc_lloyd_step(const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                    const float* C_in, float* C_out, uint8_t* codes, double* objective);

/* Symmetric distance (baseline Pre_IndexPQ_SDC, §3.2): the query is encoded
 * first; dist = sum_m ||C[m][cq[m]] - C[m][cv[m]]||^2. */
double orc_sdc(const double* C, const uint8_t* cq, const uint8_t* cv, int32_t M, int32_t K,
               int32_t ds);

/* Learning C_iFVS and w_f (§2 "Learning"); the readings are stated in
 * oracle.c.  orc_train_loss: the loss of nq queries whose candidate lists
 * cand [nq][V] hold the positives first (P of them) and then the negatives
 * (id -1 = absent), with one shared w_z [D] (non-NULL); if g_bank [B][M r],
 * g_W [M][r][K][ds] and g_wz [D] are all non-NULL they receive dL/d(bank,
 * W, w_z). */
double orc_train_loss(const uint8_t* codes, int32_t M, int32_t K, int32_t ds,
                      const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                      const float* W, const uint64_t* seeds, const float* wz,
                      const float* queries, const orc_predicate* preds, int64_t nq,
                      const int64_t* cand, int32_t P, int32_t V, double tau, double lambda,
                      double* g_bank, double* g_W, double* g_wz);
/* Hard negatives: per query the n_neg rows of the pool with the smallest
 * current distance that are not among its P positives (pos [nq][P], -1 =
 * absent), ties to the smaller row; -1 where the pool runs out. */
int orc_mine_negatives(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
                       const void* const* cols, const int32_t* types, int32_t n_attrs,
                       const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                       const float* W, const uint64_t* seeds, const float* wz,
                       const float* queries, const orc_predicate* preds, int64_t nq,
                       const int64_t* pos, int32_t P, int32_t n_neg, int64_t* neg);
/* One training step: mine negatives, loss and gradient, then plain SGD on
 * bank and W (step lr) and w_z (step lr_wz); new values rounded to float32
 * into the *_out arrays. */
int orc_train_step(const uint8_t* codes, int64_t N, int32_t M, int32_t K, int32_t ds,
                   const void* const* cols, const int32_t* types, int32_t n_attrs,
                   const float* C_pq, const float* bank, int64_t B, int32_t h, int32_t r,
                   const float* W, const uint64_t* seeds, const float* wz,
                   const float* queries, const orc_predicate* preds, int64_t nq,
                   const int64_t* pos, int32_t P, int32_t n_neg, double tau, double lambda,
                   double lr, double lr_wz, float* bank_out, float* W_out, float* wz_out,
                   int64_t* neg, double* loss);

#ifdef __cplusplus
}
#endif
#endif
