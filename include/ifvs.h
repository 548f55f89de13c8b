/*
 * ifvs.h — C ABI of the GB300 query path of iFVS (instance-optimised
 * filtered vector search, arXiv 2607.22922).
 *
 * The library answers filtered k-nearest-neighbour queries over a fixed
 * PQ-encoded dataset (the query form of Listing 1, §1: a conjunctive
 * predicate on relational attribute columns, then ORDER BY distance LIMIT k)
 * with the three stages of §2:
 *   Filter  every row's attributes are tested against the predicate, giving
 *           the candidate pool P as a pass bitmap;
 *   Rank    the query- and predicate-conditioned codebook
 *           C_iFVS = C_PQ + Delta, Delta = alpha . W, alpha = the sum of the h
 *           memory-bank rows that <q, f> hashes to, and the filter weights
 *           w_f = softplus(w_z) give each candidate the score of §2, which the
 *           library evaluates as the equivalent weighted ADC distance
 *           dist(v) = sum_m LUT[m][code_v[m]],
 *           LUT[m][k] = sum_t w_f[m ds + t] (q[m ds + t] - C_iFVS[m][k][t])^2
 *           (score(v) = sum w q^2 - dist(v): descending score is ascending
 *           distance);
 *   Select  the k candidates with the smallest (dist, row id).
 *
 * Every step runs in the library's CUDA kernels for sm_103a; there is no CPU
 * fallback.  All calls are synchronous: they return once their outputs are
 * written.  No call keeps a pointer to caller memory after it returns.
 *
 * Streams: where a call takes a stream, NULL selects a stream of the
 * library's own (the index's, or one the call creates).  Those streams are
 * blocking streams, so the call's kernels run after work the caller queued
 * on the legacy default stream.  With device I/O, inputs that the caller
 * produces on any other stream are only safe to read if that stream is
 * passed (or synchronised before the call).
 *
 * Errors: every call returns an ifvs_status.  On error the outputs are
 * unspecified and ifvs_last_error() (thread-local) describes the cause.
 * Nothing aborts the process and nothing throws across the ABI.
 *
 * Thread safety: an index may be used by one thread at a time; different
 * indexes may be used concurrently.
 */
#ifndef IFVS_H
#define IFVS_H

#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define IFVS_MAX_CLAUSES 4
#define IFVS_MAX_ATTRS 4
#define IFVS_MAX_K 256      /* largest k (and rerank depth R) per query  */
#define IFVS_MAX_M 128      /* largest number of PQ subspaces            */
#define IFVS_N_STAGES 9

typedef struct ifvs_index ifvs_index;

typedef enum {
    IFVS_OK = 0,
    IFVS_ERR_ARG = -1,          /* invalid argument (message says which)      */
    IFVS_ERR_OOM = -2,          /* device allocation failed                   */
    IFVS_ERR_CUDA = -3,         /* a CUDA runtime call or kernel failed       */
    IFVS_ERR_STATE = -4,        /* e.g. search before ifvs_load_codebooks     */
    IFVS_ERR_UNSUPPORTED = -5,  /* shape outside the supported range          */
    IFVS_ERR_TIMEOUT = -6       /* a bounded wait inside a kernel ran out; the
                                   results are incomplete, the GPU stays usable */
} ifvs_status;

/* Every entry point that allocates device memory returns IFVS_ERR_OOM when
 * an allocation fails, frees what the call had allocated, and leaves the
 * index as it was (later calls may succeed).  For tests of that path the
 * failure can be injected on the host: while the environment variable
 * IFVS_FAIL_ALLOC holds a number n >= 1, the n-th device allocation since
 * the variable took its current string fails without calling cudaMalloc.
 *
 * Kernels never wait without a bound.  The sorted-copy scan waits for its
 * bulk-copied code tiles for at most about half a second per tile; when a
 * wait runs out the search returns IFVS_ERR_TIMEOUT and the device stays
 * usable.  For tests of that path, while the environment variable
 * IFVS_TEST_STALL_COPIES is "1" every such wait runs out. */

/* Clause operators (Listing 1 uses = and >; all are intervals on integers):
 *   EQ    a == lo        RANGE lo <= a < hi     GE  a >= lo
 *   LT    a <  lo        GT    a >  lo          LE  a <= lo
 * Comparisons are exact on the column's integer values (int64 semantics). */
enum { IFVS_OP_EQ = 0, IFVS_OP_RANGE = 1, IFVS_OP_GE = 2, IFVS_OP_LT = 3,
       IFVS_OP_GT = 4, IFVS_OP_LE = 5 };

/* Attribute column element types. */
enum { IFVS_ATTR_I32 = 0, IFVS_ATTR_I16 = 1 };

typedef struct {
    int32_t col;   /* attribute column, 0 <= col < n_attrs */
    int32_t op;    /* IFVS_OP_*                            */
    int64_t lo;
    int64_t hi;    /* used by IFVS_OP_RANGE only           */
} ifvs_clause;     /* 24 bytes */

/* A predicate is the conjunction (AND) of its first n_clauses clauses;
 * n_clauses = 0 passes every row.  104 bytes. */
typedef struct {
    int32_t n_clauses;
    int32_t reserved;   /* must be 0 */
    ifvs_clause c[IFVS_MAX_CLAUSES];
} ifvs_predicate;

/* Flags of ifvs_search_params.flags and of ifvs_load_index(flags). */
#define IFVS_F_DEVICE_IO    0x1u  /* array arguments are device pointers on
                                     the index's device                       */
#define IFVS_F_STAGE_TIMING 0x2u  /* time every kernel launch with CUDA events
                                     on the launching stream (ifvs_stage_times) */
#define IFVS_F_PLAIN_PQ     0x4u  /* ignore the memory bank: Delta = 0 (plain PQ
                                     ADC, baseline Pre_IndexPQ_ADC of §3.2)   */
#define IFVS_F_PLAIN_LOADS  0x8u  /* search, M = 16 sorted-copy scan: one-query
                                     CTAs read code rows with per-lane vector
                                     loads instead of bulk copies (TMA) into
                                     shared memory; same results              */

typedef struct {
    uint32_t flags;     /* IFVS_F_*                                            */
    int32_t rerank;     /* R > 0: re-rank the R best ADC candidates by exact fp32
                           L2 on the raw vectors (needs vectors at load), then
                           keep k (k <= R <= IFVS_MAX_K).  0: off.              */
    int32_t sub_batch;  /* queries per filter/scan pass; bounds the bitmap
                           workspace to sub_batch * ceil(N/1024) * 128 bytes.
                           0: automatic (at most 1024).                        */
    int32_t chunk_blocks; /* rows per scan CTA in units of 1024 (0: automatic);
                           a tuning knob: CTAs of different queries that walk
                           the same chunk together share its codes in L2     */
    int32_t list_max_ppm; /* a query whose predicate constrains one column,
                           or, on an index of two columns, fixes one column
                           to a single value and bounds the other, takes the
                           sorted-copy scan (its pool is a position range of
                           the codes sorted by that column, or of a composite
                           copy: no filter pass, no bitmap) when the pool
                           holds at most this many rows per million of N.
                           0: default (1000000: always); -1: never.  The two
                           paths sum a row's entries in different orders, so
                           distances agree to float32 rounding.              */
    int32_t pair_min_rows; /* M = 16 sorted-copy scan: two queries on the same
                           column whose ranges share 3/4 of the longer one
                           and together span at least this many rows share a
                           CTA and one shared-memory look-up per code byte
                           (tables quantised to 11 bits; every row that can
                           reach a top-k is rescored exactly, so results
                           equal those of one query per CTA bit for bit).
                           0: default (4194304); -1: never pair.             */
    void* stream;       /* cudaStream_t to run on; NULL: the index's stream   */
} ifvs_search_params;

/* Stages reported by ifvs_stage_times (index into its arrays). */
enum {
    IFVS_STAGE_PREDICATE = 0,  /* predicate validation + canonical intervals  */
    IFVS_STAGE_FILTER = 1,     /* Filter: attribute columns -> pass bitmaps   */
    IFVS_STAGE_CONDITION = 2,  /* fingerprint, alpha, w_f                     */
    IFVS_STAGE_LUT = 3,        /* Delta, C_iFVS and the weighted ADC tables    */
    IFVS_STAGE_SCAN = 4,       /* Rank: code scan + per-CTA top-k             */
    IFVS_STAGE_MERGE = 5,      /* Select: merge of the per-CTA top-k lists    */
    IFVS_STAGE_RERANK = 6,     /* exact fp32 rerank                           */
    IFVS_STAGE_LAYOUT = 7,     /* bitmap layout conversions                   */
    IFVS_STAGE_TRAIN = 8       /* training: loss, gradient and SGD kernels    */
};

/*
 * ifvs_load_index — copy a PQ-encoded dataset to the device.
 *   out         receives the new index (free with ifvs_free)
 *   device      CUDA device ordinal
 *   codes       [N][M] uint8, row-major: code of row i in subspace m (§1:
 *               subspace m covers dimensions [m ds, (m+1) ds)); every code
 *               must be < K
 *   N           rows, 1 <= N < 2^32 - 1024
 *   M, K        subspaces (1..IFVS_MAX_M) and codewords per subspace (1..256)
 *   attr_cols   n_attrs pointers to columns of N elements (int32 or int16 as
 *               attr_types says); n_attrs in 0..IFVS_MAX_ATTRS
 *   vectors     [N][D] float32 raw vectors for the exact rerank, or NULL
 *   D           vector dimension (a multiple of M)
 *   flags       IFVS_F_DEVICE_IO: codes, columns and vectors are device
 *               pointers on `device`
 * The library copies everything; the caller keeps ownership of its buffers.
 * Codes are stored re-laid out for the scan (rows padded to a multiple of
 * 1024; each row's codes rotated so that a warp's 32 lanes read 32 distinct
 * shared-memory banks).  For every attribute column the library also keeps
 * the row ids sorted by (value, row), the sorted values and a copy of the
 * code rows in that order (8 + row_bytes bytes per row and column; the order
 * is sorted on the host at load), in which a one-column predicate's pool is
 * a contiguous position range.  An index of exactly two columns also keeps
 * two composite copies, rows by (column j, column 1 - j, row) for j = 0, 1
 * (the 8-byte key, the row id and the code row: 12 + row_bytes bytes per
 * row each), in which a predicate fixing column j to one value and bounding
 * the other column is a contiguous position range.
 */
int ifvs_load_index(ifvs_index** out, int32_t device, const uint8_t* codes, int64_t N,
                    int32_t M, int32_t K, const void* const* attr_cols,
                    const int32_t* attr_types, int32_t n_attrs, const float* vectors,
                    int32_t D, uint32_t flags);

/*
 * ifvs_load_codebooks — the base codebook and the conditioning model (§2).
 *   C_pq        [M][K][ds] float32 base codebook C_PQ (ds = D / M)
 *   bank        [B][M r] float32 memory bank (row b viewed as alpha's M x r
 *               layout), or NULL: Delta = 0 for every query
 *   B, h, r     bank rows, hash functions per query, adjustment rank
 *   W           [M][r][K][ds] float32 adjustment directions (NULL iff bank is)
 *   hash_seeds  [h] uint64: hash i of <q, f> is
 *               splitmix64_finalizer(fnv1a64(key) XOR hash_seeds[i]) mod B,
 *               key = the float32 bits of q (little-endian), n_clauses
 *               (int32) and each clause's col, op (int32), lo, hi (int64)
 * Host pointers; copied.  May be called again to replace the model.
 */
int ifvs_load_codebooks(ifvs_index* ix, const float* C_pq, int32_t ds, const float* bank,
                        int64_t B, int32_t h, int32_t r, const float* W,
                        const uint64_t* hash_seeds);

/*
 * ifvs_search_batch — the whole query path (Filter, Rank, Select of §2) for
 * nq queries.
 *   queries   [nq][D] float32
 *   preds     [nq] predicates
 *   nq        >= 0 (0 returns at once)
 *   k         1..IFVS_MAX_K results per query
 *   wz        [nq][D] float32 predicate encodings w_z (w_f = softplus(w_z)),
 *             or NULL: w_f = 1 exactly (the paper's initial state)
 *   p         options, or NULL for defaults (host I/O, index stream)
 *   ids       [nq][k] int64 out: row ids by ascending (dist, id); -1 pads
 *             when fewer than k rows pass
 *   dists     [nq][k] float32 out: weighted ADC distances (or exact L2 after
 *             a rerank); +inf pads
 *   npass     [nq] int64 out: |P| per query, or NULL
 * Array arguments are host memory unless p->flags has IFVS_F_DEVICE_IO.
 */
int ifvs_search_batch(ifvs_index* ix, const float* queries, const ifvs_predicate* preds,
                      int64_t nq, int32_t k, const float* wz, const ifvs_search_params* p,
                      int64_t* ids, float* dists, int64_t* npass);

/*
 * ifvs_filter — stage 1 alone (§2 Filter).
 *   bitmaps  [nq][ceil(N/32)] uint32 out: bit (i % 32) of word i / 32 is set
 *            iff row i passes (bits beyond N are 0)
 *   npass    [nq] int64 out, or NULL
 */
int ifvs_filter(ifvs_index* ix, const ifvs_predicate* preds, int64_t nq,
                const ifvs_search_params* p, uint32_t* bitmaps, int64_t* npass);

/*
 * ifvs_condition — the conditioning and table build of §2 alone.  Every
 * output may be NULL.
 *   bank_idx  [nq][h] uint32 out: the h bank rows <q, f> hashes to
 *   alpha     [nq][M r] float32 out: sum of those rows
 *   wf        [nq][D] float32 out: softplus(w_z) (or 1)
 *   C_ifvs    [nq][M][K][ds] float32 out: C_PQ + alpha . W
 *   lut       [nq][M][K] float32 out: weighted ADC tables
 */
int ifvs_condition(ifvs_index* ix, const float* queries, const ifvs_predicate* preds,
                   int64_t nq, const float* wz, const ifvs_search_params* p,
                   uint32_t* bank_idx, float* alpha, float* wf, float* C_ifvs, float* lut);

/*
 * ifvs_scan_topk — Rank and Select from given tables and bitmaps.
 *   lut      [nq][M][K] float32 weighted ADC tables
 *   bitmaps  [nq][ceil(N/32)] uint32 pass bitmaps in the layout ifvs_filter
 *            writes
 *   ids, dists as for ifvs_search_batch
 */
int ifvs_scan_topk(ifvs_index* ix, const float* lut, const uint32_t* bitmaps, int64_t nq,
                   int32_t k, const ifvs_search_params* p, int64_t* ids, float* dists);

/*
 * ifvs_scan_topk_static — ifvs_scan_topk without any device allocation.
 * The paper has no counterpart: this entry point exists for callers that
 * must not allocate device memory while serving queries — code whose device
 * memory belongs to another allocator (a framework's caching pool), or
 * latency-critical loops that allocate nothing after start-up, because
 * cudaMalloc / cudaFree can synchronise the whole device.
 *   lut, bitmaps, ids, dists  device pointers, shapes as for ifvs_scan_topk
 *   stream                    cudaStream_t to enqueue on (NULL: legacy stream)
 * The call only enqueues work on `stream` and returns; results are ready
 * when the stream reaches them.  Its scratch is a file-scope device array of
 * IFVS_STATIC_SCRATCH_BYTES that every GPU running the library holds until
 * the process exits; queries are processed in sub-batches that fit it.
 * Sizes beyond it (one query's lane-major bitmap, N / 8 bytes rounded up to
 * 128-byte blocks, plus its 64 KB scan table (160 KB for M > 33) and k keys,
 * above the array) return
 * IFVS_ERR_UNSUPPORTED, and so does a k whose scan needs more shared memory
 * than the device offers (as in ifvs_scan_topk).  Every call looks up the
 * array's device address on the index's device (cudaGetSymbolAddress, a
 * host-side query), so a context torn down and created again
 * (cudaDeviceReset) is followed; the first call on a device also loads the
 * library's module there: make it before any stream capture.  All calls
 * share the array: calls whose work overlaps on
 * the GPU (different streams, or threads without ordering) race.  No
 * cudaMalloc, cudaFree or allocating library routine is called.
 */
#define IFVS_STATIC_SCRATCH_BYTES (32u << 20)
int ifvs_scan_topk_static(ifvs_index* ix, const float* lut, const uint32_t* bitmaps, int64_t nq,
                          int32_t k, void* stream, int64_t* ids, float* dists);

/*
 * ifvs_rerank — exact fp32 L2 (the Pre_IndexFlatL2 distance of §3.2) of
 * candidate rows, then the k best by (dist, id).
 *   cand  [nq][R] int64 candidate row ids; -1 entries are skipped
 *   needs raw vectors given to ifvs_load_index
 */
int ifvs_rerank(ifvs_index* ix, const float* queries, const int64_t* cand, int64_t nq,
                int32_t R, int32_t k, const ifvs_search_params* p, int64_t* ids,
                float* dists);

/*
 * ifvs_merge_topk — Select (§2, stage 3) across row shards.  The paper has
 * one device; when an index is split into G row shards (rows [r_g, r_g+1)
 * on shard g, searched separately, ids offset by r_g), the k best of each
 * shard are gathered and this call keeps the k smallest by (dist, id) of the
 * G k entries of each query — the same ids and distances as one search over
 * all rows.
 *   dists   [G][nq][k] float32 per-shard distances (the layout of an
 *           all-gather of each shard's [nq][k] result)
 *   ids     [G][nq][k] int64 global row ids; -1 marks padding (sorted last)
 *   dists_out, ids_out  [nq][k] out; padded with (+inf, -1) where the
 *           shards return fewer than k rows in all
 *   flags   IFVS_F_DEVICE_IO: all arrays are device pointers on `device`
 *   stream  cudaStream_t for the work, or NULL (a stream of the call's own)
 * Shards must hold disjoint rows.  With IFVS_F_DEVICE_IO and a non-NULL
 * stream the call allocates nothing and only enqueues one kernel.  Errors:
 * IFVS_ERR_ARG (NULL, nq < 0, G < 1, k outside 1..IFVS_MAX_K, unknown flag),
 * IFVS_ERR_UNSUPPORTED (G k above 4096), IFVS_ERR_OOM, IFVS_ERR_CUDA.
 */
int ifvs_merge_topk(int32_t device, const float* dists, const int64_t* ids, int64_t nq, int32_t G,
                    int32_t k, float* dists_out, int64_t* ids_out, uint32_t flags, void* stream);

/*
 * ifvs_pq_encode — PQ encoding of raw vectors (the offline step before the
 * query path: §1's product quantisation, 16 x 8 in §3.2), on `device`.
 *   X       [n][D] float32; subspace m covers dimensions [m ds, (m+1) ds)
 *   C_pq    [M][K][ds] float32 codebook
 *   codes   [n][M] uint8 out: argmin over codewords of the float32 squared
 *           distance s = s + (x_t - c_t)^2 accumulated for t ascending with
 *           every operation rounded on its own; ties to the smallest codeword
 *   dmin    [n][M] float32 out (that minimum), or NULL
 *   flags   IFVS_F_DEVICE_IO: all arrays are device pointers
 *   stream  cudaStream_t for the work, or NULL (a stream of the call's own)
 * With IFVS_F_DEVICE_IO and a non-NULL stream the call allocates nothing,
 * only enqueues one kernel and returns; otherwise it returns when the
 * results are written.  Errors: IFVS_ERR_ARG (NULL pointer, n < 0 or
 * above 2^32 - 1, D not a multiple of M, unknown flag), IFVS_ERR_UNSUPPORTED
 * (K outside 1..256, K x ds x 8 bytes above 200 KB), IFVS_ERR_OOM, IFVS_ERR_CUDA.
 */
int ifvs_pq_encode(int32_t device, const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                   const float* C_pq, uint8_t* codes, float* dmin, uint32_t flags, void* stream);

/*
 * ifvs_pq_train — `iters` Lloyd iterations per subspace from C_init
 * (k-means training of the PQ codebook).  Each iteration assigns every row
 * as ifvs_pq_encode does, then replaces each codeword used by at least one
 * row by the fp64 mean of its rows rounded to float32; each unused
 * codeword, in increasing order, takes the row farthest from its codeword
 * (largest distance, ties to the smallest row), whose distance then counts
 * as 0.
 *   C_init     [M][K][ds] float32 start (e.g. K distinct sample rows)
 *   C_out      [M][K][ds] float32 out
 *   objective  [iters][M] fp64 out (sum of the assignment's minimum
 *              distances at each iteration, before its update), or NULL
 *   stream     cudaStream_t for the work, or NULL (a stream of the call's own)
 * The call returns when C_out (and objective) are written; it reads the
 * per-codeword counts back to the host once per iteration.  Errors as
 * ifvs_pq_encode, plus IFVS_ERR_ARG for iters < 0.
 */
int ifvs_pq_train(int32_t device, const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
                  int32_t iters, const float* C_init, float* C_out, double* objective,
                  uint32_t flags, void* stream);

/*
 * Training of the memory bank, W and w_f (§2 "Learning": at the start the
 * bank is zero (alpha = 0) and w_f = 1; each query-predicate pair scores its
 * ground-truth rows and hard negatives mined from its pool, i.e. the
 * highest-scoring rows that are not ground truth under the current
 * parameters; an anchor term keeps C_iFVS near C_PQ; gradients reach the
 * bank, W and w_f while C_PQ and the codes stay fixed).  The paper leaves the
 * loss, the regulariser weight and the optimiser open; this library reads
 * them as: score = -dist; for each positive g of a query,
 *   l_g = dist_g / tau + log( exp(-dist_g / tau) + sum_{n in N} exp(-dist_n / tau) )
 * over the query's negatives N, averaged over its positives, plus
 * lambda ||Delta||^2 (all M K ds entries); the loss L is the mean over the
 * queries; one w_z [D] is learned for all queries (w_f = softplus(w_z); the
 * predicate Transformer is not given); plain SGD, with a step size of its
 * own for w_z (at a fixed temperature, shrinking every weight lowers this
 * loss whenever positives trail hard negatives, so a jointly learned w_f
 * can collapse toward 0).  Distances are float32
 * terms summed in fp64; gradients are float32; every sum runs in a fixed
 * order, so results are deterministic.  One call handles one mini-batch of
 * at most 1024 queries; the index must hold a bank, W and seeds with
 * r <= 32.
 */
typedef struct {
    float tau;          /* softmax temperature, > 0                          */
    float lambda;       /* anchor weight, >= 0                               */
    float lr;           /* SGD step size for the bank and W, >= 0            */
    float lr_wz;        /* SGD step size for w_z, >= 0 (0 keeps w_f fixed)   */
    int32_t n_pos;      /* positives per query (P)                           */
    int32_t n_neg;      /* negatives per query; 1 <= P + n_neg <= 512
                           (<= IFVS_MAX_K when mined)                         */
    uint32_t flags;     /* IFVS_F_DEVICE_IO | IFVS_F_STAGE_TIMING            */
    void* stream;       /* cudaStream_t, or NULL for the index's stream       */
} ifvs_train_params;

/*
 * ifvs_train_grad — the loss and its gradient for given candidates, without
 * mining and without an update.
 *   queries [nq][D] float32, preds [nq], wz [D] the shared w_z
 *   cand    [nq][P + n_neg] int64: the P positives, then the negatives
 *           (-1 = absent; a query without valid positives adds only its
 *           anchor term)
 *   g_bank  [B][M r], g_W [M][r][K][ds], g_wz [D] float32 out (each may be
 *           NULL); loss: the mean loss (host double) or NULL
 * Returns when all outputs are written.  Errors: IFVS_ERR_ARG (parameters,
 * nq > 1024, NULL arrays, malformed predicate), IFVS_ERR_STATE (no bank),
 * IFVS_ERR_UNSUPPORTED (r > 32, shared memory), IFVS_ERR_OOM, IFVS_ERR_CUDA.
 */
int ifvs_train_grad(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                    const float* wz, const int64_t* cand, const ifvs_train_params* tp,
                    float* g_bank, float* g_W, float* g_wz, double* loss);

/*
 * ifvs_train_step — one SGD step on a mini-batch: mines each query's hard
 * negatives with the query path (top P + n_neg under the current bank, W and
 * w_z, positives removed, the first n_neg kept, -1 where the pool runs out),
 * computes the loss and gradient as ifvs_train_grad, then updates the
 * index's bank and W in place (theta -= lr * dL/dtheta) and wz [D] (in/out,
 * wz -= lr_wz * dL/dwz).
 *   positives  [nq][P] int64 (-1 = absent)
 *   negatives  [nq][n_neg] int64 out (the mined negatives) or NULL
 * Errors as ifvs_train_grad.
 */
int ifvs_train_step(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                    float* wz, const int64_t* positives, const ifvs_train_params* tp,
                    int64_t* negatives, double* loss);

/* ifvs_get_conditioning — copies the index's current bank [B][M r] and W
 * [M][r][K][ds] (either may be NULL) to host memory, or to device memory
 * with IFVS_F_DEVICE_IO in flags. */
int ifvs_get_conditioning(ifvs_index* ix, float* bank, float* W, uint32_t flags);

/*
 * ifvs_stage_times — device time (ms, from CUDA events recorded on the
 * launching stream around each launch) and launch counts per stage,
 * accumulated over calls made with IFVS_F_STAGE_TIMING.  Either array may be
 * NULL; reset != 0 zeroes the counters after reading.
 */
int ifvs_stage_times(ifvs_index* ix, double* ms, int64_t* launches, int32_t reset);

/*
 * ifvs_canonical_predicate — host-side helper exposing how a predicate is
 * reduced to one closed interval [lo, lo + width_m1] per attribute column
 * (clauses on the same column intersect).  Column c passes every value when
 * lo[c] is the type's minimum and width_m1[c] the type's span minus one.
 * *empty = 1 when no row can pass.  Returns IFVS_ERR_ARG for an invalid
 * predicate.
 */
int ifvs_canonical_predicate(const ifvs_predicate* p, const int32_t* attr_types,
                             int32_t n_attrs, int32_t* lo, uint32_t* width_m1, int32_t* empty);

/* ifvs_index_info — out[0..7] = N, M, K, D, ds, n_attrs, has codebooks,
 * device bytes held. */
int ifvs_index_info(const ifvs_index* ix, int64_t* out);

void ifvs_free(ifvs_index* ix);
const char* ifvs_last_error(void);
const char* ifvs_version(void);

#ifdef __cplusplus
}
#endif
#endif /* IFVS_H */
