// Internal declarations of the iFVS GB300 library (not part of the ABI).
#pragma once

#include <cuda_runtime.h>
#include <stdint.h>

#include "ifvs.h"

namespace ifvs {

// A bitmap block covers 1024 rows: 32 lane-words of 32 bits.  In the
// device ("lane-major") layout, word (b * 32 + l) bit j is row
// b * 1024 + 32 * j + l, so lane l of a warp owns rows congruent to l mod 32
// and reads its 32 pass bits of a block in one coalesced 128-byte load.
constexpr int kBlockRows = 1024;
constexpr int kWarps = 8;          // warps per CTA in the scan and filter
constexpr int kThreads = kWarps * 32;

// One predicate reduced to a closed interval per attribute column:
// row passes iff for every column c, (uint32)(a_c - lo[c]) <= wm1[c].
struct CanonPred {
    int32_t lo[IFVS_MAX_ATTRS];
    uint32_t wm1[IFVS_MAX_ATTRS];
    uint32_t used;     // bit c: column c is constrained
    int32_t empty;     // 1: no row can pass
    int32_t invalid;   // 1: malformed predicate
    int32_t pad;
};

// Reduce a predicate to per-column intervals (clauses on one column
// intersect).  Returns 0, or -1 when the predicate is malformed.
__host__ __device__ inline int canonicalize(const ifvs_predicate& p, const int32_t* types,
                                            int n_attrs, CanonPred* out) {
    int64_t lo[IFVS_MAX_ATTRS], hi[IFVS_MAX_ATTRS];
    out->used = 0;
    out->empty = 0;
    out->invalid = 0;
    out->pad = 0;
    for (int c = 0; c < IFVS_MAX_ATTRS; ++c) {
        bool i16 = c < n_attrs && types[c] == IFVS_ATTR_I16;
        lo[c] = i16 ? -32768 : -2147483648LL;
        hi[c] = i16 ? 32767 : 2147483647LL;
    }
    int bad = (p.n_clauses < 0 || p.n_clauses > IFVS_MAX_CLAUSES || p.reserved != 0);
    int nc = bad ? 0 : p.n_clauses;
    for (int i = 0; i < nc; ++i) {
        const ifvs_clause& cl = p.c[i];
        if (cl.col < 0 || cl.col >= n_attrs) { bad = 1; break; }
        int64_t a, b;
        const int64_t kMin = (-9223372036854775807LL - 1), kMax = 9223372036854775807LL;
        bool none = false;
        switch (cl.op) {
            case IFVS_OP_EQ: a = cl.lo; b = cl.lo; break;
            case IFVS_OP_RANGE:
                a = cl.lo;
                if (cl.hi == kMin) { none = true; b = kMin; } else { b = cl.hi - 1; }
                break;
            case IFVS_OP_GE: a = cl.lo; b = kMax; break;
            case IFVS_OP_LT:
                a = kMin;
                if (cl.lo == kMin) { none = true; b = kMin; } else { b = cl.lo - 1; }
                break;
            case IFVS_OP_GT:
                b = kMax;
                if (cl.lo == kMax) { none = true; a = kMax; } else { a = cl.lo + 1; }
                break;
            case IFVS_OP_LE: a = kMin; b = cl.lo; break;
            default: bad = 1; a = 0; b = 0; break;
        }
        if (bad) break;
        if (none) { out->empty = 1; continue; }
        if (a > lo[cl.col]) lo[cl.col] = a;
        if (b < hi[cl.col]) hi[cl.col] = b;
        out->used |= 1u << cl.col;
    }
    for (int c = 0; c < IFVS_MAX_ATTRS; ++c) {
        if (lo[c] > hi[c]) {
            out->empty = 1;
            out->lo[c] = 0;
            out->wm1[c] = 0;
        } else {
            out->lo[c] = (int32_t)lo[c];
            out->wm1[c] = (uint32_t)(hi[c] - lo[c]);
        }
    }
    if (bad) { out->invalid = 1; out->empty = 1; return -1; }
    return 0;
}

struct AttrCols {
    const void* col[IFVS_MAX_ATTRS];
    int32_t type[IFVS_MAX_ATTRS];
    int32_t n;
};

// ---- kernel launchers (one per translation unit) -----------------------
// Every launcher returns the cudaError_t of its launch.

// predicates -> canonical intervals; *err |= 1 for any malformed predicate
cudaError_t launch_canonicalize(const ifvs_predicate* preds, int64_t nq, AttrCols cols,
                                CanonPred* out, int* err, cudaStream_t s);

// Per-query scan plan: a predicate whose pool is one position range [a, b)
// of a sorted copy (one constrained column; or, with composite copies, one
// column fixed to a value and the other bounded) with at most max_rows rows,
// or an empty / malformed one, takes the sorted-copy scan of copy `col`; the
// rest take the bitmap path.
struct ScanPlan {
    int64_t a, b;
    int32_t col;
    int32_t list;      // 1: row-list scan
};
// Sorted copies of the codes.  Copy c < IFVS_MAX_ATTRS: the rows sorted by
// (column c's value, row); vals[c] holds the values in that order.  For an
// index of exactly two columns, copies kComposite + j (j = 0, 1) are sorted
// by (column j, column 1 - j, row), and ckeys[j] holds the composite key
// ckey(v_j, v_{1-j}) of each position: a predicate fixing column j to one
// value and bounding the other column to an interval selects one contiguous
// position range of that copy.  Every copy: position p holds row rows[p]'s
// codes, rotated by (p mod 32) mod M, row_bytes apart, padded like the index.
constexpr int kComposite = IFVS_MAX_ATTRS;
constexpr int kSortedCopies = IFVS_MAX_ATTRS + 2;

// composite key: unsigned order of the pair is signed (primary, secondary) order
__host__ __device__ inline uint64_t ckey(int32_t primary, int32_t secondary) {
    return ((uint64_t)((uint32_t)primary ^ 0x80000000u) << 32) | (uint64_t)((uint32_t)secondary ^ 0x80000000u);
}

struct SortedCols {
    const uint32_t* rows[kSortedCopies];
    const uint8_t* codes[kSortedCopies];
    const int32_t* vals[IFVS_MAX_ATTRS];
    const uint64_t* ckeys[2];
    int32_t n;
    // copy c's arrays, selected without indexing the parameter at run time
    __host__ __device__ const uint8_t* codes_of(int c) const {
        const uint8_t* r = codes[0];
#pragma unroll
        for (int i = 1; i < kSortedCopies; ++i)
            if (c == i) r = codes[i];
        return r;
    }
    __host__ __device__ const uint32_t* rows_of(int c) const {
        const uint32_t* r = rows[0];
#pragma unroll
        for (int i = 1; i < kSortedCopies; ++i)
            if (c == i) r = rows[i];
        return r;
    }
    __host__ __device__ const int32_t* vals_of(int c) const {
        const int32_t* v = vals[0];
#pragma unroll
        for (int i = 1; i < IFVS_MAX_ATTRS; ++i)
            if (c == i) v = vals[i];
        return v;
    }
    __host__ __device__ const uint64_t* ckeys_of(int j) const { return j == 0 ? ckeys[0] : ckeys[1]; }
};
// plan [nq]; writes npass of the list-path queries
cudaError_t launch_plan(const CanonPred* canon, int64_t nq, SortedCols sc, int64_t N, int64_t max_rows,
                        ScanPlan* plan, unsigned long long* npass, cudaStream_t s);

// Filter: lane-major pass bitmaps [nq][n_blocks * 32] + popcounts (added to
// npass) for the bitmap-path queries of `plan` (all queries when plan is null)
cudaError_t launch_filter(AttrCols cols, int64_t N, int64_t n_blocks, const CanonPred* canon,
                          const ScanPlan* plan, int64_t nq, uint32_t* bm, unsigned long long* npass,
                          int num_sms, cudaStream_t s);

// 32x32 bit transposes between the lane-major layout and the row-ordered
// layout of the ABI ([nq][ceil(N/32)]).  to_rows = true: lane-major -> rows.
cudaError_t launch_bitmap_layout(const uint32_t* src, uint32_t* dst, int64_t nq,
                                 int64_t n_blocks, int64_t n_words_rows, bool to_rows,
                                 cudaStream_t s);

// fingerprint + alpha (when bank != nullptr) and w_f
cudaError_t launch_condition(const float* q, const ifvs_predicate* preds, int64_t nq, int D,
                             const uint64_t* seeds, int h, int64_t B, const float* bank, int Mr,
                             const float* wz, uint32_t* idx, float* alpha, float* wf,
                             cudaStream_t s);

// Delta, C_iFVS (optional output) and the weighted ADC tables
cudaError_t launch_lut(const float* cpq, const float* W, const float* alpha, const float* q,
                       const float* wf, int64_t nq, int M, int K, int ds, int r,
                       float* lut, float* cifvs, int num_sms, cudaStream_t s);

// weighted ADC tables [nq][M][K] -> the scan's shared-memory layout
// [nq][256][S] (S = tab_words)
cudaError_t launch_tables(const float* lut, int64_t nq, int M, int K, int S, float* tab,
                          cudaStream_t s);

struct ScanShape {
    int64_t n_blocks;      // bitmap blocks (rows padded to n_blocks * 1024)
    int M, K;
    int row_bytes;         // code row stride in bytes (M rounded up to 4)
    int tab_words;         // LUT table stride in words per codeword
    int64_t blocks_per_chunk;
    int n_chunks;
    int64_t n_rows;        // N (rows of the index)
};
size_t scan_smem_bytes(int tab_words, int kp);
// CTAs of the scan resident per SM for this table stride and list size
int scan_ctas_per_sm(int tab_words, int kp);
int scan_kp(int k);
// Rank: per (query, chunk) CTA, the k best keys (dist bits << 32 | row) of
// the chunk's passing rows -> partials [nq][n_chunks][k]; `tab` holds the
// tables written by launch_tables
cudaError_t launch_scan(const uint8_t* codes, const float* tab, const uint32_t* bm,
                        const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                        uint64_t* partials, cudaStream_t s);
// One CTA's work in the M = 16 sorted-copy scan: queries qa and qb share
// it (qb = -1: qa alone; qa = -1: no work).
struct PairItem {
    int32_t qa, qb;
};
// the list-path queries of `plan`: their pool is the position range [a, b)
// of a column's sorted copy (same grid and partial layout as launch_scan).
// For M = 16, `work` (scan_list_workspace_bytes(nq) bytes) receives the
// pairs of overlapping ranges that together span at least pair_min_rows
// positions, served by a two-query kernel; a one-query kernel serves the
// other queries (all of them when work is null or M != 16).  *launches =
// kernels launched.
// M = 16 one-query CTAs bring their code rows in by bulk copies into shared
// memory when `bulk` (else by per-lane vector loads); a bounded wait that
// runs out sets bit 4 of *err.  tx_extra: bytes added to what each copy's
// barrier expects (0; positive only to exercise the timeout path).
struct ListOpts {
    int64_t pair_min_rows;
    bool bulk;
    uint32_t tx_extra;
    int* err;
};
size_t scan_list_workspace_bytes(int64_t nq);
cudaError_t launch_scan_list(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                             const ScanShape& sh, uint64_t* partials, uint8_t* work, const ListOpts& lo,
                             cudaStream_t s, int* launches);
// the sorted copy of the codes: dst position p <- row rows[p] of the index
// layout `src`, re-rotated by (p mod 32) mod M; positions >= N are zero
cudaError_t launch_relayout_sorted(const uint8_t* src, const uint32_t* rows, int64_t N, int M,
                                   int row_bytes, int64_t n_rows_pad, uint8_t* dst, cudaStream_t s);
// Select: merge [nq][n_lists][k] partial keys -> ids / dists
cudaError_t launch_merge(const uint64_t* partials, int64_t nq, int n_lists, int k,
                         int64_t* ids, float* dists, cudaStream_t s);
// exact fp32 rerank of cand [nq][R] -> k best
// Select across row shards: [G][nq][k] (dist, global id) -> [nq][k]
int shard_merge_cap();
cudaError_t launch_merge_shards(const float* dists, const int64_t* ids, int64_t nq, int G, int k,
                                float* dists_out, int64_t* ids_out, cudaStream_t s);
cudaError_t launch_rerank(const float* X, int64_t N, int D, const float* q, const int64_t* cand,
                          int64_t nq, int R, int k, int64_t* ids, float* dists, cudaStream_t s);
// codes [N][M] -> rotated rows [n_rows_pad][row_bytes]; *bad = 1 if a code >= K
cudaError_t launch_relayout_codes(const uint8_t* src, int64_t N, int M, int K, int row_bytes,
                                  int64_t n_rows_pad, uint8_t* dst, int* bad, cudaStream_t s);

// ---- PQ construction (csrc/pq.cu) --------------------------------------
// codes [n][M] and optional dmin [n][M] (float32 argmin, fixed order)
cudaError_t launch_pq_assign(const float* X, int64_t n, int D, int M, int K, const float* C,
                             uint8_t* codes, float* dmin, cudaStream_t s);
// Lloyd update: fp64 means of the members (sums [M][K][ds], counts [M][K])
cudaError_t launch_pq_update(const float* X, int64_t n, int D, int M, int K, const uint8_t* codes,
                             double* sums, unsigned long long* counts, const float* C_in,
                             float* C_out, int num_sms, cudaStream_t s);
// empty codeword c of subspace m <- the farthest row (best: 8-byte scratch)
cudaError_t launch_pq_reseed(const float* X, int64_t n, int D, int M, int K, int m, int c,
                             unsigned long long* best, float* C_out, float* dmin, int num_sms,
                             cudaStream_t s);
cudaError_t launch_pq_objective(const float* dmin, int64_t n, int M, double* objective, int num_sms,
                                cudaStream_t s);

// ---- training of bank, W, w_f (csrc/train.cu) --------------------------
constexpr int kTrainMaxR = 32;     // r per subspace handled by the gradient kernels
constexpr int kTrainMaxV = 512;    // positives + negatives per query
struct TrainQueryArgs {
    const uint8_t* codes;          // index layout (rows rotated, row_bytes apart)
    int row_bytes, M, K, ds, D, r;
    const float* C_pq;             // [M][K][ds]
    const float* W;                // [M][r][K][ds]
    const float* G;                // [M][r][r] Gram matrices (written by the gradient launch)
    const float* q;                // [n][D]
    const float* wf;               // [n][D]
    const float* alpha;            // [n][M r]
    const int64_t* pos;            // positives, row q at pos + q * pos_stride, P of them
    int64_t pos_stride;
    int P;
    const int64_t* negsrc;         // negative source, row q at negsrc + q * neg_stride, S entries
    int64_t neg_stride;
    int S, n_neg;
    int exclude;                   // 1: mined list (skip positives, stop at -1); 0: take as given
    float tau, lambda;
    int64_t n;
    int64_t N;                     // rows of the index: ids outside -1..N-1 are refused
    int* err;                      // |= 2 when a candidate id is outside -1..N-1 (then treated as absent)
    int64_t* neg_out;              // [n][n_neg] or null
    float* gC;                     // [n][M][K][ds] scratch
    float* gw;                     // [n][D] scratch: dL/dw_f per query
    float* galpha;                 // [n][M r] dL/dalpha per query (not divided by n)
    double* loss;                  // [n]
};
size_t train_query_smem(int V, int Mr, int D, int r);
// G [M][r][r] = W[m] W[m]^T
cudaError_t launch_train_gram(const float* W, int M, int r, int KD, float* G, cudaStream_t s);
// per query: candidates, distances, softmax, loss, gC (zeroed by the caller), dL/dw_f, dL/dalpha
cudaError_t launch_train_query(const TrainQueryArgs& a, cudaStream_t s);
// gW [M][r][K ds] of the mean loss (written, not accumulated); scratch of
// train_gW_scratch bytes; *launches = kernels launched
size_t train_gW_scratch(int64_t n, int M, int r, int KD);
cudaError_t launch_train_gW(const float* alpha, const float* gC, const float* W, int64_t n, int M, int r,
                            int KD, float lambda, float inv_n, float* scratch, float* gW,
                            cudaStream_t s, int* launches);

// gbank rows fetched by the batch (other rows must be zeroed by the caller)
cudaError_t launch_train_bank(const uint32_t* idx, int64_t n, int h, int Mr, const float* galpha,
                              float inv_n, float* gbank, cudaStream_t s);
cudaError_t launch_train_wz(const float* gw, int64_t n, int D, const float* wz, float inv_n, float* gwz,
                            cudaStream_t s);
cudaError_t launch_broadcast_wz(const float* wz, int D, int64_t n, float* out, cudaStream_t s);
cudaError_t launch_sgd(float* theta, const float* g, int64_t n, float lr, cudaStream_t s);

// Read-only view of a loaded index, for entry points defined outside api.cu.
struct IndexView {
    int device;
    int num_sms;
    int max_smem;  // opt-in shared memory per block on `device`, bytes
    int64_t N, n_blocks;
    int M, K, row_bytes, tab_words;
    const uint8_t* codes;
};
int index_view(const ifvs_index* ix, IndexView* out);
// Sets the thread-local message of ifvs_last_error and returns `code`.
int report_error(int code, const char* fmt, ...);

}  // namespace ifvs
