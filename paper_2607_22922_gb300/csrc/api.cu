// Host side of the C ABI declared in include/ifvs.h: argument checks,
// device memory of the index and its grow-only workspace, the launch
// sequence of the query path per sub-batch, and per-stage CUDA-event timing.
#include <stdarg.h>
#include <stdio.h>
#include <string.h>

#include <stdlib.h>

#include <algorithm>
#include <mutex>
#include <string>
#include <new>
#include <utility>
#include <cmath>
#include <vector>

#include "internal.cuh"

using namespace ifvs;

namespace {

thread_local char g_err[768] = "";

int set_err(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return code;
}

int cuda_fail(cudaError_t e, const char* what, int line) {
    cudaGetLastError();  // clear a sticky launch error where possible
    return set_err(e == cudaErrorMemoryAllocation ? IFVS_ERR_OOM : IFVS_ERR_CUDA,
                   "%s failed: %s (api.cu:%d)", what, cudaGetErrorString(e), line);
}

#define CUDA_TRY(x)                                                  \
    do {                                                             \
        cudaError_t e_ = (x);                                        \
        if (e_ != cudaSuccess) return cuda_fail(e_, #x, __LINE__);   \
    } while (0)

#define TRY(x)               \
    do {                     \
        int rc_ = (x);       \
        if (rc_ != 0) return rc_; \
    } while (0)

// Every device allocation of the library goes through device_malloc.
// Failure injection for tests of the error path (no GPU fault involved):
// while the environment variable IFVS_FAIL_ALLOC holds a number n >= 1,
// the n-th device allocation counted since the variable took its current
// value fails as if the device were out of memory (no cudaMalloc is called
// for it); the count restarts whenever the variable's string changes (so
// "1" and then "01" each fail the next allocation) or is unset.
cudaError_t device_malloc(void** p, size_t bytes) {
    static std::mutex mu;
    static std::string last;
    static long count = 0;
    {
        std::lock_guard<std::mutex> lock(mu);
        const char* v = getenv("IFVS_FAIL_ALLOC");
        const std::string cur = v ? v : "";
        if (cur != last) {
            last = cur;
            count = 0;
        }
        if (!cur.empty()) {
            const long n = strtol(cur.c_str(), nullptr, 10);
            if (n >= 1 && ++count == n) {
                *p = nullptr;
                return cudaErrorMemoryAllocation;
            }
        }
    }
    return cudaMalloc(p, bytes);
}

// Timeout injection for tests of the scan's bounded waits (no GPU fault
// involved): while the environment variable IFVS_TEST_STALL_COPIES is "1",
// the bulk-copy barriers of the sorted-copy scan expect 16 bytes more than
// their copies deliver, so every wait on them runs out after its bound and
// the search returns IFVS_ERR_TIMEOUT with the context intact.
bool stall_copies_for_tests() {
    const char* v = getenv("IFVS_TEST_STALL_COPIES");
    return v != nullptr && v[0] == '1' && v[1] == '\0';
}

struct DevBuf {
    void* p = nullptr;
    size_t cap = 0;
    template <class T> T* as() const { return reinterpret_cast<T*>(p); }
};

int ensure(DevBuf& b, size_t bytes) {
    if (bytes == 0) bytes = 16;
    if (bytes <= b.cap) return 0;
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
    cudaError_t e = device_malloc(&b.p, bytes);
    if (e != cudaSuccess) {
        cudaGetLastError();
        b.p = nullptr;
        return set_err(IFVS_ERR_OOM, "device allocation of %zu bytes failed: %s", bytes, cudaGetErrorString(e));
    }
    b.cap = bytes;
    return 0;
}

void release(DevBuf& b) {
    if (b.p) cudaFree(b.p);
    b.p = nullptr;
    b.cap = 0;
}

struct DeviceGuard {
    int prev = -1;
    bool ok = true;
    explicit DeviceGuard(int dev) {
        if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
        if (prev != dev) ok = cudaSetDevice(dev) == cudaSuccess;
    }
    ~DeviceGuard() {
        int cur = -1;
        if (prev >= 0 && cudaGetDevice(&cur) == cudaSuccess && cur != prev) cudaSetDevice(prev);
    }
};

int64_t round_up(int64_t a, int64_t b) { return (a + b - 1) / b * b; }

}  // namespace

struct ifvs_index {
    int device = 0;
    int num_sms = 0;
    int max_smem = 0;
    cudaStream_t stream = nullptr;
    int64_t N = 0, n_blocks = 0, n_rows_pad = 0;
    int M = 0, K = 0, D = 0, ds = 0, row_bytes = 0, tab_words = 0;
    int n_attrs = 0;
    int32_t types[IFVS_MAX_ATTRS] = {0, 0, 0, 0};
    void* d_attr[IFVS_MAX_ATTRS] = {nullptr, nullptr, nullptr, nullptr};
    // sorted copies (see SortedCols): row ids in copy order, the codes in
    // that order; the values of the one-column copies; the composite keys
    uint32_t* d_srt_rows[kSortedCopies] = {};
    uint8_t* d_srt_codes[kSortedCopies] = {};
    int32_t* d_srt_vals[IFVS_MAX_ATTRS] = {};
    uint64_t* d_ckeys[2] = {};
    uint8_t* d_codes = nullptr;
    float* d_vec = nullptr;
    bool has_cb = false;
    float* d_cpq = nullptr;
    float* d_bank = nullptr;
    float* d_W = nullptr;
    uint64_t* d_seeds = nullptr;
    int64_t B = 0;
    int h = 0, r = 0;
    size_t bytes = 0;
    // workspace
    DevBuf w_q, w_wz, w_preds, w_canon, w_err, w_bm, w_rows, w_npass, w_idx, w_alpha, w_wf,
        w_lut, w_cifvs, w_part, w_ids, w_dists, w_cand, w_cdist, w_tab, w_plan, w_items;
    // training workspace
    DevBuf t_cand, t_pos, t_mined, t_mdist, t_gC, t_gw, t_loss, t_G, t_gW, t_gWpart, t_galpha,
        t_gbank, t_gwz, t_wz, t_neg;
    // timing
    double stage_ms[IFVS_N_STAGES] = {0};
    int64_t stage_launches[IFVS_N_STAGES] = {0};
    std::vector<cudaEvent_t> ev_free;
    std::vector<std::pair<int, std::pair<cudaEvent_t, cudaEvent_t>>> pending;

    SortedCols sorted() const {
        SortedCols c;
        for (int i = 0; i < kSortedCopies; ++i) {
            c.rows[i] = d_srt_rows[i];
            c.codes[i] = d_srt_codes[i];
        }
        for (int i = 0; i < IFVS_MAX_ATTRS; ++i) c.vals[i] = d_srt_vals[i];
        c.ckeys[0] = d_ckeys[0];
        c.ckeys[1] = d_ckeys[1];
        c.n = n_attrs;
        return c;
    }
    AttrCols cols() const {
        AttrCols c;
        for (int i = 0; i < IFVS_MAX_ATTRS; ++i) {
            c.col[i] = d_attr[i];
            c.type[i] = types[i];
        }
        c.n = n_attrs;
        return c;
    }
    cudaEvent_t event() {
        if (!ev_free.empty()) {
            cudaEvent_t e = ev_free.back();
            ev_free.pop_back();
            return e;
        }
        cudaEvent_t e = nullptr;
        if (cudaEventCreate(&e) != cudaSuccess) return nullptr;
        return e;
    }
    void collect() {
        for (auto& pr : pending) {
            float ms = 0.f;
            if (cudaEventElapsedTime(&ms, pr.second.first, pr.second.second) == cudaSuccess)
                stage_ms[pr.first] += ms;
            ev_free.push_back(pr.second.first);
            ev_free.push_back(pr.second.second);
        }
        pending.clear();
        cudaGetLastError();
    }
};

namespace {

void free_index(ifvs_index* ix) {
    if (!ix) return;
    DeviceGuard g(ix->device);
    if (ix->stream) cudaStreamSynchronize(ix->stream);
    for (int i = 0; i < IFVS_MAX_ATTRS; ++i) {
        if (ix->d_attr[i]) cudaFree(ix->d_attr[i]);
        if (ix->d_srt_vals[i]) cudaFree(ix->d_srt_vals[i]);
    }
    for (int i = 0; i < kSortedCopies; ++i) {
        if (ix->d_srt_rows[i]) cudaFree(ix->d_srt_rows[i]);
        if (ix->d_srt_codes[i]) cudaFree(ix->d_srt_codes[i]);
    }
    for (int j = 0; j < 2; ++j)
        if (ix->d_ckeys[j]) cudaFree(ix->d_ckeys[j]);
    void* ptrs[] = {ix->d_codes, ix->d_vec, ix->d_cpq, ix->d_bank, ix->d_W, ix->d_seeds};
    for (void* p : ptrs)
        if (p) cudaFree(p);
    DevBuf* bufs[] = {&ix->w_q, &ix->w_wz, &ix->w_preds, &ix->w_canon, &ix->w_err, &ix->w_bm,
                      &ix->w_rows, &ix->w_npass, &ix->w_idx, &ix->w_alpha, &ix->w_wf,
                      &ix->w_lut, &ix->w_cifvs, &ix->w_part, &ix->w_ids, &ix->w_dists,
                      &ix->w_cand, &ix->w_cdist, &ix->w_tab, &ix->w_plan, &ix->w_items, &ix->t_cand, &ix->t_pos,
                      &ix->t_mined, &ix->t_mdist, &ix->t_gC, &ix->t_gw, &ix->t_loss, &ix->t_G,
                      &ix->t_gW, &ix->t_gWpart, &ix->t_galpha, &ix->t_gbank, &ix->t_gwz, &ix->t_wz, &ix->t_neg};
    for (DevBuf* b : bufs) release(*b);
    for (auto& pr : ix->pending) {
        ix->ev_free.push_back(pr.second.first);
        ix->ev_free.push_back(pr.second.second);
    }
    for (cudaEvent_t e : ix->ev_free)
        if (e) cudaEventDestroy(e);
    if (ix->stream) cudaStreamDestroy(ix->stream);
    delete ix;
}

int dev_alloc(ifvs_index* ix, void** p, size_t bytes) {
    cudaError_t e = device_malloc(p, bytes ? bytes : 16);
    if (e != cudaSuccess) {
        cudaGetLastError();
        *p = nullptr;
        return set_err(IFVS_ERR_OOM, "device allocation of %zu bytes failed: %s", bytes, cudaGetErrorString(e));
    }
    ix->bytes += bytes;
    return 0;
}

// A column's values as int32 on the host (device columns are copied back).
int column_values(const void* col, int32_t type, bool dio, int64_t N, std::vector<int32_t>& out) {
    const size_t es = type == IFVS_ATTR_I16 ? 2 : 4;
    std::vector<uint8_t> raw;
    const uint8_t* src = (const uint8_t*)col;
    if (dio) {
        raw.resize((size_t)N * es);
        CUDA_TRY(cudaMemcpy(raw.data(), col, (size_t)N * es, cudaMemcpyDeviceToHost));
        src = raw.data();
    }
    out.resize((size_t)N);
    for (int64_t i = 0; i < N; ++i) {
        if (type == IFVS_ATTR_I16) {
            int16_t h;
            memcpy(&h, src + i * 2, 2);
            out[(size_t)i] = h;
        } else {
            memcpy(&out[(size_t)i], src + i * 4, 4);
        }
    }
    return 0;
}

// One stable counting-sort pass of (key, row) by the 16-bit digit of key at
// bit `shift` (least significant digit first: the passes compose into a
// stable sort by the whole key, ties in row order).
template <class Key>
void radix_pass(std::vector<Key>& key, std::vector<uint32_t>& row, std::vector<Key>& key2,
                std::vector<uint32_t>& row2, int shift, std::vector<int64_t>& cnt) {
    const size_t n = key.size();
    std::fill(cnt.begin(), cnt.end(), 0);
    for (size_t i = 0; i < n; ++i) ++cnt[(size_t)((key[i] >> shift) & 0xFFFFu) + 1];
    for (int d = 0; d < 65536; ++d) cnt[d + 1] += cnt[d];
    for (size_t i = 0; i < n; ++i) {
        const int64_t at = cnt[(size_t)((key[i] >> shift) & 0xFFFFu)]++;
        key2[(size_t)at] = key[i];
        row2[(size_t)at] = row[i];
    }
    key.swap(key2);
    row.swap(row2);
}

// Uploads a sorted copy's row order and lays out its codes.
int upload_copy(ifvs_index* ix, int c, const std::vector<uint32_t>& row) {
    const int64_t N = ix->N;
    void* p = nullptr;
    TRY(dev_alloc(ix, &p, sizeof(uint32_t) * (size_t)N));
    ix->d_srt_rows[c] = (uint32_t*)p;
    CUDA_TRY(cudaMemcpy(p, row.data(), sizeof(uint32_t) * (size_t)N, cudaMemcpyHostToDevice));
    TRY(dev_alloc(ix, &p, (size_t)ix->n_rows_pad * ix->row_bytes));
    ix->d_srt_codes[c] = (uint8_t*)p;
    CUDA_TRY(launch_relayout_sorted(ix->d_codes, ix->d_srt_rows[c], N, ix->M, ix->row_bytes, ix->n_rows_pad,
                                    ix->d_srt_codes[c], ix->stream));
    CUDA_TRY(cudaStreamSynchronize(ix->stream));
    return 0;
}

// Sorted copy of column c: rows by (value, row) — a stable host radix sort
// of the values with the sign bit flipped (unsigned order is signed order)
// — the values in that order, and the code rows in that order.
int build_sorted_column(ifvs_index* ix, int c, const std::vector<int32_t>& vals) {
    const int64_t N = ix->N;
    std::vector<uint32_t> key((size_t)N), row((size_t)N), key2((size_t)N), row2((size_t)N);
    for (int64_t i = 0; i < N; ++i) {
        key[(size_t)i] = (uint32_t)vals[(size_t)i] ^ 0x80000000u;
        row[(size_t)i] = (uint32_t)i;
    }
    std::vector<int64_t> cnt(65537);
    radix_pass(key, row, key2, row2, 0, cnt);
    radix_pass(key, row, key2, row2, 16, cnt);
    for (int64_t i = 0; i < N; ++i) key[(size_t)i] ^= 0x80000000u;   // back to the signed value bits
    void* p = nullptr;
    TRY(dev_alloc(ix, &p, sizeof(int32_t) * (size_t)N));
    ix->d_srt_vals[c] = (int32_t*)p;
    CUDA_TRY(cudaMemcpy(p, key.data(), sizeof(int32_t) * (size_t)N, cudaMemcpyHostToDevice));
    return upload_copy(ix, c, row);
}

// Composite copy j of a two-column index: rows by (column j, column 1 - j,
// row) — four radix passes over the 64-bit composite key — and that key of
// each position (ckey).
int build_composite(ifvs_index* ix, int j, const std::vector<int32_t>& primary,
                    const std::vector<int32_t>& secondary) {
    const int64_t N = ix->N;
    std::vector<uint64_t> key((size_t)N), key2((size_t)N);
    std::vector<uint32_t> row((size_t)N), row2((size_t)N);
    for (int64_t i = 0; i < N; ++i) {
        key[(size_t)i] = ckey(primary[(size_t)i], secondary[(size_t)i]);
        row[(size_t)i] = (uint32_t)i;
    }
    std::vector<int64_t> cnt(65537);
    for (int shift = 0; shift < 64; shift += 16) radix_pass(key, row, key2, row2, shift, cnt);
    void* p = nullptr;
    TRY(dev_alloc(ix, &p, sizeof(uint64_t) * (size_t)N));
    ix->d_ckeys[j] = (uint64_t*)p;
    CUDA_TRY(cudaMemcpy(p, key.data(), sizeof(uint64_t) * (size_t)N, cudaMemcpyHostToDevice));
    return upload_copy(ix, kComposite + j, row);
}

// Records a CUDA event pair around one launch on the launching stream when
// timing is on; counts launches per stage always.
struct Stage {
    ifvs_index* ix;
    cudaStream_t s;
    bool on;
    int stage;
    cudaEvent_t a = nullptr;
    Stage(ifvs_index* ix_, cudaStream_t s_, bool on_, int st) : ix(ix_), s(s_), on(on_), stage(st) {
        if (on) {
            a = ix->event();
            if (a) cudaEventRecord(a, s);
        }
    }
    cudaError_t end(cudaError_t launch_err, int launches = 1) {
        ix->stage_launches[stage] += launches;
        if (on && a) {
            cudaEvent_t b = ix->event();
            if (b) {
                cudaEventRecord(b, s);
                ix->pending.push_back({stage, {a, b}});
            } else {
                ix->ev_free.push_back(a);
            }
        }
        return launch_err;
    }
};

struct Opts {
    bool dio = false, timing = false, plain = false, plain_loads = false;
    int R = 0;
    int64_t sub_batch = 0;
    int64_t chunk_blocks = 0;
    int32_t list_max_ppm = 0;
    int32_t pair_min_rows = 0;
    cudaStream_t stream = nullptr;
};

// one-column predicates take the sorted-copy scan at any pool size unless
// the caller sets a threshold: it read fewer bytes and ran faster than the
// bitmap path in every measured selectivity bin, for M = 16 and for the
// generic-M loop (10^6 x 120 codes)
constexpr int32_t kListDefaultPpm = 1000000;

// two-query CTAs for ranges that together span at least 2^22 rows: on the
// 10^8-row workload pairs were faster at 10 % and 100 % of the rows
// (10^7, 10^8) and slower at 0.1 % and 1 % (10^5, 10^6) than one query per
// CTA, which holds two or three CTAs per SM
constexpr int64_t kPairDefaultMinRows = int64_t(1) << 22;

int parse_opts(const ifvs_search_params* p, Opts* o) {
    if (!p) return 0;
    if (p->flags & ~(IFVS_F_DEVICE_IO | IFVS_F_STAGE_TIMING | IFVS_F_PLAIN_PQ | IFVS_F_PLAIN_LOADS))
        return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", p->flags);
    if (p->chunk_blocks < 0) return set_err(IFVS_ERR_ARG, "chunk_blocks must be >= 0");
    if (p->rerank < 0 || p->rerank > IFVS_MAX_K)
        return set_err(IFVS_ERR_ARG, "rerank depth %d outside 0..%d", p->rerank, IFVS_MAX_K);
    if (p->sub_batch < 0) return set_err(IFVS_ERR_ARG, "sub_batch must be >= 0");
    if (p->list_max_ppm < -1 || p->list_max_ppm > 1000000)
        return set_err(IFVS_ERR_ARG, "list_max_ppm = %d outside -1..1000000", p->list_max_ppm);
    if (p->pair_min_rows < -1) return set_err(IFVS_ERR_ARG, "pair_min_rows = %d below -1", p->pair_min_rows);
    o->dio = p->flags & IFVS_F_DEVICE_IO;
    o->timing = p->flags & IFVS_F_STAGE_TIMING;
    o->plain = p->flags & IFVS_F_PLAIN_PQ;
    o->plain_loads = p->flags & IFVS_F_PLAIN_LOADS;
    o->R = p->rerank;
    o->sub_batch = p->sub_batch;
    o->chunk_blocks = p->chunk_blocks;
    o->list_max_ppm = p->list_max_ppm;
    o->pair_min_rows = p->pair_min_rows;
    o->stream = reinterpret_cast<cudaStream_t>(p->stream);
    return 0;
}

int64_t pick_sub_batch(const ifvs_index* ix, const Opts& o, int64_t nq) {
    if (o.sub_batch > 0) return o.sub_batch < nq ? o.sub_batch : nq;
    // bound the lane-major bitmaps to ~16 GiB and the batch to 1024 queries
    const int64_t per_q = ix->n_blocks * 128;
    int64_t sb = (int64_t(16) << 30) / (per_q > 0 ? per_q : 1);
    if (sb > 1024) sb = 1024;
    if (sb < 1) sb = 1;
    return sb < nq ? sb : nq;
}

ScanShape scan_shape(const ifvs_index* ix, int64_t n, int kk, int64_t chunk_blocks) {
    ScanShape sh;
    sh.n_blocks = ix->n_blocks;
    sh.n_rows = ix->N;
    sh.M = ix->M;
    sh.K = ix->K;
    sh.row_bytes = ix->row_bytes;
    sh.tab_words = ix->tab_words;
    // Rows per scan CTA.  Every CTA pays a fixed cost (its table, its
    // lists and their merge, one more partial list per query for k_merge),
    // so a batch takes as few chunks as keep the GPU busy: about two waves
    // of CTAs from the queries alone, and chunks of at most 65 536 blocks
    // (6.7e7 rows), which keeps the long CTAs of 10^8-row dense bins from
    // leaving a ragged last wave.  Measured with 1024-query batches:
    // 10^8 rows 2 chunks 28.1k queries/s (1: 25.3k, 3: 27.2k, 4: 27.5k,
    // 12 L2-sized chunks, the earlier rule: 25.4k); 10^6 rows 1 chunk 795k
    // (2: 723k, 3: 693k).
    const int64_t resident = (int64_t)ix->num_sms * scan_ctas_per_sm(ix->tab_words, scan_kp(kk));
    int64_t chunks = (resident * 2 + n - 1) / n;
    const int64_t by_rows = (ix->n_blocks + 65535) / 65536;
    if (chunks < by_rows) chunks = by_rows;
    int64_t max_chunks = ix->n_blocks / 16;
    if (max_chunks < 1) max_chunks = 1;
    const int64_t key_cap = 32768 / kk;  // bounds the merge's input per query
    if (max_chunks > key_cap) max_chunks = key_cap > 0 ? key_cap : 1;
    if (max_chunks > 65535) max_chunks = 65535;
    if (chunks > max_chunks) chunks = max_chunks;
    if (chunks < 1) chunks = 1;
    if (chunk_blocks > 0) {
        chunks = (ix->n_blocks + chunk_blocks - 1) / chunk_blocks;
        if (chunks > 65535) chunks = 65535;
    }
    sh.blocks_per_chunk = (ix->n_blocks + chunks - 1) / chunks;
    sh.n_chunks = (int)((ix->n_blocks + sh.blocks_per_chunk - 1) / sh.blocks_per_chunk);
    return sh;
}

// The query path for one sub-batch of n queries whose inputs are on the
// device.  Writes k ids / dists per query to out_ids / out_dists (device)
// and the pass counts to npass_u64 (device, zeroed here).
int run_path(ifvs_index* ix, cudaStream_t s, const Opts& o, const float* dq,
             const ifvs_predicate* dp, const float* dwz, int64_t n, int k, int64_t* out_ids,
             float* out_dists, unsigned long long* npass_u64) {
    const int kk = o.R > 0 ? o.R : k;
    const int Mr = ix->M * ix->r;
    const bool cond = !o.plain && ix->d_bank != nullptr;
    // Which queries take the bitmap path is decided on the device (k_plan),
    // but with the sorted-copy path on for every pool size and one attribute
    // column none can: every predicate then constrains at most that column.
    // Such batches need no bitmap workspace (N / 8 bytes per query) and no
    // filter or bitmap-scan launch.
    const bool list_on = o.list_max_ppm >= 0 && ix->n_attrs > 0;
    const int64_t ppm = o.list_max_ppm > 0 ? o.list_max_ppm : kListDefaultPpm;
    const bool bitmaps = !(list_on && ppm >= 1000000 && ix->n_attrs == 1);
    TRY(ensure(ix->w_canon, sizeof(CanonPred) * n));
    if (bitmaps) TRY(ensure(ix->w_bm, (size_t)n * ix->n_blocks * 32 * 4));
    TRY(ensure(ix->w_idx, sizeof(uint32_t) * n * (ix->h > 0 ? ix->h : 1)));
    TRY(ensure(ix->w_alpha, sizeof(float) * n * (Mr > 0 ? Mr : 1)));
    TRY(ensure(ix->w_wf, sizeof(float) * n * ix->D));
    TRY(ensure(ix->w_lut, sizeof(float) * n * ix->M * ix->K));
    TRY(ensure(ix->w_tab, sizeof(float) * n * 256 * ix->tab_words));
    const ScanShape sh = scan_shape(ix, n, kk, o.chunk_blocks);
    TRY(ensure(ix->w_part, sizeof(uint64_t) * n * sh.n_chunks * kk));
    if (o.R > 0) {
        TRY(ensure(ix->w_cand, sizeof(int64_t) * n * kk));
        TRY(ensure(ix->w_cdist, sizeof(float) * n * kk));
    }
    CUDA_TRY(cudaMemsetAsync(npass_u64, 0, sizeof(unsigned long long) * n, s));
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_PREDICATE);
        CUDA_TRY(st.end(launch_canonicalize(dp, n, ix->cols(), ix->w_canon.as<CanonPred>(),
                                            ix->w_err.as<int>(), s)));
    }
    // one-column predicates take the sorted-copy scan (up to the threshold)
    const ScanPlan* plan = nullptr;
    if (list_on) {
        const int64_t max_rows = ppm >= 1000000 ? ix->N : ix->N * ppm / 1000000;
        TRY(ensure(ix->w_plan, sizeof(ScanPlan) * n));
        TRY(ensure(ix->w_items, scan_list_workspace_bytes(n)));   // query groups of the sorted-copy scan
        Stage st(ix, s, o.timing, IFVS_STAGE_FILTER);
        CUDA_TRY(st.end(launch_plan(ix->w_canon.as<CanonPred>(), n, ix->sorted(), ix->N, max_rows,
                                    ix->w_plan.as<ScanPlan>(), npass_u64, s)));
        plan = ix->w_plan.as<ScanPlan>();
    }
    if (bitmaps) {
        Stage st(ix, s, o.timing, IFVS_STAGE_FILTER);
        CUDA_TRY(st.end(launch_filter(ix->cols(), ix->N, ix->n_blocks, ix->w_canon.as<CanonPred>(),
                                      plan, n, ix->w_bm.as<uint32_t>(), npass_u64, ix->num_sms, s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_CONDITION);
        CUDA_TRY(st.end(launch_condition(dq, dp, n, ix->D, ix->d_seeds, ix->h, ix->B,
                                         cond ? ix->d_bank : nullptr, Mr, dwz,
                                         ix->w_idx.as<uint32_t>(), ix->w_alpha.as<float>(),
                                         ix->w_wf.as<float>(), s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_LUT);
        CUDA_TRY(st.end(launch_lut(ix->d_cpq, ix->d_W, cond ? ix->w_alpha.as<float>() : nullptr,
                                   dq, ix->w_wf.as<float>(), n, ix->M, ix->K, ix->ds, ix->r,
                                   ix->w_lut.as<float>(), nullptr, ix->num_sms, s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_LUT);
        CUDA_TRY(st.end(launch_tables(ix->w_lut.as<float>(), n, ix->M, ix->K, ix->tab_words,
                                      ix->w_tab.as<float>(), s)));
    }
    if (bitmaps) {
        Stage st(ix, s, o.timing, IFVS_STAGE_SCAN);
        CUDA_TRY(st.end(launch_scan(ix->d_codes, ix->w_tab.as<float>(), ix->w_bm.as<uint32_t>(), plan,
                                    n, kk, sh, ix->w_part.as<uint64_t>(), s)));
    }
    if (plan) {
        Stage st(ix, s, o.timing, IFVS_STAGE_SCAN);
        int nl = 0;
        ListOpts lo;
        lo.pair_min_rows = o.pair_min_rows > 0 ? o.pair_min_rows : kPairDefaultMinRows;
        lo.bulk = !o.plain_loads;
        lo.tx_extra = stall_copies_for_tests() ? 16u : 0u;
        lo.err = ix->w_err.as<int>();
        const cudaError_t e = launch_scan_list(ix->w_tab.as<float>(), ix->sorted(), plan, n, kk, sh,
                                               ix->w_part.as<uint64_t>(),
                                               o.pair_min_rows < 0 ? nullptr : ix->w_items.as<uint8_t>(),
                                               lo, s, &nl);
        CUDA_TRY(st.end(e, nl));
    }
    int64_t* m_ids = o.R > 0 ? ix->w_cand.as<int64_t>() : out_ids;
    float* m_dists = o.R > 0 ? ix->w_cdist.as<float>() : out_dists;
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_MERGE);
        CUDA_TRY(st.end(launch_merge(ix->w_part.as<uint64_t>(), n, sh.n_chunks, kk, m_ids, m_dists, s)));
    }
    if (o.R > 0) {
        Stage st(ix, s, o.timing, IFVS_STAGE_RERANK);
        CUDA_TRY(st.end(launch_rerank(ix->d_vec, ix->N, ix->D, dq, m_ids, n, o.R, k, out_ids,
                                      out_dists, s)));
    }
    return 0;
}

// The scan keeps the table and per-warp lists of the next power of two >= k
// in shared memory; large M leaves room for smaller k only.
int check_scan_fits(const ifvs_index* ix, int kk) {
    const size_t need = scan_smem_bytes(ix->tab_words, scan_kp(kk));
    if (need > (size_t)ix->max_smem)
        return set_err(IFVS_ERR_UNSUPPORTED,
                       "k = %d with M = %d needs %zu bytes of shared memory per CTA (device: %d)",
                       kk, ix->M, need, ix->max_smem);
    return 0;
}

int check_index(const ifvs_index* ix, bool need_cb) {
    if (!ix) return set_err(IFVS_ERR_ARG, "index is NULL");
    if (need_cb && !ix->has_cb)
        return set_err(IFVS_ERR_STATE, "ifvs_load_codebooks has not been called on this index");
    return 0;
}

// Stage inputs of one sub-batch on the device (copies unless device I/O).
int stage_inputs(ifvs_index* ix, cudaStream_t s, const Opts& o, int64_t q0, int64_t n,
                 const float* queries, const ifvs_predicate* preds, const float* wz,
                 const float** dq, const ifvs_predicate** dp, const float** dwz) {
    const int D = ix->D;
    if (o.dio) {
        if (dq) *dq = queries ? queries + q0 * D : nullptr;
        if (dp) *dp = preds ? preds + q0 : nullptr;
        if (dwz) *dwz = wz ? wz + q0 * D : nullptr;
        return 0;
    }
    if (dq) {
        *dq = nullptr;
        if (queries) {
            TRY(ensure(ix->w_q, sizeof(float) * n * D));
            CUDA_TRY(cudaMemcpyAsync(ix->w_q.p, queries + q0 * D, sizeof(float) * n * D,
                                     cudaMemcpyHostToDevice, s));
            *dq = ix->w_q.as<float>();
        }
    }
    if (dp) {
        *dp = nullptr;
        if (preds) {
            TRY(ensure(ix->w_preds, sizeof(ifvs_predicate) * n));
            CUDA_TRY(cudaMemcpyAsync(ix->w_preds.p, preds + q0, sizeof(ifvs_predicate) * n,
                                     cudaMemcpyHostToDevice, s));
            *dp = ix->w_preds.as<ifvs_predicate>();
        }
    }
    if (dwz) {
        *dwz = nullptr;
        if (wz) {
            TRY(ensure(ix->w_wz, sizeof(float) * n * D));
            CUDA_TRY(cudaMemcpyAsync(ix->w_wz.p, wz + q0 * D, sizeof(float) * n * D,
                                     cudaMemcpyHostToDevice, s));
            *dwz = ix->w_wz.as<float>();
        }
    }
    return 0;
}

int copy_out(cudaStream_t s, bool dio, void* dst, const void* src, size_t bytes) {
    if (bytes == 0) return 0;
    CUDA_TRY(cudaMemcpyAsync(dst, src, bytes, dio ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, s));
    return 0;
}

// Synchronise, fold the timing events, and report a malformed predicate.
int finish(ifvs_index* ix, cudaStream_t s, bool check_preds) {
    CUDA_TRY(cudaStreamSynchronize(s));
    ix->collect();
    if (check_preds) {
        int err = 0;
        CUDA_TRY(cudaMemcpy(&err, ix->w_err.p, sizeof(int), cudaMemcpyDeviceToHost));
        if (err & 4)
            return set_err(IFVS_ERR_TIMEOUT, "a bounded wait of the scan for its bulk-copied code tiles ran out; "
                                             "the results are incomplete");
        if (err & 2) return set_err(IFVS_ERR_ARG, "a candidate row id is outside -1..N-1");
        if (err) return set_err(IFVS_ERR_ARG, "a predicate is malformed (n_clauses outside 0..4, "
                                              "reserved != 0, column out of range or unknown operator)");
    }
    return 0;
}

int reset_err_flag(ifvs_index* ix, cudaStream_t s) {
    TRY(ensure(ix->w_err, sizeof(int)));
    CUDA_TRY(cudaMemsetAsync(ix->w_err.p, 0, sizeof(int), s));
    return 0;
}

// ---- training (§2 "Learning") ----------------------------------------

int train_check(ifvs_index* ix, const ifvs_train_params* tp, int64_t nq, bool step, Opts* o) {
    TRY(check_index(ix, true));
    if (!tp) return set_err(IFVS_ERR_ARG, "training parameters are NULL");
    if (!ix->d_bank) return set_err(IFVS_ERR_STATE, "training needs a memory bank, W and seeds (ifvs_load_codebooks)");
    if (tp->flags & ~(IFVS_F_DEVICE_IO | IFVS_F_STAGE_TIMING))
        return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", tp->flags);
    if (!(tp->tau > 0.f) || !std::isfinite(tp->tau)) return set_err(IFVS_ERR_ARG, "tau must be finite and > 0");
    if (!(tp->lambda >= 0.f) || !std::isfinite(tp->lambda)) return set_err(IFVS_ERR_ARG, "lambda must be finite and >= 0");
    if (step && (!(tp->lr >= 0.f) || !std::isfinite(tp->lr) || !(tp->lr_wz >= 0.f) || !std::isfinite(tp->lr_wz)))
        return set_err(IFVS_ERR_ARG, "lr and lr_wz must be finite and >= 0");
    const int V = tp->n_pos + tp->n_neg;
    if (tp->n_pos < 0 || tp->n_neg < 0 || V < 1 || V > kTrainMaxV)
        return set_err(IFVS_ERR_ARG, "n_pos = %d, n_neg = %d: need n_pos, n_neg >= 0 and 1 <= n_pos + n_neg <= %d",
                       tp->n_pos, tp->n_neg, kTrainMaxV);
    if (step && V > IFVS_MAX_K)
        return set_err(IFVS_ERR_ARG, "mining n_pos + n_neg = %d rows per query exceeds %d", V, IFVS_MAX_K);
    if (step) TRY(check_scan_fits(ix, V));
    if (nq < 0 || nq > 1024) return set_err(IFVS_ERR_ARG, "nq = %lld outside 0..1024 (one mini-batch per call)", (long long)nq);
    if (ix->r > kTrainMaxR) return set_err(IFVS_ERR_UNSUPPORTED, "training supports r <= %d (index: %d)", kTrainMaxR, ix->r);
    if (train_query_smem(V, ix->M * ix->r, ix->D, ix->r) > (size_t)ix->max_smem)
        return set_err(IFVS_ERR_UNSUPPORTED, "D = %d, M r = %d with %d candidates exceed shared memory",
                       ix->D, ix->M * ix->r, V);
    o->dio = tp->flags & IFVS_F_DEVICE_IO;
    o->timing = tp->flags & IFVS_F_STAGE_TIMING;
    o->stream = reinterpret_cast<cudaStream_t>(tp->stream);
    return 0;
}

// Stages queries, predicates and the shared w_z (a device copy in t_wz and a
// per-query broadcast in w_wz), and validates the predicates.
int train_stage(ifvs_index* ix, cudaStream_t s, const Opts& o, int64_t n, const float* queries,
                const ifvs_predicate* preds, const float* wz, const float** dq,
                const ifvs_predicate** dp) {
    TRY(stage_inputs(ix, s, o, 0, n, queries, preds, nullptr, dq, dp, nullptr));
    TRY(ensure(ix->t_wz, sizeof(float) * ix->D));
    CUDA_TRY(cudaMemcpyAsync(ix->t_wz.p, wz, sizeof(float) * ix->D,
                             o.dio ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice, s));
    TRY(ensure(ix->w_wz, sizeof(float) * n * ix->D));
    CUDA_TRY(launch_broadcast_wz(ix->t_wz.as<float>(), ix->D, n, ix->w_wz.as<float>(), s));
    TRY(ensure(ix->w_canon, sizeof(CanonPred) * n));
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_PREDICATE);
        CUDA_TRY(st.end(launch_canonicalize(*dp, n, ix->cols(), ix->w_canon.as<CanonPred>(),
                                            ix->w_err.as<int>(), s)));
    }
    return 0;
}

// Loss and gradients of one mini-batch into the t_* buffers (gW, gbank, gwz).
int train_gradient(ifvs_index* ix, cudaStream_t s, const Opts& o, const TrainQueryArgs& a) {
    const int Mr = ix->M * ix->r, KD = ix->K * ix->ds;
    const float inv_n = 1.f / (float)a.n;
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_train_gram(ix->d_W, ix->M, ix->r, KD, ix->t_G.as<float>(), s)));
    }
    CUDA_TRY(cudaMemsetAsync(a.gC, 0, sizeof(float) * (size_t)a.n * ix->M * KD, s));
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_train_query(a, s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        int nl = 0;
        const cudaError_t e = launch_train_gW(a.alpha, a.gC, ix->d_W, a.n, ix->M, ix->r, KD, a.lambda,
                                              inv_n, ix->t_gWpart.as<float>(), ix->t_gW.as<float>(), s, &nl);
        CUDA_TRY(st.end(e, nl));
    }
    CUDA_TRY(cudaMemsetAsync(ix->t_gbank.p, 0, sizeof(float) * (size_t)ix->B * Mr, s));
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_train_bank(ix->w_idx.as<uint32_t>(), a.n, ix->h, Mr,
                                          ix->t_galpha.as<float>(), inv_n, ix->t_gbank.as<float>(), s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_train_wz(a.gw, a.n, ix->D, ix->t_wz.as<float>(), inv_n,
                                        ix->t_gwz.as<float>(), s)));
    }
    return 0;
}

int train_buffers(ifvs_index* ix, int64_t n, int V) {
    const int64_t Mr = (int64_t)ix->M * ix->r, KD = (int64_t)ix->K * ix->ds;
    TRY(ensure(ix->t_gC, sizeof(float) * n * ix->M * KD));
    TRY(ensure(ix->t_gw, sizeof(float) * n * ix->D));
    TRY(ensure(ix->t_loss, sizeof(double) * n));
    TRY(ensure(ix->t_G, sizeof(float) * ix->M * ix->r * ix->r));
    TRY(ensure(ix->t_gW, sizeof(float) * ix->M * ix->r * KD));
    TRY(ensure(ix->t_gWpart, train_gW_scratch(n, ix->M, ix->r, (int)KD)));
    TRY(ensure(ix->t_galpha, sizeof(float) * n * Mr));
    TRY(ensure(ix->t_gbank, sizeof(float) * ix->B * Mr));
    TRY(ensure(ix->t_gwz, sizeof(float) * ix->D));
    TRY(ensure(ix->w_idx, sizeof(uint32_t) * n * ix->h));
    TRY(ensure(ix->w_alpha, sizeof(float) * n * Mr));
    TRY(ensure(ix->w_wf, sizeof(float) * n * ix->D));
    (void)V;
    return 0;
}

TrainQueryArgs train_args(ifvs_index* ix, const ifvs_train_params* tp, int64_t n, const float* dq) {
    TrainQueryArgs a{};
    a.codes = ix->d_codes;
    a.row_bytes = ix->row_bytes;
    a.M = ix->M;
    a.K = ix->K;
    a.ds = ix->ds;
    a.D = ix->D;
    a.r = ix->r;
    a.C_pq = ix->d_cpq;
    a.W = ix->d_W;
    a.G = ix->t_G.as<float>();
    a.q = dq;
    a.wf = ix->w_wf.as<float>();
    a.alpha = ix->w_alpha.as<float>();
    a.P = tp->n_pos;
    a.n_neg = tp->n_neg;
    a.tau = tp->tau;
    a.lambda = tp->lambda;
    a.n = n;
    a.N = ix->N;
    a.err = ix->w_err.as<int>();
    a.gC = ix->t_gC.as<float>();
    a.gw = ix->t_gw.as<float>();
    a.galpha = ix->t_galpha.as<float>();
    a.loss = ix->t_loss.as<double>();
    return a;
}

// Mean of the per-query losses, summed in query order on the host.
int train_loss_out(ifvs_index* ix, cudaStream_t s, int64_t n, double* loss) {
    if (!loss) return 0;
    std::vector<double> l((size_t)n);
    CUDA_TRY(cudaMemcpyAsync(l.data(), ix->t_loss.p, sizeof(double) * n, cudaMemcpyDeviceToHost, s));
    CUDA_TRY(cudaStreamSynchronize(s));
    double t = 0.0;
    for (double v : l) t += v;
    *loss = t / (double)n;
    return 0;
}

}  // namespace

// ============================================================== internal

int ifvs::index_view(const ifvs_index* ix, IndexView* out) {
    if (!ix) return set_err(IFVS_ERR_ARG, "index is NULL");
    out->device = ix->device;
    out->num_sms = ix->num_sms;
    out->max_smem = ix->max_smem;
    out->N = ix->N;
    out->n_blocks = ix->n_blocks;
    out->M = ix->M;
    out->K = ix->K;
    out->row_bytes = ix->row_bytes;
    out->tab_words = ix->tab_words;
    out->codes = ix->d_codes;
    return 0;
}

int ifvs::report_error(int code, const char* fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_err, sizeof g_err, fmt, ap);
    va_end(ap);
    return code;
}

// ============================================================== C ABI

extern "C" {

const char* ifvs_last_error(void) { return g_err; }

const char* ifvs_version(void) { return "ifvs-gb300 0.1 (sm_103a)"; }

int ifvs_canonical_predicate(const ifvs_predicate* p, const int32_t* attr_types, int32_t n_attrs,
                             int32_t* lo, uint32_t* width_m1, int32_t* empty) {
    if (!p || (n_attrs > 0 && !attr_types) || n_attrs < 0 || n_attrs > IFVS_MAX_ATTRS)
        return set_err(IFVS_ERR_ARG, "invalid arguments");
    int32_t t[IFVS_MAX_ATTRS] = {0, 0, 0, 0};
    for (int i = 0; i < n_attrs; ++i) t[i] = attr_types[i];
    CanonPred c;
    int rc = canonicalize(*p, t, n_attrs, &c);
    for (int i = 0; i < n_attrs; ++i) {
        if (lo) lo[i] = c.lo[i];
        if (width_m1) width_m1[i] = c.wm1[i];
    }
    if (empty) *empty = c.empty;
    if (rc != 0) return set_err(IFVS_ERR_ARG, "malformed predicate");
    return IFVS_OK;
}

int ifvs_load_index(ifvs_index** out, int32_t device, const uint8_t* codes, int64_t N, int32_t M,
                    int32_t K, const void* const* attr_cols, const int32_t* attr_types,
                    int32_t n_attrs, const float* vectors, int32_t D, uint32_t flags) {
    if (!out) return set_err(IFVS_ERR_ARG, "out is NULL");
    *out = nullptr;
    if (!codes) return set_err(IFVS_ERR_ARG, "codes is NULL");
    if (N < 1 || N > (int64_t)0xFFFFFFFFLL - 2048)
        return set_err(IFVS_ERR_ARG, "N = %lld outside 1..2^32-2049", (long long)N);
    if (M < 1 || M > IFVS_MAX_M) return set_err(IFVS_ERR_UNSUPPORTED, "M = %d outside 1..%d", M, IFVS_MAX_M);
    if (K < 1 || K > 256) return set_err(IFVS_ERR_UNSUPPORTED, "K = %d outside 1..256", K);
    if (n_attrs < 0 || n_attrs > IFVS_MAX_ATTRS)
        return set_err(IFVS_ERR_ARG, "n_attrs = %d outside 0..%d", n_attrs, IFVS_MAX_ATTRS);
    if (n_attrs > 0 && (!attr_cols || !attr_types)) return set_err(IFVS_ERR_ARG, "attribute arrays are NULL");
    for (int i = 0; i < n_attrs; ++i) {
        if (!attr_cols[i]) return set_err(IFVS_ERR_ARG, "attribute column %d is NULL", i);
        if (attr_types[i] != IFVS_ATTR_I32 && attr_types[i] != IFVS_ATTR_I16)
            return set_err(IFVS_ERR_ARG, "attribute column %d has unknown type %d", i, attr_types[i]);
    }
    if (D < 0 || (D > 0 && D % M != 0)) return set_err(IFVS_ERR_ARG, "D = %d is not a multiple of M = %d", D, M);
    if (vectors && D == 0) return set_err(IFVS_ERR_ARG, "raw vectors need D > 0");
    if (flags & ~IFVS_F_DEVICE_IO) return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", flags);
    const bool dio = flags & IFVS_F_DEVICE_IO;

    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
        cudaGetLastError();
        return set_err(IFVS_ERR_CUDA, "no CUDA device is available");
    }
    if (device < 0 || device >= ndev) return set_err(IFVS_ERR_ARG, "device %d outside 0..%d", device, ndev - 1);
    DeviceGuard g(device);
    if (!g.ok) return set_err(IFVS_ERR_CUDA, "cudaSetDevice(%d) failed", device);

    ifvs_index* ix = new (std::nothrow) ifvs_index();
    if (!ix) return set_err(IFVS_ERR_OOM, "host allocation failed");
    ix->device = device;
    int rc = 0;
    auto fail = [&](int code) {
        free_index(ix);
        return code;
    };
    if (cudaDeviceGetAttribute(&ix->num_sms, cudaDevAttrMultiProcessorCount, device) != cudaSuccess ||
        cudaDeviceGetAttribute(&ix->max_smem, cudaDevAttrMaxSharedMemoryPerBlockOptin, device) != cudaSuccess)
        return fail(cuda_fail(cudaGetLastError(), "cudaDeviceGetAttribute", __LINE__));
    // a blocking stream: work the caller put on the legacy default stream
    // (NULL) before a call is ordered before the call's kernels
    if (cudaStreamCreateWithFlags(&ix->stream, cudaStreamDefault) != cudaSuccess)
        return fail(cuda_fail(cudaGetLastError(), "cudaStreamCreateWithFlags", __LINE__));
    ix->N = N;
    ix->M = M;
    ix->K = K;
    ix->D = D;
    ix->ds = D > 0 ? D / M : 0;
    ix->n_blocks = (N + kBlockRows - 1) / kBlockRows;
    ix->n_rows_pad = ix->n_blocks * kBlockRows;
    // rows of 9 to 16 subspaces take 16 bytes (one vector load per row, and
    // the scan loops compiled for M = 12 and 16); others M rounded up to 4
    ix->row_bytes = (M > 8 && M <= 16) ? 16 : (int)round_up(M, 4);
    ix->tab_words = (int)round_up(M + 31, 32);
    if (scan_smem_bytes(ix->tab_words, scan_kp(1)) > (size_t)ix->max_smem)
        return fail(set_err(IFVS_ERR_UNSUPPORTED, "M = %d needs %zu bytes of shared memory (device: %d)",
                            M, scan_smem_bytes(ix->tab_words, scan_kp(1)), ix->max_smem));
    cudaStream_t s = ix->stream;
    const cudaMemcpyKind h2d = dio ? cudaMemcpyDeviceToDevice : cudaMemcpyHostToDevice;

    // codes -> rotated rows
    void* tmp = nullptr;
    const uint8_t* src = codes;
    if (!dio) {
        if ((rc = dev_alloc(ix, &tmp, (size_t)N * M))) return fail(rc);
        ix->bytes -= (size_t)N * M;
        if (cudaMemcpyAsync(tmp, codes, (size_t)N * M, cudaMemcpyHostToDevice, s) != cudaSuccess) {
            cudaFree(tmp);
            return fail(cuda_fail(cudaGetLastError(), "cudaMemcpyAsync(codes)", __LINE__));
        }
        src = (const uint8_t*)tmp;
    }
    void* dcodes = nullptr;
    if ((rc = dev_alloc(ix, &dcodes, (size_t)ix->n_rows_pad * ix->row_bytes))) {
        if (tmp) cudaFree(tmp);
        return fail(rc);
    }
    ix->d_codes = (uint8_t*)dcodes;
    if ((rc = ensure(ix->w_err, sizeof(int)))) {
        if (tmp) cudaFree(tmp);
        return fail(rc);
    }
    cudaMemsetAsync(ix->w_err.p, 0, sizeof(int), s);
    cudaError_t e = launch_relayout_codes(src, N, M, K, ix->row_bytes, ix->n_rows_pad, ix->d_codes,
                                          ix->w_err.as<int>(), s);
    if (e == cudaSuccess) e = cudaStreamSynchronize(s);
    if (tmp) cudaFree(tmp);
    if (e != cudaSuccess) return fail(cuda_fail(e, "code re-layout", __LINE__));
    int bad = 0;
    if (cudaMemcpy(&bad, ix->w_err.p, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess)
        return fail(cuda_fail(cudaGetLastError(), "cudaMemcpy(flag)", __LINE__));
    if (bad) return fail(set_err(IFVS_ERR_ARG, "a code is >= K = %d", K));

    // attribute columns, padded with zeros to n_rows_pad
    ix->n_attrs = n_attrs;
    for (int i = 0; i < n_attrs; ++i) {
        ix->types[i] = attr_types[i];
        const size_t es = attr_types[i] == IFVS_ATTR_I16 ? 2 : 4;
        if ((rc = dev_alloc(ix, &ix->d_attr[i], es * ix->n_rows_pad))) return fail(rc);
        if (cudaMemsetAsync(ix->d_attr[i], 0, es * ix->n_rows_pad, s) != cudaSuccess ||
            cudaMemcpyAsync(ix->d_attr[i], attr_cols[i], es * N, h2d, s) != cudaSuccess)
            return fail(cuda_fail(cudaGetLastError(), "attribute copy", __LINE__));
    }
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(cuda_fail(e, "attribute upload", __LINE__));
    {
        std::vector<std::vector<int32_t>> vals((size_t)n_attrs);
        for (int i = 0; i < n_attrs; ++i) {
            if ((rc = column_values(attr_cols[i], attr_types[i], dio, N, vals[(size_t)i]))) return fail(rc);
            if ((rc = build_sorted_column(ix, i, vals[(size_t)i]))) return fail(rc);
        }
        // two columns: both composite orders, so that a predicate fixing
        // either column and bounding the other reads one position range
        if (n_attrs == 2)
            for (int jj = 0; jj < 2; ++jj)
                if ((rc = build_composite(ix, jj, vals[(size_t)jj], vals[(size_t)(1 - jj)]))) return fail(rc);
    }
    if (vectors) {
        void* v = nullptr;
        if ((rc = dev_alloc(ix, &v, sizeof(float) * N * D))) return fail(rc);
        ix->d_vec = (float*)v;
        if (cudaMemcpyAsync(v, vectors, sizeof(float) * N * D, h2d, s) != cudaSuccess)
            return fail(cuda_fail(cudaGetLastError(), "vector copy", __LINE__));
    }
    e = cudaStreamSynchronize(s);
    if (e != cudaSuccess) return fail(cuda_fail(e, "index upload", __LINE__));
    *out = ix;
    return IFVS_OK;
}

int ifvs_load_codebooks(ifvs_index* ix, const float* C_pq, int32_t ds, const float* bank, int64_t B,
                        int32_t h, int32_t r, const float* W, const uint64_t* hash_seeds) {
    TRY(check_index(ix, false));
    if (!C_pq) return set_err(IFVS_ERR_ARG, "C_pq is NULL");
    if (ds < 1) return set_err(IFVS_ERR_ARG, "ds = %d must be >= 1", ds);
    if (ix->D > 0 && ix->D != ix->M * ds)
        return set_err(IFVS_ERR_ARG, "ds = %d does not match D = %d and M = %d", ds, ix->D, ix->M);
    if (bank) {
        if (B < 1 || B > 0xFFFFFFFFLL) return set_err(IFVS_ERR_ARG, "B = %lld outside 1..2^32-1", (long long)B);
        if (h < 1 || h > 64) return set_err(IFVS_ERR_ARG, "h = %d outside 1..64", h);
        if (r < 1 || r > 256) return set_err(IFVS_ERR_ARG, "r = %d outside 1..256", r);
        if (!W || !hash_seeds) return set_err(IFVS_ERR_ARG, "W and hash_seeds are required with a bank");
    }
    DeviceGuard g(ix->device);
    cudaStream_t s = ix->stream;
    CUDA_TRY(cudaStreamSynchronize(s));
    void* old[] = {ix->d_cpq, ix->d_bank, ix->d_W, ix->d_seeds};
    for (void* p : old)
        if (p) cudaFree(p);
    ix->d_cpq = nullptr;
    ix->d_bank = nullptr;
    ix->d_W = nullptr;
    ix->d_seeds = nullptr;
    ix->has_cb = false;
    ix->ds = ds;
    ix->D = ix->M * ds;
    const size_t ncb = (size_t)ix->M * ix->K * ds;
    void* p = nullptr;
    TRY(dev_alloc(ix, &p, sizeof(float) * ncb));
    ix->d_cpq = (float*)p;
    CUDA_TRY(cudaMemcpyAsync(p, C_pq, sizeof(float) * ncb, cudaMemcpyHostToDevice, s));
    if (bank) {
        ix->B = B;
        ix->h = h;
        ix->r = r;
        TRY(dev_alloc(ix, &p, sizeof(float) * (size_t)B * ix->M * r));
        ix->d_bank = (float*)p;
        CUDA_TRY(cudaMemcpyAsync(p, bank, sizeof(float) * (size_t)B * ix->M * r, cudaMemcpyHostToDevice, s));
        TRY(dev_alloc(ix, &p, sizeof(float) * ncb * r));
        ix->d_W = (float*)p;
        CUDA_TRY(cudaMemcpyAsync(p, W, sizeof(float) * ncb * r, cudaMemcpyHostToDevice, s));
        TRY(dev_alloc(ix, &p, sizeof(uint64_t) * h));
        ix->d_seeds = (uint64_t*)p;
        CUDA_TRY(cudaMemcpyAsync(p, hash_seeds, sizeof(uint64_t) * h, cudaMemcpyHostToDevice, s));
    } else {
        ix->B = 0;
        ix->h = 0;
        ix->r = 0;
    }
    CUDA_TRY(cudaStreamSynchronize(s));
    ix->has_cb = true;
    return IFVS_OK;
}

int ifvs_search_batch(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                      int32_t k, const float* wz, const ifvs_search_params* p, int64_t* ids,
                      float* dists, int64_t* npass) {
    TRY(check_index(ix, true));
    Opts o;
    TRY(parse_opts(p, &o));
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (k < 1 || k > IFVS_MAX_K) return set_err(IFVS_ERR_ARG, "k = %d outside 1..%d", k, IFVS_MAX_K);
    if (o.R > 0 && o.R < k) return set_err(IFVS_ERR_ARG, "rerank depth %d is below k = %d", o.R, k);
    if (o.R > 0 && !ix->d_vec) return set_err(IFVS_ERR_STATE, "rerank needs raw vectors at load time");
    TRY(check_scan_fits(ix, o.R > 0 ? o.R : k));
    if (nq == 0) return IFVS_OK;
    if (!queries || !preds || !ids || !dists) return set_err(IFVS_ERR_ARG, "an array argument is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const int64_t sb = pick_sub_batch(ix, o, nq);
    TRY(reset_err_flag(ix, s));
    TRY(ensure(ix->w_npass, sizeof(unsigned long long) * sb));
    if (!o.dio) {
        TRY(ensure(ix->w_ids, sizeof(int64_t) * sb * k));
        TRY(ensure(ix->w_dists, sizeof(float) * sb * k));
    }
    for (int64_t q0 = 0; q0 < nq; q0 += sb) {
        const int64_t n = sb < nq - q0 ? sb : nq - q0;
        const float *dq, *dwz;
        const ifvs_predicate* dp;
        TRY(stage_inputs(ix, s, o, q0, n, queries, preds, wz, &dq, &dp, &dwz));
        int64_t* oid = o.dio ? ids + q0 * k : ix->w_ids.as<int64_t>();
        float* odi = o.dio ? dists + q0 * k : ix->w_dists.as<float>();
        TRY(run_path(ix, s, o, dq, dp, dwz, n, k, oid, odi, ix->w_npass.as<unsigned long long>()));
        if (!o.dio) {
            TRY(copy_out(s, false, ids + q0 * k, oid, sizeof(int64_t) * n * k));
            TRY(copy_out(s, false, dists + q0 * k, odi, sizeof(float) * n * k));
        }
        if (npass) TRY(copy_out(s, o.dio, npass + q0, ix->w_npass.p, sizeof(int64_t) * n));
        if (!o.dio && q0 + sb < nq) CUDA_TRY(cudaStreamSynchronize(s));
    }
    return finish(ix, s, true);
}

int ifvs_filter(ifvs_index* ix, const ifvs_predicate* preds, int64_t nq, const ifvs_search_params* p,
                uint32_t* bitmaps, int64_t* npass) {
    TRY(check_index(ix, false));
    Opts o;
    TRY(parse_opts(p, &o));
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (nq == 0) return IFVS_OK;
    if (!preds || !bitmaps) return set_err(IFVS_ERR_ARG, "an array argument is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const int64_t sb = pick_sub_batch(ix, o, nq);
    const int64_t wrows = (ix->N + 31) / 32;
    TRY(reset_err_flag(ix, s));
    TRY(ensure(ix->w_npass, sizeof(unsigned long long) * sb));
    TRY(ensure(ix->w_canon, sizeof(CanonPred) * sb));
    TRY(ensure(ix->w_bm, (size_t)sb * ix->n_blocks * 128));
    if (!o.dio) TRY(ensure(ix->w_rows, (size_t)sb * wrows * 4));
    for (int64_t q0 = 0; q0 < nq; q0 += sb) {
        const int64_t n = sb < nq - q0 ? sb : nq - q0;
        const ifvs_predicate* dp;
        TRY(stage_inputs(ix, s, o, q0, n, nullptr, preds, nullptr, nullptr, &dp, nullptr));
        CUDA_TRY(cudaMemsetAsync(ix->w_npass.p, 0, sizeof(unsigned long long) * n, s));
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_PREDICATE);
            CUDA_TRY(st.end(launch_canonicalize(dp, n, ix->cols(), ix->w_canon.as<CanonPred>(),
                                                ix->w_err.as<int>(), s)));
        }
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_FILTER);
            CUDA_TRY(st.end(launch_filter(ix->cols(), ix->N, ix->n_blocks, ix->w_canon.as<CanonPred>(),
                                          nullptr, n, ix->w_bm.as<uint32_t>(),
                                          ix->w_npass.as<unsigned long long>(), ix->num_sms, s)));
        }
        uint32_t* rows = o.dio ? bitmaps + q0 * wrows : ix->w_rows.as<uint32_t>();
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_LAYOUT);
            CUDA_TRY(st.end(launch_bitmap_layout(ix->w_bm.as<uint32_t>(), rows, n, ix->n_blocks, wrows,
                                                 true, s)));
        }
        if (!o.dio) TRY(copy_out(s, false, bitmaps + q0 * wrows, rows, sizeof(uint32_t) * n * wrows));
        if (npass) TRY(copy_out(s, o.dio, npass + q0, ix->w_npass.p, sizeof(int64_t) * n));
        if (q0 + sb < nq) CUDA_TRY(cudaStreamSynchronize(s));
    }
    return finish(ix, s, true);
}

int ifvs_condition(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                   const float* wz, const ifvs_search_params* p, uint32_t* bank_idx, float* alpha,
                   float* wf, float* C_ifvs, float* lut) {
    TRY(check_index(ix, true));
    Opts o;
    TRY(parse_opts(p, &o));
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (nq == 0) return IFVS_OK;
    if (!queries || !preds) return set_err(IFVS_ERR_ARG, "queries / preds is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const bool cond = !o.plain && ix->d_bank != nullptr;
    const int Mr = ix->M * ix->r;
    const int64_t sb = nq < 1024 ? nq : 1024;
    TRY(reset_err_flag(ix, s));
    TRY(ensure(ix->w_canon, sizeof(CanonPred) * sb));
    TRY(ensure(ix->w_idx, sizeof(uint32_t) * sb * (ix->h > 0 ? ix->h : 1)));
    TRY(ensure(ix->w_alpha, sizeof(float) * sb * (Mr > 0 ? Mr : 1)));
    TRY(ensure(ix->w_wf, sizeof(float) * sb * ix->D));
    TRY(ensure(ix->w_lut, sizeof(float) * sb * ix->M * ix->K));
    if (C_ifvs) TRY(ensure(ix->w_cifvs, sizeof(float) * sb * ix->M * ix->K * ix->ds));
    for (int64_t q0 = 0; q0 < nq; q0 += sb) {
        const int64_t n = sb < nq - q0 ? sb : nq - q0;
        const float *dq, *dwz;
        const ifvs_predicate* dp;
        TRY(stage_inputs(ix, s, o, q0, n, queries, preds, wz, &dq, &dp, &dwz));
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_PREDICATE);
            CUDA_TRY(st.end(launch_canonicalize(dp, n, ix->cols(), ix->w_canon.as<CanonPred>(),
                                                ix->w_err.as<int>(), s)));
        }
        if (!cond) {
            CUDA_TRY(cudaMemsetAsync(ix->w_idx.p, 0, sizeof(uint32_t) * n * (ix->h > 0 ? ix->h : 1), s));
            CUDA_TRY(cudaMemsetAsync(ix->w_alpha.p, 0, sizeof(float) * n * (Mr > 0 ? Mr : 1), s));
        }
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_CONDITION);
            CUDA_TRY(st.end(launch_condition(dq, dp, n, ix->D, ix->d_seeds, ix->h, ix->B,
                                             cond ? ix->d_bank : nullptr, Mr, dwz,
                                             ix->w_idx.as<uint32_t>(), ix->w_alpha.as<float>(),
                                             ix->w_wf.as<float>(), s)));
        }
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_LUT);
            CUDA_TRY(st.end(launch_lut(ix->d_cpq, ix->d_W, cond ? ix->w_alpha.as<float>() : nullptr, dq,
                                       ix->w_wf.as<float>(), n, ix->M, ix->K, ix->ds, ix->r,
                                       ix->w_lut.as<float>(), C_ifvs ? ix->w_cifvs.as<float>() : nullptr,
                                       ix->num_sms, s)));
        }
        if (bank_idx && ix->h > 0)
            TRY(copy_out(s, o.dio, bank_idx + q0 * ix->h, ix->w_idx.p, sizeof(uint32_t) * n * ix->h));
        if (alpha && Mr > 0) TRY(copy_out(s, o.dio, alpha + q0 * Mr, ix->w_alpha.p, sizeof(float) * n * Mr));
        if (wf) TRY(copy_out(s, o.dio, wf + q0 * ix->D, ix->w_wf.p, sizeof(float) * n * ix->D));
        if (lut)
            TRY(copy_out(s, o.dio, lut + q0 * ix->M * ix->K, ix->w_lut.p, sizeof(float) * n * ix->M * ix->K));
        if (C_ifvs)
            TRY(copy_out(s, o.dio, C_ifvs + q0 * ix->M * ix->K * ix->ds, ix->w_cifvs.p,
                         sizeof(float) * n * ix->M * ix->K * ix->ds));
        if (q0 + sb < nq) CUDA_TRY(cudaStreamSynchronize(s));
    }
    return finish(ix, s, true);
}

int ifvs_scan_topk(ifvs_index* ix, const float* lut, const uint32_t* bitmaps, int64_t nq, int32_t k,
                   const ifvs_search_params* p, int64_t* ids, float* dists) {
    TRY(check_index(ix, false));
    Opts o;
    TRY(parse_opts(p, &o));
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (k < 1 || k > IFVS_MAX_K) return set_err(IFVS_ERR_ARG, "k = %d outside 1..%d", k, IFVS_MAX_K);
    TRY(check_scan_fits(ix, k));
    if (nq == 0) return IFVS_OK;
    if (!lut || !bitmaps || !ids || !dists) return set_err(IFVS_ERR_ARG, "an array argument is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const int64_t sb = pick_sub_batch(ix, o, nq);
    const int64_t wrows = (ix->N + 31) / 32;
    const size_t lut_n = (size_t)ix->M * ix->K;
    TRY(ensure(ix->w_bm, (size_t)sb * ix->n_blocks * 128));
    if (!o.dio) {
        TRY(ensure(ix->w_rows, (size_t)sb * wrows * 4));
        TRY(ensure(ix->w_lut, sizeof(float) * sb * lut_n));
        TRY(ensure(ix->w_ids, sizeof(int64_t) * sb * k));
        TRY(ensure(ix->w_dists, sizeof(float) * sb * k));
    }
    for (int64_t q0 = 0; q0 < nq; q0 += sb) {
        const int64_t n = sb < nq - q0 ? sb : nq - q0;
        const float* dl = lut + q0 * lut_n;
        const uint32_t* drows = bitmaps + q0 * wrows;
        if (!o.dio) {
            CUDA_TRY(cudaMemcpyAsync(ix->w_lut.p, dl, sizeof(float) * n * lut_n, cudaMemcpyHostToDevice, s));
            CUDA_TRY(cudaMemcpyAsync(ix->w_rows.p, drows, sizeof(uint32_t) * n * wrows, cudaMemcpyHostToDevice, s));
            dl = ix->w_lut.as<float>();
            drows = ix->w_rows.as<uint32_t>();
        }
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_LAYOUT);
            CUDA_TRY(st.end(launch_bitmap_layout(drows, ix->w_bm.as<uint32_t>(), n, ix->n_blocks, wrows,
                                                 false, s)));
        }
        const ScanShape sh = scan_shape(ix, n, k, o.chunk_blocks);
        TRY(ensure(ix->w_part, sizeof(uint64_t) * n * sh.n_chunks * k));
        TRY(ensure(ix->w_tab, sizeof(float) * n * 256 * ix->tab_words));
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_LUT);
            CUDA_TRY(st.end(launch_tables(dl, n, ix->M, ix->K, ix->tab_words, ix->w_tab.as<float>(), s)));
        }
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_SCAN);
            CUDA_TRY(st.end(launch_scan(ix->d_codes, ix->w_tab.as<float>(), ix->w_bm.as<uint32_t>(), nullptr,
                                        n, k, sh, ix->w_part.as<uint64_t>(), s)));
        }
        int64_t* oid = o.dio ? ids + q0 * k : ix->w_ids.as<int64_t>();
        float* odi = o.dio ? dists + q0 * k : ix->w_dists.as<float>();
        {
            Stage st(ix, s, o.timing, IFVS_STAGE_MERGE);
            CUDA_TRY(st.end(launch_merge(ix->w_part.as<uint64_t>(), n, sh.n_chunks, k, oid, odi, s)));
        }
        if (!o.dio) {
            TRY(copy_out(s, false, ids + q0 * k, oid, sizeof(int64_t) * n * k));
            TRY(copy_out(s, false, dists + q0 * k, odi, sizeof(float) * n * k));
            CUDA_TRY(cudaStreamSynchronize(s));
        }
    }
    return finish(ix, s, false);
}

int ifvs_rerank(ifvs_index* ix, const float* queries, const int64_t* cand, int64_t nq, int32_t R,
                int32_t k, const ifvs_search_params* p, int64_t* ids, float* dists) {
    TRY(check_index(ix, false));
    Opts o;
    TRY(parse_opts(p, &o));
    if (!ix->d_vec) return set_err(IFVS_ERR_STATE, "rerank needs raw vectors at load time");
    if (ix->D <= 0) return set_err(IFVS_ERR_STATE, "vector dimension unknown");
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (R < 1 || R > IFVS_MAX_K) return set_err(IFVS_ERR_ARG, "R = %d outside 1..%d", R, IFVS_MAX_K);
    if (k < 1 || k > R) return set_err(IFVS_ERR_ARG, "k = %d outside 1..R", k);
    if (nq == 0) return IFVS_OK;
    if (!queries || !cand || !ids || !dists) return set_err(IFVS_ERR_ARG, "an array argument is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const float* dq = queries;
    const int64_t* dc = cand;
    int64_t* oid = ids;
    float* odi = dists;
    if (!o.dio) {
        TRY(ensure(ix->w_q, sizeof(float) * nq * ix->D));
        TRY(ensure(ix->w_cand, sizeof(int64_t) * nq * R));
        TRY(ensure(ix->w_ids, sizeof(int64_t) * nq * k));
        TRY(ensure(ix->w_dists, sizeof(float) * nq * k));
        CUDA_TRY(cudaMemcpyAsync(ix->w_q.p, queries, sizeof(float) * nq * ix->D, cudaMemcpyHostToDevice, s));
        CUDA_TRY(cudaMemcpyAsync(ix->w_cand.p, cand, sizeof(int64_t) * nq * R, cudaMemcpyHostToDevice, s));
        dq = ix->w_q.as<float>();
        dc = ix->w_cand.as<int64_t>();
        oid = ix->w_ids.as<int64_t>();
        odi = ix->w_dists.as<float>();
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_RERANK);
        CUDA_TRY(st.end(launch_rerank(ix->d_vec, ix->N, ix->D, dq, dc, nq, R, k, oid, odi, s)));
    }
    if (!o.dio) {
        TRY(copy_out(s, false, ids, oid, sizeof(int64_t) * nq * k));
        TRY(copy_out(s, false, dists, odi, sizeof(float) * nq * k));
    }
    return finish(ix, s, false);
}

// ---- PQ construction ----------------------------------------------------------

namespace {

struct PqArgs {
    int device = 0, num_sms = 0;
    cudaStream_t s = nullptr;
    bool own_stream = false;
    std::vector<void*> owned;
    ~PqArgs() {
        if (s && (own_stream || !owned.empty())) cudaStreamSynchronize(s);
        for (void* p : owned) cudaFree(p);
        if (s && own_stream) cudaStreamDestroy(s);
    }
    int alloc(void** p, size_t bytes) {
        cudaError_t e = device_malloc(p, bytes ? bytes : 16);
        if (e != cudaSuccess) {
            cudaGetLastError();
            *p = nullptr;
            return set_err(IFVS_ERR_OOM, "device allocation of %zu bytes failed: %s", bytes, cudaGetErrorString(e));
        }
        owned.push_back(*p);
        return 0;
    }
    // device copy of a host input (or the pointer itself with device I/O)
    int input(const void* host, size_t bytes, bool dio, const void** out) {
        if (dio) {
            *out = host;
            return 0;
        }
        void* p = nullptr;
        TRY(alloc(&p, bytes));
        CUDA_TRY(cudaMemcpyAsync(p, host, bytes, cudaMemcpyHostToDevice, s));
        *out = p;
        return 0;
    }
};

int pq_check(int32_t device, const float* X, int64_t n, int32_t D, int32_t M, int32_t K,
             uint32_t flags, void* stream, PqArgs* a) {
    if (n < 0) return set_err(IFVS_ERR_ARG, "n < 0");
    if (n > 0 && !X) return set_err(IFVS_ERR_ARG, "X is NULL");
    if (n > (int64_t)0xFFFFFFFFLL) return set_err(IFVS_ERR_ARG, "n = %lld above 2^32 - 1", (long long)n);
    if (M < 1 || D < M || D % M != 0) return set_err(IFVS_ERR_ARG, "D = %d must be a positive multiple of M = %d", D, M);
    if (K < 1 || K > 256) return set_err(IFVS_ERR_UNSUPPORTED, "K = %d outside 1..256", K);
    if ((size_t)K * (D / M) * sizeof(double) + (size_t)K * 8 > 200 * 1024)
        return set_err(IFVS_ERR_UNSUPPORTED, "K x ds too large for the shared-memory codebook");
    if (flags & ~IFVS_F_DEVICE_IO) return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", flags);
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
        cudaGetLastError();
        return set_err(IFVS_ERR_CUDA, "no CUDA device is available");
    }
    if (device < 0 || device >= ndev) return set_err(IFVS_ERR_ARG, "device %d outside 0..%d", device, ndev - 1);
    a->device = device;
    CUDA_TRY(cudaDeviceGetAttribute(&a->num_sms, cudaDevAttrMultiProcessorCount, device));
    if (stream) {
        a->s = (cudaStream_t)stream;
    } else {
        // blocking: ordered after the caller's work on the legacy default stream
        CUDA_TRY(cudaStreamCreateWithFlags(&a->s, cudaStreamDefault));
        a->own_stream = true;
    }
    return 0;
}

}  // namespace

extern "C" int ifvs_merge_topk(int32_t device, const float* dists, const int64_t* ids, int64_t nq, int32_t G,
                               int32_t k, float* dists_out, int64_t* ids_out, uint32_t flags, void* stream) {
    if (nq < 0) return set_err(IFVS_ERR_ARG, "nq < 0");
    if (G < 1) return set_err(IFVS_ERR_ARG, "G = %d < 1", G);
    if (k < 1 || k > IFVS_MAX_K) return set_err(IFVS_ERR_ARG, "k = %d outside 1..%d", k, IFVS_MAX_K);
    if ((int64_t)G * k > shard_merge_cap())
        return set_err(IFVS_ERR_UNSUPPORTED, "G x k = %lld above %d", (long long)G * k, shard_merge_cap());
    if (flags & ~IFVS_F_DEVICE_IO) return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", flags);
    if (nq == 0) return IFVS_OK;
    if (!dists || !ids || !dists_out || !ids_out) return set_err(IFVS_ERR_ARG, "an array argument is NULL");
    int ndev = 0;
    if (cudaGetDeviceCount(&ndev) != cudaSuccess || ndev == 0) {
        cudaGetLastError();
        return set_err(IFVS_ERR_CUDA, "no CUDA device is available");
    }
    if (device < 0 || device >= ndev) return set_err(IFVS_ERR_ARG, "device %d outside 0..%d", device, ndev - 1);
    DeviceGuard g(device);
    PqArgs a;
    a.device = device;
    if (stream) {
        a.s = (cudaStream_t)stream;
    } else {
        CUDA_TRY(cudaStreamCreateWithFlags(&a.s, cudaStreamDefault));
        a.own_stream = true;
    }
    const bool dio = flags & IFVS_F_DEVICE_IO;
    const size_t n_in = (size_t)G * nq * k, n_out = (size_t)nq * k;
    const void *dd, *di;
    TRY(a.input(dists, sizeof(float) * n_in, dio, &dd));
    TRY(a.input(ids, sizeof(int64_t) * n_in, dio, &di));
    float* od = dists_out;
    int64_t* oi = ids_out;
    if (!dio) {
        void* p;
        TRY(a.alloc(&p, sizeof(float) * n_out));
        od = (float*)p;
        TRY(a.alloc(&p, sizeof(int64_t) * n_out));
        oi = (int64_t*)p;
    }
    CUDA_TRY(launch_merge_shards((const float*)dd, (const int64_t*)di, nq, G, k, od, oi, a.s));
    if (!dio) {
        CUDA_TRY(cudaMemcpyAsync(dists_out, od, sizeof(float) * n_out, cudaMemcpyDeviceToHost, a.s));
        CUDA_TRY(cudaMemcpyAsync(ids_out, oi, sizeof(int64_t) * n_out, cudaMemcpyDeviceToHost, a.s));
    }
    if (a.own_stream || !dio) CUDA_TRY(cudaStreamSynchronize(a.s));
    return IFVS_OK;
}

extern "C" int ifvs_pq_encode(int32_t device, const float* X, int64_t n, int32_t D, int32_t M,
                              int32_t K, const float* C_pq, uint8_t* codes, float* dmin,
                              uint32_t flags, void* stream) {
    if (!C_pq || (n > 0 && !codes)) return set_err(IFVS_ERR_ARG, "C_pq / codes is NULL");
    DeviceGuard g(device);
    PqArgs a;
    TRY(pq_check(device, X, n, D, M, K, flags, stream, &a));
    if (n == 0) return IFVS_OK;
    const bool dio = flags & IFVS_F_DEVICE_IO;
    const int ds = D / M;
    const void *dX, *dC;
    TRY(a.input(X, sizeof(float) * n * D, dio, &dX));
    TRY(a.input(C_pq, sizeof(float) * M * K * ds, dio, &dC));
    uint8_t* dcodes = codes;
    float* ddmin = dmin;
    if (!dio) {
        void* p;
        TRY(a.alloc(&p, (size_t)n * M));
        dcodes = (uint8_t*)p;
        ddmin = nullptr;
        if (dmin) {
            TRY(a.alloc(&p, sizeof(float) * n * M));
            ddmin = (float*)p;
        }
    }
    CUDA_TRY(launch_pq_assign((const float*)dX, n, D, M, K, (const float*)dC, dcodes, ddmin, a.s));
    if (!dio) {
        CUDA_TRY(cudaMemcpyAsync(codes, dcodes, (size_t)n * M, cudaMemcpyDeviceToHost, a.s));
        if (dmin) CUDA_TRY(cudaMemcpyAsync(dmin, ddmin, sizeof(float) * n * M, cudaMemcpyDeviceToHost, a.s));
    }
    if (a.own_stream || !dio) CUDA_TRY(cudaStreamSynchronize(a.s));
    return IFVS_OK;
}

extern "C" int ifvs_pq_train(int32_t device, const float* X, int64_t n, int32_t D, int32_t M,
                             int32_t K, int32_t iters, const float* C_init, float* C_out,
                             double* objective, uint32_t flags, void* stream) {
    if (!C_init || !C_out) return set_err(IFVS_ERR_ARG, "C_init / C_out is NULL");
    if (iters < 0) return set_err(IFVS_ERR_ARG, "iters < 0");
    DeviceGuard g(device);
    PqArgs a;
    TRY(pq_check(device, X, n, D, M, K, flags, stream, &a));
    const bool dio = flags & IFVS_F_DEVICE_IO;
    const int ds = D / M;
    const size_t cb_bytes = sizeof(float) * (size_t)M * K * ds;
    const void *dX = nullptr, *dC0;
    if (n > 0) TRY(a.input(X, sizeof(float) * n * D, dio, &dX));
    TRY(a.input(C_init, cb_bytes, dio, &dC0));
    void *cA, *cB, *codes, *dmin, *sums, *counts, *best, *obj;
    TRY(a.alloc(&cA, cb_bytes));
    TRY(a.alloc(&cB, cb_bytes));
    TRY(a.alloc(&codes, (size_t)(n > 0 ? n : 1) * M));
    TRY(a.alloc(&dmin, sizeof(float) * (size_t)(n > 0 ? n : 1) * M));
    TRY(a.alloc(&sums, sizeof(double) * (size_t)M * K * ds));
    TRY(a.alloc(&counts, sizeof(unsigned long long) * (size_t)M * K));
    TRY(a.alloc(&best, sizeof(unsigned long long)));
    TRY(a.alloc(&obj, sizeof(double) * M));
    CUDA_TRY(cudaMemcpyAsync(cA, dC0, cb_bytes, cudaMemcpyDeviceToDevice, a.s));
    std::vector<unsigned long long> cnt((size_t)M * K);
    for (int it = 0; it < iters && n > 0; ++it) {
        CUDA_TRY(launch_pq_assign((const float*)dX, n, D, M, K, (const float*)cA, (uint8_t*)codes,
                                  (float*)dmin, a.s));
        if (objective) {
            CUDA_TRY(launch_pq_objective((const float*)dmin, n, M, (double*)obj, a.num_sms, a.s));
            CUDA_TRY(cudaMemcpyAsync(objective + (size_t)it * M, obj, sizeof(double) * M,
                                     dio ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, a.s));
        }
        CUDA_TRY(launch_pq_update((const float*)dX, n, D, M, K, (const uint8_t*)codes, (double*)sums,
                                  (unsigned long long*)counts, (const float*)cA, (float*)cB,
                                  a.num_sms, a.s));
        CUDA_TRY(cudaMemcpyAsync(cnt.data(), counts, sizeof(unsigned long long) * cnt.size(),
                                 cudaMemcpyDeviceToHost, a.s));
        CUDA_TRY(cudaStreamSynchronize(a.s));
        for (int m = 0; m < M; ++m)
            for (int c = 0; c < K; ++c)
                if (cnt[(size_t)m * K + c] == 0)
                    CUDA_TRY(launch_pq_reseed((const float*)dX, n, D, M, K, m, c,
                                              (unsigned long long*)best, (float*)cB, (float*)dmin,
                                              a.num_sms, a.s));
        std::swap(cA, cB);
    }
    CUDA_TRY(cudaMemcpyAsync(C_out, cA, cb_bytes, dio ? cudaMemcpyDeviceToDevice : cudaMemcpyDeviceToHost, a.s));
    CUDA_TRY(cudaStreamSynchronize(a.s));
    return IFVS_OK;
}

int ifvs_train_grad(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                    const float* wz, const int64_t* cand, const ifvs_train_params* tp, float* g_bank,
                    float* g_W, float* g_wz, double* loss) {
    Opts o;
    TRY(train_check(ix, tp, nq, false, &o));
    if (nq == 0) {
        if (loss) *loss = 0.0;
        return IFVS_OK;
    }
    if (!queries || !preds || !wz || !cand) return set_err(IFVS_ERR_ARG, "an input array is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const int V = tp->n_pos + tp->n_neg;
    const int64_t Mr = (int64_t)ix->M * ix->r;
    TRY(reset_err_flag(ix, s));
    const float* dq;
    const ifvs_predicate* dp;
    TRY(train_stage(ix, s, o, nq, queries, preds, wz, &dq, &dp));
    TRY(train_buffers(ix, nq, V));
    const int64_t* dcand = cand;
    if (!o.dio) {
        TRY(ensure(ix->t_cand, sizeof(int64_t) * nq * V));
        CUDA_TRY(cudaMemcpyAsync(ix->t_cand.p, cand, sizeof(int64_t) * nq * V, cudaMemcpyHostToDevice, s));
        dcand = ix->t_cand.as<int64_t>();
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_CONDITION);
        CUDA_TRY(st.end(launch_condition(dq, dp, nq, ix->D, ix->d_seeds, ix->h, ix->B, ix->d_bank,
                                         (int)Mr, ix->w_wz.as<float>(), ix->w_idx.as<uint32_t>(),
                                         ix->w_alpha.as<float>(), ix->w_wf.as<float>(), s)));
    }
    TrainQueryArgs a = train_args(ix, tp, nq, dq);
    a.pos = dcand;
    a.pos_stride = V;
    a.negsrc = dcand + tp->n_pos;
    a.neg_stride = V;
    a.S = tp->n_neg;
    a.exclude = 0;
    TRY(train_gradient(ix, s, o, a));
    const size_t nW = sizeof(float) * (size_t)ix->M * ix->r * ix->K * ix->ds;
    if (g_bank) TRY(copy_out(s, o.dio, g_bank, ix->t_gbank.p, sizeof(float) * ix->B * Mr));
    if (g_W) TRY(copy_out(s, o.dio, g_W, ix->t_gW.p, nW));
    if (g_wz) TRY(copy_out(s, o.dio, g_wz, ix->t_gwz.p, sizeof(float) * ix->D));
    TRY(train_loss_out(ix, s, nq, loss));
    return finish(ix, s, true);
}

int ifvs_train_step(ifvs_index* ix, const float* queries, const ifvs_predicate* preds, int64_t nq,
                    float* wz, const int64_t* positives, const ifvs_train_params* tp,
                    int64_t* negatives, double* loss) {
    Opts o;
    TRY(train_check(ix, tp, nq, true, &o));
    if (nq == 0) {
        if (loss) *loss = 0.0;
        return IFVS_OK;
    }
    if (!queries || !preds || !wz || (tp->n_pos > 0 && !positives))
        return set_err(IFVS_ERR_ARG, "an input array is NULL");
    DeviceGuard g(ix->device);
    cudaStream_t s = o.stream ? o.stream : ix->stream;
    const int P = tp->n_pos, kk = tp->n_pos + tp->n_neg;
    const int64_t Mr = (int64_t)ix->M * ix->r;
    TRY(reset_err_flag(ix, s));
    const float* dq;
    const ifvs_predicate* dp;
    TRY(train_stage(ix, s, o, nq, queries, preds, wz, &dq, &dp));
    TRY(train_buffers(ix, nq, kk));
    const int64_t* dpos = positives;
    if (!o.dio && P > 0) {
        TRY(ensure(ix->t_pos, sizeof(int64_t) * nq * P));
        CUDA_TRY(cudaMemcpyAsync(ix->t_pos.p, positives, sizeof(int64_t) * nq * P, cudaMemcpyHostToDevice, s));
        dpos = ix->t_pos.as<int64_t>();
    }
    // hard negatives: the query path with the current bank, W and w_z, top n_pos + n_neg
    TRY(ensure(ix->t_mined, sizeof(int64_t) * nq * kk));
    TRY(ensure(ix->t_mdist, sizeof(float) * nq * kk));
    TRY(ensure(ix->w_npass, sizeof(unsigned long long) * nq));
    Opts mo = o;
    mo.dio = true;
    mo.plain = false;
    mo.R = 0;
    mo.sub_batch = 0;
    mo.chunk_blocks = 0;
    TRY(run_path(ix, s, mo, dq, dp, ix->w_wz.as<float>(), nq, kk, ix->t_mined.as<int64_t>(),
                 ix->t_mdist.as<float>(), ix->w_npass.as<unsigned long long>()));
    TRY(ensure(ix->t_neg, sizeof(int64_t) * nq * (tp->n_neg > 0 ? tp->n_neg : 1)));
    TrainQueryArgs a = train_args(ix, tp, nq, dq);
    a.pos = dpos;
    a.pos_stride = P;
    a.negsrc = ix->t_mined.as<int64_t>();
    a.neg_stride = kk;
    a.S = kk;
    a.exclude = 1;
    a.neg_out = ix->t_neg.as<int64_t>();
    TRY(train_gradient(ix, s, o, a));
    // plain SGD on the bank, W and the shared w_z
    const int64_t nW = (int64_t)ix->M * ix->r * ix->K * ix->ds;
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_sgd(ix->d_bank, ix->t_gbank.as<float>(), ix->B * Mr, tp->lr, s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_sgd(ix->d_W, ix->t_gW.as<float>(), nW, tp->lr, s)));
    }
    {
        Stage st(ix, s, o.timing, IFVS_STAGE_TRAIN);
        CUDA_TRY(st.end(launch_sgd(ix->t_wz.as<float>(), ix->t_gwz.as<float>(), ix->D, tp->lr_wz, s)));
    }
    TRY(copy_out(s, o.dio, wz, ix->t_wz.p, sizeof(float) * ix->D));
    if (negatives && tp->n_neg > 0)
        TRY(copy_out(s, o.dio, negatives, ix->t_neg.p, sizeof(int64_t) * nq * tp->n_neg));
    TRY(train_loss_out(ix, s, nq, loss));
    return finish(ix, s, true);
}

int ifvs_get_conditioning(ifvs_index* ix, float* bank, float* W, uint32_t flags) {
    TRY(check_index(ix, true));
    if (!ix->d_bank) return set_err(IFVS_ERR_STATE, "the index has no memory bank");
    if (flags & ~IFVS_F_DEVICE_IO) return set_err(IFVS_ERR_ARG, "unknown flag bits 0x%x", flags);
    const bool dio = flags & IFVS_F_DEVICE_IO;
    DeviceGuard g(ix->device);
    cudaStream_t s = ix->stream;
    const size_t nW = sizeof(float) * (size_t)ix->M * ix->r * ix->K * ix->ds;
    if (bank) TRY(copy_out(s, dio, bank, ix->d_bank, sizeof(float) * ix->B * ix->M * ix->r));
    if (W) TRY(copy_out(s, dio, W, ix->d_W, nW));
    CUDA_TRY(cudaStreamSynchronize(s));
    return IFVS_OK;
}

int ifvs_stage_times(ifvs_index* ix, double* ms, int64_t* launches, int32_t reset) {
    TRY(check_index(ix, false));
    for (int i = 0; i < IFVS_N_STAGES; ++i) {
        if (ms) ms[i] = ix->stage_ms[i];
        if (launches) launches[i] = ix->stage_launches[i];
        if (reset) {
            ix->stage_ms[i] = 0.0;
            ix->stage_launches[i] = 0;
        }
    }
    return IFVS_OK;
}

int ifvs_index_info(const ifvs_index* ix, int64_t* out) {
    if (!ix || !out) return set_err(IFVS_ERR_ARG, "NULL argument");
    out[0] = ix->N;
    out[1] = ix->M;
    out[2] = ix->K;
    out[3] = ix->D;
    out[4] = ix->ds;
    out[5] = ix->n_attrs;
    out[6] = ix->has_cb ? 1 : 0;
    out[7] = (int64_t)ix->bytes;
    return IFVS_OK;
}

void ifvs_free(ifvs_index* ix) { free_index(ix); }

}  // extern "C"
