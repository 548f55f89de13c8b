// ifvs_scan_topk_static: the Rank + Select launches of ifvs_scan_topk with
// their scratch memory in a file-scope device array instead of memory the
// library allocates, for callers that must not allocate device memory while
// they serve queries: code whose device memory is owned by another
// allocator (a framework's caching pool), and latency-critical loops that
// allocate nothing after start-up, because cudaMalloc / cudaFree may
// synchronise the whole device.
//
// The array below is part of the library's device image: every GPU on which
// the library's kernels are loaded holds IFVS_STATIC_SCRATCH_BYTES of it
// until the process exits.  Host code must not pass `g_scan_scratch` itself
// to a kernel (on the host that name is only a stand-in for the symbol);
// its device address comes from cudaGetSymbolAddress with the index's
// device current.  Every call repeats that host-side lookup instead of
// caching it, so a context that was torn down and created again
// (cudaDeviceReset) never leaves a stale address behind; the first call on
// a device also loads the library's module there.
//
// Every call reuses the same array and leaves the last call's contents in
// it.  Within one call every scratch byte is written before it is read (the
// lane-major bitmaps by the layout kernel, the per-CTA lists by the scan),
// so nothing needs clearing; two calls whose work overlaps on the GPU (on
// different streams, or from different threads without ordering) race on
// the array.
#include "internal.cuh"

namespace ifvs {
namespace {

constexpr size_t kScratchBytes = (size_t)IFVS_STATIC_SCRATCH_BYTES;
__device__ __align__(256) unsigned char g_scan_scratch[kScratchBytes];

// Device address of g_scan_scratch on the current device.
int scratch_address(unsigned char** out) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_scan_scratch);
    if (e != cudaSuccess || p == nullptr) {
        cudaGetLastError();
        return report_error(IFVS_ERR_CUDA, "cudaGetSymbolAddress(scratch) failed: %s",
                            cudaGetErrorString(e));
    }
    *out = static_cast<unsigned char*>(p);
    return 0;
}

// Chunks per query for n queries: the allocating path's rule (about two
// waves of CTAs from the queries alone, chunks of at most 65 536 blocks, at
// least 16 blocks per chunk, at most 32768 keys per query for the merge).
int64_t chunks_for(const IndexView& v, int64_t n, int k) {
    const int64_t resident = (int64_t)v.num_sms * scan_ctas_per_sm(v.tab_words, scan_kp(k));
    int64_t c = (resident * 2 + n - 1) / n;
    const int64_t by_rows = (v.n_blocks + 65535) / 65536;
    if (c < by_rows) c = by_rows;
    int64_t cap = v.n_blocks / 16;
    if (cap < 1) cap = 1;
    if (cap > 32768 / k) cap = 32768 / k > 0 ? 32768 / k : 1;
    if (cap > 65535) cap = 65535;
    if (c > cap) c = cap;
    if (c < 1) c = 1;
    return c;
}

size_t footprint(const IndexView& v, int64_t n, int64_t chunks, int k) {
    const size_t bm = (size_t)n * v.n_blocks * 128;
    const size_t tab = (size_t)n * 256 * v.tab_words * sizeof(float);
    return bm + tab + (size_t)n * chunks * k * sizeof(uint64_t);
}

}  // namespace
}  // namespace ifvs

using namespace ifvs;

extern "C" int ifvs_scan_topk_static(ifvs_index* ix, const float* lut, const uint32_t* bitmaps,
                                     int64_t nq, int32_t k, void* stream, int64_t* ids,
                                     float* dists) {
    IndexView v;
    int rc = index_view(ix, &v);
    if (rc != 0) return rc;
    if (nq < 0) return report_error(IFVS_ERR_ARG, "nq < 0");
    if (k < 1 || k > IFVS_MAX_K) return report_error(IFVS_ERR_ARG, "k = %d outside 1..%d", k, IFVS_MAX_K);
    // the scan CTA's shared memory for this k and table stride, as in ifvs_scan_topk
    if (scan_smem_bytes(v.tab_words, scan_kp(k)) > (size_t)v.max_smem)
        return report_error(IFVS_ERR_UNSUPPORTED,
                            "k = %d with M = %d needs %zu bytes of shared memory per CTA (device: %d)",
                            k, v.M, scan_smem_bytes(v.tab_words, scan_kp(k)), v.max_smem);
    if (nq == 0) return IFVS_OK;
    if (!lut || !bitmaps || !ids || !dists) return report_error(IFVS_ERR_ARG, "an array argument is NULL");
    // one query must fit: its lane-major bitmap, its table and one list of k keys
    if (footprint(v, 1, 1, k) > kScratchBytes)
        return report_error(IFVS_ERR_UNSUPPORTED,
                            "N = %lld needs %zu bytes of scratch per query; the static scratch "
                            "holds %zu (IFVS_STATIC_SCRATCH_BYTES)",
                            (long long)v.N, footprint(v, 1, 1, k), kScratchBytes);
    int prev = -1;
    if (cudaGetDevice(&prev) != cudaSuccess) prev = -1;
    if (prev != v.device && cudaSetDevice(v.device) != cudaSuccess) {
        cudaGetLastError();
        return report_error(IFVS_ERR_CUDA, "cudaSetDevice(%d) failed", v.device);
    }
    cudaStream_t s = static_cast<cudaStream_t>(stream);
    unsigned char* base = nullptr;
    rc = scratch_address(&base);
    const int64_t wrows = (v.N + 31) / 32;
    const size_t lut_n = (size_t)v.M * v.K;
    // largest sub-batch (halving from nq) whose bitmaps, tables and lists fit
    // the scratch with the allocating path's chunk split
    int64_t sb = nq;
    while (rc == 0 && sb > 1 && footprint(v, sb, chunks_for(v, sb, k), k) > kScratchBytes) sb = (sb + 1) / 2;
    for (int64_t q0 = 0; rc == 0 && q0 < nq; q0 += sb) {
        const int64_t n = sb < nq - q0 ? sb : nq - q0;
        // where even one query's lists with that split overflow, use fewer
        // chunks (one chunk always fits: checked above)
        int64_t chunks = chunks_for(v, n, k);
        while (chunks > 1 && footprint(v, n, chunks, k) > kScratchBytes) chunks = (chunks + 1) / 2;
        uint32_t* bm = reinterpret_cast<uint32_t*>(base);
        float* tab = reinterpret_cast<float*>(base + (size_t)n * v.n_blocks * 128);
        uint64_t* part = reinterpret_cast<uint64_t*>(base + (size_t)n * v.n_blocks * 128 +
                                                     (size_t)n * 256 * v.tab_words * sizeof(float));
        ScanShape sh;
        sh.n_blocks = v.n_blocks;
        sh.n_rows = v.N;
        sh.M = v.M;
        sh.K = v.K;
        sh.row_bytes = v.row_bytes;
        sh.tab_words = v.tab_words;
        sh.blocks_per_chunk = (v.n_blocks + chunks - 1) / chunks;
        sh.n_chunks = (int)((v.n_blocks + sh.blocks_per_chunk - 1) / sh.blocks_per_chunk);
        cudaError_t e = launch_bitmap_layout(bitmaps + q0 * wrows, bm, n, v.n_blocks, wrows, false, s);
        if (e == cudaSuccess) e = launch_tables(lut + q0 * lut_n, n, v.M, v.K, v.tab_words, tab, s);
        if (e == cudaSuccess) e = launch_scan(v.codes, tab, bm, nullptr, n, k, sh, part, s);
        if (e == cudaSuccess) e = launch_merge(part, n, sh.n_chunks, k, ids + q0 * k, dists + q0 * k, s);
        if (e != cudaSuccess) {
            cudaGetLastError();
            rc = report_error(IFVS_ERR_CUDA, "ifvs_scan_topk_static launch failed: %s", cudaGetErrorString(e));
        }
    }
    if (prev >= 0 && prev != v.device) cudaSetDevice(prev);
    return rc == 0 ? IFVS_OK : rc;
}
