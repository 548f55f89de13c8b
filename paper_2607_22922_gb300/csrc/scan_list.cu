// Rank (§2 stage 2) over a one-column predicate's pool read as a position
// range of that column's sorted copy of the codes: the one-query kernel
// k_scan_list, and the launcher that first pairs overlapping ranges for the
// two-query kernel (scan_pair.cu).  Design notes in scan_common.cuh.
#include "scan_common.cuh"

namespace ifvs {

// ---- sorted-copy scan ---------------------------------------------------
//
// For a query of the list path (ScanPlan) the pool is the position range
// [a, b) of one column's sorted copy of the codes, whose position p holds
// row rows[p]'s codes rotated by (p mod 32) mod M.  CTA (query, chunk) walks
// the chunk's 1024-position blocks that meet [a, b) exactly as the bitmap
// path walks dense blocks: lane l takes the positions = l (mod 32), so its
// look-ups hit banks (l + s) mod 32 and the code loads are coalesced; blocks
// cut by a or b mask their positions.  No bitmap, no per-row bit handling,
// and the CTAs of one chunk share its codes in L2.  The row id, needed for
// the key, is loaded only for positions whose distance can enter the top-k.
// The sum order (the subspaces from (p mod 32) mod M on) differs from the
// bitmap path's, so the two agree to float32 rounding.

size_t scan_list_smem_bytes(int tab_words, int kp) {
    return (size_t)256 * tab_words * 4 + (size_t)kScanWarps * 2 * kp * 8 + 16;
}

template <int KP, int MM, bool FAST>
__device__ __forceinline__ void scan_positions(const uint8_t* __restrict__ codes, const uint32_t* __restrict__ rows,
                                               int64_t a, int64_t b, int64_t blk0, int64_t blk1, int wstride,
                                               const ScanShape& sh, const float* tab, WarpTopK<KP>& tk,
                                               int lane, int warp) {
    const int M = MM > 0 ? MM : sh.M;
    const int S = MM > 0 ? 64 : sh.tab_words;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    const uint32_t tb = 4u * (uint32_t)lane;
    const uint64_t keep = policy_evict_last();
    // positions fit in 32 bits: N < 2^32 - 2048
    const uint32_t a32 = (uint32_t)a, b32 = (uint32_t)b;
    for (int64_t blk = blk0 + warp; blk < blk1; blk += wstride) {
        const uint32_t p0 = (uint32_t)(blk * kBlockRows);
        const bool full = p0 >= a32 && p0 + kBlockRows <= b32;
#pragma unroll 1
        for (int j0 = 0; j0 < 32; j0 += kU) {
            tk.refresh(lane);
            uint32_t pos[kU];
            unsigned valid = 0u;
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                pos[u] = p0 + 32u * (uint32_t)(j0 + u) + (uint32_t)lane;
                valid |= (unsigned)(full || (pos[u] >= a32 && pos[u] < b32)) << u;
            }
            float d[kU];
            if constexpr (MM > 0) {
                uint4 c[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u)
                    c[u] = (valid >> u & 1u) ? ldg_nc_v4(codes + (size_t)pos[u] * 16, keep) : make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int u = 0; u < kU; u += 2) lookup2<MM, FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
            } else {
                lookup_rows<kU>(codes, pos, valid, sh.row_bytes, M, S, tab, lane, d);
            }
            // a position can enter the top-k only if its distance is at most
            // the current k-th one; only those load their row id
            const uint32_t thr_hi = (uint32_t)(tk.thr >> 32);
            bool cand_any = false;
#pragma unroll
            for (int u = 0; u < kU; ++u) cand_any |= (valid >> u & 1u) && __float_as_uint(d[u]) <= thr_hi;
            if (!__any_sync(0xFFFFFFFFu, cand_any)) continue;
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const bool cand = (valid >> u & 1u) && __float_as_uint(d[u]) <= thr_hi;
                const uint32_t row = cand ? __ldg(rows + pos[u]) : 0u;
                const uint64_t key = ((uint64_t)__float_as_uint(d[u]) << 32) | row;
                tk.offer(key, cand && key < tk.thr, lane);
            }
        }
    }
}

template <int KP, int MM, int MINB>
__global__ void __launch_bounds__(kScanThreads, MINB)
k_scan_list(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan, int64_t nq,
            int k, ScanShape sh, uint64_t* __restrict__ partials, const uint8_t* __restrict__ paired) {
    extern __shared__ __align__(256) uint8_t smem[];
    const int S = MM > 0 ? 64 : sh.tab_words;
    float* tab = reinterpret_cast<float*>(smem);
    uint64_t* tkbuf = reinterpret_cast<uint64_t*>(smem + (size_t)256 * S * 4);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t q = blockIdx.x;
    const int chunk = blockIdx.y;
    const ScanPlan p = plan[q];
    if (!p.list) return;                               // k_scan covers this query
    if (paired != nullptr && paired[q]) return;        // k_scan_list_pair covers it
    const int64_t c0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t c1 = min(sh.n_blocks, c0 + sh.blocks_per_chunk);
    const int64_t blk0 = max(c0, p.a / kBlockRows);
    const int64_t blk1 = min(c1, (p.b + kBlockRows - 1) / kBlockRows);
    uint64_t* out = partials + (q * sh.n_chunks + chunk) * (int64_t)k;
    if (p.a >= p.b || blk0 >= blk1) {
        for (int i = threadIdx.x; i < k; i += kScanThreads) out[i] = ~0ull;
        return;
    }
    {
        const float4* src = reinterpret_cast<const float4*>(tables + q * (int64_t)256 * S);
        float4* dst = reinterpret_cast<float4*>(tab);
        for (int i = threadIdx.x; i < 64 * S; i += kScanThreads) dst[i] = __ldg(src + i);
    }
    uint64_t* cta = tkbuf + kScanWarps * 2 * KP;
    if (threadIdx.x == 0) *cta = ~0ull;
    WarpTopK<KP> tk;
    tk.init(tkbuf + warp * 2 * KP, k, lane, cta);
    __syncthreads();
    const uint8_t* codes = sc.codes_of(p.col);
    const uint32_t* rows = sc.rows_of(p.col);
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    if constexpr (MM > 0) {
        if (base == kDynSmemBase)
            scan_positions<KP, MM, true>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
        else
            scan_positions<KP, MM, false>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
    } else {
        scan_positions<KP, 0, false>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
    }
    tk.flush(lane);
#pragma unroll 1
    for (int step = 1; step < kScanWarps; step <<= 1) {
        __syncthreads();
        if ((warp & (2 * step - 1)) == 0) {
            const uint64_t* other = tkbuf + (warp + step) * 2 * KP;
            for (int i = lane; i < k; i += 32) tk.buf[KP + i] = other[i];
            __syncwarp();
            tk.flush(lane);
        }
    }
    if (warp == 0)
        for (int i = lane; i < k; i += 32) out[i] = tk.buf[i];
}

// ---- sorted-copy scan with bulk-copied code tiles (M = 16) ------------------
//
// The walk of k_scan_list with the code rows of every round brought into
// shared memory by the bulk-copy engine (cp.async.bulk, the untiled form of
// TMA) instead of per-lane vector loads.  A warp's round is 256 consecutive
// positions (lane l takes positions 32u + l, u < kU = 8): 4 KB of codes, one
// copy.  Each warp owns a ring of NST such tiles with an mbarrier each; lane
// 0 issues the copy of round r + NST as soon as round r's rows sit in
// registers, so a warp keeps NST rounds of codes in flight while it
// computes, in shared memory rather than in registers.  A warp whose tile
// has not arrived within the bounded wait sets bit 4 of *err (the search
// returns IFVS_ERR_TIMEOUT), waits (bounded again) for its copies still in
// flight, and stops scanning; its CTA still merges and writes its lists.
// tx_extra (0 in normal use) is added to the bytes each barrier expects; a
// positive value makes every wait run out, which exercises that path.
// One tile per warp (NST = 1) keeps two 8-warp CTAs per SM; measured on the
// 10^8-row workload it beat vector loads by 3 % (0.1 % pools) and 7 % (1 %),
// while two or four tiles per warp (one CTA per SM) lost 38 % and 36 %.

#ifndef IFVS_BULK_STAGES
#define IFVS_BULK_STAGES 1
#endif
constexpr int kBulkStages = IFVS_BULK_STAGES;
constexpr uint32_t kTileBytes = 32u * kU * 16u;    // one warp round: 256 positions x 16 bytes
static_assert(32 % kU == 0, "whole rounds per block");
constexpr int kRoundsPerBlock = 32 / kU;

__host__ __device__ constexpr size_t bulk_ring_offset(int kp) {
    return ((size_t)256 * 64 * 4 + (size_t)kScanWarps * 2 * kp * 8 + 16 + 127) / 128 * 128;
}

// tiles, one barrier per tile, and the barrier of the table copy
size_t scan_bulk_smem_bytes(int kp) {
    return bulk_ring_offset(kp) + (size_t)kScanWarps * kBulkStages * (kTileBytes + 8) + 16;
}

template <int KP, int MM, bool FAST>
__device__ __forceinline__ void scan_positions_bulk(const uint8_t* __restrict__ codes,
                                                    const uint32_t* __restrict__ rows, int64_t a, int64_t b,
                                                    int64_t blk0, int64_t blk1, const float* tab, uint8_t* ring,
                                                    uint64_t* bars, uint32_t tx_extra, int* err, WarpTopK<KP>& tk,
                                                    int lane, int warp) {
    constexpr int NST = kBulkStages;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    const uint32_t tb = 4u * (uint32_t)lane;
    const uint64_t keep = policy_evict_last();
    const uint32_t a32 = (uint32_t)a, b32 = (uint32_t)b;   // positions fit in 32 bits
    const int64_t first = blk0 + warp;
    const int nblk = first < blk1 ? (int)((blk1 - first + kScanWarps - 1) / kScanWarps) : 0;
    const int R = kRoundsPerBlock * nblk;
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring);
    const uint32_t bar_s = (uint32_t)__cvta_generic_to_shared(bars);
    // first position of round r of this warp
    auto tile_pos = [&](int r) -> uint32_t {
        return (uint32_t)((first + (int64_t)(r / kRoundsPerBlock) * kScanWarps) * kBlockRows) +
               (uint32_t)(r % kRoundsPerBlock) * (32u * kU);
    };
    auto issue = [&](int r) {
        const uint32_t st = (uint32_t)(r % NST);
        mbar_arrive_expect_tx(bar_s + 8u * st, kTileBytes + tx_extra);
        bulk_g2s(ring_s + st * kTileBytes, codes + (size_t)tile_pos(r) * 16, kTileBytes, bar_s + 8u * st, keep);
    };
    if (lane == 0)
        for (int r = 0; r < NST && r < R; ++r) issue(r);
#pragma unroll 1
    for (int r = 0; r < R; ++r) {
        const int st = r % NST;
        if (!mbar_wait_warp(bar_s + 8u * (uint32_t)st, (uint32_t)(r / NST) & 1u)) {
            if (lane == 0) atomicOr(err, 4);
            // rounds r .. min(R, r + NST) - 1 were issued and not consumed
            for (int q = r; q < R && q < r + NST; ++q)
                mbar_wait_warp(bar_s + 8u * (uint32_t)(q % NST), (uint32_t)(q / NST) & 1u);
            return;
        }
        tk.refresh(lane);
        const uint32_t P = tile_pos(r);
        const uint4* tile = reinterpret_cast<const uint4*>(ring + (size_t)st * kTileBytes);
        uint4 c[kU];
#pragma unroll
        for (int u = 0; u < kU; ++u) c[u] = tile[32 * u + lane];
        __syncwarp();
        if (lane == 0 && r + NST < R) {
            fence_proxy_async_smem();
            issue(r + NST);
        }
        const bool full = P >= a32 && P + 32u * kU <= b32;
        uint32_t pos[kU];
        unsigned valid = 0u;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            pos[u] = P + 32u * (uint32_t)u + (uint32_t)lane;
            valid |= (unsigned)(full || (pos[u] >= a32 && pos[u] < b32)) << u;
        }
        float d[kU];
#pragma unroll
        for (int u = 0; u < kU; u += 2) lookup2<MM, FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
        // as in scan_positions: only candidates load their row id
        const uint32_t thr_hi = (uint32_t)(tk.thr >> 32);
        bool cand_any = false;
#pragma unroll
        for (int u = 0; u < kU; ++u) cand_any |= (valid >> u & 1u) && __float_as_uint(d[u]) <= thr_hi;
        if (!__any_sync(0xFFFFFFFFu, cand_any)) continue;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            const bool cand = (valid >> u & 1u) && __float_as_uint(d[u]) <= thr_hi;
            const uint32_t row = cand ? __ldg(rows + pos[u]) : 0u;
            const uint64_t key = ((uint64_t)__float_as_uint(d[u]) << 32) | row;
            tk.offer(key, cand && key < tk.thr, lane);
        }
    }
}

template <int KP, int MM, int MINB>
__global__ void __launch_bounds__(kScanThreads, MINB)
k_scan_list_bulk(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan, int64_t nq,
                 int k, ScanShape sh, uint64_t* __restrict__ partials, const uint8_t* __restrict__ paired,
                 uint32_t tx_extra, int* __restrict__ err) {
    extern __shared__ __align__(256) uint8_t smem[];
    float* tab = reinterpret_cast<float*>(smem);
    uint64_t* tkbuf = reinterpret_cast<uint64_t*>(smem + (size_t)256 * 64 * 4);
    uint8_t* ring_all = smem + bulk_ring_offset(KP);
    uint64_t* bars_all = reinterpret_cast<uint64_t*>(ring_all + (size_t)kScanWarps * kBulkStages * kTileBytes);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t q = blockIdx.x;
    const int chunk = blockIdx.y;
    const ScanPlan p = plan[q];
    if (!p.list) return;                               // k_scan covers this query
    if (paired != nullptr && paired[q]) return;        // k_scan_list_pair covers it
    const int64_t c0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t c1 = min(sh.n_blocks, c0 + sh.blocks_per_chunk);
    const int64_t blk0 = max(c0, p.a / kBlockRows);
    const int64_t blk1 = min(c1, (p.b + kBlockRows - 1) / kBlockRows);
    uint64_t* out = partials + (q * sh.n_chunks + chunk) * (int64_t)k;
    if (p.a >= p.b || blk0 >= blk1) {
        for (int i = threadIdx.x; i < k; i += kScanThreads) out[i] = ~0ull;
        return;
    }
    uint8_t* ring = ring_all + (size_t)warp * kBulkStages * kTileBytes;
    uint64_t* bars = bars_all + warp * kBulkStages;
    const uint32_t tbar = (uint32_t)__cvta_generic_to_shared(bars_all + kScanWarps * kBulkStages);
    if (lane == 0) {
        for (int i = 0; i < kBulkStages; ++i) mbar_init((uint32_t)__cvta_generic_to_shared(bars + i), 1u);
        if (threadIdx.x == 0) mbar_init(tbar, 1u);
        fence_mbar_init();
    }
    // the query's 64 KB table (rows replicated and rotated, as k_tables
    // wrote it) in one bulk copy, while the lists are set up
    if (threadIdx.x == 0) {
        mbar_arrive_expect_tx(tbar, 256u * 64u * 4u);
        bulk_g2s((uint32_t)__cvta_generic_to_shared(tab), tables + q * (int64_t)256 * 64, 256u * 64u * 4u, tbar,
                 policy_evict_first());
    }
    uint64_t* cta = tkbuf + kScanWarps * 2 * KP;
    if (threadIdx.x == 0) *cta = ~0ull;
    WarpTopK<KP> tk;
    tk.init(tkbuf + warp * 2 * KP, k, lane, cta);
    __syncthreads();
    if (!mbar_wait_warp(tbar, 0u)) {
        if (lane == 0) atomicOr(err, 4);
        mbar_wait_warp(tbar, 0u);   // the copy may still be in flight
        merge_warps<KP, kScanWarps>(tk, tkbuf, k, lane, warp, out);
        return;
    }
    const uint8_t* codes = sc.codes_of(p.col);
    const uint32_t* rows = sc.rows_of(p.col);
    if ((uint32_t)__cvta_generic_to_shared(tab) == kDynSmemBase)
        scan_positions_bulk<KP, MM, true>(codes, rows, p.a, p.b, blk0, blk1, tab, ring, bars, tx_extra, err, tk, lane,
                                      warp);
    else
        scan_positions_bulk<KP, MM, false>(codes, rows, p.a, p.b, blk0, blk1, tab, ring, bars, tx_extra, err, tk, lane,
                                       warp);
    merge_warps<KP, kScanWarps>(tk, tkbuf, k, lane, warp, out);
}

// ---- generic M: one row per lane and round from a bulk-copied tile ---------
//
// For M other than 12 and 16 the code rows are M rounded up to 4 bytes (120
// for gist1m), and per-lane loads of a row's words touch one 32-byte sector
// per lane per word: about one L1 wavefront per row and word, several times
// the look-ups' own shared-memory wavefronts.  Here a warp's round is 32
// consecutive positions (one per lane), 32 x row_bytes contiguous bytes (at
// most 4 KB), brought into the warp's shared tile by one bulk copy; each lane
// then reads its own row's words from shared memory.  A row's entries are
// added for s ascending from its rotated first subspace, as in lookup_rows,
// so the results equal the vector-load kernel's bit for bit.
__host__ __device__ inline size_t bulkg_ring_offset(int tab_words, int kp) {
    return ((size_t)256 * tab_words * 4 + (size_t)kScanWarps * 2 * kp * 8 + 16 + 127) / 128 * 128;
}

size_t scan_bulkg_smem_bytes(int tab_words, int kp, int row_bytes) {
    return bulkg_ring_offset(tab_words, kp) + (size_t)kScanWarps * kBulkStages * (32u * row_bytes + 8) + 16;
}

// code words of a row whose look-ups are unrolled together (gist1m, M = 120:
// 8 words 86.9k queries/s, 4 words 85.8k, 2 words 78.0k)
#ifndef IFVS_BULKG_UNROLL
#define IFVS_BULKG_UNROLL 8
#endif
constexpr int kBulkgUnroll = IFVS_BULKG_UNROLL;

template <int KP>
__device__ __forceinline__ void scan_positions_bulkg(const uint8_t* __restrict__ codes,
                                                     const uint32_t* __restrict__ rows, int64_t a, int64_t b,
                                                     int64_t blk0, int64_t blk1, const ScanShape& sh,
                                                     const float* tab, uint8_t* ring, uint64_t* bars,
                                                     uint32_t tx_extra, int* err, WarpTopK<KP>& tk, int lane,
                                                     int warp) {
    constexpr int NST = kBulkStages;
    const int M = sh.M, S = sh.tab_words, rb = sh.row_bytes, nw = sh.row_bytes / 4;
    const uint32_t tile_bytes = 32u * (uint32_t)rb;
    const uint64_t keep = policy_evict_last();
    const uint32_t a32 = (uint32_t)a, b32 = (uint32_t)b;
    const int64_t first = blk0 + warp;
    const int nblk = first < blk1 ? (int)((blk1 - first + kScanWarps - 1) / kScanWarps) : 0;
    const int R = 32 * nblk;   // one row per lane per round: 32 rounds per block
    const uint32_t ring_s = (uint32_t)__cvta_generic_to_shared(ring);
    const uint32_t bar_s = (uint32_t)__cvta_generic_to_shared(bars);
    auto tile_pos = [&](int r) -> uint32_t {
        return (uint32_t)((first + (int64_t)(r >> 5) * kScanWarps) * kBlockRows) + 32u * (uint32_t)(r & 31);
    };
    auto issue = [&](int r) {
        const uint32_t st = (uint32_t)(r % NST);
        mbar_arrive_expect_tx(bar_s + 8u * st, tile_bytes + tx_extra);
        bulk_g2s(ring_s + st * tile_bytes, codes + (size_t)tile_pos(r) * rb, tile_bytes, bar_s + 8u * st, keep);
    };
    if (lane == 0)
        for (int r = 0; r < NST && r < R; ++r) issue(r);
    const float* tw = tab + lane;
#pragma unroll 1
    for (int r = 0; r < R; ++r) {
        const int st = r % NST;
        if (!mbar_wait_warp(bar_s + 8u * (uint32_t)st, (uint32_t)(r / NST) & 1u)) {
            if (lane == 0) atomicOr(err, 4);
            for (int q = r; q < R && q < r + NST; ++q)
                mbar_wait_warp(bar_s + 8u * (uint32_t)(q % NST), (uint32_t)(q / NST) & 1u);
            return;
        }
        tk.refresh(lane);
        const uint32_t pos = tile_pos(r) + (uint32_t)lane;
        const bool valid = pos >= a32 && pos < b32;
        const uint32_t* row = reinterpret_cast<const uint32_t*>(ring + (size_t)st * tile_bytes) + lane * nw;
        float acc = 0.f;
#pragma unroll kBulkgUnroll
        for (int w = 0; w < nw; ++w) {
            const uint32_t wd = row[w];
#pragma unroll
            for (int bb = 0; bb < 4; ++bb) {
                const int s = 4 * w + bb;
                if (s < M) acc += tw[(int)((wd >> (8 * bb)) & 0xFFu) * S + s];
            }
        }
        __syncwarp();   // every lane has read its row: the tile can be refilled
        if (lane == 0 && r + NST < R) {
            fence_proxy_async_smem();
            issue(r + NST);
        }
        const bool cand = valid && __float_as_uint(acc) <= (uint32_t)(tk.thr >> 32);
        if (!__any_sync(0xFFFFFFFFu, cand)) continue;
        const uint32_t id = cand ? __ldg(rows + pos) : 0u;
        const uint64_t key = ((uint64_t)__float_as_uint(acc) << 32) | id;
        tk.offer(key, cand && key < tk.thr, lane);
    }
}

template <int KP>
__global__ void __launch_bounds__(kScanThreads, 1)
k_scan_list_bulkg(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan, int64_t nq,
                  int k, ScanShape sh, uint64_t* __restrict__ partials, const uint8_t* __restrict__ paired,
                  uint32_t tx_extra, int* __restrict__ err) {
    extern __shared__ __align__(256) uint8_t smem[];
    const int S = sh.tab_words;
    float* tab = reinterpret_cast<float*>(smem);
    uint64_t* tkbuf = reinterpret_cast<uint64_t*>(smem + (size_t)256 * S * 4);
    const uint32_t tile_bytes = 32u * (uint32_t)sh.row_bytes;
    uint8_t* ring_all = smem + bulkg_ring_offset(S, KP);
    uint64_t* bars_all = reinterpret_cast<uint64_t*>(ring_all + (size_t)kScanWarps * kBulkStages * tile_bytes);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t q = blockIdx.x;
    const int chunk = blockIdx.y;
    const ScanPlan p = plan[q];
    if (!p.list) return;
    if (paired != nullptr && paired[q]) return;
    const int64_t c0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t c1 = min(sh.n_blocks, c0 + sh.blocks_per_chunk);
    const int64_t blk0 = max(c0, p.a / kBlockRows);
    const int64_t blk1 = min(c1, (p.b + kBlockRows - 1) / kBlockRows);
    uint64_t* out = partials + (q * sh.n_chunks + chunk) * (int64_t)k;
    if (p.a >= p.b || blk0 >= blk1) {
        for (int i = threadIdx.x; i < k; i += kScanThreads) out[i] = ~0ull;
        return;
    }
    uint8_t* ring = ring_all + (size_t)warp * kBulkStages * tile_bytes;
    uint64_t* bars = bars_all + warp * kBulkStages;
    const uint32_t tbar = (uint32_t)__cvta_generic_to_shared(bars_all + kScanWarps * kBulkStages);
    if (lane == 0) {
        for (int i = 0; i < kBulkStages; ++i) mbar_init((uint32_t)__cvta_generic_to_shared(bars + i), 1u);
        if (threadIdx.x == 0) mbar_init(tbar, 1u);
        fence_mbar_init();
    }
    if (threadIdx.x == 0) {
        const uint32_t tb = 256u * (uint32_t)S * 4u;
        mbar_arrive_expect_tx(tbar, tb);
        bulk_g2s((uint32_t)__cvta_generic_to_shared(tab), tables + q * (int64_t)256 * S, tb, tbar,
                 policy_evict_first());
    }
    uint64_t* cta = tkbuf + kScanWarps * 2 * KP;
    if (threadIdx.x == 0) *cta = ~0ull;
    WarpTopK<KP> tk;
    tk.init(tkbuf + warp * 2 * KP, k, lane, cta);
    __syncthreads();
    if (!mbar_wait_warp(tbar, 0u)) {
        if (lane == 0) atomicOr(err, 4);
        mbar_wait_warp(tbar, 0u);
        merge_warps<KP, kScanWarps>(tk, tkbuf, k, lane, warp, out);
        return;
    }
    scan_positions_bulkg<KP>(sc.codes_of(p.col), sc.rows_of(p.col), p.a, p.b, blk0, blk1, sh, tab, ring, bars,
                             tx_extra, err, tk, lane, warp);
    merge_warps<KP, kScanWarps>(tk, tkbuf, k, lane, warp, out);
}

template <int KP>
static cudaError_t launch_list_bulkg(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                                     const ScanShape& sh, uint64_t* partials, const uint8_t* paired, size_t smem,
                                     uint32_t tx_extra, int* err, cudaStream_t s) {
    cudaError_t e =
        cudaFuncSetAttribute(k_scan_list_bulkg<KP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan_list_bulkg<KP><<<grid, kScanThreads, smem, s>>>(tab, sc, plan, nq, k, sh, partials, paired, tx_extra, err);
    return cudaGetLastError();
}

template <int KP, int MM, int MINB>
static cudaError_t launch_list_bulk(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                                    const ScanShape& sh, uint64_t* partials, const uint8_t* paired, size_t smem,
                                    uint32_t tx_extra, int* err, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(k_scan_list_bulk<KP, MM, MINB>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan_list_bulk<KP, MM, MINB><<<grid, kScanThreads, smem, s>>>(tab, sc, plan, nq, k, sh, partials, paired,
                                                                tx_extra, err);
    return cudaGetLastError();
}

template <int KP, int MM, int MINB>
static cudaError_t launch_list_one(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq,
                                   int k, const ScanShape& sh, uint64_t* partials, const uint8_t* paired,
                                   size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(k_scan_list<KP, MM, MINB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan_list<KP, MM, MINB><<<grid, kScanThreads, smem, s>>>(tab, sc, plan, nq, k, sh, partials, paired);
    return cudaGetLastError();
}

template <int KP>
static cudaError_t launch_list_kp(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq,
                                  int k, const ScanShape& sh, uint64_t* partials, uint8_t* work,
                                  const ListOpts& lo, int* launches, cudaStream_t s) {
    const int mm = fixed_m(sh);
    const uint8_t* paired = nullptr;
    int nl = 0;
    if (mm == 16 && work != nullptr) {
        // M = 16: long, overlapping ranges are paired and served by the
        // two-query kernel; the one-query kernel takes the rest
        const cudaError_t e =
            launch_pairs(tab, sc, plan, nq, k, sh, partials, work, lo.pair_min_rows, s, &paired, &nl);
        if (e != cudaSuccess) return e;
    }
    if (launches) *launches = nl + 1;
    if (mm > 0 && lo.bulk) {
        const size_t smem = scan_bulk_smem_bytes(KP);
        if (smem <= (size_t)max_smem_optin()) {
            const bool two = (size_t)233472 / (smem + 1024) >= 2;
            if (mm == 16)
                return two ? launch_list_bulk<KP, 16, 2>(tab, sc, plan, nq, k, sh, partials, paired, smem,
                                                         lo.tx_extra, lo.err, s)
                           : launch_list_bulk<KP, 16, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem,
                                                         lo.tx_extra, lo.err, s);
            return two ? launch_list_bulk<KP, 12, 2>(tab, sc, plan, nq, k, sh, partials, paired, smem, lo.tx_extra,
                                                     lo.err, s)
                       : launch_list_bulk<KP, 12, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, lo.tx_extra,
                                                     lo.err, s);
        }
    }
    if (mm == 0 && lo.bulk && sh.row_bytes <= 128 && sh.row_bytes % 4 == 0) {
        const size_t smem = scan_bulkg_smem_bytes(sh.tab_words, KP, sh.row_bytes);
        if (smem <= (size_t)max_smem_optin())
            return launch_list_bulkg<KP>(tab, sc, plan, nq, k, sh, partials, paired, smem, lo.tx_extra, lo.err, s);
    }
    const size_t smem = scan_list_smem_bytes(sh.tab_words, KP);
    const bool two = (size_t)233472 / (smem + 1024) >= 2;
    if (mm == 16)
        return two ? launch_list_one<KP, 16, 2>(tab, sc, plan, nq, k, sh, partials, paired, smem, s)
                   : launch_list_one<KP, 16, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
    if (mm == 12)
        return two ? launch_list_one<KP, 12, 2>(tab, sc, plan, nq, k, sh, partials, paired, smem, s)
                   : launch_list_one<KP, 12, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
    return launch_list_one<KP, 0, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
}

cudaError_t launch_scan_list(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                             const ScanShape& sh, uint64_t* partials, uint8_t* work, const ListOpts& lo,
                             cudaStream_t s, int* launches) {
    if (launches) *launches = 0;
    if (nq <= 0) return cudaSuccess;
    switch (scan_kp(k)) {
        case 32: return launch_list_kp<32>(tab, sc, plan, nq, k, sh, partials, work, lo, launches, s);
        case 64: return launch_list_kp<64>(tab, sc, plan, nq, k, sh, partials, work, lo, launches, s);
        case 128: return launch_list_kp<128>(tab, sc, plan, nq, k, sh, partials, work, lo, launches, s);
        default: return launch_list_kp<256>(tab, sc, plan, nq, k, sh, partials, work, lo, launches, s);
    }
}
}  // namespace ifvs
