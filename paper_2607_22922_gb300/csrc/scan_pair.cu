// Rank (§2 stage 2) for two queries per CTA on the sorted copy of the codes
// (M = 16): the pairing kernel k_pair_items and the two-query kernel
// k_scan_list_pair.  Design notes in scan_common.cuh.
#include "scan_common.cuh"

namespace ifvs {

// ---- two queries per CTA on the sorted copy --------------------------------
//
// When k_pair_items (below) pairs two queries on the sorted copy of the same
// column (M = 16), one CTA serves both, and one shared-memory load serves
// both queries' look-ups.  A 64 KB table with the rows, replication and rotation
// of the float32 one holds, in word w of codeword row c, the pair
// qA[w mod 16][c] | qB[w mod 16][c] << 16 of 11-bit quantised entries,
// q[m][c] = floor((LUT[m][c] - lo_m) * inv), lo_m the smallest entry of
// subspace m, inv = 2047 / (the widest subspace's range).  Sixteen entries
// sum to at most 32752, so one integer add accumulates both queries with no
// carry between the halves (and bit 15 of each half stays free for the
// candidate test, pack_bounds), and a row's sum S bounds its float32 distance
// from below (quant_bound).  A row whose S exceeds the bound of its query's
// current k-th key cannot enter that top-k and is dropped; every other row
// gets its exact float32 distance from the query's unreplicated table,
// added in the order of the one-query loop (subspace (p mod 32) mod 16
// first), so the top-k receives the keys the one-query loop would give it.
// Since the dropped rows are decided by integers, the shared-memory traffic
// of the dense loop is half that of two float32 tables.  Blocks that meet
// one query's range only run the same loop with the other query masked.
// 16 warps, one CTA per SM.
constexpr int kPairWarps = 16;
constexpr int kPairThreads = kPairWarps * 32;
constexpr uint32_t kTabBytes16 = 256u * 64u * 4u;    // one replicated M = 16 table
constexpr uint32_t kExactBytes16 = 256u * 16u * 4u;  // one unreplicated table, [c][m]
constexpr int kQMax = 2047;                           // 16 * 2047 < 2^15

// Deferred rescoring.  The rows of a round that pass a query's quantised
// test (about 0.5 % of the rows on the dense bins, but in a third of the
// warps' rounds) are not rescored where they are found, which ran the exact
// sum for one or two lanes of the warp at a time; each warp appends them
// (codes, position, query flags) to a buffer of kCandCap entries in shared
// memory, and every 32 entries the warp rescores them with one entry per
// lane.  The exact sums, the keys and the offers are the same as in place
// (the offers only in another order, which the exact top-k does not see).
// Lists of KP = 256 leave no room for the buffer: they rescore in place.
#ifndef IFVS_PAIR_DEFER
#define IFVS_PAIR_DEFER 1
#endif
constexpr int kCandCap = 64;   // a warp drains at 32: at most 31 + 32 entries are held
constexpr size_t kCandWarpBytes = (size_t)kCandCap * (16 + 4 + 4);

__host__ __device__ constexpr bool pair_defers(int kp) { return IFVS_PAIR_DEFER != 0 && kp <= 128; }

// packed table, two exact tables, extremes + the two shared bounds, lists,
// the candidate buffers, the current work item (no static shared memory:
// it would move the dynamic window off the base the look-ups' immediate
// offsets assume)
size_t scan_pair_smem_bytes(int kp) {
    return (size_t)kTabBytes16 + 2 * (size_t)kExactBytes16 + 64 * 4 + 16 + (size_t)kPairWarps * 2 * 2 * kp * 8 +
           (pair_defers(kp) ? (size_t)kPairWarps * kCandWarpBytes : 0) + 16;
}

template <int IMM>
__device__ __forceinline__ uint32_t lds_u32_imm(uint32_t addr) {
    uint32_t v;
    asm volatile("ld.shared.u32 %0, [%1+%2];" : "=r"(v) : "r"(addr), "n"(IMM));
    return v;
}

__device__ __forceinline__ uint32_t quant12(float L, float lo, float inv) {
    const float y = __fmul_rn(__fsub_rn(L, lo), inv);
    return (uint32_t)fminf((float)kQMax, fmaxf(0.f, y));   // truncation: floor of y >= 0
}

// The largest quantised sum S a row can have and still reach a top-k whose
// k-th key is thr (INT_MAX: every row; -1: none).  With u = 2^-24 and
// entries L >= 0 (so lo_m >= 0): the float32 distance d, sixteen rounded
// additions from 0, is at least (sum_m L_m)(1 - 15u); each q_m is at most
// (L_m - lo_m)(1 + u)^2 inv (two roundings, then floor); so
// S <= (1 + u)^2 inv (d / (1 - 15u) - sum_m lo_m).  At d = dist(thr) the
// bound below is at least that: each of its float32 steps carries a factor
// 1 +- 2^-12 beyond its rounding, and sl, the float32 sum of the lo_m, is at
// most (1 + 15u) sum_m lo_m.  A row with S above it has d > dist(thr).
__device__ __forceinline__ int quant_bound(uint64_t thr, float sl, float inv) {
    const uint32_t hi = (uint32_t)(thr >> 32);
    if (inv == 0.f || hi >= 0x7F800000u) return INT_MAX;   // list not full, inf, NaN or -0
    const float a = __fmul_rn(__uint_as_float(hi), 1.f + 0x1p-12f);
    const float b = __fmul_rn(sl, 1.f - 0x1p-12f);
    const float t = __fmul_rn(__fsub_rn(a, b), __fmul_rn(inv, 1.f + 0x1p-12f));
    if (!(t < 1.0e9f)) return INT_MAX;
    return t < 0.f ? -1 : (int)t;
}

// Quantised sums of two M = 16 rows (codes ca, cb), both queries at once:
// the addresses of lookup2, integer loads and adds.
template <bool FAST>
__device__ __forceinline__ void lookup16x2_q(const uint4 ca, const uint4 cb, uint32_t tb, uint32_t base,
                                             uint32_t& sa, uint32_t& sb) {
    const uint32_t wa[4] = {ca.x, ca.y, ca.z, ca.w};
    const uint32_t wb[4] = {cb.x, cb.y, cb.z, cb.w};
    uint32_t va[16], vb[16];
#pragma unroll
    for (int s = 0; s < 16; ++s) {
        const uint32_t sel = 0x5504u | ((uint32_t)(s & 3) << 4);
        uint32_t oa = __byte_perm(wa[s >> 2], tb, sel);
        uint32_t ob = __byte_perm(wb[s >> 2], tb, sel);
        if (!FAST) {
            oa += base;
            ob += base;
        }
        constexpr uint32_t B0 = FAST ? kDynSmemBase : 0u;
        switch (s) {
#define IFVS_LDQ_CASE(S)                         \
    case S:                                      \
        va[S] = lds_u32_imm<B0 + 4 * S>(oa);     \
        vb[S] = lds_u32_imm<B0 + 4 * S>(ob);     \
        break;
            IFVS_LDQ_CASE(0) IFVS_LDQ_CASE(1) IFVS_LDQ_CASE(2) IFVS_LDQ_CASE(3)
            IFVS_LDQ_CASE(4) IFVS_LDQ_CASE(5) IFVS_LDQ_CASE(6) IFVS_LDQ_CASE(7)
            IFVS_LDQ_CASE(8) IFVS_LDQ_CASE(9) IFVS_LDQ_CASE(10) IFVS_LDQ_CASE(11)
            IFVS_LDQ_CASE(12) IFVS_LDQ_CASE(13) IFVS_LDQ_CASE(14) IFVS_LDQ_CASE(15)
#undef IFVS_LDQ_CASE
            default: break;
        }
    }
    uint32_t xa = 0u, xb = 0u;
#pragma unroll
    for (int s = 0; s < 16; ++s) {
        xa += va[s];
        xb += vb[s];
    }
    sa = xa;
    sb = xb;
}

// Exact float32 distance of one M = 16 row of the sorted copy from an
// unreplicated table ex[c * 16 + m]: byte s holds subspace (s + rot) mod 16,
// rot = (p mod 32) mod 16, added for s ascending from 0, as lookup2 does.
// Called for the rare candidate rows only: kept out of line, the round's
// code is smaller (measured 1-2 % faster than inlining its eight copies).
__device__ __noinline__ float exact16(const uint4 c, const float* ex, int rot) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    float d = 0.f;
#pragma unroll
    for (int s = 0; s < 16; ++s) {
        const uint32_t code = (w[s >> 2] >> (8 * (s & 3))) & 0xFFu;
        d = __fadd_rn(d, ex[code * 16u + (uint32_t)((s + rot) & 15)]);
    }
    return d;
}

// Both queries' bounds in one word: half h holds bound_h + 0x8000, bound_h
// clamped to [-1, 0x7FFF].  A row's packed sums (each half <= 16 * 2047 <
// 0x8000) are candidates where (packed bounds - sums) keeps bit 15 (query A)
// or bit 31 (query B): no borrow crosses the halves.
__device__ __forceinline__ uint32_t pack_bounds(int ta, int tb) {
    ta = ta > 0x7FFF ? 0x7FFF : ta;
    tb = tb > 0x7FFF ? 0x7FFF : tb;
    return (uint32_t)(ta + 0x8000) | (uint32_t)(tb + 0x8000) << 16;
}

constexpr uint32_t kCandA = 0x00008000u, kCandB = 0x80000000u;

// kU2 rows per lane per round in the paired loop.  Measured on the 10^8-row
// dense bin with candidates rescored in batches: 8 rows 137.4 ms, 4 rows
// 142.1 ms, 2 rows 200.1 ms per batch; 16 rows spill at the 128-register cap
// of a 16-warp CTA.  (With in-place rescoring 4 rows had been the fastest.)
#ifndef IFVS_PAIR_ROWS
#define IFVS_PAIR_ROWS 8
#endif
constexpr int kU2 = IFVS_PAIR_ROWS;
static_assert(kU2 % 2 == 0 && 32 % kU2 == 0, "rows in pairs, whole rounds per block");

// A warp's candidate buffer (shared memory): entry i = codes[i], pos[i],
// flags[i] (kCandA | kCandB for the queries whose test it passed).
struct CandBuf {
    uint4* codes;
    uint32_t* pos;
    uint32_t* flags;
    int cnt;
};

// Rescoring of entries [first, first + n) (n <= 32), entry first + l by lane
// l: the exact float32 distance of each flagged query in the one-query
// kernel's order, the row id for those within the query's k-th key, the
// offers (warp-collective).
template <int KP>
__device__ __forceinline__ void rescore_entries(const CandBuf& cbuf, int first, int n,
                                                const uint32_t* __restrict__ rows, WarpTopK<KP>& tkA,
                                                WarpTopK<KP>& tkB, const float* exA, const float* exB, int lane) {
    uint4 c = make_uint4(0, 0, 0, 0);
    uint32_t pos = 0u, f = 0u;
    if (lane < n) {
        c = cbuf.codes[first + lane];
        pos = cbuf.pos[first + lane];
        f = cbuf.flags[first + lane];
    }
    const int rot = (int)(pos & 15u);   // the lane that met position pos: pos mod 32
    bool cA = (f & kCandA) != 0u;
    bool cB = (f & kCandB) != 0u;
    float dA = 0.f, dB = 0.f;
    if (cA) dA = exact16(c, exA, rot);
    if (cB) dB = exact16(c, exB, rot);
    cA = cA && __float_as_uint(dA) <= (uint32_t)(tkA.thr >> 32);
    cB = cB && __float_as_uint(dB) <= (uint32_t)(tkB.thr >> 32);
    const uint32_t row = (cA || cB) ? __ldg(rows + pos) : 0u;
    const uint64_t kA = ((uint64_t)__float_as_uint(dA) << 32) | row;
    const uint64_t kB = ((uint64_t)__float_as_uint(dB) << 32) | row;
    tkA.offer(kA, cA && kA < tkA.thr, lane);
    tkB.offer(kB, cB && kB < tkB.thr, lane);
}

// Codes of a round's kU2 positions.  mask[] holds kCandA / kCandB for the
// positions inside each query's range; MASKED: it differs between positions
// (a cut block), so only positions inside a range load codes.
template <bool MASKED>
__device__ __forceinline__ void pair_load(const uint8_t* __restrict__ codes, uint32_t pos0,
                                          const uint32_t (&mask)[kU2], uint64_t keep, uint4 (&c)[kU2]) {
#pragma unroll
    for (int u = 0; u < kU2; ++u) {
        const uint32_t pos = pos0 + 32u * (uint32_t)u;
        c[u] = (!MASKED || mask[u] != 0u) ? ldg_nc_v4(codes + (size_t)pos * 16, keep) : make_uint4(0, 0, 0, 0);
    }
}

// One round of kU2 positions of a block: the shared bounds refreshed,
// quantised sums of both queries, candidates by the packed bounds, exact
// distances and top-k offers for the candidates.
template <int KP, bool FAST, bool MASKED>
__device__ __forceinline__ void pair_round(const uint4 (&c)[kU2], const uint32_t* __restrict__ rows,
                                           uint32_t pos0, const uint32_t (&mask)[kU2], WarpTopK<KP>& tkA,
                                           WarpTopK<KP>& tkB, const float* exA, const float* exB, float slA,
                                           float invA, float slB, float invB, uint32_t tb, uint32_t base,
                                           int rot, int lane, uint32_t& Tpk, CandBuf& cbuf) {
    {
        const uint64_t oa = tkA.thr, ob = tkB.thr;
        tkA.refresh(lane);
        tkB.refresh(lane);
        if (tkA.thr != oa || tkB.thr != ob)
            Tpk = pack_bounds(quant_bound(tkA.thr, slA, invA), quant_bound(tkB.thr, slB, invB));
    }
    uint32_t sq[kU2];
#pragma unroll
    for (int u = 0; u < kU2; u += 2) lookup16x2_q<FAST>(c[u], c[u + 1], tb, base, sq[u], sq[u + 1]);
    uint32_t cb[kU2], any = 0u;
#pragma unroll
    for (int u = 0; u < kU2; ++u) {
        cb[u] = (Tpk - sq[u]) & mask[u];
        any |= cb[u];
    }
    if (!__any_sync(0xFFFFFFFFu, any != 0u)) return;
    if constexpr (pair_defers(KP)) {
        const unsigned lt = (1u << lane) - 1u;
#pragma unroll
        for (int u = 0; u < kU2; ++u) {
            const unsigned ball = __ballot_sync(0xFFFFFFFFu, cb[u] != 0u);
            if (ball == 0u) continue;
            if (cb[u] != 0u) {
                const int at = cbuf.cnt + __popc(ball & lt);
                cbuf.codes[at] = c[u];
                cbuf.pos[at] = pos0 + 32u * (uint32_t)u;
                cbuf.flags[at] = cb[u];
            }
            cbuf.cnt += __popc(ball);
            if (cbuf.cnt >= 32) {
                __syncwarp();
                cbuf.cnt -= 32;
                rescore_entries<KP>(cbuf, cbuf.cnt, 32, rows, tkA, tkB, exA, exB, lane);
                __syncwarp();   // the drained slots take the next entries
                Tpk = pack_bounds(quant_bound(tkA.thr, slA, invA), quant_bound(tkB.thr, slB, invB));
            }
        }
        return;
    }
#pragma unroll
    for (int u = 0; u < kU2; ++u) {
        const uint32_t pos = pos0 + 32u * (uint32_t)u;
        bool cA = (cb[u] & kCandA) != 0u;
        bool cB = (cb[u] & kCandB) != 0u;
        float dA = 0.f, dB = 0.f;
        if (cA) dA = exact16(c[u], exA, rot);
        if (cB) dB = exact16(c[u], exB, rot);
        cA = cA && __float_as_uint(dA) <= (uint32_t)(tkA.thr >> 32);
        cB = cB && __float_as_uint(dB) <= (uint32_t)(tkB.thr >> 32);
        const uint32_t row = (cA || cB) ? __ldg(rows + pos) : 0u;
        const uint64_t kA = ((uint64_t)__float_as_uint(dA) << 32) | row;
        const uint64_t kB = ((uint64_t)__float_as_uint(dB) << 32) | row;
        tkA.offer(kA, cA && kA < tkA.thr, lane);
        tkB.offer(kB, cB && kB < tkB.thr, lane);
    }
    Tpk = pack_bounds(quant_bound(tkA.thr, slA, invA), quant_bound(tkB.thr, slB, invB));
}

template <int KP, bool FAST>
__device__ __forceinline__ void scan_positions_pair(const uint8_t* __restrict__ codes,
                                                    const uint32_t* __restrict__ rows, int64_t aA,
                                                    int64_t bA, int64_t aB, int64_t bB, int64_t blk0,
                                                    int64_t blk1, WarpTopK<KP>& tkA, WarpTopK<KP>& tkB,
                                                    const float* exA, const float* exB, float slA, float invA,
                                                    float slB, float invB, uint32_t base, int lane, int warp,
                                                    CandBuf& cbuf) {
    const uint32_t tb = 4u * (uint32_t)lane;
    const int rot = lane & 15;
    const uint64_t keep = policy_evict_last();
    const uint32_t a1 = (uint32_t)aA, b1 = (uint32_t)bA, a2 = (uint32_t)aB, b2 = (uint32_t)bB;
    uint32_t Tpk = pack_bounds(quant_bound(tkA.thr, slA, invA), quant_bound(tkB.thr, slB, invB));
    for (int64_t blk = blk0 + warp; blk < blk1; blk += kPairWarps) {
        const uint32_t p0 = (uint32_t)(blk * kBlockRows);
        const uint32_t pe = p0 + kBlockRows;
        const bool inA = p0 < b1 && pe > a1, inB = p0 < b2 && pe > a2;
        if (!(inA || inB)) continue;
        const bool fullA = inA && p0 >= a1 && pe <= b1, fullB = inB && p0 >= a2 && pe <= b2;
        if ((fullA || !inA) && (fullB || !inB)) {
            // each query takes all or none of the block: one mask for all rows
            const uint32_t mc = (fullA ? kCandA : 0u) | (fullB ? kCandB : 0u);
            uint32_t mask[kU2];
#pragma unroll
            for (int u = 0; u < kU2; ++u) mask[u] = mc;
            const uint32_t pb = p0 + (uint32_t)lane;
#pragma unroll 1
            for (int j0 = 0; j0 < 32; j0 += kU2) {
                uint4 c[kU2];
                pair_load<false>(codes, pb + 32u * (uint32_t)j0, mask, keep, c);
                pair_round<KP, FAST, false>(c, rows, pb + 32u * (uint32_t)j0, mask, tkA, tkB, exA, exB, slA, invA,
                                            slB, invB, tb, base, rot, lane, Tpk, cbuf);
            }
            continue;
        }
#pragma unroll 1
        for (int j0 = 0; j0 < 32; j0 += kU2) {
            const uint32_t pos0 = p0 + 32u * (uint32_t)j0 + (uint32_t)lane;
            uint32_t mask[kU2];
#pragma unroll
            for (int u = 0; u < kU2; ++u) {
                const uint32_t pos = pos0 + 32u * (uint32_t)u;
                mask[u] = ((fullA || (inA && pos >= a1 && pos < b1)) ? kCandA : 0u) |
                          ((fullB || (inB && pos >= a2 && pos < b2)) ? kCandB : 0u);
            }
            uint4 c[kU2];
            pair_load<true>(codes, pos0, mask, keep, c);
            pair_round<KP, FAST, true>(c, rows, pos0, mask, tkA, tkB, exA, exB, slA, invA, slB, invB, tb, base,
                                       rot, lane, Tpk, cbuf);
        }
    }
    if constexpr (pair_defers(KP)) {
        if (cbuf.cnt > 0) {   // warp-uniform
            __syncwarp();
            rescore_entries<KP>(cbuf, 0, cbuf.cnt, rows, tkA, tkB, exA, exB, lane);
            cbuf.cnt = 0;
        }
    }
}
// Quantisation parameters of one query from the per-subspace extremes
// lo[16], hi[16]: inv (0 turns the test off: every row is rescored) and sl.
__device__ __forceinline__ void quant_params(const float* lo, const float* hi, float& inv, float& sl) {
    float r = 0.f, s = 0.f;
    bool ok = true;
#pragma unroll
    for (int m = 0; m < 16; ++m) {
        r = fmaxf(r, __fsub_rn(hi[m], lo[m]));
        s = __fadd_rn(s, lo[m]);
        ok = ok && lo[m] >= 0.f;
    }
    inv = __fdiv_rn((float)kQMax, r);
    if (!(ok && r > 0.f && isfinite(inv) && isfinite(s))) inv = 0.f;
    sl = s;
}

// ---- pairing of the sorted-copy queries of a batch -------------------------
//
// Two queries are worth one CTA when they read the same column's copy, their
// ranges mostly coincide (at least 3/4 of the longer range is common to both;
// the rows of only one range then run with the other query masked) and the
// two ranges together span at least min_rows positions (the caller's choice:
// for short ranges the one-query kernel, with two or three CTAs per SM, was
// measured faster).
// k_pair_items sorts the list-path queries of each segment of kPairSeg by
// (column, range start, query) and pairs sorted neighbours (2j, 2j + 1) that
// qualify.  Pairs fill the segment's item slots in sorted order and the
// unused slots get qa = -1, so the pair kernel's CTA x serves item x (or
// nothing); `paired` marks the queries of the pairs, and k_scan_list serves
// every other list-path query.
constexpr int kPairSeg = 2048;
static_assert(kSortedCopies <= 8, "the pairing key keeps 3 bits of the sorted copy");
constexpr int kPairSortThreads = 1024;

__device__ __forceinline__ bool pairable(const ScanPlan& x, const ScanPlan& y, int64_t min_rows) {
    if (!x.list || !y.list || x.col != y.col) return false;
    const int64_t lx = x.b - x.a, ly = y.b - y.a;
    if (lx <= 0 || ly <= 0) return false;
    const int64_t common = min(x.b, y.b) - max(x.a, y.a);
    const int64_t span = max(x.b, y.b) - min(x.a, y.a);
    return 4 * common >= 3 * max(lx, ly) && span >= min_rows;
}

// exclusive prefix of v over the block's threads (in thread order) and the
// total; wsum holds one int per warp
__device__ __forceinline__ int block_prefix(int v, int* wsum, int& total) {
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    int incl = v;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
        const int t = __shfl_up_sync(0xFFFFFFFFu, incl, o);
        if (lane >= o) incl += t;
    }
    __syncthreads();
    if (lane == 31) wsum[warp] = incl;
    __syncthreads();
    int before = 0;
    total = 0;
    for (int w = 0; w < (int)(blockDim.x >> 5); ++w) {
        const int t = wsum[w];
        before += w < warp ? t : 0;
        total += t;
    }
    return before + incl - v;
}

__global__ void __launch_bounds__(kPairSortThreads)
k_pair_items(const ScanPlan* __restrict__ plan, int64_t nq, int64_t min_rows, PairItem* __restrict__ items,
             uint8_t* __restrict__ paired, unsigned* __restrict__ counter) {
    if (blockIdx.x == 0 && threadIdx.x == 0) *counter = 0u;   // work counter of the two-query kernel
    __shared__ uint64_t key[kPairSeg];
    __shared__ int wsum[kPairSortThreads / 32];
    const int64_t q0 = (int64_t)blockIdx.x * kPairSeg;
    const int n = (int)min((int64_t)kPairSeg, nq - q0);
    // key = copy (3 bits) | range start (32 bits) | index in the segment (11 bits);
    // queries of the bitmap path sort last as all ones
    for (int i = threadIdx.x; i < kPairSeg; i += kPairSortThreads) {
        uint64_t kk = ~0ull;
        if (i < n) {
            const ScanPlan p = plan[q0 + i];
            if (p.list) kk = ((uint64_t)(p.col & 7) << 43) | ((uint64_t)(uint32_t)p.a << 11) | (uint64_t)i;
        }
        key[i] = kk;
    }
    // block bitonic sort, ascending
    for (int size = 2; size <= kPairSeg; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < kPairSeg / 2; t += kPairSortThreads) {
                const int i = 2 * t - (t & (stride - 1));
                const int j = i + stride;
                const bool up = (i & size) == 0;
                const uint64_t x = key[i], y = key[j];
                if ((x > y) == up) {
                    key[i] = y;
                    key[j] = x;
                }
            }
        }
    __syncthreads();
    // sorted neighbours (2j, 2j + 1) that qualify make an item; positions by
    // a block-wide exclusive scan of the counts, in sorted order
    static_assert(kPairSeg == 2 * kPairSortThreads, "one neighbour pair per thread");
    const int j = threadIdx.x;
    const uint64_t ka = key[2 * j], kb = key[2 * j + 1];
    int qa = -1, qb = -1, cnt = 0;
    if (ka != ~0ull && kb != ~0ull) {
        qa = (int)(q0 + (int64_t)(ka & 2047u));
        qb = (int)(q0 + (int64_t)(kb & 2047u));
        cnt = pairable(plan[qa], plan[qb], min_rows) ? 1 : 0;
    }
    for (int i = j; i < n; i += kPairSortThreads) paired[q0 + i] = 0;
    __syncthreads();
    if (cnt) paired[qa] = paired[qb] = 1;
    // segment s owns item slots [s kPairSeg / 2, + ceil(n / 2)): at most one
    // pair per two of its queries
    int total = 0;
    const int at = block_prefix(cnt, wsum, total);
    PairItem* its = items + q0 / 2;
    if (cnt) its[at] = PairItem{qa, qb};
    for (int i = total + j; i < (n + 1) / 2; i += kPairSortThreads) its[i] = PairItem{-1, -1};
}

// Offset of the current work item in the two-query kernel's shared memory.
__host__ __device__ constexpr size_t scan_pair_item_offset(int kp) {
    return (size_t)kTabBytes16 + 2 * (size_t)kExactBytes16 + 64 * 4 + 16 + (size_t)kPairWarps * 2 * 2 * kp * 8 +
           (pair_defers(kp) ? (size_t)kPairWarps * kCandWarpBytes : 0);
}

// One work item of the two-query kernel: pair slot `slot` on chunk `chunk`.
template <int KP>
__device__ __forceinline__ void pair_item(uint8_t* smem, const float* __restrict__ tables, const SortedCols& sc,
                                          const ScanPlan* __restrict__ plan, const PairItem* __restrict__ items,
                                          int k, const ScanShape& sh, uint64_t* __restrict__ partials, int slot,
                                          int chunk) {
    uint32_t* ptab = reinterpret_cast<uint32_t*>(smem);
    float* exA = reinterpret_cast<float*>(smem + kTabBytes16);
    float* exB = reinterpret_cast<float*>(smem + kTabBytes16 + kExactBytes16);
    float* prm = reinterpret_cast<float*>(smem + kTabBytes16 + 2 * kExactBytes16);   // lo/hi of A, lo/hi of B
    uint64_t* ctab = reinterpret_cast<uint64_t*>(smem + kTabBytes16 + 2 * kExactBytes16 + 64 * 4);   // A, B
    uint64_t* tkbufA = reinterpret_cast<uint64_t*>(smem + kTabBytes16 + 2 * kExactBytes16 + 64 * 4 + 16);
    uint64_t* tkbufB = tkbufA + kPairWarps * 2 * KP;
    float* red = reinterpret_cast<float*>(tkbufA);   // [warp][4][16], before the lists are set up
    uint8_t* cand_base = reinterpret_cast<uint8_t*>(tkbufB + kPairWarps * 2 * KP);   // 16-byte aligned
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const PairItem it = items[slot];
    if (it.qa < 0) return;
    const int64_t qA = it.qa;
    const bool hasB = it.qb >= 0;
    const int64_t qB = hasB ? it.qb : it.qa;   // a single query: B mirrors A's table, with no range
    const ScanPlan pA = plan[qA];
    ScanPlan pB = plan[qB];
    if (!hasB) pB.a = pB.b = 0;
    const int64_t c0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t c1 = min(sh.n_blocks, c0 + sh.blocks_per_chunk);
    auto range = [&](const ScanPlan& p, int64_t& lo, int64_t& hi) {
        lo = max(c0, p.a / kBlockRows);
        hi = min(c1, (p.b + kBlockRows - 1) / kBlockRows);
        if (p.a >= p.b || lo >= hi) lo = hi = 0;
    };
    int64_t lA, hA, lB, hB;
    range(pA, lA, hA);
    range(pB, lB, hB);
    uint64_t* outA = partials + (qA * sh.n_chunks + chunk) * (int64_t)k;
    uint64_t* outB = hasB ? partials + (qB * sh.n_chunks + chunk) * (int64_t)k : nullptr;
    if (lA == hA && lB == hB) {
        for (int i = threadIdx.x; i < k; i += kPairThreads) {
            outA[i] = ~0ull;
            if (outB) outB[i] = ~0ull;
        }
        return;
    }
    // 1) unreplicated float32 tables ex[c * 16 + m] (from the replicated
    //    tables of k_tables: word m < 16 of row c is LUT[m][c]) and the
    //    extremes of each subspace; a thread keeps one subspace m
    {
        const float* srcA = tables + qA * (int64_t)256 * 64;
        const float* srcB = tables + qB * (int64_t)256 * 64;
        const int m = threadIdx.x & 15;
        float loA = INFINITY, hiA = -INFINITY, loB = INFINITY, hiB = -INFINITY;
        for (int i = threadIdx.x; i < 4096; i += kPairThreads) {
            const int c = i >> 4;
            const float x = __ldg(srcA + c * 64 + m), y = __ldg(srcB + c * 64 + m);
            exA[i] = x;
            exB[i] = y;
            loA = fminf(loA, x);
            hiA = fmaxf(hiA, x);
            loB = fminf(loB, y);
            hiB = fmaxf(hiB, y);
        }
        loA = fminf(loA, __shfl_xor_sync(0xFFFFFFFFu, loA, 16));
        hiA = fmaxf(hiA, __shfl_xor_sync(0xFFFFFFFFu, hiA, 16));
        loB = fminf(loB, __shfl_xor_sync(0xFFFFFFFFu, loB, 16));
        hiB = fmaxf(hiB, __shfl_xor_sync(0xFFFFFFFFu, hiB, 16));
        if (lane < 16) {
            red[warp * 64 + m] = loA;
            red[warp * 64 + 16 + m] = hiA;
            red[warp * 64 + 32 + m] = loB;
            red[warp * 64 + 48 + m] = hiB;
        }
    }
    __syncthreads();
    if (threadIdx.x < 64) {
        const int j = threadIdx.x;   // 0-15 lo A, 16-31 hi A, 32-47 lo B, 48-63 hi B
        const bool is_lo = (j & 16) == 0;
        float v = red[j];
        for (int w = 1; w < kPairWarps; ++w) v = is_lo ? fminf(v, red[w * 64 + j]) : fmaxf(v, red[w * 64 + j]);
        prm[j] = v;
    }
    __syncthreads();
    float invA, slA, invB, slB;
    quant_params(prm, prm + 16, invA, slA);
    quant_params(prm + 32, prm + 48, invB, slB);
    // 2) the packed table: word w of row c = qA[w mod 16][c] | qB[..] << 16
    for (int i = threadIdx.x; i < 256 * 64; i += kPairThreads) {
        const int c = i >> 6, m = i & 15;
        ptab[i] = quant12(exA[c * 16 + m], prm[m], invA) | quant12(exB[c * 16 + m], prm[32 + m], invB) << 16;
    }
    __syncthreads();   // the reduction scratch becomes the lists
    if (threadIdx.x < 2) ctab[threadIdx.x] = ~0ull;
    WarpTopK<KP> tkA, tkB;
    tkA.init(tkbufA + warp * 2 * KP, k, lane, ctab);
    tkB.init(tkbufB + warp * 2 * KP, k, lane, ctab + 1);
    __syncthreads();
    const int64_t lo = (lA == hA) ? lB : ((lB == hB) ? lA : min(lA, lB));
    const int64_t hi = max(hA, hB);
    CandBuf cbuf;
    {
        uint8_t* wb = cand_base + (size_t)warp * kCandWarpBytes;
        cbuf.codes = reinterpret_cast<uint4*>(wb);
        cbuf.pos = reinterpret_cast<uint32_t*>(wb + kCandCap * 16);
        cbuf.flags = reinterpret_cast<uint32_t*>(wb + kCandCap * 20);
        cbuf.cnt = 0;
    }
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(ptab);
    if (base == kDynSmemBase)
        scan_positions_pair<KP, true>(sc.codes_of(pA.col), sc.rows_of(pA.col), pA.a, pA.b, pB.a, pB.b, lo, hi,
                                      tkA, tkB, exA, exB, slA, invA, slB, invB, base, lane, warp, cbuf);
    else
        scan_positions_pair<KP, false>(sc.codes_of(pA.col), sc.rows_of(pA.col), pA.a, pA.b, pB.a, pB.b, lo, hi,
                                       tkA, tkB, exA, exB, slA, invA, slB, invB, base, lane, warp, cbuf);
    merge_warps<KP, kPairWarps>(tkA, tkbufA, k, lane, warp, outA);
    merge_warps<KP, kPairWarps>(tkB, tkbufB, k, lane, warp, outB);
}

// Persistent: one CTA per SM takes work items (pair slot, chunk) in the
// order of a (slot, chunk) grid, chunk-major, from a counter that
// k_pair_items zeroes: the CTAs that run together still walk the same chunk,
// and no SM idles through a ragged last wave of long items (a 1024-CTA grid
// over 152 SMs left 0.26 of its last wave empty on the dense bin).
template <int KP>
__global__ void __launch_bounds__(kPairThreads, 1)
k_scan_list_pair(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan,
                 const PairItem* __restrict__ items, int n_slots, unsigned* __restrict__ counter, int k,
                 ScanShape sh, uint64_t* __restrict__ partials) {
    extern __shared__ __align__(256) uint8_t smem[];
    volatile unsigned* s_item = reinterpret_cast<volatile unsigned*>(smem + scan_pair_item_offset(KP));
    const unsigned total = (unsigned)n_slots * (unsigned)sh.n_chunks;
    for (;;) {
        if (threadIdx.x == 0) *s_item = atomicAdd(counter, 1u);
        __syncthreads();
        const unsigned w = *s_item;
        __syncthreads();   // read by all before thread 0 takes the next item
        if (w >= total) break;
        pair_item<KP>(smem, tables, sc, plan, items, k, sh, partials, (int)(w % (unsigned)n_slots),
                      (int)(w / (unsigned)n_slots));
        __syncthreads();   // the next item reuses the shared memory
    }
}

size_t scan_list_workspace_bytes(int64_t nq) {
    // pair slots (each segment rounds its count up), a flag per query, the
    // two-query kernel's work counter
    return (size_t)(nq + 2 * kPairSeg) * sizeof(PairItem) + (size_t)nq + 64;
}

template <int KP>
static cudaError_t launch_pairs_kp(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                                   const ScanShape& sh, uint64_t* partials, uint8_t* work, int64_t pair_min_rows,
                                   cudaStream_t s, const uint8_t** paired, int* launches) {
    const size_t ps = scan_pair_smem_bytes(KP);
    if (ps > (size_t)max_smem_optin()) return cudaSuccess;   // no pairs: one query per CTA
    PairItem* items = reinterpret_cast<PairItem*>(work);
    uint8_t* pd = reinterpret_cast<uint8_t*>(items + nq + 2 * kPairSeg);
    unsigned* counter = reinterpret_cast<unsigned*>(work + (((size_t)(nq + 2 * kPairSeg) * sizeof(PairItem) +
                                                             (size_t)nq + 15) / 16) * 16);
    const unsigned segs = (unsigned)((nq + kPairSeg - 1) / kPairSeg);
    k_pair_items<<<segs, kPairSortThreads, 0, s>>>(plan, nq, pair_min_rows, items, pd, counter);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    if ((e = cudaFuncSetAttribute(k_scan_list_pair<KP>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)ps)) !=
        cudaSuccess)
        return e;
    int dev = 0, sms = 0;
    if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
    if ((e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
    const int n_slots = (int)((nq + 1) / 2);   // at most nq / 2 pairs
    const long long items_total = (long long)n_slots * sh.n_chunks;
    const int grid = (int)(items_total < sms ? items_total : sms);   // one CTA per SM
    k_scan_list_pair<KP><<<grid, kPairThreads, ps, s>>>(tab, sc, plan, items, n_slots, counter, k, sh, partials);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    *paired = pd;
    *launches += 2;
    return cudaSuccess;
}

cudaError_t launch_pairs(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                         const ScanShape& sh, uint64_t* partials, uint8_t* work, int64_t pair_min_rows,
                         cudaStream_t s, const uint8_t** paired, int* launches) {
    *paired = nullptr;
    if (nq <= 0) return cudaSuccess;
    switch (scan_kp(k)) {
        case 32: return launch_pairs_kp<32>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, s, paired, launches);
        case 64: return launch_pairs_kp<64>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, s, paired, launches);
        case 128: return launch_pairs_kp<128>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, s, paired, launches);
        default: return launch_pairs_kp<256>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, s, paired, launches);
    }
}

}  // namespace ifvs
