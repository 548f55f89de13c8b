// Stage 2 of §2 (Rank) with the per-CTA part of stage 3 (Select): every
// passing row v gets dist(v) = sum_m LUT[m][code_v[m]] (the weighted ADC
// form of the printed score), and each CTA keeps the k smallest
// (dist, row id) of its chunk exactly.
//
// Work split.  CTA (query q, chunk c), 8 warps; blockIdx.x runs over the
// queries so that the CTAs resident together walk the same code chunk and
// share it through L2.  Warp w of the CTA owns bitmap blocks c0 + w,
// c0 + w + 8, ...; lane l owns, in each of them, the 32 rows
// b*1024 + 32*j + l, whose pass bits form its lane-major bitmap word.
//
// LUT placement.  The scan issues one shared-memory load per code byte, so
// bank conflicts set its speed.  The table of query q is stored as 256 rows
// (one per codeword) of S words, S a multiple of 32, word w of row c holding
// LUT[w mod M][c] for w < M + 31.  Row i's codes are stored rotated by
// (i mod 32) mod M, so the lane that owns row i (lane i mod 32) reads at
// step s the code of subspace (l + s) mod M and finds its entry at word
// l + s of that codeword's row: bank (l + s) mod 32, distinct across the
// warp whatever the codes.  For M = 16 the row stride is 256 bytes and the
// address is one byte permute, code * 256 + 4l, with the table base and the
// step 4s in the load's immediate offset (the table starts the CTA's dynamic
// shared memory, whose address the kernel checks).
//
// Compaction.  Each lane visits only its own passing rows, so it keeps its
// residue class and the conflict-free banks at any selectivity.  The warp's
// bitmap words sit in a ring of 16 blocks in shared memory (lane l's word in
// bank l); lanes advance through the ring at their own pace, eight rows per
// round, and the ring is refilled by halves, from words prefetched into
// registers, once every lane has left the older half.  When every lane
// holds a full word of the same block the warp takes the block in lockstep
// without per-row bit handling.
//
// Top-k.  Each warp keeps a sorted list of its KP best keys and a candidate
// area of KP slots; a key (dist bits << 32 | row) enters the area when it
// is below the warp's current k-th key, and a full area is merged by a warp
// bitonic sort.  Keys are unique (row ids are), so the result is exact and
// independent of scheduling.  At the end the warps' lists are merged
// pairwise and warp 0 writes the CTA's k keys.
//
// The tile constants (warps per CTA, ring depth, rows per round) were chosen
// by measurement on the 10^8-row workload; the macros below only exist to
// rebuild variants for such sweeps.
#include <climits>

#include "internal.cuh"

namespace ifvs {

#ifndef IFVS_SCAN_WARPS
#define IFVS_SCAN_WARPS 8
#endif
#ifndef IFVS_SCAN_RING
#define IFVS_SCAN_RING 16
#endif
#ifndef IFVS_SCAN_ROWS
#define IFVS_SCAN_ROWS 8
#endif
constexpr int kScanWarps = IFVS_SCAN_WARPS;
constexpr int kScanThreads = kScanWarps * 32;
constexpr int kRing = IFVS_SCAN_RING;    // bitmap words per lane in the ring
constexpr int kHalf = kRing / 2;
constexpr int kU = IFVS_SCAN_ROWS;       // rows per lane per round (even)

int scan_kp(int k) { return k <= 32 ? 32 : (k <= 64 ? 64 : (k <= 128 ? 128 : 256)); }

size_t scan_smem_bytes(int tab_words, int kp) {
    return (size_t)256 * tab_words * 4 + (size_t)kScanWarps * 2 * kp * 8 +
           (size_t)kScanWarps * kRing * 32 * 4;
}

int scan_ctas_per_sm(int tab_words, int kp) {
    const size_t per_cta = scan_smem_bytes(tab_words, kp) + 1024;
    const int by_smem = (int)((size_t)233472 / per_cta);
    const int by_threads = 2048 / kScanThreads;
    int n = by_smem < by_threads ? by_smem : by_threads;
    return n < 1 ? 1 : n;
}

__device__ __forceinline__ void warp_sort(uint64_t* a, int n, int lane) {
    for (int size = 2; size <= n; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncwarp();
            for (int t = lane; t < (n >> 1); t += 32) {
                const int i = 2 * t - (t & (stride - 1));
                const int j = i + stride;
                const bool up = (i & size) == 0;
                const uint64_t x = a[i], y = a[j];
                if ((x > y) == up) {
                    a[i] = y;
                    a[j] = x;
                }
            }
        }
    __syncwarp();
}

// The warps of a CTA that serve one query share a bound `cta` (shared
// memory): the smallest k-th key any of them has published.  A warp's list
// holds k distinct rows, so its k-th key is at least the CTA's true k-th
// key, and a row whose key is above some warp's k-th key cannot be in the
// CTA's top-k: each warp offers only keys below min(own k-th, cta).  The
// warps' lists then still contain every row of the CTA's top-k, and the
// shared bound lets every warp drop rows as early as the whole CTA could.
template <int KP>
struct WarpTopK {
    uint64_t* buf;   // [0, KP): sorted best keys; [KP, 2KP): candidates
    uint64_t* cta;   // shared bound of the CTA's warps for this query, or null
    int cnt;
    int k;
    uint64_t thr;    // keys below thr are offered: min(own k-th key, *cta)

    __device__ __forceinline__ void init(uint64_t* b, int k_, int lane, uint64_t* cta_ = nullptr) {
        buf = b;
        cta = cta_;
        k = k_;
        cnt = 0;
        thr = ~0ull;
        for (int i = lane; i < 2 * KP; i += 32) buf[i] = ~0ull;
        __syncwarp();
    }
    // lower thr to the shared bound: every lane loads the same word in one
    // broadcast (measured faster than a lane-0 load and a shuffle); any value
    // a lane sees is a valid bound, so thr stays correct in every lane
    __device__ __forceinline__ void refresh(int) {
        if (cta == nullptr) return;
        const uint64_t t = *reinterpret_cast<volatile uint64_t*>(cta);
        if (t < thr) thr = t;
    }
    __device__ __forceinline__ void flush(int lane) {
        warp_sort(buf, 2 * KP, lane);
        thr = buf[k - 1];
        for (int i = KP + lane; i < 2 * KP; i += 32) buf[i] = ~0ull;
        if (cta != nullptr && lane == 0 && thr != ~0ull) atomicMin(reinterpret_cast<unsigned long long*>(cta), thr);
        __syncwarp();
        cnt = 0;
        refresh(lane);
    }
    __device__ __forceinline__ void offer(uint64_t key, bool want, int lane) {
        const unsigned ball = __ballot_sync(0xFFFFFFFFu, want);
        if (ball == 0) return;
        if (want) buf[KP + cnt + __popc(ball & ((1u << lane) - 1u))] = key;
        cnt += __popc(ball);
        if (cnt > KP - 32) {
            __syncwarp();
            flush(lane);
        }
    }
};

// L2 policies: code rows are read by every query of a batch (keep them, so
// the CTAs that walk the same chunk share them); bitmap words are read once.
__device__ __forceinline__ uint64_t policy_evict_last() {
    uint64_t pol;
    asm("createpolicy.fractional.L2::evict_last.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ uint64_t policy_evict_first() {
    uint64_t pol;
    asm volatile("createpolicy.fractional.L2::evict_first.b64 %0, 1.0;" : "=l"(pol));
    return pol;
}

__device__ __forceinline__ uint4 ldg_nc_v4(const uint8_t* p, uint64_t pol) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.v4.u32 {%0, %1, %2, %3}, [%4], %5;"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p), "l"(pol));
    return v;
}

__device__ __forceinline__ uint32_t ldg_nc_u32(const uint32_t* p, uint64_t pol) {
    uint32_t v;
    asm volatile("ld.global.nc.L1::no_allocate.L2::cache_hint.u32 %0, [%1], %2;"
                 : "=r"(v) : "l"(p), "l"(pol));
    return v;
}

template <int IMM>
__device__ __forceinline__ float lds_imm(uint32_t addr) {
    float v;
    asm volatile("ld.shared.f32 %0, [%1+%2];" : "=f"(v) : "r"(addr), "n"(IMM));
    return v;
}

// Two packed fp32 additions at once (Blackwell f32x2 pipe).
__device__ __forceinline__ uint64_t add_f32x2(uint64_t acc, float a, float b) {
    uint64_t r;
    asm("{\n\t.reg .b64 t;\n\tmov.b64 t, {%1, %2};\n\tadd.rn.f32x2 %0, %3, t;\n\t}"
        : "=l"(r) : "f"(a), "f"(b), "l"(acc));
    return r;
}

__device__ __forceinline__ void unpack_f32x2(uint64_t v, float& a, float& b) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(a), "=f"(b) : "l"(v));
}

// Shared address at which the dynamic shared memory of a CTA begins on this
// architecture (after the 1 KB the hardware reserves); the kernel checks it.
constexpr uint32_t kDynSmemBase = 0x400u;

// Distances of two M = 16 rows (codes ca, cb).  One byte permute forms
// code * 256 + 4 * w0, w0 = the row's index mod 32 (the lane that owns it in
// the bitmap path); FAST (table at kDynSmemBase): the table base and the step
// go into the load's immediate offset; otherwise the base is added.
template <bool FAST>
__device__ __forceinline__ void lookup16x2(const uint4 ca, const uint4 cb, uint32_t tba, uint32_t tbb,
                                           uint32_t base, float& da, float& db) {
    const uint32_t wa[4] = {ca.x, ca.y, ca.z, ca.w};
    const uint32_t wb[4] = {cb.x, cb.y, cb.z, cb.w};
    uint64_t acc = 0ull;
#pragma unroll
    for (int s = 0; s < 16; ++s) {
        const uint32_t sel = 0x5504u | ((uint32_t)(s & 3) << 4);
        uint32_t oa = __byte_perm(wa[s >> 2], tba, sel);
        uint32_t ob = __byte_perm(wb[s >> 2], tbb, sel);
        if (!FAST) {
            oa += base;
            ob += base;
        }
        constexpr uint32_t B0 = FAST ? kDynSmemBase : 0u;
        float va, vb;
        switch (s) {
#define IFVS_LDS_CASE(S)                  \
    case S:                               \
        va = lds_imm<B0 + 4 * S>(oa);     \
        vb = lds_imm<B0 + 4 * S>(ob);     \
        break;
            IFVS_LDS_CASE(0) IFVS_LDS_CASE(1) IFVS_LDS_CASE(2) IFVS_LDS_CASE(3)
            IFVS_LDS_CASE(4) IFVS_LDS_CASE(5) IFVS_LDS_CASE(6) IFVS_LDS_CASE(7)
            IFVS_LDS_CASE(8) IFVS_LDS_CASE(9) IFVS_LDS_CASE(10) IFVS_LDS_CASE(11)
            IFVS_LDS_CASE(12) IFVS_LDS_CASE(13) IFVS_LDS_CASE(14) IFVS_LDS_CASE(15)
#undef IFVS_LDS_CASE
            default: va = 0.f; vb = 0.f; break;
        }
        acc = add_f32x2(acc, va, vb);
    }
    unpack_f32x2(acc, da, db);
}

// Distance of one row for any M (runtime loop; row_bytes a multiple of 4);
// w0 = the row's index mod 32.
__device__ __forceinline__ float lookup_any(const uint8_t* rp, bool pass, int M, int S,
                                            const float* tab, int w0) {
    float acc = 0.f;
    for (int w = 0; w * 4 < M; ++w) {
        const uint32_t wd = pass ? __ldg(reinterpret_cast<const uint32_t*>(rp) + w) : 0u;
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) {
            const int s = 4 * w + bb;
            if (s < M) acc += tab[(int)((wd >> (8 * bb)) & 0xFFu) * S + w0 + s];
        }
    }
    return acc;
}

// Distances of NU rows for any M, all owned by one lane (so they share the
// table word offset w0 = the lane): the rows' code words are read together
// and their look-ups go into NU/2 packed f32x2 chains, independent of each
// other; each row's entries are still added for s ascending, as in
// lookup_any.  Rows whose bit in `valid` is clear read no codes.
template <int NU>
__device__ __forceinline__ void lookup_rows(const uint8_t* __restrict__ codes, const uint32_t (&idx)[NU],
                                            unsigned valid, int row_bytes, int M, int S, const float* tab,
                                            int w0, float (&d)[NU]) {
    static_assert(NU % 2 == 0, "rows in pairs");
    uint64_t acc[NU / 2];
#pragma unroll
    for (int u = 0; u < NU / 2; ++u) acc[u] = 0ull;
    const float* tw = tab + w0;
    for (int w = 0; w * 4 < M; ++w) {
        uint32_t wd[NU];
#pragma unroll
        for (int u = 0; u < NU; ++u)
            wd[u] = (valid >> u & 1u)
                        ? __ldg(reinterpret_cast<const uint32_t*>(codes + (size_t)idx[u] * row_bytes) + w)
                        : 0u;
#pragma unroll
        for (int bb = 0; bb < 4; ++bb) {
            const int s = 4 * w + bb;
            if (s < M) {
#pragma unroll
                for (int u = 0; u < NU; u += 2) {
                    const float va = tw[(int)((wd[u] >> (8 * bb)) & 0xFFu) * S + s];
                    const float vb = tw[(int)((wd[u + 1] >> (8 * bb)) & 0xFFu) * S + s];
                    acc[u / 2] = add_f32x2(acc[u / 2], va, vb);
                }
            }
        }
    }
#pragma unroll
    for (int u = 0; u < NU; u += 2) unpack_f32x2(acc[u / 2], d[u], d[u + 1]);
}

template <int KP, bool M16, bool FAST>
__device__ __forceinline__ void scan_chunk(const uint8_t* __restrict__ codes,
                                           const uint32_t* __restrict__ bmq, const ScanShape& sh,
                                           int64_t b0, int64_t b1, const float* tab,
                                           uint32_t* ring, WarpTopK<KP>& tk, int lane, int warp) {
    const int M = M16 ? 16 : sh.M;
    const int S = M16 ? 64 : sh.tab_words;
    const int row_bytes = sh.row_bytes;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    const uint32_t tb = 4u * (uint32_t)lane;

    const uint64_t keep = policy_evict_last();
    const int64_t first = b0 + warp;
    const int T = first < b1 ? (int)((b1 - first + kScanWarps - 1) / kScanWarps) : 0;
    auto word_addr = [&](int t) { return bmq + (first + (int64_t)t * kScanWarps) * 32 + lane; };

    // ring: words of the blocks t in [F - kRing, F) in slot t % kRing
    int F = T < kRing ? T : kRing;
#pragma unroll
    for (int i = 0; i < kRing; ++i)
        if (i < F) ring[i * 32 + lane] = ldg_nc_u32(word_addr(i), policy_evict_first());
    uint32_t pf[kHalf];
    int npf = T - F < kHalf ? T - F : kHalf;
#pragma unroll
    for (int i = 0; i < kHalf; ++i) pf[i] = i < npf ? ldg_nc_u32(word_addr(F + i), policy_evict_first()) : 0u;
    __syncwarp();
    int pos = 0;
    uint32_t cur = F > 0 ? ring[lane] : 0u;

    for (;;) {
        const int slow = (int)__reduce_min_sync(0xFFFFFFFFu, (unsigned)pos);
        if (npf > 0 && slow >= F - kHalf) {
#pragma unroll
            for (int i = 0; i < kHalf; ++i)
                if (i < npf) ring[((F + i) % kRing) * 32 + lane] = pf[i];
            F += npf;
            npf = T - F < kHalf ? T - F : kHalf;
            const uint64_t once = policy_evict_first();
#pragma unroll
            for (int i = 0; i < kHalf; ++i) pf[i] = i < npf ? ldg_nc_u32(word_addr(F + i), once) : 0u;
            __syncwarp();
        }
        // lanes whose word is used up move on before the mode is chosen
        while (cur == 0u && pos + 1 < F) {
            ++pos;
            cur = ring[(pos % kRing) * 32 + lane];
        }
        const bool dense = __all_sync(0xFFFFFFFFu, cur == 0xFFFFFFFFu) &&
                           __reduce_min_sync(0xFFFFFFFFu, (unsigned)pos) ==
                               __reduce_max_sync(0xFFFFFFFFu, (unsigned)pos);
        if (dense) {
            // every lane holds all 32 rows of the same block: lockstep rows
            const uint32_t rb = (uint32_t)((first + (int64_t)pos * kScanWarps) * kBlockRows) + lane;
#pragma unroll 1
            for (int j0 = 0; j0 < 32; j0 += kU) {
                uint32_t row[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u) row[u] = rb + 32u * (uint32_t)(j0 + u);
                if constexpr (M16) {
                    uint4 c[kU];
#pragma unroll
                    for (int u = 0; u < kU; ++u) c[u] = ldg_nc_v4(codes + (size_t)row[u] * 16, keep);
                    float d[kU];
#pragma unroll
                    for (int u = 0; u < kU; u += 2) lookup16x2<FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
                    uint64_t key[kU];
                    bool want = false;
#pragma unroll
                    for (int u = 0; u < kU; ++u) {
                        key[u] = ((uint64_t)__float_as_uint(d[u]) << 32) | row[u];
                        want |= key[u] < tk.thr;
                    }
                    if (__any_sync(0xFFFFFFFFu, want)) {
#pragma unroll
                        for (int u = 0; u < kU; ++u) tk.offer(key[u], key[u] < tk.thr, lane);
                    }
                } else {
                    float d[kU];
                    lookup_rows<kU>(codes, row, (1u << kU) - 1u, row_bytes, M, S, tab, lane, d);
#pragma unroll
                    for (int u = 0; u < kU; ++u) {
                        const uint64_t key = ((uint64_t)__float_as_uint(d[u]) << 32) | row[u];
                        tk.offer(key, key < tk.thr, lane);
                    }
                }
            }
            cur = 0u;
            continue;
        }
        // up to kU passing rows of this lane
        uint32_t row[kU];
        unsigned valid = 0u;
#pragma unroll
        for (int u = 0; u < kU; ++u) {
            while (cur == 0u && pos + 1 < F) {
                ++pos;
                cur = ring[(pos % kRing) * 32 + lane];
            }
            row[u] = 0u;
            if (cur != 0u) {
                const int j = __ffs(cur) - 1;
                cur &= cur - 1u;
                row[u] = (uint32_t)((first + (int64_t)pos * kScanWarps) * kBlockRows) + 32u * (uint32_t)j + lane;
                valid |= 1u << u;
            }
        }
        if (__ballot_sync(0xFFFFFFFFu, valid != 0u) == 0u) {
            if (F >= T) break;   // every word loaded and consumed
            continue;            // lanes wait for the next refill
        }
        if constexpr (M16) {
            uint4 c[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u)
                c[u] = (valid >> u & 1u) ? ldg_nc_v4(codes + (size_t)row[u] * 16, keep) : make_uint4(0, 0, 0, 0);
            float d[kU];
#pragma unroll
            for (int u = 0; u < kU; u += 2) lookup16x2<FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
            uint64_t key[kU];
            bool want = false;
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                key[u] = ((uint64_t)__float_as_uint(d[u]) << 32) | row[u];
                want |= (valid >> u & 1u) && key[u] < tk.thr;
            }
            if (__any_sync(0xFFFFFFFFu, want)) {
#pragma unroll
                for (int u = 0; u < kU; ++u) tk.offer(key[u], (valid >> u & 1u) && key[u] < tk.thr, lane);
            }
        } else {
            float d[kU];
            lookup_rows<kU>(codes, row, valid, row_bytes, M, S, tab, lane, d);
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const bool pass = valid >> u & 1u;
                const uint64_t key = ((uint64_t)__float_as_uint(d[u]) << 32) | row[u];
                tk.offer(key, pass && key < tk.thr, lane);
            }
        }
    }
}

template <int KP, bool M16, int MINB>
__global__ void __launch_bounds__(kScanThreads, MINB)
k_scan(const uint8_t* __restrict__ codes, const float* __restrict__ tables,
       const uint32_t* __restrict__ bm, const ScanPlan* __restrict__ plan, int64_t nq, int k,
       ScanShape sh, uint64_t* __restrict__ partials) {
    extern __shared__ __align__(256) uint8_t smem[];
    const int S = M16 ? 64 : sh.tab_words;
    float* tab = reinterpret_cast<float*>(smem);
    uint64_t* tkbuf = reinterpret_cast<uint64_t*>(smem + (size_t)256 * S * 4);
    uint32_t* ringbase = reinterpret_cast<uint32_t*>(smem + (size_t)256 * S * 4 +
                                                     (size_t)kScanWarps * 2 * KP * 8);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t q = blockIdx.x;
    const int chunk = blockIdx.y;
    if (plan != nullptr && plan[q].list) return;   // k_scan_list covers this query

    // 1) the query's table, replicated and rotated (see the file comment),
    //    as written by k_tables: a straight 16-byte-wide copy
    {
        const float4* src = reinterpret_cast<const float4*>(tables + q * (int64_t)256 * S);
        float4* dst = reinterpret_cast<float4*>(tab);
        for (int i = threadIdx.x; i < 64 * S; i += kScanThreads) dst[i] = __ldg(src + i);
    }
    WarpTopK<KP> tk;
    tk.init(tkbuf + warp * 2 * KP, k, lane);
    __syncthreads();

    // 2) the chunk's blocks
    const int64_t b0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t b1 = min(sh.n_blocks, b0 + sh.blocks_per_chunk);
    const uint32_t* bmq = bm + q * sh.n_blocks * 32;
    uint32_t* ring = ringbase + warp * kRing * 32;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    const bool fast = base == kDynSmemBase;
    if constexpr (M16) {
        if (fast)
            scan_chunk<KP, true, true>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
        else
            scan_chunk<KP, true, false>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
    } else {
        scan_chunk<KP, false, false>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
    }

    // 3) merge the warps' lists pairwise (4 levels); warp 0 writes the
    //    CTA's k best keys
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
    if (warp == 0) {
        uint64_t* out = partials + (q * sh.n_chunks + chunk) * (int64_t)k;
        for (int i = lane; i < k; i += 32) out[i] = tk.buf[i];
    }
}

template <int KP, bool M16, int MINB>
static cudaError_t launch_one(const uint8_t* codes, const float* tab, const uint32_t* bm,
                              const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                              uint64_t* partials, size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(k_scan<KP, M16, MINB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan<KP, M16, MINB><<<grid, kScanThreads, smem, s>>>(codes, tab, bm, plan, nq, k, sh, partials);
    return cudaGetLastError();
}

template <int KP>
static cudaError_t launch_scan_kp(const uint8_t* codes, const float* tab, const uint32_t* bm,
                                  const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                                  uint64_t* partials, cudaStream_t s) {
    const bool m16 = sh.M == 16 && sh.row_bytes == 16 && sh.tab_words == 64;
    const size_t smem = scan_smem_bytes(sh.tab_words, KP);
    if (m16) {
#ifndef IFVS_SCAN_ONE_CTA
        if (scan_ctas_per_sm(sh.tab_words, KP) >= 2)
#else
        if (false)
#endif
            return launch_one<KP, true, 2>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
        return launch_one<KP, true, 1>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
    }
    return launch_one<KP, false, 1>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
}

cudaError_t launch_scan(const uint8_t* codes, const float* tab, const uint32_t* bm,
                        const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                        uint64_t* partials, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    switch (scan_kp(k)) {
        case 32: return launch_scan_kp<32>(codes, tab, bm, plan, nq, k, sh, partials, s);
        case 64: return launch_scan_kp<64>(codes, tab, bm, plan, nq, k, sh, partials, s);
        case 128: return launch_scan_kp<128>(codes, tab, bm, plan, nq, k, sh, partials, s);
        default: return launch_scan_kp<256>(codes, tab, bm, plan, nq, k, sh, partials, s);
    }
}

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

template <int KP, bool M16, bool FAST>
__device__ __forceinline__ void scan_positions(const uint8_t* __restrict__ codes, const uint32_t* __restrict__ rows,
                                               int64_t a, int64_t b, int64_t blk0, int64_t blk1, int wstride,
                                               const ScanShape& sh, const float* tab, WarpTopK<KP>& tk,
                                               int lane, int warp) {
    const int M = M16 ? 16 : sh.M;
    const int S = M16 ? 64 : sh.tab_words;
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
            if constexpr (M16) {
                uint4 c[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u)
                    c[u] = (valid >> u & 1u) ? ldg_nc_v4(codes + (size_t)pos[u] * 16, keep) : make_uint4(0, 0, 0, 0);
#pragma unroll
                for (int u = 0; u < kU; u += 2) lookup16x2<FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
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

template <int KP, bool M16, int MINB>
__global__ void __launch_bounds__(kScanThreads, MINB)
k_scan_list(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan, int64_t nq,
            int k, ScanShape sh, uint64_t* __restrict__ partials, const uint8_t* __restrict__ paired) {
    extern __shared__ __align__(256) uint8_t smem[];
    const int S = M16 ? 64 : sh.tab_words;
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
    if constexpr (M16) {
        if (base == kDynSmemBase)
            scan_positions<KP, true, true>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
        else
            scan_positions<KP, true, false>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
    } else {
        scan_positions<KP, false, false>(codes, rows, p.a, p.b, blk0, blk1, kScanWarps, sh, tab, tk, lane, warp);
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

// packed table, two exact tables, extremes + the two shared bounds, lists
size_t scan_pair_smem_bytes(int kp) {
    return (size_t)kTabBytes16 + 2 * (size_t)kExactBytes16 + 64 * 4 + 16 + (size_t)kPairWarps * 2 * 2 * kp * 8;
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
// the addresses of lookup16x2, integer loads and adds.
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
// rot = (p mod 32) mod 16, added for s ascending from 0, as lookup16x2 does.
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

// kU2 rows per lane per round in the paired loop (measured: 2 rows, 8 rows,
// and loading the next round's codes before this round's look-ups are all
// slower at the 128-register cap of a 16-warp CTA)
constexpr int kU2 = 4;

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
                                           int rot, int lane, uint32_t& Tpk) {
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
                                                    float slB, float invB, uint32_t base, int lane, int warp) {
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
                                            slB, invB, tb, base, rot, lane, Tpk);
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
                                       rot, lane, Tpk);
        }
    }
}

// merge the warps' lists of one query pairwise; warp 0 writes k keys
template <int KP, int WARPS>
__device__ __forceinline__ void merge_warps(WarpTopK<KP>& tk, uint64_t* tkbuf, int k, int lane, int warp,
                                            uint64_t* out) {
    tk.flush(lane);
#pragma unroll 1
    for (int step = 1; step < WARPS; step <<= 1) {
        __syncthreads();
        if ((warp & (2 * step - 1)) == 0 && warp + step < WARPS) {
            const uint64_t* other = tkbuf + (warp + step) * 2 * KP;
            for (int i = lane; i < k; i += 32) tk.buf[KP + i] = other[i];
            __syncwarp();
            tk.flush(lane);
        }
    }
    if (warp == 0 && out != nullptr)
        for (int i = lane; i < k; i += 32) out[i] = tk.buf[i];
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
static_assert(IFVS_MAX_ATTRS <= 4, "the pairing key keeps 2 bits of the column");
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
             uint8_t* __restrict__ paired) {
    __shared__ uint64_t key[kPairSeg];
    __shared__ int wsum[kPairSortThreads / 32];
    const int64_t q0 = (int64_t)blockIdx.x * kPairSeg;
    const int n = (int)min((int64_t)kPairSeg, nq - q0);
    // key = col (2 bits) | range start (32 bits) | index in the segment (11 bits);
    // queries of the bitmap path sort last as all ones
    for (int i = threadIdx.x; i < kPairSeg; i += kPairSortThreads) {
        uint64_t kk = ~0ull;
        if (i < n) {
            const ScanPlan p = plan[q0 + i];
            if (p.list) kk = ((uint64_t)(p.col & 3) << 43) | ((uint64_t)(uint32_t)p.a << 11) | (uint64_t)i;
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

template <int KP>
__global__ void __launch_bounds__(kPairThreads, 1)
k_scan_list_pair(const float* __restrict__ tables, SortedCols sc, const ScanPlan* __restrict__ plan,
                 const PairItem* __restrict__ items, int k, ScanShape sh, uint64_t* __restrict__ partials) {
    extern __shared__ __align__(256) uint8_t smem[];
    uint32_t* ptab = reinterpret_cast<uint32_t*>(smem);
    float* exA = reinterpret_cast<float*>(smem + kTabBytes16);
    float* exB = reinterpret_cast<float*>(smem + kTabBytes16 + kExactBytes16);
    float* prm = reinterpret_cast<float*>(smem + kTabBytes16 + 2 * kExactBytes16);   // lo/hi of A, lo/hi of B
    uint64_t* ctab = reinterpret_cast<uint64_t*>(smem + kTabBytes16 + 2 * kExactBytes16 + 64 * 4);   // A, B
    uint64_t* tkbufA = reinterpret_cast<uint64_t*>(smem + kTabBytes16 + 2 * kExactBytes16 + 64 * 4 + 16);
    uint64_t* tkbufB = tkbufA + kPairWarps * 2 * KP;
    float* red = reinterpret_cast<float*>(tkbufA);   // [warp][4][16], before the lists are set up
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const PairItem it = items[blockIdx.x];
    if (it.qa < 0) return;
    const int64_t qA = it.qa;
    const bool hasB = it.qb >= 0;
    const int64_t qB = hasB ? it.qb : it.qa;   // a single query: B mirrors A's table, with no range
    const int chunk = blockIdx.y;
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
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(ptab);
    if (base == kDynSmemBase)
        scan_positions_pair<KP, true>(sc.codes_of(pA.col), sc.rows_of(pA.col), pA.a, pA.b, pB.a, pB.b, lo, hi,
                                      tkA, tkB, exA, exB, slA, invA, slB, invB, base, lane, warp);
    else
        scan_positions_pair<KP, false>(sc.codes_of(pA.col), sc.rows_of(pA.col), pA.a, pA.b, pB.a, pB.b, lo, hi,
                                       tkA, tkB, exA, exB, slA, invA, slB, invB, base, lane, warp);
    merge_warps<KP, kPairWarps>(tkA, tkbufA, k, lane, warp, outA);
    merge_warps<KP, kPairWarps>(tkB, tkbufB, k, lane, warp, outB);
}

template <int KP, bool M16, int MINB>
static cudaError_t launch_list_one(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq,
                                   int k, const ScanShape& sh, uint64_t* partials, const uint8_t* paired,
                                   size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(k_scan_list<KP, M16, MINB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan_list<KP, M16, MINB><<<grid, kScanThreads, smem, s>>>(tab, sc, plan, nq, k, sh, partials, paired);
    return cudaGetLastError();
}

static int max_smem_optin() {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
    return v;
}

size_t scan_list_workspace_bytes(int64_t nq) {
    // pair slots (each segment rounds its count up), a flag per query
    return (size_t)(nq + 2 * kPairSeg) * sizeof(PairItem) + (size_t)nq + 64;
}

template <int KP>
static cudaError_t launch_list_kp(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq,
                                  int k, const ScanShape& sh, uint64_t* partials, uint8_t* work,
                                  int64_t pair_min_rows, int* launches, cudaStream_t s) {
    const bool m16 = sh.M == 16 && sh.row_bytes == 16 && sh.tab_words == 64;
    const size_t ps = scan_pair_smem_bytes(KP);
    const uint8_t* paired = nullptr;
    int nl = 0;
    if (m16 && work != nullptr && ps <= (size_t)max_smem_optin()) {
        // M = 16: long, overlapping ranges are paired by k_pair_items and
        // served by the two-query kernel; the one-query kernel takes the rest
        PairItem* items = reinterpret_cast<PairItem*>(work);
        uint8_t* pd = reinterpret_cast<uint8_t*>(items + nq + 2 * kPairSeg);
        const unsigned segs = (unsigned)((nq + kPairSeg - 1) / kPairSeg);
        k_pair_items<<<segs, kPairSortThreads, 0, s>>>(plan, nq, pair_min_rows, items, pd);
        cudaError_t e = cudaGetLastError();
        if (e != cudaSuccess) return e;
        if ((e = cudaFuncSetAttribute(k_scan_list_pair<KP>, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                      (int)ps)) != cudaSuccess)
            return e;
        dim3 grid((unsigned)((nq + 1) / 2), (unsigned)sh.n_chunks);   // at most nq / 2 pairs
        k_scan_list_pair<KP><<<grid, kPairThreads, ps, s>>>(tab, sc, plan, items, k, sh, partials);
        if ((e = cudaGetLastError()) != cudaSuccess) return e;
        paired = pd;
        nl = 2;
    }
    const size_t smem = scan_list_smem_bytes(sh.tab_words, KP);
    if (launches) *launches = nl + 1;
    if (m16) {
        if ((size_t)233472 / (smem + 1024) >= 2)
            return launch_list_one<KP, true, 2>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
        return launch_list_one<KP, true, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
    }
    return launch_list_one<KP, false, 1>(tab, sc, plan, nq, k, sh, partials, paired, smem, s);
}

cudaError_t launch_scan_list(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                             const ScanShape& sh, uint64_t* partials, uint8_t* work, int64_t pair_min_rows,
                             cudaStream_t s, int* launches) {
    if (launches) *launches = 0;
    if (nq <= 0) return cudaSuccess;
    switch (scan_kp(k)) {
        case 32: return launch_list_kp<32>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, launches, s);
        case 64: return launch_list_kp<64>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, launches, s);
        case 128: return launch_list_kp<128>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, launches, s);
        default: return launch_list_kp<256>(tab, sc, plan, nq, k, sh, partials, work, pair_min_rows, launches, s);
    }
}

// sorted copy: position p <- row rows[p] (stored rotated by (row mod 32) mod M)
// re-rotated by (p mod 32) mod M
__global__ void k_relayout_sorted(const uint8_t* __restrict__ src, const uint32_t* __restrict__ rows,
                                  int64_t N, int M, int row_bytes, int64_t n_rows_pad,
                                  uint8_t* __restrict__ dst) {
    const int64_t p = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (p >= n_rows_pad) return;
    uint8_t* out = dst + p * row_bytes;
    if (p >= N) {
        for (int s = 0; s < row_bytes; ++s) out[s] = 0;
        return;
    }
    const uint32_t row = rows[p];
    const uint8_t* in = src + (int64_t)row * row_bytes;
    const int rot_r = (int)(row & 31u) % M;
    const int rot_p = (int)(p & 31) % M;
    for (int s = 0; s < row_bytes; ++s) {
        uint8_t v = 0;
        if (s < M) {
            // byte s must hold subspace (s + rot_p) mod M, stored in `in` at
            // byte (s + rot_p - rot_r) mod M
            int t = s + rot_p - rot_r;
            t %= M;
            if (t < 0) t += M;
            v = in[t];
        }
        out[s] = v;
    }
}

cudaError_t launch_relayout_sorted(const uint8_t* src, const uint32_t* rows, int64_t N, int M,
                                   int row_bytes, int64_t n_rows_pad, uint8_t* dst, cudaStream_t s) {
    const int threads = 256;
    const int64_t blocks = (n_rows_pad + threads - 1) / threads;
    k_relayout_sorted<<<(unsigned)blocks, threads, 0, s>>>(src, rows, N, M, row_bytes, n_rows_pad, dst);
    return cudaGetLastError();
}

// ---- index layout -----------------------------------------------------------

__global__ void k_relayout_codes(const uint8_t* __restrict__ src, int64_t N, int M, int K,
                                 int row_bytes, int64_t n_rows_pad, uint8_t* __restrict__ dst,
                                 int* __restrict__ bad) {
    const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= n_rows_pad) return;
    uint8_t* out = dst + i * row_bytes;
    if (i >= N) {
        for (int s = 0; s < row_bytes; ++s) out[s] = 0;
        return;
    }
    const int rot = (int)(i & 31) % M;
    const uint8_t* in = src + i * M;
    int any_bad = 0;
    for (int s = 0; s < row_bytes; ++s) {
        uint8_t v = 0;
        if (s < M) {
            int m = s + rot;
            if (m >= M) m -= M;
            v = in[m];
            any_bad |= (int)v >= K;
        }
        out[s] = v;
    }
    if (any_bad) atomicOr(bad, 1);
}

cudaError_t launch_relayout_codes(const uint8_t* src, int64_t N, int M, int K, int row_bytes,
                                  int64_t n_rows_pad, uint8_t* dst, int* bad, cudaStream_t s) {
    const int threads = 256;
    const int64_t blocks = (n_rows_pad + threads - 1) / threads;
    k_relayout_codes<<<(unsigned)blocks, threads, 0, s>>>(src, N, M, K, row_bytes, n_rows_pad,
                                                         dst, bad);
    return cudaGetLastError();
}

}  // namespace ifvs
