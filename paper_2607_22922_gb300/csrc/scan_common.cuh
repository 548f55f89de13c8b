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
// registers, once every lane has left the older half.  Lanes at different
// blocks read rows that lie far apart, one cache line per lane; a block
// with at least kDenseRows passing rows (of 1024) is therefore taken in
// lockstep instead: each lane stops at it until the whole warp has arrived,
// then the warp walks its 32 columns, 32 neighbouring rows per load, with
// the lanes whose row fails masked.
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
#pragma once
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
#ifndef IFVS_SCAN_DENSE
#define IFVS_SCAN_DENSE 448
#endif
constexpr int kScanWarps = IFVS_SCAN_WARPS;
constexpr int kScanThreads = kScanWarps * 32;
constexpr int kRing = IFVS_SCAN_RING;    // bitmap words per lane in the ring
constexpr int kHalf = kRing / 2;
constexpr int kU = IFVS_SCAN_ROWS;       // rows per lane per round (even)
constexpr int kDenseRows = IFVS_SCAN_DENSE;   // passing rows from which a block goes in lockstep
static_assert(kRing <= 32 && 32 % kU == 0, "one mask bit per ring slot; whole column groups");

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

// a[0, n) and a[n, 2n) ascending (n a power of two) -> a[0, n) holds the n
// smallest keys of both, ascending; a[n, 2n) is left unspecified.  The first
// step pairs a[i] with a[2n-1-i] (the second run read backwards, which makes
// the 2n keys one bitonic sequence) and keeps the smaller key: the n smallest
// of the union, as a bitonic sequence; the half-cleaners of a bitonic merge
// then sort it.
__device__ __forceinline__ void warp_merge_low(uint64_t* a, int n, int lane) {
    __syncwarp();
    for (int i = lane; i < n; i += 32) {
        const uint64_t x = a[i], y = a[2 * n - 1 - i];
        if (y < x) a[i] = y;
    }
    for (int stride = n >> 1; stride > 0; stride >>= 1) {
        __syncwarp();
        for (int t = lane; t < (n >> 1); t += 32) {
            const int i = 2 * t - (t & (stride - 1));
            const int j = i + stride;
            const uint64_t x = a[i], y = a[j];
            if (x > y) {
                a[i] = y;
                a[j] = x;
            }
        }
    }
    __syncwarp();
}

// Merges a warp's candidates [KP, 2KP) of buf into its sorted list [0, KP),
// clears the candidates, publishes the new k-th key to the CTA's bound (if
// any) and returns it.  For KP >= 64 the candidates are sorted and the KP
// smallest of both runs kept by one bitonic merge (half the compare-
// exchanges of one sort of 2 KP); for KP = 32 both take the same number of
// steps and one sort of 64 measured faster (sift1m 693k against 599k
// queries/s; 10^8 rows at KP = 128: 0.1 % and 1 % bins 1.51 -> 1.41 and
// 4.33 -> 4.04 ms with the merge).  Out of line: the scan loops offer keys
// at many sites and flush rarely, and one copy of the sort keeps their code
// small (instruction-fetch stalls led the two-query kernel's profile).
template <int KP>
#ifndef IFVS_FLUSH_INLINE
__device__ __noinline__
#else
__device__ __forceinline__
#endif
uint64_t flush_list(uint64_t* buf, int k, uint64_t* cta, int lane) {
    if constexpr (KP <= 32) {
        warp_sort(buf, 2 * KP, lane);
    } else {
        warp_sort(buf + KP, KP, lane);
        warp_merge_low(buf, KP, lane);
    }
    const uint64_t thr = buf[k - 1];
    for (int i = KP + lane; i < 2 * KP; i += 32) buf[i] = ~0ull;
    if (cta != nullptr && lane == 0 && thr != ~0ull) atomicMin(reinterpret_cast<unsigned long long*>(cta), thr);
    __syncwarp();
    return thr;
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
        thr = flush_list<KP>(buf, k, cta, lane);
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

// Distances of two rows of MM <= 16 subspaces (codes ca, cb: 16-byte rows,
// table rows of 64 words).  One byte permute forms code * 256 + 4 * w0, w0 =
// the row's index mod 32 (the lane that owns it in the bitmap path); FAST
// (table at kDynSmemBase): the table base and the step go into the load's
// immediate offset; otherwise the base is added.
template <int MM, bool FAST>
__device__ __forceinline__ void lookup2(const uint4 ca, const uint4 cb, uint32_t tba, uint32_t tbb,
                                        uint32_t base, float& da, float& db) {
    static_assert(MM >= 1 && MM <= 16, "16-byte rows");
    const uint32_t wa[4] = {ca.x, ca.y, ca.z, ca.w};
    const uint32_t wb[4] = {cb.x, cb.y, cb.z, cb.w};
    uint64_t acc = 0ull;
#pragma unroll
    for (int s = 0; s < MM; ++s) {
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

// ---- bulk copies into shared memory (cp.async.bulk) and their mbarriers ----
//
// The untiled form of TMA: one instruction copies a contiguous, 16-byte
// aligned run of global memory into shared memory and reports its bytes to
// an mbarrier (complete_tx); threads wait on the barrier's phase parity.
// Every wait is bounded (kWaitCycles SM cycles, about half a second at
// 2 GHz): a wait that runs out returns false and the kernel reports it.

constexpr long long kWaitCycles = 1ll << 30;

__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
    asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}

// makes barrier initialisations visible to the bulk-copy (async) proxy
__device__ __forceinline__ void fence_mbar_init() {
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}

// orders this thread's earlier shared-memory accesses before later
// bulk-copy writes to the same bytes
__device__ __forceinline__ void fence_proxy_async_smem() {
    asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// one arrival that also announces `bytes` of bulk-copy traffic
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
    asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes) : "memory");
}

// global -> shared copy of `bytes` (a multiple of 16, both addresses 16-byte
// aligned), completion counted on `bar`, with an L2 cache policy
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes, uint32_t bar,
                                         uint64_t pol) {
    asm volatile(
        "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes.L2::cache_hint [%0], [%1], %2, [%3], "
        "%4;" ::"r"(dst),
        "l"(src), "r"(bytes), "r"(bar), "l"(pol)
        : "memory");
}

// a thread whose phase has not completed may sleep in the instruction for
// up to kSuspendNs (it wakes when the phase completes) instead of spinning;
// 0: no hint (the hardware's own time limit)
#ifndef IFVS_SUSPEND_NS
#define IFVS_SUSPEND_NS 20000
#endif
constexpr uint32_t kSuspendNs = IFVS_SUSPEND_NS;

__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
    uint32_t ok;
    if constexpr (kSuspendNs > 0) {
        asm volatile(
            "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\tselp.u32 %0, 1, 0, "
            "p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity), "n"(kSuspendNs)
            : "memory");
    } else {
        asm volatile(
            "{\n\t.reg .pred p;\n\tmbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\tselp.u32 %0, 1, 0, p;\n\t}"
            : "=r"(ok)
            : "r"(bar), "r"(parity)
            : "memory");
    }
    return ok != 0u;
}

// Waits, with every lane of the warp, until the barrier's phase of parity
// `parity` has completed; false (for the whole warp) when kWaitCycles pass
// first.
__device__ __forceinline__ bool mbar_wait_warp(uint32_t bar, uint32_t parity) {
    const long long t0 = clock64();
    for (;;) {
        const bool ok = mbar_try_wait(bar, parity);
        if (__all_sync(0xFFFFFFFFu, ok)) return true;
        if (__any_sync(0xFFFFFFFFu, clock64() - t0 > kWaitCycles)) return false;
    }
}

// largest dynamic shared memory per CTA the current device allows (opt-in)
inline int max_smem_optin() {
    int dev = 0, v = 0;
    if (cudaGetDevice(&dev) != cudaSuccess) return 0;
    if (cudaDeviceGetAttribute(&v, cudaDevAttrMaxSharedMemoryPerBlockOptin, dev) != cudaSuccess) return 0;
    return v;
}

// Subspace count the fixed-M scan loops are compiled for when the index
// stores 16-byte rows with 64-word tables (M = 12 rows padded to 16 bytes,
// or M = 16); 0: the generic-M loop.
inline int fixed_m(const ScanShape& sh) {
    if (sh.row_bytes != 16 || sh.tab_words != 64) return 0;
    return (sh.M == 16 || sh.M == 12) ? sh.M : 0;
}

// Two-query scan of the sorted copy (scan_pair.cu): pairs the list-path
// queries of `plan` whose ranges overlap enough (k_pair_items) and serves
// the pairs; `work` receives the pair items and a flag per query, *paired
// points at the flags (null when no pair kernel ran), *launches += kernels.
cudaError_t launch_pairs(const float* tab, SortedCols sc, const ScanPlan* plan, int64_t nq, int k,
                         const ScanShape& sh, uint64_t* partials, uint8_t* work, int64_t pair_min_rows,
                         cudaStream_t s, const uint8_t** paired, int* launches);

}  // namespace ifvs
