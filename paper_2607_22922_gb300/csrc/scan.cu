// Rank (§2 stage 2) over a pass bitmap, with the per-CTA part of Select:
// the bitmap-path scan kernel k_scan, and the re-layout kernels that build
// the code rows the scans read (the index layout and the sorted copies).
// The design shared by all scan kernels is described in scan_common.cuh.
#include "scan_common.cuh"

namespace ifvs {

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

template <int KP, int MM, bool FAST>
__device__ __forceinline__ void scan_chunk(const uint8_t* __restrict__ codes,
                                           const uint32_t* __restrict__ bmq, const ScanShape& sh,
                                           int64_t b0, int64_t b1, const float* tab,
                                           uint32_t* ring, WarpTopK<KP>& tk, int lane, int warp) {
    const int M = MM > 0 ? MM : sh.M;
    const int S = MM > 0 ? 64 : sh.tab_words;
    const int row_bytes = sh.row_bytes;
    const uint32_t base = (uint32_t)__cvta_generic_to_shared(tab);
    const uint32_t tb = 4u * (uint32_t)lane;

    const uint64_t keep = policy_evict_last();
    const int64_t first = b0 + warp;
    const int T = first < b1 ? (int)((b1 - first + kScanWarps - 1) / kScanWarps) : 0;
    auto word_addr = [&](int t) { return bmq + (first + (int64_t)t * kScanWarps) * 32 + lane; };

    // ring: words of the blocks t in [F - kRing, F) in slot t % kRing;
    // dense: bit t % kRing set when block t has at least kDenseRows passing
    // rows (warp-uniform)
    uint32_t dense = 0u;
    auto mark = [&](int t, uint32_t w) {
        const unsigned n = __reduce_add_sync(0xFFFFFFFFu, (unsigned)__popc(w));
        const uint32_t bit = 1u << (t % kRing);
        dense = n >= (unsigned)kDenseRows ? (dense | bit) : (dense & ~bit);
    };
    int F = T < kRing ? T : kRing;
#pragma unroll
    for (int i = 0; i < kRing; ++i)
        if (i < F) {
            const uint32_t w = ldg_nc_u32(word_addr(i), policy_evict_first());
            ring[i * 32 + lane] = w;
            mark(i, w);
        }
    uint32_t pf[kHalf];
    int npf = T - F < kHalf ? T - F : kHalf;
#pragma unroll
    for (int i = 0; i < kHalf; ++i) pf[i] = i < npf ? ldg_nc_u32(word_addr(F + i), policy_evict_first()) : 0u;
    __syncwarp();
    // a lane stops at every dense block (held) until the whole warp has
    // reached it, so all lanes wait at the same block
    int pos = 0;
    uint32_t cur = F > 0 ? ring[lane] : 0u;
    bool held = F > 0 && (dense & 1u) != 0u;
    auto advance = [&]() {
        while (cur == 0u && !held && pos + 1 < F) {
            ++pos;
            cur = ring[(pos % kRing) * 32 + lane];
            held = (dense >> (pos % kRing) & 1u) != 0u;
        }
    };

    int col = -1;   // >= 0: the warp is in the dense block at pos, at this column
    for (;;) {
        uint32_t row[kU];
        unsigned valid = 0u;
        if (col < 0) {
            const int slow = (int)__reduce_min_sync(0xFFFFFFFFu, (unsigned)pos);
            if (npf > 0 && slow >= F - kHalf) {
#pragma unroll
                for (int i = 0; i < kHalf; ++i)
                    if (i < npf) {
                        ring[((F + i) % kRing) * 32 + lane] = pf[i];
                        mark(F + i, pf[i]);
                    }
                F += npf;
                npf = T - F < kHalf ? T - F : kHalf;
                const uint64_t once = policy_evict_first();
#pragma unroll
                for (int i = 0; i < kHalf; ++i) pf[i] = i < npf ? ldg_nc_u32(word_addr(F + i), once) : 0u;
                __syncwarp();
            }
            // lanes whose word is used up move on before the mode is chosen
            advance();
            if (__all_sync(0xFFFFFFFFu, held)) col = 0;
        }
        if (col >= 0) {
            // a dense block in lockstep: kU columns, 32 neighbouring rows
            // per column, lanes whose row fails masked
            const uint32_t rb = (uint32_t)((first + (int64_t)pos * kScanWarps) * kBlockRows) + 32u * (uint32_t)col + lane;
#pragma unroll
            for (int u = 0; u < kU; ++u) row[u] = rb + 32u * (uint32_t)u;
            valid = cur >> col & ((1u << kU) - 1u);
            col += kU;
            if (col == 32) {
                col = -1;
                cur = 0u;
                held = false;
            }
        } else {
            // up to kU passing rows of this lane
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                advance();
                row[u] = 0u;
                if (cur != 0u && !held) {
                    const int j = __ffs(cur) - 1;
                    cur &= cur - 1u;
                    row[u] = (uint32_t)((first + (int64_t)pos * kScanWarps) * kBlockRows) + 32u * (uint32_t)j + lane;
                    valid |= 1u << u;
                }
            }
            if (__ballot_sync(0xFFFFFFFFu, valid != 0u) == 0u) {
                // every lane is held at a dense block or out of words
                if (F >= T && !__any_sync(0xFFFFFFFFu, held)) break;
                continue;
            }
        }
        // rows whose bit is clear are read too, unmasked (a row of the
        // block in lockstep, row 0 otherwise), but never offered
        if constexpr (MM > 0) {
            uint4 c[kU];
#pragma unroll
            for (int u = 0; u < kU; ++u) c[u] = ldg_nc_v4(codes + (size_t)row[u] * 16, keep);
            float d[kU];
#pragma unroll
            for (int u = 0; u < kU; u += 2) lookup2<MM, FAST>(c[u], c[u + 1], tb, tb, base, d[u], d[u + 1]);
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
            lookup_rows<kU>(codes, row, (1u << kU) - 1u, row_bytes, M, S, tab, lane, d);
#pragma unroll
            for (int u = 0; u < kU; ++u) {
                const bool pass = valid >> u & 1u;
                const uint64_t key = ((uint64_t)__float_as_uint(d[u]) << 32) | row[u];
                tk.offer(key, pass && key < tk.thr, lane);
            }
        }
    }
}

template <int KP, int MM, int MINB>
__global__ void __launch_bounds__(kScanThreads, MINB)
k_scan(const uint8_t* __restrict__ codes, const float* __restrict__ tables,
       const uint32_t* __restrict__ bm, const ScanPlan* __restrict__ plan, int64_t nq, int k,
       ScanShape sh, uint64_t* __restrict__ partials) {
    extern __shared__ __align__(256) uint8_t smem[];
    const int S = MM > 0 ? 64 : sh.tab_words;
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
    if constexpr (MM > 0) {
        if (fast)
            scan_chunk<KP, MM, true>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
        else
            scan_chunk<KP, MM, false>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
    } else {
        scan_chunk<KP, 0, false>(codes, bmq, sh, b0, b1, tab, ring, tk, lane, warp);
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

template <int KP, int MM, int MINB>
static cudaError_t launch_one(const uint8_t* codes, const float* tab, const uint32_t* bm,
                              const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                              uint64_t* partials, size_t smem, cudaStream_t s) {
    cudaError_t e = cudaFuncSetAttribute(k_scan<KP, MM, MINB>,
                                         cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    k_scan<KP, MM, MINB><<<grid, kScanThreads, smem, s>>>(codes, tab, bm, plan, nq, k, sh, partials);
    return cudaGetLastError();
}

template <int KP>
static cudaError_t launch_scan_kp(const uint8_t* codes, const float* tab, const uint32_t* bm,
                                  const ScanPlan* plan, int64_t nq, int k, const ScanShape& sh,
                                  uint64_t* partials, cudaStream_t s) {
    const int mm = fixed_m(sh);
    const size_t smem = scan_smem_bytes(sh.tab_words, KP);
    const bool two = scan_ctas_per_sm(sh.tab_words, KP) >= 2;
    if (mm == 16)
        return two ? launch_one<KP, 16, 2>(codes, tab, bm, plan, nq, k, sh, partials, smem, s)
                   : launch_one<KP, 16, 1>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
    if (mm == 12)
        return two ? launch_one<KP, 12, 2>(codes, tab, bm, plan, nq, k, sh, partials, smem, s)
                   : launch_one<KP, 12, 1>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
    return launch_one<KP, 0, 1>(codes, tab, bm, plan, nq, k, sh, partials, smem, s);
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
