// Stage 1 of §2 (Filter): every row's attribute values are tested against
// the query's predicate (the conjunctive form of Listing 1), giving the
// candidate pool P as a pass bitmap.
//
// One warp owns one 1024-row block: lane l holds the 32 attribute values of
// rows b*1024 + 32*j + l (j = 0..31), loaded with 32 coalesced 128-byte
// column reads, and then evaluates every query of its group against them,
// so the columns are read once per query group.  The lane's 32 pass bits
// form its word of the lane-major bitmap directly (no ballot needed), one
// 128-byte store per warp and query.  Popcounts go through a warp reduction
// into npass.
#include "internal.cuh"

namespace ifvs {

__global__ void k_canonicalize(const ifvs_predicate* __restrict__ preds, int64_t nq,
                               AttrCols cols, CanonPred* __restrict__ out, int* __restrict__ err) {
    int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (i >= nq) return;
    ifvs_predicate p = preds[i];
    CanonPred c;
    if (canonicalize(p, cols.type, cols.n, &c) != 0) atomicOr(err, 1);
    out[i] = c;
}

cudaError_t launch_canonicalize(const ifvs_predicate* preds, int64_t nq, AttrCols cols,
                                CanonPred* out, int* err, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    int threads = 128;
    int64_t blocks = (nq + threads - 1) / threads;
    k_canonicalize<<<(unsigned)blocks, threads, 0, s>>>(preds, nq, cols, out, err);
    return cudaGetLastError();
}

// Scan plan.  A predicate that constrains one column selects, for that
// column's canonical interval [lo, lo + wm1], a contiguous segment of the
// rows sorted by (value, row): two binary searches give it, and its length
// is the exact pool size.  Pools up to max_rows take the row-list scan (no
// filter pass, no bitmap); empty and malformed predicates take it with an
// empty segment, and a predicate that constrains no column (every row
// passes) takes it with all N positions of column 0's copy; every other
// query takes the bitmap path.
__device__ __forceinline__ int64_t first_not_below(const int32_t* __restrict__ v, int64_t n, int64_t x) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if ((int64_t)v[mid] < x)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

__device__ __forceinline__ int64_t first_key_not_below(const uint64_t* __restrict__ v, int64_t n, uint64_t x) {
    int64_t lo = 0, hi = n;
    while (lo < hi) {
        const int64_t mid = (lo + hi) >> 1;
        if (v[mid] < x)
            lo = mid + 1;
        else
            hi = mid;
    }
    return lo;
}

__global__ void k_plan(const CanonPred* __restrict__ canon, int64_t nq, SortedCols sc, int64_t N,
                       int64_t max_rows, ScanPlan* __restrict__ plan,
                       unsigned long long* __restrict__ npass) {
    const int64_t q = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= nq) return;
    const CanonPred cp = canon[q];
    ScanPlan p;
    p.a = 0;
    p.b = 0;
    p.col = 0;
    p.list = 0;
    if (cp.empty) {
        p.list = 1;
    } else if (cp.used == 0u) {
        if (sc.n > 0 && sc.vals_of(0) != nullptr && N <= max_rows) {
            p.b = N;
            p.list = 1;
        }
    } else if (__popc(cp.used) == 1) {
        const int c = __ffs(cp.used) - 1;
        const int32_t* vals = sc.vals_of(c);
        if (c < sc.n && vals != nullptr) {
            int64_t lo = 0, wm1 = 0;
#pragma unroll
            for (int i = 0; i < IFVS_MAX_ATTRS; ++i)
                if (c == i) {
                    lo = cp.lo[i];
                    wm1 = cp.wm1[i];
                }
            const int64_t hi = lo + wm1;
            const int64_t a = first_not_below(vals, N, lo);
            const int64_t b = first_not_below(vals, N, hi + 1);
            if (b - a <= max_rows) {
                p.a = a;
                p.b = b;
                p.col = c;
                p.list = 1;
            }
        }
    } else if (cp.used == 3u && sc.ckeys[0] != nullptr && (cp.wm1[0] == 0u || cp.wm1[1] == 0u)) {
        // columns 0 and 1, one of them fixed to a value: a position range of
        // the composite copy keyed by that column first
        const int j = cp.wm1[0] == 0u ? 0 : 1;
        const int32_t v = cp.lo[j];
        const int32_t lo2 = cp.lo[1 - j];
        const uint32_t w2 = cp.wm1[1 - j];
        const uint64_t* keys = sc.ckeys_of(j);
        const int64_t a = first_key_not_below(keys, N, ckey(v, lo2));
        // one past (v, lo2 + w2): the next composite key (carries into the
        // primary half when the secondary value is the largest int32)
        const uint64_t kh = ckey(v, (int32_t)((uint32_t)lo2 + w2));
        const int64_t b = kh == ~0ull ? N : first_key_not_below(keys, N, kh + 1ull);
        if (b - a <= max_rows) {
            p.a = a;
            p.b = b;
            p.col = kComposite + j;
            p.list = 1;
        }
    }
    plan[q] = p;
    if (p.list) npass[q] = (unsigned long long)(p.b - p.a);
}

cudaError_t launch_plan(const CanonPred* canon, int64_t nq, SortedCols sc, int64_t N, int64_t max_rows,
                        ScanPlan* plan, unsigned long long* npass, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    k_plan<<<(unsigned)((nq + 127) / 128), 128, 0, s>>>(canon, nq, sc, N, max_rows, plan, npass);
    return cudaGetLastError();
}

// Fail bits of 8 rows against one interval, shifted into `fail` (row j0 + 7
// first, so that after four calls bit j is row j).  For each row:
// off = v - lo (mod 2^32); the carry out of off + ~wm1 is 1 exactly when
// off > wm1, i.e. when the row fails; addc shifts the carry in.  The carry
// never leaves the asm block.
__device__ __forceinline__ uint32_t fail8(uint32_t fail, const int32_t* v, int32_t lo, uint32_t nwm1) {
    asm("{\n\t.reg .u32 t;\n\t"
        "sub.u32 t, %8, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %7, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %6, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %5, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %4, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %3, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %2, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "sub.u32 t, %1, %9;\n\tadd.cc.u32 t, t, %10;\n\taddc.u32 %0, %0, %0;\n\t"
        "}"
        : "+r"(fail)
        : "r"(v[0]), "r"(v[1]), "r"(v[2]), "r"(v[3]), "r"(v[4]), "r"(v[5]), "r"(v[6]), "r"(v[7]),
          "r"(lo), "r"(nwm1));
    return fail;
}

constexpr int kFilterQ = 256;   // queries staged in shared memory at a time

template <int NA>
__global__ void __launch_bounds__(kThreads) k_filter(AttrCols cols, int64_t N, int64_t n_blocks,
                                                     const CanonPred* __restrict__ canon,
                                                     const ScanPlan* __restrict__ plan,
                                                     int64_t nq, int q_per_cta,
                                                     uint32_t* __restrict__ bm,
                                                     unsigned long long* __restrict__ npass) {
    static_assert(kThreads >= kFilterQ, "one staging pass per query group");
    __shared__ int2 s_iv[kFilterQ][NA];      // (lo, ~wm1) per query and column
    __shared__ uint32_t s_keep[kFilterQ];    // 0 for a predicate no row can pass
    __shared__ uint32_t s_used[kFilterQ];
    __shared__ int s_q[kFilterQ];            // query (offset from the group start)
    __shared__ int s_wcnt[kWarps];
    const int lane = threadIdx.x & 31;
    const int64_t b = (int64_t)blockIdx.x * kWarps + (threadIdx.x >> 5);
    const bool live = b < n_blocks;
    const int64_t q0 = (int64_t)blockIdx.y * q_per_cta;
    const int64_t q1 = min(nq, q0 + (int64_t)q_per_cta);
    const int64_t row0 = (live ? b : 0) * kBlockRows + lane;

    // rows beyond N keep their bits at 0 (columns are padded, so the loads
    // themselves stay inside the allocation)
    uint32_t valid = 0xFFFFFFFFu;
    if (b * kBlockRows + kBlockRows > N) {
        valid = 0;
#pragma unroll
        for (int j = 0; j < 32; ++j) valid |= (uint32_t)(row0 + 32 * j < N) << j;
    }

    int32_t v[NA][32];
#pragma unroll
    for (int c = 0; c < NA; ++c) {
        if (cols.type[c] == IFVS_ATTR_I16) {
            const int16_t* col = (const int16_t*)cols.col[c] + row0;
#pragma unroll
            for (int j = 0; j < 32; ++j) v[c][j] = __ldg(col + 32 * j);
        } else {
            const int32_t* col = (const int32_t*)cols.col[c] + row0;
#pragma unroll
            for (int j = 0; j < 32; ++j) v[c][j] = __ldg(col + 32 * j);
        }
    }

    const int64_t words = n_blocks * 32;
    const int warp = threadIdx.x >> 5;
    for (int64_t g0 = q0; g0 < q1; g0 += kFilterQ) {
        const int ng = (int)min((int64_t)kFilterQ, q1 - g0);
        __syncthreads();
        // stage the group's bitmap-path queries, in order (list-path queries
        // need no bitmap and cost nothing here)
        const int t = threadIdx.x;
        const bool mine = t < ng && (plan == nullptr || !plan[g0 + t].list);
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, mine);
        if (lane == 0) s_wcnt[warp] = __popc(bal);
        __syncthreads();
        int pos = __popc(bal & ((1u << lane) - 1u));
        for (int w = 0; w < warp; ++w) pos += s_wcnt[w];
        int ngd = 0;
        for (int w = 0; w < kWarps; ++w) ngd += s_wcnt[w];
        if (mine) {
            const CanonPred cp = canon[g0 + t];
#pragma unroll
            for (int c = 0; c < NA; ++c) s_iv[pos][c] = make_int2(cp.lo[c], (int32_t)~cp.wm1[c]);
            s_keep[pos] = cp.empty ? 0u : 0xFFFFFFFFu;
            s_used[pos] = cp.used;
            s_q[pos] = t;
        }
        __syncthreads();
        if (!live) continue;
        for (int i = 0; i < ngd; ++i) {
            uint32_t m = valid & s_keep[i];
            const uint32_t used = s_used[i];
#pragma unroll
            for (int c = 0; c < NA; ++c) {
                if (NA == 1 || (used >> c & 1u)) {
                    const int2 iv = s_iv[i][c];
                    uint32_t fail = 0;
#pragma unroll
                    for (int j8 = 24; j8 >= 0; j8 -= 8) fail = fail8(fail, &v[c][j8], iv.x, (uint32_t)iv.y);
                    m &= ~fail;
                }
            }
            const int64_t q = g0 + s_q[i];
            bm[q * words + b * 32 + lane] = m;
            const unsigned cnt = __reduce_add_sync(0xFFFFFFFFu, (unsigned)__popc(m));
            if (lane == 0 && cnt) atomicAdd(npass + q, (unsigned long long)cnt);
        }
    }
}

cudaError_t launch_filter(AttrCols cols, int64_t N, int64_t n_blocks, const CanonPred* canon,
                          const ScanPlan* plan, int64_t nq, uint32_t* bm, unsigned long long* npass,
                          int num_sms, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    const int64_t tiles = (n_blocks + kWarps - 1) / kWarps;
    // enough CTAs to fill the GPU a few times over; each CTA walks a group
    // of queries so that a column tile is read once per group
    const int64_t target = (int64_t)num_sms * 8;
    int64_t groups = (target + tiles - 1) / tiles;
    if (groups < 1) groups = 1;
    if (groups > nq) groups = nq;
    if (groups > 65535) groups = 65535;
    const int64_t qpc = (nq + groups - 1) / groups;
    groups = (nq + qpc - 1) / qpc;
    dim3 grid((unsigned)tiles, (unsigned)groups);
    int na = cols.n < 1 ? 1 : cols.n;
    switch (na) {
        case 1: k_filter<1><<<grid, kThreads, 0, s>>>(cols, N, n_blocks, canon, plan, nq, (int)qpc, bm, npass); break;
        case 2: k_filter<2><<<grid, kThreads, 0, s>>>(cols, N, n_blocks, canon, plan, nq, (int)qpc, bm, npass); break;
        case 3: k_filter<3><<<grid, kThreads, 0, s>>>(cols, N, n_blocks, canon, plan, nq, (int)qpc, bm, npass); break;
        default: k_filter<4><<<grid, kThreads, 0, s>>>(cols, N, n_blocks, canon, plan, nq, (int)qpc, bm, npass); break;
    }
    return cudaGetLastError();
}

// ---- layout conversion ---------------------------------------------------

// Transpose the 32x32 bit matrix held one row per lane (lane l, bit j =
// element (l, j)) so that lane l ends up with column l.  Five butterfly
// stages swap the off-diagonal s x s sub-blocks for s = 16, 8, 4, 2, 1.
__device__ __forceinline__ uint32_t transpose32(uint32_t x, int lane) {
    const uint32_t masks[5] = {0x0000FFFFu, 0x00FF00FFu, 0x0F0F0F0Fu, 0x33333333u, 0x55555555u};
#pragma unroll
    for (int i = 0; i < 5; ++i) {
        const int s = 16 >> i;
        const uint32_t mk = masks[i];
        const uint32_t y = __shfl_xor_sync(0xFFFFFFFFu, x, s);
        x = (lane & s) ? ((x & ~mk) | ((y >> s) & mk)) : ((x & mk) | ((y & mk) << s));
    }
    return x;
}

__global__ void k_bitmap_layout(const uint32_t* __restrict__ src, uint32_t* __restrict__ dst,
                                int64_t nq, int64_t n_blocks, int64_t n_words_rows,
                                bool to_rows) {
    const int lane = threadIdx.x & 31;
    const int64_t gw = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    if (gw >= nq * n_blocks) return;
    const int64_t q = gw / n_blocks, b = gw - q * n_blocks;
    const int64_t lm = q * n_blocks * 32 + b * 32 + lane;
    const int64_t ri = b * 32 + lane;
    const int64_t rows_off = q * n_words_rows + ri;
    uint32_t x;
    if (to_rows) {
        x = src[lm];
    } else {
        x = ri < n_words_rows ? src[rows_off] : 0u;
    }
    // lane-major word (b, l) bit j == row-ordered word (b*32 + j) bit l
    x = transpose32(x, lane);
    if (to_rows) {
        if (ri < n_words_rows) dst[rows_off] = x;
    } else {
        dst[lm] = x;
    }
}

cudaError_t launch_bitmap_layout(const uint32_t* src, uint32_t* dst, int64_t nq,
                                 int64_t n_blocks, int64_t n_words_rows, bool to_rows,
                                 cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    const int64_t warps = nq * n_blocks;
    const int threads = 256;
    const int64_t blocks = (warps * 32 + threads - 1) / threads;
    k_bitmap_layout<<<(unsigned)blocks, threads, 0, s>>>(src, dst, nq, n_blocks, n_words_rows,
                                                        to_rows);
    return cudaGetLastError();
}

}  // namespace ifvs
