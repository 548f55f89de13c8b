// Stage 3 of §2 (Select) across CTAs, and the optional exact rerank.
//
// k_merge: one CTA per query folds the per-chunk lists of k keys
// (dist bits << 32 | row) into the query's k smallest with a block bitonic
// sort in shared memory; keys are unique, so ties in distance fall to the
// smaller row id exactly as the definition asks.
//
// k_merge_shards: Select across row shards.  Each of G shards returns its
// k best (dist, global row id) per query; one CTA per query sorts the G k
// entries by (dist, id) — a block bitonic sort on an order-preserving
// integer image of the distance and the id (padding, id -1, sorts last) —
// and keeps the k smallest.
//
// k_rerank: one CTA per query computes the exact fp32 squared L2 distance
// (the Pre_IndexFlatL2 distance of §3.2) between the query and each
// candidate's raw vector — one warp per candidate, lanes over dimensions,
// a fixed-order shuffle reduction — and keeps the k best the same way.
#include <math.h>

#include "internal.cuh"

namespace ifvs {

__device__ __forceinline__ void block_sort(uint64_t* a, int n) {
    for (int size = 2; size <= n; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < (n >> 1); t += blockDim.x) {
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
    __syncthreads();
}

__device__ __forceinline__ void write_key(uint64_t key, int64_t* id, float* d) {
    if (key == ~0ull) {
        *id = -1;
        *d = INFINITY;
    } else {
        *id = (int64_t)(uint32_t)(key & 0xFFFFFFFFull);
        *d = __uint_as_float((uint32_t)(key >> 32));
    }
}

constexpr int kMergeCap = 4096;

__global__ void __launch_bounds__(256) k_merge(const uint64_t* __restrict__ partials, int n_lists,
                                               int k, int kp, int cap,
                                               int64_t* __restrict__ ids,
                                               float* __restrict__ dists) {
    __shared__ uint64_t a[kMergeCap];
    const int64_t q = blockIdx.x;
    const int64_t total = (int64_t)n_lists * k;
    const uint64_t* src = partials + q * total;
    for (int i = threadIdx.x; i < kp; i += blockDim.x) a[i] = ~0ull;
    for (int64_t pos = 0; pos < total; pos += cap - kp) {
        for (int i = threadIdx.x; i < cap - kp; i += blockDim.x)
            a[kp + i] = pos + i < total ? src[pos + i] : ~0ull;
        block_sort(a, cap);
    }
    __syncthreads();
    for (int i = threadIdx.x; i < k; i += blockDim.x) write_key(a[i], ids + q * k + i, dists + q * k + i);
}

cudaError_t launch_merge(const uint64_t* partials, int64_t nq, int n_lists, int k, int64_t* ids,
                         float* dists, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    int kp = 32;
    while (kp < k) kp <<= 1;
    int cap = 64;
    const int64_t need = (int64_t)n_lists * k + kp;
    while (cap < need && cap < kMergeCap) cap <<= 1;
    if (cap < 2 * kp) cap = 2 * kp;
    k_merge<<<(unsigned)nq, 256, 0, s>>>(partials, n_lists, k, kp, cap, ids, dists);
    return cudaGetLastError();
}

constexpr int kShardMergeCap = 4096;   // G * k entries per query, at most

// float -> uint32 whose unsigned order is the float order (NaN aside)
__device__ __forceinline__ uint32_t float_order(float x) {
    const uint32_t b = __float_as_uint(x);
    return (b & 0x80000000u) ? ~b : (b | 0x80000000u);
}

__global__ void __launch_bounds__(512) k_merge_shards(const float* __restrict__ dists, const int64_t* __restrict__ ids,
                                                      int64_t nq, int G, int k, int n,
                                                      float* __restrict__ dists_out, int64_t* __restrict__ ids_out) {
    __shared__ uint32_t dk[kShardMergeCap];
    __shared__ uint64_t ik[kShardMergeCap];
    const int64_t q = blockIdx.x;
    for (int i = threadIdx.x; i < n; i += blockDim.x) {
        uint32_t d = 0xFFFFFFFFu;
        uint64_t id = ~0ull;
        if (i < G * k) {
            const int g = i / k, j = i - g * k;
            const int64_t at = ((int64_t)g * nq + q) * k + j;
            const int64_t r = ids[at];
            if (r >= 0) {
                d = float_order(dists[at]);
                id = (uint64_t)r;
            }
        }
        dk[i] = d;
        ik[i] = id;
    }
    for (int size = 2; size <= n; size <<= 1)
        for (int stride = size >> 1; stride > 0; stride >>= 1) {
            __syncthreads();
            for (int t = threadIdx.x; t < (n >> 1); t += blockDim.x) {
                const int i = 2 * t - (t & (stride - 1));
                const int j = i + stride;
                const bool up = (i & size) == 0;
                const uint32_t dx = dk[i], dy = dk[j];
                const uint64_t ix = ik[i], iy = ik[j];
                const bool gt = dx > dy || (dx == dy && ix > iy);
                if (gt == up) {
                    dk[i] = dy;
                    dk[j] = dx;
                    ik[i] = iy;
                    ik[j] = ix;
                }
            }
        }
    __syncthreads();
    for (int i = threadIdx.x; i < k; i += blockDim.x) {
        const bool pad = ik[i] == ~0ull;
        const uint32_t b = dk[i];
        ids_out[q * k + i] = pad ? -1 : (int64_t)ik[i];
        dists_out[q * k + i] = pad ? INFINITY : __uint_as_float((b & 0x80000000u) ? (b & 0x7FFFFFFFu) : ~b);
    }
}

int shard_merge_cap() { return kShardMergeCap; }

cudaError_t launch_merge_shards(const float* dists, const int64_t* ids, int64_t nq, int G, int k,
                                float* dists_out, int64_t* ids_out, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    int n = 2;
    while (n < G * k) n <<= 1;
    k_merge_shards<<<(unsigned)nq, 512, 0, s>>>(dists, ids, nq, G, k, n, dists_out, ids_out);
    return cudaGetLastError();
}

__global__ void __launch_bounds__(256) k_rerank(const float* __restrict__ X, int64_t N, int D,
                                                const float* __restrict__ q,
                                                const int64_t* __restrict__ cand, int R, int k,
                                                int rp, int64_t* __restrict__ ids,
                                                float* __restrict__ dists) {
    __shared__ uint64_t a[IFVS_MAX_K];
    const int64_t qi = blockIdx.x;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    for (int i = threadIdx.x; i < rp; i += blockDim.x) a[i] = ~0ull;
    __syncthreads();
    const float* qv = q + qi * D;
    for (int j = warp; j < R; j += 8) {
        const int64_t id = cand[qi * R + j];
        if (id < 0 || id >= N) continue;
        const float* x = X + id * D;
        float s = 0.f;
        for (int d = lane; d < D; d += 32) {
            const float diff = qv[d] - x[d];
            s = fmaf(diff, diff, s);
        }
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        if (lane == 0) a[j] = ((uint64_t)__float_as_uint(s) << 32) | (uint64_t)(uint32_t)id;
    }
    block_sort(a, rp);
    for (int i = threadIdx.x; i < k; i += blockDim.x) write_key(a[i], ids + qi * k + i, dists + qi * k + i);
}

cudaError_t launch_rerank(const float* X, int64_t N, int D, const float* q, const int64_t* cand,
                          int64_t nq, int R, int k, int64_t* ids, float* dists, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    int rp = 32;
    while (rp < R) rp <<= 1;
    k_rerank<<<(unsigned)nq, 256, 0, s>>>(X, N, D, q, cand, R, k, rp, ids, dists);
    return cudaGetLastError();
}

}  // namespace ifvs
