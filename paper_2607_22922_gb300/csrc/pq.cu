// Building the PQ index on the GPU (the offline step before the query path
// of §2: the base codebook C_PQ and the uint8 codes stay fixed afterwards).
//
// k_pq_assign: one thread per row; the whole codebook of the current
// subspace sits in shared memory and every lane of a warp reads the same
// codeword (broadcast); two codewords are measured at once with packed
// float32 differences and squares.  The distance to a codeword is accumulated in
// float32 in a fixed order — s = s + (x_t - c_t)^2 for t ascending, every
// operation rounded on its own (no fused multiply-add) — and the argmin
// keeps the smallest codeword on ties, so the codes are bit-exact with the
// same decision made in float32 on the CPU.
//
// k_pq_accumulate: one Lloyd update per subspace.  Each CTA adds its rows'
// vectors into per-codeword fp64 sums in shared memory, then adds those into
// the global sums (one atomic per accumulator per CTA).  k_pq_finalize turns
// the sums into float32 means; an empty codeword keeps its old value until
// the host gives it the farthest point (k_pq_farthest: largest float32
// distance, ties to the smallest row, by a 64-bit atomic max on
// (distance bits << 32 | ~row)).
#include "internal.cuh"

namespace ifvs {

constexpr int kPqThreads = 256;

// packed float32 pairs: each half is rounded on its own, as two scalar
// operations with the same rounding would be (explicit .rn: never fused)
__device__ __forceinline__ unsigned long long f2_sub(unsigned long long a, unsigned long long b) {
    unsigned long long d;
    asm("sub.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long f2_mul(unsigned long long a, unsigned long long b) {
    unsigned long long d;
    asm("mul.rn.f32x2 %0, %1, %2;" : "=l"(d) : "l"(a), "l"(b));
    return d;
}
__device__ __forceinline__ unsigned long long f2_dup(float x) {
    unsigned long long d;
    asm("mov.b64 %0, {%1, %1};" : "=l"(d) : "f"(x));
    return d;
}
__device__ __forceinline__ void f2_split(unsigned long long v, float& lo, float& hi) {
    asm("mov.b64 {%0, %1}, %2;" : "=f"(lo), "=f"(hi) : "l"(v));
}

// Codewords 2p and 2p+1 of one subspace are interleaved in shared memory as
// [p][t][2], so one 16-byte broadcast load gives both codewords' values at
// t and t+1; an odd K keeps its last codeword in plain [t] order after the
// pairs.  Differences and squares of both codewords run packed; the two
// sums stay scalar: a packed multiply feeding a packed add is compiled into
// a fused multiply-add (one rounding instead of two) even with explicit
// .rn, volatile asm and -fmad=false, which would change the float32 sums.
// The first term needs no add (0 + sq = sq exactly).
template <int DS>
__device__ __forceinline__ void pair_dist(const float* __restrict__ cbp,
                                          const unsigned long long (&xx)[DS], float& s0,
                                          float& s1) {
    static_assert(DS % 2 == 0, "pairs of dimensions");
    const ulonglong2* c = reinterpret_cast<const ulonglong2*>(cbp);
#pragma unroll
    for (int t = 0; t < DS; t += 2) {
        const ulonglong2 cc = c[t / 2];
        const unsigned long long d0 = f2_sub(xx[t], cc.x);
        const unsigned long long d1 = f2_sub(xx[t + 1], cc.y);
        float a0, b0, a1, b1;
        f2_split(f2_mul(d0, d0), a0, b0);
        f2_split(f2_mul(d1, d1), a1, b1);
        if (t == 0) {
            s0 = a0;
            s1 = b0;
        } else {
            s0 = __fadd_rn(s0, a0);
            s1 = __fadd_rn(s1, b0);
        }
        s0 = __fadd_rn(s0, a1);
        s1 = __fadd_rn(s1, b1);
    }
}

template <int DS>
__global__ void __launch_bounds__(kPqThreads) k_pq_assign(const float* __restrict__ X, int64_t n,
                                                          int D, int M, int K,
                                                          const float* __restrict__ C,
                                                          uint8_t* __restrict__ codes,
                                                          float* __restrict__ dmin) {
    extern __shared__ __align__(16) float cb[];   // K * DS floats of one subspace, pairs interleaved
    const int64_t i = (int64_t)blockIdx.x * kPqThreads + threadIdx.x;
    const int KP = K >> 1;
    for (int m = 0; m < M; ++m) {
        __syncthreads();
        for (int e = threadIdx.x; e < K * DS; e += kPqThreads) {
            const int k = e / DS, t = e - k * DS;
            const int dst = k < 2 * KP ? ((k >> 1) * DS + t) * 2 + (k & 1) : e;
            cb[dst] = C[(int64_t)m * K * DS + e];
        }
        __syncthreads();
        if (i >= n) continue;
        unsigned long long xx[DS];
#pragma unroll
        for (int t = 0; t < DS; ++t) xx[t] = f2_dup(__ldg(X + i * D + m * DS + t));
        float best = 0.f;
        int bk = 0;
        if (KP > 0) {
            float s0, s1;
            pair_dist<DS>(cb, xx, s0, s1);
            best = s0;
            if (s1 < best) {
                best = s1;
                bk = 1;
            }
        }
#pragma unroll 4
        for (int p = 1; p < KP; ++p) {
            float s0, s1;
            pair_dist<DS>(cb + p * DS * 2, xx, s0, s1);
            if (s0 < best) {
                best = s0;
                bk = 2 * p;
            }
            if (s1 < best) {
                best = s1;
                bk = 2 * p + 1;
            }
        }
        if (K & 1) {
            const float* c = cb + (K - 1) * DS;
            float s = 0.f;
#pragma unroll
            for (int t = 0; t < DS; ++t) {
                float x, unused;
                f2_split(xx[t], x, unused);
                const float d = __fsub_rn(x, c[t]);
                s = __fadd_rn(s, __fmul_rn(d, d));
            }
            if (KP == 0 || s < best) {
                best = s;
                bk = K - 1;
            }
        }
        codes[i * M + m] = (uint8_t)bk;
        if (dmin != nullptr) dmin[i * M + m] = best;
    }
}

// any ds: the same arithmetic with a runtime loop
__global__ void __launch_bounds__(kPqThreads) k_pq_assign_any(const float* __restrict__ X, int64_t n,
                                                              int D, int M, int K, int ds,
                                                              const float* __restrict__ C,
                                                              uint8_t* __restrict__ codes,
                                                              float* __restrict__ dmin) {
    extern __shared__ __align__(16) float cb[];
    const int64_t i = (int64_t)blockIdx.x * kPqThreads + threadIdx.x;
    for (int m = 0; m < M; ++m) {
        __syncthreads();
        for (int e = threadIdx.x; e < K * ds; e += kPqThreads) cb[e] = C[(int64_t)m * K * ds + e];
        __syncthreads();
        if (i >= n) continue;
        const float* x = X + i * D + m * ds;
        float best = 0.f;
        int bk = 0;
        for (int k = 0; k < K; ++k) {
            float s = 0.f;
            for (int t = 0; t < ds; ++t) {
                const float d = __fsub_rn(__ldg(x + t), cb[k * ds + t]);
                s = __fadd_rn(s, __fmul_rn(d, d));
            }
            if (k == 0 || s < best) {
                best = s;
                bk = k;
            }
        }
        codes[i * M + m] = (uint8_t)bk;
        if (dmin != nullptr) dmin[i * M + m] = best;
    }
}

cudaError_t launch_pq_assign(const float* X, int64_t n, int D, int M, int K, const float* C,
                             uint8_t* codes, float* dmin, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    const int ds = D / M;
    const size_t smem = (size_t)K * ds * sizeof(float);
    const int64_t blocks = (n + kPqThreads - 1) / kPqThreads;
    cudaError_t e;
    if (ds == 8) {
        e = cudaFuncSetAttribute(k_pq_assign<8>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_pq_assign<8><<<(unsigned)blocks, kPqThreads, smem, s>>>(X, n, D, M, K, C, codes, dmin);
    } else {
        e = cudaFuncSetAttribute(k_pq_assign_any, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_pq_assign_any<<<(unsigned)blocks, kPqThreads, smem, s>>>(X, n, D, M, K, ds, C, codes, dmin);
    }
    return cudaGetLastError();
}

// sums [M][K][ds] fp64 and counts [M][K] (zeroed by the caller)
__global__ void __launch_bounds__(kPqThreads) k_pq_accumulate(const float* __restrict__ X, int64_t n,
                                                              int D, int M, int K, int ds,
                                                              int64_t rows_per_cta,
                                                              const uint8_t* __restrict__ codes,
                                                              double* __restrict__ sums,
                                                              unsigned long long* __restrict__ counts) {
    extern __shared__ __align__(16) double acc[];   // K * ds sums, then K counts
    unsigned long long* cnt = reinterpret_cast<unsigned long long*>(acc + (size_t)K * ds);
    const int64_t r0 = (int64_t)blockIdx.x * rows_per_cta;
    const int64_t r1 = min(n, r0 + rows_per_cta);
    for (int m = 0; m < M; ++m) {
        __syncthreads();
        for (int e = threadIdx.x; e < K * ds; e += kPqThreads) acc[e] = 0.0;
        for (int e = threadIdx.x; e < K; e += kPqThreads) cnt[e] = 0ull;
        __syncthreads();
        for (int64_t i = r0 + threadIdx.x; i < r1; i += kPqThreads) {
            const int c = codes[i * M + m];
            atomicAdd(cnt + c, 1ull);
            for (int t = 0; t < ds; ++t) atomicAdd(acc + c * ds + t, (double)__ldg(X + i * D + m * ds + t));
        }
        __syncthreads();
        for (int e = threadIdx.x; e < K * ds; e += kPqThreads)
            if (acc[e] != 0.0) atomicAdd(sums + (int64_t)m * K * ds + e, acc[e]);
        for (int e = threadIdx.x; e < K; e += kPqThreads)
            if (cnt[e] != 0ull) atomicAdd(counts + (int64_t)m * K + e, cnt[e]);
    }
}

__global__ void k_pq_finalize(const double* __restrict__ sums,
                              const unsigned long long* __restrict__ counts, int M, int K, int ds,
                              const float* __restrict__ C_in, float* __restrict__ C_out) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e >= (int64_t)M * K * ds) return;
    const int64_t mk = e / ds;
    const unsigned long long c = counts[mk];
    C_out[e] = c > 0 ? (float)(sums[e] / (double)c) : C_in[e];
}

// key = (float bits of dmin[i][m] << 32) | ~i (32-bit); the max is the
// largest distance, ties to the smallest row
__global__ void k_pq_farthest(const float* __restrict__ dmin, int64_t n, int M, int m,
                              unsigned long long* __restrict__ best) {
    unsigned long long local = 0ull;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x) {
        const unsigned long long key =
            ((unsigned long long)__float_as_uint(dmin[i * M + m]) << 32) |
            (unsigned long long)(0xFFFFFFFFu - (uint32_t)i);
        local = key > local ? key : local;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long other = __shfl_xor_sync(0xFFFFFFFFu, local, o);
        local = other > local ? other : local;
    }
    if ((threadIdx.x & 31) == 0) atomicMax(best, local);
}

// the empty codeword c of subspace m takes row `far`; its distance becomes 0
__global__ void k_pq_reseed(const float* __restrict__ X, int D, int M, int K, int ds, int m, int c,
                            const unsigned long long* __restrict__ best, float* __restrict__ C_out,
                            float* __restrict__ dmin) {
    const int64_t far = (int64_t)(0xFFFFFFFFu - (uint32_t)(*best & 0xFFFFFFFFull));
    const int t = threadIdx.x;
    if (t < ds) C_out[((int64_t)m * K + c) * ds + t] = X[far * D + m * ds + t];
    __syncthreads();
    if (t == 0) dmin[far * M + m] = 0.f;
}

cudaError_t launch_pq_update(const float* X, int64_t n, int D, int M, int K, const uint8_t* codes,
                             double* sums, unsigned long long* counts, const float* C_in,
                             float* C_out, int num_sms, cudaStream_t s) {
    const int ds = D / M;
    cudaError_t e = cudaMemsetAsync(sums, 0, sizeof(double) * (size_t)M * K * ds, s);
    if (e == cudaSuccess) e = cudaMemsetAsync(counts, 0, sizeof(unsigned long long) * (size_t)M * K, s);
    if (e != cudaSuccess) return e;
    if (n > 0) {
        const size_t smem = (size_t)K * ds * sizeof(double) + (size_t)K * sizeof(unsigned long long);
        e = cudaFuncSetAttribute(k_pq_accumulate, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        const int64_t ctas = (int64_t)num_sms * 2;
        int64_t rows = (n + ctas - 1) / ctas;
        if (rows < kPqThreads) rows = kPqThreads;
        const int64_t grid = (n + rows - 1) / rows;
        k_pq_accumulate<<<(unsigned)grid, kPqThreads, smem, s>>>(X, n, D, M, K, ds, rows, codes, sums, counts);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    const int64_t total = (int64_t)M * K * ds;
    k_pq_finalize<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(sums, counts, M, K, ds, C_in, C_out);
    return cudaGetLastError();
}

cudaError_t launch_pq_reseed(const float* X, int64_t n, int D, int M, int K, int m, int c,
                             unsigned long long* best, float* C_out, float* dmin, int num_sms,
                             cudaStream_t s) {
    const int ds = D / M;
    cudaError_t e = cudaMemsetAsync(best, 0, sizeof(unsigned long long), s);
    if (e != cudaSuccess) return e;
    int64_t grid = (n + 255) / 256;
    if (grid > (int64_t)num_sms * 8) grid = (int64_t)num_sms * 8;
    if (grid < 1) grid = 1;
    k_pq_farthest<<<(unsigned)grid, 256, 0, s>>>(dmin, n, M, m, best);
    e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    k_pq_reseed<<<1, ds < 32 ? 32 : ds, 0, s>>>(X, D, M, K, ds, m, c, best, C_out, dmin);
    return cudaGetLastError();
}

// objective[m] += sum over rows of dmin[i][m] (fp64), objective zeroed by the caller
__global__ void k_pq_objective(const float* __restrict__ dmin, int64_t n, int M,
                               double* __restrict__ objective) {
    const int m = blockIdx.y;
    double local = 0.0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n;
         i += (int64_t)gridDim.x * blockDim.x)
        local += (double)dmin[i * M + m];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) local += __shfl_xor_sync(0xFFFFFFFFu, local, o);
    if ((threadIdx.x & 31) == 0 && local != 0.0) atomicAdd(objective + m, local);
}

cudaError_t launch_pq_objective(const float* dmin, int64_t n, int M, double* objective, int num_sms,
                                cudaStream_t s) {
    cudaError_t e = cudaMemsetAsync(objective, 0, sizeof(double) * M, s);
    if (e != cudaSuccess || n <= 0) return e;
    int64_t gx = (n + 255) / 256;
    if (gx > (int64_t)num_sms * 4) gx = (int64_t)num_sms * 4;
    dim3 grid((unsigned)gx, (unsigned)M);
    k_pq_objective<<<grid, 256, 0, s>>>(dmin, n, M, objective);
    return cudaGetLastError();
}

}  // namespace ifvs
