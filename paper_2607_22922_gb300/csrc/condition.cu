// Conditioning and table build of §2.
//
// k_condition (one CTA per query): the pair <q, f> is fingerprinted by h
// hash functions into the memory bank (FNV-1a-64 of the key bytes, then the
// SplitMix64 finalizer of base XOR seed_i, mod B — the paper names no hash
// function), alpha = sum of the h fetched bank rows, and the filter weights
// w_f = softplus(w_z) (w_f = 1 when no w_z is given: the paper's initial
// state).
//
// k_lut (grid: subspace m x query group; thread = codeword k): the
// adjustment Delta[m][k][:] = sum_j alpha[m][j] W[m][j][k][:] is formed with
// the thread's slice of W held in registers across the whole query group,
// C_iFVS = C_PQ + Delta, and the weighted ADC table
// LUT[m][k] = sum_t w_f[m ds + t] (q[m ds + t] - C_iFVS[m][k][t])^2, which
// turns the Rank score of §2 into an additive distance (score = sum w q^2 -
// dist).  C_iFVS is only written out on request.
#include "internal.cuh"

namespace ifvs {

__device__ __forceinline__ uint64_t fnv_byte(uint64_t h, uint32_t byte) {
    return (h ^ (uint64_t)byte) * 1099511628211ull;
}

__device__ __forceinline__ uint64_t fnv_word(uint64_t h, uint64_t v, int nbytes) {
    for (int b = 0; b < nbytes; ++b) h = fnv_byte(h, (uint32_t)(v >> (8 * b)) & 0xFFu);
    return h;
}

__device__ __forceinline__ uint64_t splitmix64_finalizer(uint64_t z) {
    z = (z ^ (z >> 30)) * 0xbf58476d1ce4e5b9ull;
    z = (z ^ (z >> 27)) * 0x94d049bb133111ebull;
    return z ^ (z >> 31);
}

__device__ __forceinline__ float softplus_f32(float x) {
    // log(1 + e^x) without overflow on either side
    return x > 0.f ? x + log1pf(expf(-x)) : log1pf(expf(x));
}

__global__ void k_condition(const float* __restrict__ q, const ifvs_predicate* __restrict__ preds,
                            int64_t nq, int D, const uint64_t* __restrict__ seeds, int h,
                            int64_t B, const float* __restrict__ bank, int Mr,
                            const float* __restrict__ wz, uint32_t* __restrict__ idx_out,
                            float* __restrict__ alpha, float* __restrict__ wf) {
    const int64_t qi = blockIdx.x;
    __shared__ uint32_t s_idx[64];
    const float* qv = q + qi * D;
    if (bank != nullptr) {
        if (threadIdx.x == 0) {
            uint64_t hsh = 14695981039346656037ull;
            for (int d = 0; d < D; ++d) hsh = fnv_word(hsh, __float_as_uint(qv[d]), 4);
            const ifvs_predicate& p = preds[qi];
            int nc = p.n_clauses;
            hsh = fnv_word(hsh, (uint32_t)nc, 4);
            if (nc < 0) nc = 0;
            if (nc > IFVS_MAX_CLAUSES) nc = IFVS_MAX_CLAUSES;
            for (int i = 0; i < nc; ++i) {
                hsh = fnv_word(hsh, (uint32_t)p.c[i].col, 4);
                hsh = fnv_word(hsh, (uint32_t)p.c[i].op, 4);
                hsh = fnv_word(hsh, (uint64_t)p.c[i].lo, 8);
                hsh = fnv_word(hsh, (uint64_t)p.c[i].hi, 8);
            }
            for (int i = 0; i < h; ++i)
                s_idx[i] = (uint32_t)(splitmix64_finalizer(hsh ^ seeds[i]) % (uint64_t)B);
        }
        __syncthreads();
        if (idx_out != nullptr)
            for (int i = threadIdx.x; i < h; i += blockDim.x) idx_out[qi * h + i] = s_idx[i];
        for (int t = threadIdx.x; t < Mr; t += blockDim.x) {
            float a = 0.f;
            for (int i = 0; i < h; ++i) a += bank[(int64_t)s_idx[i] * Mr + t];
            alpha[qi * Mr + t] = a;
        }
    }
    for (int d = threadIdx.x; d < D; d += blockDim.x)
        wf[qi * D + d] = wz != nullptr ? softplus_f32(wz[qi * D + d]) : 1.0f;
}

cudaError_t launch_condition(const float* q, const ifvs_predicate* preds, int64_t nq, int D,
                             const uint64_t* seeds, int h, int64_t B, const float* bank, int Mr,
                             const float* wz, uint32_t* idx, float* alpha, float* wf,
                             cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    k_condition<<<(unsigned)nq, 128, 0, s>>>(q, preds, nq, D, seeds, h, B, bank, Mr, wz, idx,
                                             alpha, wf);
    return cudaGetLastError();
}

// Fixed (ds, r): the thread keeps W[m][:][k][:] and C_PQ[m][k][:] in registers.
template <int DS, int R>
__global__ void __launch_bounds__(256) k_lut_fixed(const float* __restrict__ cpq,
                                                   const float* __restrict__ W,
                                                   const float* __restrict__ alpha,
                                                   const float* __restrict__ q,
                                                   const float* __restrict__ wf, int64_t nq,
                                                   int M, int K, int q_per_cta,
                                                   float* __restrict__ lut,
                                                   float* __restrict__ cifvs) {
    const int m = blockIdx.x;
    const int k = threadIdx.x;
    if (k >= K) return;
    const int D = M * DS;
    float c0[DS];
    float w[R][DS];
#pragma unroll
    for (int t = 0; t < DS; ++t) c0[t] = cpq[((int64_t)m * K + k) * DS + t];
    if (alpha != nullptr) {
#pragma unroll
        for (int j = 0; j < R; ++j)
#pragma unroll
            for (int t = 0; t < DS; ++t) w[j][t] = W[(((int64_t)m * R + j) * K + k) * DS + t];
    }
    const int64_t q0 = (int64_t)blockIdx.y * q_per_cta;
    const int64_t q1 = min(nq, q0 + (int64_t)q_per_cta);
    for (int64_t qi = q0; qi < q1; ++qi) {
        float c[DS];
        if (alpha != nullptr) {
            float a[R];
#pragma unroll
            for (int j = 0; j < R; ++j) a[j] = alpha[(qi * M + m) * R + j];
#pragma unroll
            for (int t = 0; t < DS; ++t) {
                float delta = 0.f;
#pragma unroll
                for (int j = 0; j < R; ++j) delta = fmaf(a[j], w[j][t], delta);
                c[t] = c0[t] + delta;
            }
        } else {
#pragma unroll
            for (int t = 0; t < DS; ++t) c[t] = c0[t];
        }
        float s = 0.f;
#pragma unroll
        for (int t = 0; t < DS; ++t) {
            const float diff = q[qi * D + m * DS + t] - c[t];
            s = fmaf(wf[qi * D + m * DS + t] * diff, diff, s);
        }
        lut[(qi * M + m) * K + k] = s;
        if (cifvs != nullptr) {
#pragma unroll
            for (int t = 0; t < DS; ++t) cifvs[((qi * M + m) * K + k) * DS + t] = c[t];
        }
    }
}

// Any (ds, r): W and C_PQ are read through the cache inside the query loop.
__global__ void __launch_bounds__(256) k_lut_any(const float* __restrict__ cpq,
                                                 const float* __restrict__ W,
                                                 const float* __restrict__ alpha,
                                                 const float* __restrict__ q,
                                                 const float* __restrict__ wf, int64_t nq, int M,
                                                 int K, int ds, int r, int q_per_cta,
                                                 float* __restrict__ lut,
                                                 float* __restrict__ cifvs) {
    const int m = blockIdx.x;
    const int k = threadIdx.x;
    if (k >= K) return;
    const int D = M * ds;
    const int64_t q0 = (int64_t)blockIdx.y * q_per_cta;
    const int64_t q1 = min(nq, q0 + (int64_t)q_per_cta);
    for (int64_t qi = q0; qi < q1; ++qi) {
        float s = 0.f;
        for (int t = 0; t < ds; ++t) {
            float delta = 0.f;
            if (alpha != nullptr)
                for (int j = 0; j < r; ++j)
                    delta = fmaf(alpha[(qi * M + m) * r + j],
                                 __ldg(W + (((int64_t)m * r + j) * K + k) * ds + t), delta);
            const float c = __ldg(cpq + ((int64_t)m * K + k) * ds + t) + delta;
            const float diff = q[qi * D + m * ds + t] - c;
            s = fmaf(wf[qi * D + m * ds + t] * diff, diff, s);
            if (cifvs != nullptr) cifvs[((qi * M + m) * K + k) * ds + t] = c;
        }
        lut[(qi * M + m) * K + k] = s;
    }
}

cudaError_t launch_lut(const float* cpq, const float* W, const float* alpha, const float* q,
                       const float* wf, int64_t nq, int M, int K, int ds, int r, float* lut,
                       float* cifvs, int num_sms, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    // query groups: enough CTAs to cover the GPU, while each CTA reuses its
    // registers' W slice across as many queries as possible
    int64_t groups = ((int64_t)num_sms * 4 + M - 1) / M;
    if (groups > nq) groups = nq;
    if (groups < 1) groups = 1;
    if (groups > 65535) groups = 65535;
    const int64_t qpc = (nq + groups - 1) / groups;
    groups = (nq + qpc - 1) / qpc;
    dim3 grid((unsigned)M, (unsigned)groups);
    const int threads = K <= 32 ? 32 : (K <= 64 ? 64 : (K <= 128 ? 128 : 256));
    if (ds == 8 && (r == 8 || alpha == nullptr))
        k_lut_fixed<8, 8><<<grid, threads, 0, s>>>(cpq, W, alpha, q, wf, nq, M, K, (int)qpc,
                                                   lut, cifvs);
    else
        k_lut_any<<<grid, threads, 0, s>>>(cpq, W, alpha, q, wf, nq, M, K, ds, r, (int)qpc, lut,
                                           cifvs);
    return cudaGetLastError();
}

// ---- scan tables -------------------------------------------------------------
//
// The scan keeps each query's table in shared memory as 256 rows (one per
// codeword) of S words, word w of row c = LUT[w mod M][c] for w < M + 31
// (zero above).  This kernel writes that layout once per query so that every
// scan CTA fetches it with coalesced 16-byte loads.  Grid: query x 32-codeword
// tile; the tile passes through shared memory padded to 33 words per row so
// that both the coalesced reads and the rotated writes are conflict-free.
__global__ void __launch_bounds__(256) k_tables(const float* __restrict__ lut, int M, int K, int S,
                                                float* __restrict__ tab) {
    __shared__ float st[IFVS_MAX_M * 33];
    const int64_t q = blockIdx.x;
    const int c0 = blockIdx.y * 32;
    const float* src = lut + q * (int64_t)M * K;
    for (int i = threadIdx.x; i < M * 32; i += blockDim.x) {
        const int m = i >> 5, cc = i & 31, c = c0 + cc;
        st[m * 33 + cc] = c < K ? src[(int64_t)m * K + c] : 0.f;
    }
    __syncthreads();
    float* dst = tab + q * (int64_t)256 * S + (int64_t)c0 * S;
    const int wu = M + 31;
    for (int i = threadIdx.x; i < 32 * S; i += blockDim.x) {
        const int cc = i / S, w = i - cc * S;
        dst[i] = w < wu ? st[(w % M) * 33 + cc] : 0.f;
    }
}

cudaError_t launch_tables(const float* lut, int64_t nq, int M, int K, int S, float* tab,
                          cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    dim3 grid((unsigned)nq, 8);
    k_tables<<<grid, 256, 0, s>>>(lut, M, K, S, tab);
    return cudaGetLastError();
}

}  // namespace ifvs
