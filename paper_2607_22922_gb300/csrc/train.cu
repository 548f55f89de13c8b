// Learning the memory bank, W and w_f (§2 "Learning"), one mini-batch of
// queries per step.  The loss (per positive g: softmax cross-entropy of g
// against the mined hard negatives N at temperature tau, averaged over the
// query's positives; plus lambda ||Delta||^2; averaged over the queries) and
// its gradient:
//   dL/ddist_g = (1 - p_g) / tau / |G|,   dL/ddist_n = -sum_g p_n(g) / tau / |G|
//   dL/dC[m][c_v[m]][t] = sum_v gamma_v (-2 w_f (q - C))        (gC, sparse)
//   dL/dw_f[d]          = sum_v gamma_v (q - C)^2
//   dL/dDelta           = gC + 2 lambda Delta,   Delta = alpha . W
//   dL/dW[m][j]         = sum_q alpha_q[m][j] gC_q[m] + 2 lambda sum_j' A_m[j][j'] W[m][j']
//                         with A_m = sum_q alpha_q[m] alpha_q[m]^T
//   dL/dalpha_q[m][j]   = <gC_q[m], W[m][j]> + 2 lambda sum_j' G_m[j][j'] alpha_q[m][j']
//                         with the Gram matrix G_m = W[m] W[m]^T
//   dL/dbank[b]         = sum over the fetches (q, i) with idx_i(q) = b of dL/dalpha_q
//   dL/dw_z             = dL/dw_f sigmoid(w_z)
// (each divided by the number of queries).  Every sum runs in a fixed order
// (no atomics), so a step is deterministic.
#include "internal.cuh"

namespace ifvs {

namespace {
constexpr int kTrainThreads = 256;
constexpr int kTrainWarps = kTrainThreads / 32;

__device__ __forceinline__ double warp_sum(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v += __shfl_xor_sync(0xFFFFFFFFu, v, o);
    return v;
}
__device__ __forceinline__ double warp_min(double v) {
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) v = fmin(v, __shfl_xor_sync(0xFFFFFFFFu, v, o));
    return v;
}
}  // namespace

__global__ void k_broadcast_wz(const float* __restrict__ wz, int D, int64_t n, float* __restrict__ out) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e < n * D) out[e] = wz[e % D];
}

// G[m][j][j'] = sum over (k, t) of W[m][j][k][t] W[m][j'][k][t]; one CTA per entry
__global__ void __launch_bounds__(kTrainThreads) k_train_gram(const float* __restrict__ W, int M,
                                                              int r, int KD, float* __restrict__ G) {
    __shared__ float part[kTrainWarps];
    const int b = blockIdx.x;
    const int m = b / (r * r), j = (b / r) % r, j2 = b % r;
    const float* a = W + ((int64_t)m * r + j) * KD;
    const float* c = W + ((int64_t)m * r + j2) * KD;
    float s = 0.f;
    for (int e = threadIdx.x; e < KD; e += kTrainThreads) s += a[e] * c[e];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < kTrainWarps; ++w) t += part[w];
        G[b] = t;
    }
}

// One CTA per query: candidate list, distances, softmax weights, loss, the
// scatter of dL/dC into the query's dense gC slice and dL/dw_f.  Each thread
// owns the dimensions d = tid + i * blockDim, so every gC address (m, *, t)
// is written by one thread only, in candidate order.
__global__ void __launch_bounds__(kTrainThreads) k_train_query(TrainQueryArgs a) {
    extern __shared__ __align__(16) unsigned char sm[];
    const int V = a.P + a.n_neg;
    const int Mr = a.M * a.r;
    int64_t* cand = reinterpret_cast<int64_t*>(sm);
    double* part = reinterpret_cast<double*>(cand + V);       // [V][warps]
    double* dist = part + (size_t)V * kTrainWarps;            // [V]
    double* gam = dist + V;                                   // [V]
    double* red = gam + V;                                    // [warps]
    float* alpha = reinterpret_cast<float*>(red + kTrainWarps);   // [Mr]
    const int64_t q = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;

    if (tid == 0) {
        const int64_t* pos = a.pos + q * a.pos_stride;
        for (int g = 0; g < a.P; ++g) cand[g] = pos[g];
        const int64_t* src = a.negsrc + q * a.neg_stride;
        int got = 0;
        for (int s = 0; s < a.S && got < a.n_neg; ++s) {
            const int64_t id = src[s];
            if (a.exclude) {
                if (id < 0) break;
                bool is_pos = false;
                for (int g = 0; g < a.P; ++g) is_pos |= pos[g] == id;
                if (is_pos) continue;
            }
            cand[a.P + got++] = id;
        }
        for (; got < a.n_neg; ++got) cand[a.P + got] = -1;
        for (int v = 0; v < V; ++v)
            if (cand[v] < -1 || cand[v] >= a.N) {
                atomicOr(a.err, 2);
                cand[v] = -1;
            }
        if (a.neg_out)
            for (int n = 0; n < a.n_neg; ++n) a.neg_out[q * a.n_neg + n] = cand[a.P + n];
    }
    for (int e = tid; e < Mr; e += blockDim.x) alpha[e] = a.alpha[q * Mr + e];
    __syncthreads();

    const float* qv = a.q + q * a.D;
    const float* wf = a.wf + q * a.D;
    const int64_t KD = (int64_t)a.K * a.ds;

    // C_iFVS[m][c][t] = C_PQ + sum_j alpha[m][j] W[m][j][c][t] for the code of
    // candidate `id` in the subspace of dimension d; returns q_d - C
    auto diff_of = [&](int64_t id, int d, int* code) -> float {
        const int m = d / a.ds, t = d - m * a.ds;
        const int rot = (int)(id & 31) % a.M;
        int s = m - rot;
        if (s < 0) s += a.M;
        const int c = a.codes[id * a.row_bytes + s];
        *code = c;
        const int64_t e = (int64_t)c * a.ds + t;
        float C = a.C_pq[(int64_t)m * KD + e];
        for (int j = 0; j < a.r; ++j) C += alpha[m * a.r + j] * a.W[((int64_t)m * a.r + j) * KD + e];
        return qv[d] - C;
    };

    // pass 1: weighted distances (float32 terms, fp64 sums)
    for (int v = 0; v < V; ++v) {
        const int64_t id = cand[v];
        double acc = 0.0;
        if (id >= 0)
            for (int d = tid; d < a.D; d += blockDim.x) {
                int c;
                const float df = diff_of(id, d, &c);
                acc += (double)(wf[d] * df * df);
            }
        acc = warp_sum(acc);
        if (lane == 0) part[v * kTrainWarps + warp] = acc;
    }
    __syncthreads();
    for (int v = tid; v < V; v += blockDim.x) {
        double s = 0.0;
        for (int w = 0; w < kTrainWarps; ++w) s += part[v * kTrainWarps + w];
        dist[v] = s;
        gam[v] = 0.0;
    }
    __syncthreads();

    // softmax of each positive against the negatives (warp 0)
    if (warp == 0) {
        int npos = 0;
        double lpos = 0.0;
        for (int g = 0; g < a.P; ++g) {
            if (cand[g] < 0) continue;
            ++npos;
            double dm = dist[g];
            for (int n = a.P + lane; n < V; n += 32)
                if (cand[n] >= 0) dm = fmin(dm, dist[n]);
            dm = warp_min(dm);
            double z = 0.0;
            for (int n = a.P + lane; n < V; n += 32)
                if (cand[n] >= 0) z += exp(-(dist[n] - dm) / a.tau);
            z = warp_sum(z) + exp(-(dist[g] - dm) / a.tau);
            lpos += dist[g] / a.tau - dm / a.tau + log(z);
            for (int n = a.P + lane; n < V; n += 32)
                if (cand[n] >= 0) gam[n] -= exp(-(dist[n] - dm) / a.tau) / z / a.tau;
            if (lane == 0) gam[g] += (1.0 - exp(-(dist[g] - dm) / a.tau) / z) / a.tau;
            __syncwarp();
        }
        if (npos > 0) {
            for (int v = lane; v < V; v += 32) gam[v] /= npos;
            lpos /= npos;
        }
        if (lane == 0) red[0] = lpos;
    }
    // anchor ||Delta||^2 = sum_m alpha[m]^T G_m alpha[m]
    double an = 0.0;
    for (int m = tid; m < a.M; m += blockDim.x) {
        const float* Gm = a.G + (int64_t)m * a.r * a.r;
        for (int j = 0; j < a.r; ++j)
            for (int j2 = 0; j2 < a.r; ++j2)
                an += (double)alpha[m * a.r + j] * (double)Gm[j * a.r + j2] * (double)alpha[m * a.r + j2];
    }
    an = warp_sum(an);
    __syncthreads();
    const double lpos = red[0];
    __syncthreads();
    if (lane == 0) red[warp] = an;
    __syncthreads();
    if (tid == 0) {
        double s = 0.0;
        for (int w = 0; w < kTrainWarps; ++w) s += red[w];
        a.loss[q] = lpos + (double)a.lambda * s;
    }

    // pass 2: gC scatter and dL/dw_f
    float* gC = a.gC + q * (int64_t)a.M * KD;
    for (int d = tid; d < a.D; d += blockDim.x) {
        const int m = d / a.ds, t = d - m * a.ds;
        double gw = 0.0;
        for (int v = 0; v < V; ++v) {
            const int64_t id = cand[v];
            if (id < 0) continue;
            int c;
            const float df = diff_of(id, d, &c);
            const float gv = (float)gam[v];
            gC[(int64_t)m * KD + (int64_t)c * a.ds + t] += gv * (-2.f * wf[d] * df);
            gw += gam[v] * (double)(df * df);
        }
        a.gw[q * a.D + d] = (float)gw;
    }
}

// dL/dW[m][j][e] = inv_n (sum_q alpha_q[m][j] gC_q[m][e] + 2 lambda sum_j' A_m[j][j'] W[m][j'][e]);
// grid (M, ceil(KD / 256)); r <= kTrainMaxR
__global__ void __launch_bounds__(kTrainThreads) k_train_gW(const float* __restrict__ alpha,
                                                            const float* __restrict__ gC,
                                                            const float* __restrict__ W, int64_t n,
                                                            int M, int r, int KD, float lambda,
                                                            float inv_n, float* __restrict__ gW) {
    __shared__ float A[kTrainMaxR * kTrainMaxR];
    __shared__ float as[kTrainThreads * kTrainMaxR / 8];   // alpha of a chunk of queries
    const int m = blockIdx.x;
    const int e = blockIdx.y * kTrainThreads + threadIdx.x;
    const int Mr = M * r;
    for (int t = threadIdx.x; t < r * r; t += kTrainThreads) {
        const int j = t / r, j2 = t % r;
        float s = 0.f;
        for (int64_t q = 0; q < n; ++q) s += alpha[q * Mr + m * r + j] * alpha[q * Mr + m * r + j2];
        A[t] = s;
    }
    float acc[kTrainMaxR];
#pragma unroll
    for (int j = 0; j < kTrainMaxR; ++j) acc[j] = 0.f;
    const int qc = (kTrainThreads * kTrainMaxR / 8) / r;   // queries per staged chunk
    for (int64_t q0 = 0; q0 < n; q0 += qc) {
        const int nc = (int)min((int64_t)qc, n - q0);
        __syncthreads();
        for (int t = threadIdx.x; t < nc * r; t += kTrainThreads)
            as[t] = alpha[(q0 + t / r) * Mr + m * r + t % r];
        __syncthreads();
        if (e < KD)
            for (int i = 0; i < nc; ++i) {
                const float g = gC[((q0 + i) * M + m) * (int64_t)KD + e];
#pragma unroll
                for (int j = 0; j < kTrainMaxR; ++j)
                    if (j < r) acc[j] += as[i * r + j] * g;
            }
    }
    __syncthreads();
    if (e >= KD) return;
#pragma unroll
    for (int j = 0; j < kTrainMaxR; ++j) {
        if (j >= r) break;
        float an = 0.f;
        for (int j2 = 0; j2 < r; ++j2) an += A[j * r + j2] * W[((int64_t)m * r + j2) * KD + e];
        gW[((int64_t)m * r + j) * KD + e] = (acc[j] + 2.f * lambda * an) * inv_n;
    }
}

// dL/dalpha_q[m][j] = <gC_q[m], W[m][j]> + 2 lambda sum_j' G_m[j][j'] alpha_q[m][j'];
// grid (n, M)
__global__ void __launch_bounds__(kTrainThreads) k_train_galpha(const float* __restrict__ gC,
                                                                const float* __restrict__ W,
                                                                const float* __restrict__ G,
                                                                const float* __restrict__ alpha,
                                                                int M, int r, int KD, float lambda,
                                                                float* __restrict__ galpha) {
    __shared__ float part[kTrainWarps][kTrainMaxR];
    const int64_t q = blockIdx.x;
    const int m = blockIdx.y;
    const int Mr = M * r;
    const float* g = gC + (q * M + m) * (int64_t)KD;
    float acc[kTrainMaxR];
#pragma unroll
    for (int j = 0; j < kTrainMaxR; ++j) acc[j] = 0.f;
    for (int e = threadIdx.x; e < KD; e += kTrainThreads) {
        const float ge = g[e];
        if (ge == 0.f) continue;
#pragma unroll
        for (int j = 0; j < kTrainMaxR; ++j)
            if (j < r) acc[j] += ge * W[((int64_t)m * r + j) * KD + e];
    }
#pragma unroll
    for (int j = 0; j < kTrainMaxR; ++j) {
        float s = acc[j];
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
        if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5][j] = s;
    }
    __syncthreads();
    if (threadIdx.x < r) {
        const int j = threadIdx.x;
        float s = 0.f;
        for (int w = 0; w < kTrainWarps; ++w) s += part[w][j];
        float an = 0.f;
        for (int j2 = 0; j2 < r; ++j2) an += G[((int64_t)m * r + j) * r + j2] * alpha[q * Mr + m * r + j2];
        galpha[q * Mr + m * r + j] = s + 2.f * lambda * an;
    }
}

// dL/dbank: one CTA per fetch p = (q, i); the first fetch of each bank row
// sums, in fetch order, the dL/dalpha of every fetch of that row
__global__ void k_train_bank(const uint32_t* __restrict__ idx, int64_t n_fetch, int h, int Mr,
                             const float* __restrict__ galpha, float inv_n, float* __restrict__ gbank) {
    const int64_t p = blockIdx.x;
    const uint32_t b = idx[p];
    for (int64_t p2 = 0; p2 < p; ++p2)
        if (idx[p2] == b) return;
    for (int e = threadIdx.x; e < Mr; e += blockDim.x) {
        float s = 0.f;
        for (int64_t p2 = p; p2 < n_fetch; ++p2)
            if (idx[p2] == b) s += galpha[(p2 / h) * Mr + e];
        gbank[(int64_t)b * Mr + e] = s * inv_n;
    }
}

// dL/dw_z[d] = inv_n sum_q dL/dw_f[q][d] sigmoid(w_z[d])
__global__ void k_train_wz(const float* __restrict__ gw, int64_t n, int D, const float* __restrict__ wz,
                           float inv_n, float* __restrict__ gwz) {
    const int d = blockIdx.x * blockDim.x + threadIdx.x;
    if (d >= D) return;
    double s = 0.0;
    for (int64_t q = 0; q < n; ++q) s += (double)gw[q * D + d];
    const float x = wz[d];
    const float sg = x >= 0.f ? 1.f / (1.f + expf(-x)) : expf(x) / (1.f + expf(x));
    gwz[d] = (float)s * sg * inv_n;
}

// theta <- theta - lr * g
__global__ void k_sgd(float* __restrict__ theta, const float* __restrict__ g, int64_t n, float lr) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e < n) theta[e] = theta[e] - lr * g[e];
}

size_t train_query_smem(int V, int Mr) {
    return sizeof(int64_t) * V + sizeof(double) * ((size_t)V * kTrainWarps + 2 * V + kTrainWarps) +
           sizeof(float) * Mr;
}

cudaError_t launch_train_gram(const float* W, int M, int r, int KD, float* G, cudaStream_t s) {
    k_train_gram<<<(unsigned)(M * r * r), kTrainThreads, 0, s>>>(W, M, r, KD, G);
    return cudaGetLastError();
}

cudaError_t launch_train_query(const TrainQueryArgs& a, cudaStream_t s) {
    const size_t smem = train_query_smem(a.P + a.n_neg, a.M * a.r);
    cudaError_t e = cudaFuncSetAttribute(k_train_query, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    k_train_query<<<(unsigned)a.n, kTrainThreads, smem, s>>>(a);
    return cudaGetLastError();
}

cudaError_t launch_train_gW(const float* alpha, const float* gC, const float* W, int64_t n, int M, int r,
                            int KD, float lambda, float inv_n, float* gW, cudaStream_t s) {
    dim3 grid((unsigned)M, (unsigned)((KD + kTrainThreads - 1) / kTrainThreads));
    k_train_gW<<<grid, kTrainThreads, 0, s>>>(alpha, gC, W, n, M, r, KD, lambda, inv_n, gW);
    return cudaGetLastError();
}

cudaError_t launch_train_galpha(const float* gC, const float* W, const float* G, const float* alpha,
                                int64_t n, int M, int r, int KD, float lambda, float* galpha,
                                cudaStream_t s) {
    dim3 grid((unsigned)n, (unsigned)M);
    k_train_galpha<<<grid, kTrainThreads, 0, s>>>(gC, W, G, alpha, M, r, KD, lambda, galpha);
    return cudaGetLastError();
}

cudaError_t launch_train_bank(const uint32_t* idx, int64_t n, int h, int Mr, const float* galpha,
                              float inv_n, float* gbank, cudaStream_t s) {
    const int threads = Mr < 256 ? ((Mr + 31) / 32) * 32 : 256;
    k_train_bank<<<(unsigned)(n * h), threads, 0, s>>>(idx, n * h, h, Mr, galpha, inv_n, gbank);
    return cudaGetLastError();
}

cudaError_t launch_train_wz(const float* gw, int64_t n, int D, const float* wz, float inv_n, float* gwz,
                            cudaStream_t s) {
    k_train_wz<<<(unsigned)((D + 127) / 128), 128, 0, s>>>(gw, n, D, wz, inv_n, gwz);
    return cudaGetLastError();
}

cudaError_t launch_broadcast_wz(const float* wz, int D, int64_t n, float* out, cudaStream_t s) {
    const int64_t total = n * D;
    k_broadcast_wz<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(wz, D, n, out);
    return cudaGetLastError();
}

cudaError_t launch_sgd(float* theta, const float* g, int64_t n, float lr, cudaStream_t s) {
    if (n <= 0) return cudaSuccess;
    k_sgd<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(theta, g, n, lr);
    return cudaGetLastError();
}

}  // namespace ifvs
