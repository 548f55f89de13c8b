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
//                         with the Gram matrix G_m = W[m] W[m]^T, formed per candidate
//                         while gC is scattered (the W values are already loaded)
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
template <int RMAX>
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
    float* gas = alpha + Mr;                                      // [D][r]: dL/dalpha per dimension
    const int64_t q = blockIdx.x;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const int nwarps = blockDim.x >> 5;

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
        for (int w = 0; w < nwarps; ++w) s += part[v * kTrainWarps + w];
        dist[v] = s;
    }
    __syncthreads();

    // Softmax of each positive g against the negatives N, with the shift
    // m_g = min(dist_g, m_N), m_N = min over N:
    //   Z_g = exp(-(d_g - m_g)/tau) + exp(-(m_N - m_g)/tau) S,  S = sum_n u_n,
    //   u_n = exp(-(d_n - m_N)/tau),  p_n(g) = u_n exp(-(m_N - m_g)/tau) / Z_g,
    // so each negative's exponential is shared by all positives (warp 0).
    if (warp == 0) {
        double mN = INFINITY;
        for (int n = a.P + lane; n < V; n += 32)
            if (cand[n] >= 0) mN = fmin(mN, dist[n]);
        mN = warp_min(mN);
        double S = 0.0;
        for (int n = a.P + lane; n < V; n += 32) {
            const double u = cand[n] >= 0 ? exp(-(dist[n] - mN) / a.tau) : 0.0;
            gam[n] = u;
            S += u;
        }
        S = warp_sum(S);
        double lpos = 0.0, csum = 0.0;
        int npos = 0;
        for (int g = lane; g < a.P; g += 32) {
            gam[g] = 0.0;
            if (cand[g] < 0) continue;
            ++npos;
            const double mg = fmin(dist[g], mN);
            const double eg = exp(-(dist[g] - mg) / a.tau);
            const double en = S > 0.0 ? exp(-(mN - mg) / a.tau) : 0.0;
            const double z = eg + en * S;
            lpos += dist[g] / a.tau - mg / a.tau + log(z);
            gam[g] = (1.0 - eg / z) / a.tau;
            csum += en / z;
        }
        lpos = warp_sum(lpos);
        csum = warp_sum(csum);
        npos = __reduce_add_sync(0xFFFFFFFFu, npos);
        __syncwarp();
        const double inv = npos > 0 ? 1.0 / npos : 0.0;
        for (int n = a.P + lane; n < V; n += 32) gam[n] = -gam[n] * csum / a.tau * inv;
        for (int g = lane; g < a.P; g += 32) gam[g] *= inv;
        if (lane == 0) red[0] = npos > 0 ? lpos * inv : 0.0;
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
        for (int w = 0; w < nwarps; ++w) s += red[w];
        a.loss[q] = lpos + (double)a.lambda * s;
    }

    // pass 2: gC scatter, dL/dw_f, and dL/dalpha through the same W values:
    // dL/dalpha[m][j] = sum over (v, t) of gC contribution x W[m][j][c_v][t]
    float* gC = a.gC + q * (int64_t)a.M * KD;
    for (int d = tid; d < a.D; d += blockDim.x) {
        const int m = d / a.ds, t = d - m * a.ds;
        double gw = 0.0;
        float ga[RMAX];
#pragma unroll
        for (int j = 0; j < RMAX; ++j) ga[j] = 0.f;
        for (int v = 0; v < V; ++v) {
            const int64_t id = cand[v];
            if (id < 0) continue;
            int c;
            const float df = diff_of(id, d, &c);
            const float ge = (float)gam[v] * (-2.f * wf[d] * df);
            const int64_t e = (int64_t)c * a.ds + t;
            gC[(int64_t)m * KD + e] += ge;
            gw += gam[v] * (double)(df * df);
            const float* Wc = a.W + (int64_t)m * a.r * KD + e;
#pragma unroll
            for (int j = 0; j < RMAX; ++j)
                if (j < a.r) ga[j] += ge * Wc[(int64_t)j * KD];
        }
        a.gw[q * a.D + d] = (float)gw;
#pragma unroll
        for (int j = 0; j < RMAX; ++j)
            if (j < a.r) gas[d * a.r + j] = ga[j];
    }
    __syncthreads();
    // sum over the subspace's dimensions in order, plus the anchor 2 lambda G_m alpha[m]
    for (int x = tid; x < Mr; x += blockDim.x) {
        const int m = x / a.r, j = x - m * a.r;
        float sg = 0.f;
        for (int t = 0; t < a.ds; ++t) sg += gas[(m * a.ds + t) * a.r + j];
        float an = 0.f;
        for (int j2 = 0; j2 < a.r; ++j2) an += a.G[((int64_t)m * a.r + j) * a.r + j2] * alpha[m * a.r + j2];
        a.galpha[q * Mr + x] = sg + 2.f * a.lambda * an;
    }
}

// A[m][j][j'] = sum over the queries of alpha_q[m][j] alpha_q[m][j'] (one CTA per entry)
__global__ void __launch_bounds__(kTrainThreads) k_train_acov(const float* __restrict__ alpha, int64_t n,
                                                              int M, int r, float* __restrict__ A) {
    __shared__ float part[kTrainWarps];
    const int b = blockIdx.x;
    const int m = b / (r * r), j = (b / r) % r, j2 = b % r;
    const int Mr = M * r;
    float s = 0.f;
    for (int64_t q = threadIdx.x; q < n; q += kTrainThreads)
        s += alpha[q * Mr + m * r + j] * alpha[q * Mr + m * r + j2];
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xFFFFFFFFu, s, o);
    if ((threadIdx.x & 31) == 0) part[threadIdx.x >> 5] = s;
    __syncthreads();
    if (threadIdx.x == 0) {
        float t = 0.f;
        for (int w = 0; w < kTrainWarps; ++w) t += part[w];
        A[b] = t;
    }
}

// Partial sums of alpha_q[m][j] gC_q[m][e] over one slice of kGWQueries
// queries: grid (M, ceil(KD / 256), slices); part [slices][M][r][KD]
constexpr int kGWQueries = 64;
template <int RMAX>
__global__ void __launch_bounds__(kTrainThreads) k_train_gW_part(const float* __restrict__ alpha,
                                                                 const float* __restrict__ gC, int64_t n,
                                                                 int M, int r, int KD,
                                                                 float* __restrict__ part) {
    __shared__ float as[kGWQueries * kTrainMaxR];
    const int m = blockIdx.x;
    const int e = blockIdx.y * kTrainThreads + threadIdx.x;
    const int64_t q0 = (int64_t)blockIdx.z * kGWQueries;
    const int nc = (int)min((int64_t)kGWQueries, n - q0);
    const int Mr = M * r;
    for (int t = threadIdx.x; t < nc * r; t += kTrainThreads)
        as[t] = alpha[(q0 + t / r) * Mr + m * r + t % r];
    __syncthreads();
    if (e >= KD) return;
    float acc[RMAX];
#pragma unroll
    for (int j = 0; j < RMAX; ++j) acc[j] = 0.f;
#pragma unroll 8
    for (int i = 0; i < nc; ++i) {
        const float g = gC[((q0 + i) * M + m) * (int64_t)KD + e];
#pragma unroll
        for (int j = 0; j < RMAX; ++j)
            if (j < r) acc[j] += as[i * r + j] * g;
    }
    float* out = part + (((int64_t)blockIdx.z * M + m) * r) * KD + e;
#pragma unroll
    for (int j = 0; j < RMAX; ++j)
        if (j < r) out[(int64_t)j * KD] = acc[j];
}

// dL/dW[m][j][e] = inv_n (sum over slices of part + 2 lambda sum_j' A_m[j][j'] W[m][j'][e]),
// slices summed in order
__global__ void k_train_gW_sum(const float* __restrict__ part, int slices, const float* __restrict__ A,
                               const float* __restrict__ W, int M, int r, int KD, float lambda,
                               float inv_n, float* __restrict__ gW) {
    const int64_t total = (int64_t)M * r * KD;
    const int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (x >= total) return;
    const int e = (int)(x % KD);
    const int j = (int)((x / KD) % r);
    const int m = (int)(x / ((int64_t)KD * r));
    float s = 0.f;
    for (int z = 0; z < slices; ++z) s += part[(int64_t)z * total + x];
    float an = 0.f;
    for (int j2 = 0; j2 < r; ++j2)
        an += A[((int64_t)m * r + j) * r + j2] * W[((int64_t)m * r + j2) * KD + e];
    gW[x] = (s + 2.f * lambda * an) * inv_n;
}

// dL/dbank: one CTA per fetch p = (q, i).  The first fetch of each bank row
// gathers, in fetch order, the fetches of that row and sums their dL/dalpha.
constexpr int kBankList = 512;
__global__ void __launch_bounds__(kTrainThreads) k_train_bank(const uint32_t* __restrict__ idx,
                                                              int64_t n_fetch, int h, int Mr,
                                                              const float* __restrict__ galpha,
                                                              float inv_n, float* __restrict__ gbank) {
    __shared__ int64_t list[kBankList];
    __shared__ int wcnt[kTrainWarps];
    __shared__ int total;
    const int64_t p = blockIdx.x;
    const uint32_t b = idx[p];
    int earlier = 0;
    for (int64_t p2 = threadIdx.x; p2 < p; p2 += blockDim.x) earlier |= idx[p2] == b;
    if (__syncthreads_or(earlier)) return;
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, nw = blockDim.x >> 5;
    if (threadIdx.x == 0) total = 0;
    __syncthreads();
    for (int64_t c0 = p; c0 < n_fetch; c0 += blockDim.x) {
        const int64_t p2 = c0 + threadIdx.x;
        const bool f = p2 < n_fetch && idx[p2] == b;
        const unsigned bal = __ballot_sync(0xFFFFFFFFu, f);
        if (lane == 0) wcnt[warp] = __popc(bal);
        __syncthreads();
        int off = total;
        for (int w = 0; w < warp; ++w) off += wcnt[w];
        off += __popc(bal & ((1u << lane) - 1u));
        if (f && off < kBankList) list[off] = p2;
        __syncthreads();
        if (threadIdx.x == 0)
            for (int w = 0; w < nw; ++w) total += wcnt[w];
        __syncthreads();
    }
    const int cnt = total;
    for (int e = threadIdx.x; e < Mr; e += blockDim.x) {
        float s = 0.f;
        if (cnt <= kBankList) {
            for (int i = 0; i < cnt; ++i) s += galpha[(list[i] / h) * Mr + e];
        } else {
            for (int64_t p2 = p; p2 < n_fetch; ++p2)
                if (idx[p2] == b) s += galpha[(p2 / h) * Mr + e];
        }
        gbank[(int64_t)b * Mr + e] = s * inv_n;
    }
}

// dL/dw_z[d] = inv_n sum_q dL/dw_f[q][d] sigmoid(w_z[d]); block (32 dims, 32
// query lanes), lane y sums the queries q = y (mod 32) in order, then the 32
// lanes are added in order
__global__ void __launch_bounds__(1024) k_train_wz(const float* __restrict__ gw, int64_t n, int D,
                                                   const float* __restrict__ wz, float inv_n,
                                                   float* __restrict__ gwz) {
    __shared__ double part[32][33];
    const int d = blockIdx.x * 32 + threadIdx.x;
    double s = 0.0;
    if (d < D)
        for (int64_t q = threadIdx.y; q < n; q += 32) s += (double)gw[q * D + d];
    part[threadIdx.y][threadIdx.x] = s;
    __syncthreads();
    if (threadIdx.y != 0 || d >= D) return;
    double t = 0.0;
    for (int y = 0; y < 32; ++y) t += part[y][threadIdx.x];
    const float x = wz[d];
    const float sg = x >= 0.f ? 1.f / (1.f + expf(-x)) : expf(x) / (1.f + expf(x));
    gwz[d] = (float)t * sg * inv_n;
}

// theta <- theta - lr * g
__global__ void k_sgd(float* __restrict__ theta, const float* __restrict__ g, int64_t n, float lr) {
    const int64_t e = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
    if (e < n) theta[e] = theta[e] - lr * g[e];
}

size_t train_query_smem(int V, int Mr, int D, int r) {
    return sizeof(int64_t) * V + sizeof(double) * ((size_t)V * kTrainWarps + 2 * V + kTrainWarps) +
           sizeof(float) * (Mr + (size_t)D * r);
}

cudaError_t launch_train_gram(const float* W, int M, int r, int KD, float* G, cudaStream_t s) {
    k_train_gram<<<(unsigned)(M * r * r), kTrainThreads, 0, s>>>(W, M, r, KD, G);
    return cudaGetLastError();
}

cudaError_t launch_train_query(const TrainQueryArgs& a, cudaStream_t s) {
    const size_t smem = train_query_smem(a.P + a.n_neg, a.M * a.r, a.D, a.r);
    // threads own dimensions: no more threads than (32-rounded) dimensions
    const int threads = a.D >= kTrainThreads ? kTrainThreads : ((a.D + 31) / 32) * 32;
    auto kern = a.r <= 8 ? k_train_query<8> : k_train_query<kTrainMaxR>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
    if (e != cudaSuccess) return e;
    kern<<<(unsigned)a.n, threads, smem, s>>>(a);
    return cudaGetLastError();
}

size_t train_gW_scratch(int64_t n, int M, int r, int KD) {
    const int64_t slices = (n + kGWQueries - 1) / kGWQueries;
    return sizeof(float) * (size_t)(slices * M * r * KD + M * r * r);
}

cudaError_t launch_train_gW(const float* alpha, const float* gC, const float* W, int64_t n, int M, int r,
                            int KD, float lambda, float inv_n, float* scratch, float* gW,
                            cudaStream_t s, int* launches) {
    const int slices = (int)((n + kGWQueries - 1) / kGWQueries);
    float* A = scratch;
    float* part = scratch + M * r * r;
    k_train_acov<<<(unsigned)(M * r * r), kTrainThreads, 0, s>>>(alpha, n, M, r, A);
    cudaError_t e = cudaGetLastError();
    if (e != cudaSuccess) return e;
    dim3 grid((unsigned)M, (unsigned)((KD + kTrainThreads - 1) / kTrainThreads), (unsigned)slices);
    if (r <= 8)
        k_train_gW_part<8><<<grid, kTrainThreads, 0, s>>>(alpha, gC, n, M, r, KD, part);
    else
        k_train_gW_part<kTrainMaxR><<<grid, kTrainThreads, 0, s>>>(alpha, gC, n, M, r, KD, part);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
    const int64_t total = (int64_t)M * r * KD;
    k_train_gW_sum<<<(unsigned)((total + 255) / 256), 256, 0, s>>>(part, slices, A, W, M, r, KD, lambda,
                                                                    inv_n, gW);
    if (launches) *launches = 3;
    return cudaGetLastError();
}

cudaError_t launch_train_bank(const uint32_t* idx, int64_t n, int h, int Mr, const float* galpha,
                              float inv_n, float* gbank, cudaStream_t s) {
    const int threads = Mr < kTrainThreads ? ((Mr + 31) / 32) * 32 : kTrainThreads;
    k_train_bank<<<(unsigned)(n * h), threads, 0, s>>>(idx, n * h, h, Mr, galpha, inv_n, gbank);
    return cudaGetLastError();
}

cudaError_t launch_train_wz(const float* gw, int64_t n, int D, const float* wz, float inv_n, float* gwz,
                            cudaStream_t s) {
    k_train_wz<<<(unsigned)((D + 31) / 32), dim3(32, 32), 0, s>>>(gw, n, D, wz, inv_n, gwz);
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
