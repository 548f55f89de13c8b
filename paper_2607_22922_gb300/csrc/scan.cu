// Stage 2 of §2 (Rank) with the per-CTA part of stage 3 (Select): every
// passing row v gets dist(v) = sum_m LUT[m][code_v[m]] (the weighted ADC
// form of the printed score), and each CTA keeps the k smallest
// (dist, row id) of its chunk exactly.
//
// Work split: CTA (query q, chunk c) — blockIdx.x runs over queries so that
// the CTAs resident together share the same code chunk through L2.  Inside
// a CTA, warp w walks bitmap blocks c0 + w, c0 + w + 8, ...; lane l of a warp
// owns rows b*1024 + 32*j + l (the lane-major bitmap gives it its 32 pass
// bits in one load) and reads a row's codes with one 16-byte load (M = 16).
//
// LUT placement: the scan issues one shared-memory load per code byte, so
// bank conflicts decide its speed.  The table of query q is stored as 256
// rows (one per codeword) of S words, S a multiple of 32, word w of row c
// holding LUT[w mod M][c] for w < M + 31.  Row i's codes are stored rotated
// by rot(i) = (i mod 32) mod M, so lane l (i = l mod 32) reads at step s the
// code of subspace (l + s) mod M and finds its entry at word l + s of that
// codeword's row: bank (l + s) mod 32, distinct across the warp for any
// codes.  For M = 16 the row stride is 256 bytes and the byte address is
// formed by one byte permute: code * 256 + 4 * l (+ 4 * s as an immediate).
//
// Top-k: each warp keeps a sorted list of its KP best keys and a candidate
// area of KP slots in shared memory; a key (dist bits << 32 | row) enters
// the area when it is below the warp's current k-th key, and a full area is
// merged by a warp bitonic sort.  Keys are unique (row ids are), so the
// result is exact and independent of timing.  At the end warp 0 merges the
// other warps' lists and writes the CTA's k keys.
#include "internal.cuh"

namespace ifvs {

int scan_kp(int k) { return k <= 32 ? 32 : (k <= 64 ? 64 : (k <= 128 ? 128 : 256)); }

size_t scan_smem_bytes(int tab_words, int kp) {
    return (size_t)256 * tab_words * 4 + (size_t)kWarps * 2 * kp * 8;
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

template <int KP>
struct WarpTopK {
    uint64_t* buf;   // [0, KP): sorted best keys; [KP, 2KP): candidates
    int cnt;
    int k;
    uint64_t thr;    // current k-th best key (all ones while fewer than k)

    __device__ __forceinline__ void init(uint64_t* b, int k_, int lane) {
        buf = b;
        k = k_;
        cnt = 0;
        thr = ~0ull;
        for (int i = lane; i < 2 * KP; i += 32) buf[i] = ~0ull;
        __syncwarp();
    }
    __device__ __forceinline__ void flush(int lane) {
        warp_sort(buf, 2 * KP, lane);
        thr = buf[k - 1];
        for (int i = KP + lane; i < 2 * KP; i += 32) buf[i] = ~0ull;
        __syncwarp();
        cnt = 0;
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

__device__ __forceinline__ uint4 ldg_nc_v4(const uint8_t* p) {
    uint4 v;
    asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0, %1, %2, %3}, [%4];"
                 : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
                 : "l"(p));
    return v;
}

// 16 look-ups of one M = 16 row (row stride of the table: 256 bytes)
__device__ __forceinline__ float lookup16(const uint4 c, const char* tab, uint32_t lane4) {
    const uint32_t w[4] = {c.x, c.y, c.z, c.w};
    float acc0 = 0.f, acc1 = 0.f;
#pragma unroll
    for (int s = 0; s < 16; ++s) {
        // bytes: [4*lane, code, 0, 0] -> code * 256 + 4 * lane
        const uint32_t off = __byte_perm(w[s >> 2], lane4, 0x5504u | ((uint32_t)(s & 3) << 4));
        const float v = *reinterpret_cast<const float*>(tab + off + 4 * s);
        if (s & 1) acc1 += v; else acc0 += v;
    }
    return acc0 + acc1;
}

constexpr int kU = 4;   // rows per lane in flight

template <int KP, bool M16>
__global__ void __launch_bounds__(kThreads, 2)
k_scan(const uint8_t* __restrict__ codes, const float* __restrict__ luts,
       const uint32_t* __restrict__ bm, int64_t nq, int k, ScanShape sh,
       uint64_t* __restrict__ partials) {
    extern __shared__ __align__(16) uint8_t smem[];
    const int M = M16 ? 16 : sh.M;
    const int S = M16 ? 64 : sh.tab_words;
    const int K = sh.K;
    float* tab = reinterpret_cast<float*>(smem);
    uint64_t* tkbuf = reinterpret_cast<uint64_t*>(smem + (size_t)256 * S * 4);
    const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
    const int64_t q = blockIdx.x;
    const int chunk = blockIdx.y;

    // 1) the query's table, replicated and rotated (see the file comment)
    const float* lut = luts + q * (int64_t)M * K;
    const int wu = M + 31;
    for (int e = threadIdx.x; e < 256 * wu; e += kThreads) {
        const int c = e / wu, w = e - c * wu;
        const int m = w % M;
        tab[c * S + w] = c < K ? __ldg(lut + (int64_t)m * K + c) : 0.f;
    }
    WarpTopK<KP> tk;
    tk.init(tkbuf + warp * 2 * KP, k, lane);
    __syncthreads();

    // 2) the chunk's blocks
    const int64_t b0 = (int64_t)chunk * sh.blocks_per_chunk;
    const int64_t b1 = min(sh.n_blocks, b0 + sh.blocks_per_chunk);
    const uint32_t* bmq = bm + q * sh.n_blocks * 32;
    const uint32_t lane4 = (uint32_t)lane * 4u;
    const char* tabc = reinterpret_cast<const char*>(tab);
    const int row_bytes = sh.row_bytes;

    for (int64_t b = b0 + warp; b < b1; b += kWarps) {
        const uint32_t mword = __ldg(bmq + b * 32 + lane);
        if (__ballot_sync(0xFFFFFFFFu, mword != 0u) == 0u) continue;
        const int64_t rbase = b * kBlockRows + lane;
        for (int j0 = 0; j0 < 32; j0 += kU) {
            const uint32_t bits = (mword >> j0) & ((1u << kU) - 1u);
            if (__ballot_sync(0xFFFFFFFFu, bits != 0u) == 0u) continue;
            if (M16) {
                uint4 c[kU];
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int64_t row = rbase + 32 * (j0 + u);
                    c[u] = (bits >> u & 1u) ? ldg_nc_v4(codes + row * 16) : make_uint4(0, 0, 0, 0);
                }
#pragma unroll
                for (int u = 0; u < kU; ++u) {
                    const int64_t row = rbase + 32 * (j0 + u);
                    const float d = lookup16(c[u], tabc, lane4);
                    const uint64_t key = ((uint64_t)__float_as_uint(d) << 32) | (uint64_t)(uint32_t)row;
                    tk.offer(key, (bits >> u & 1u) && key < tk.thr, lane);
                }
            } else {
#pragma unroll 1
                for (int u = 0; u < kU; ++u) {
                    const int64_t row = rbase + 32 * (j0 + u);
                    const bool pass = bits >> u & 1u;
                    const uint8_t* rp = codes + row * row_bytes;
                    float acc = 0.f;
                    for (int w = 0; w * 4 < M; ++w) {
                        const uint32_t wd = pass ? __ldg(reinterpret_cast<const uint32_t*>(rp) + w) : 0u;
#pragma unroll
                        for (int bb = 0; bb < 4; ++bb) {
                            const int s = 4 * w + bb;
                            if (s < M) acc += tab[(int)((wd >> (8 * bb)) & 0xFFu) * S + lane + s];
                        }
                    }
                    const uint64_t key = ((uint64_t)__float_as_uint(acc) << 32) | (uint64_t)(uint32_t)row;
                    tk.offer(key, pass && key < tk.thr, lane);
                }
            }
        }
    }

    // 3) merge the warps' lists; warp 0 writes the CTA's k best keys
    tk.flush(lane);
    __syncthreads();
    if (warp == 0) {
        for (int w = 1; w < kWarps; ++w) {
            const uint64_t* other = tkbuf + w * 2 * KP;
            for (int i = lane; i < k; i += 32) tk.buf[KP + i] = other[i];
            __syncwarp();
            tk.flush(lane);
        }
        uint64_t* out = partials + (q * sh.n_chunks + chunk) * (int64_t)k;
        for (int i = lane; i < k; i += 32) out[i] = tk.buf[i];
    }
}

template <int KP>
static cudaError_t launch_scan_kp(const uint8_t* codes, const float* lut, const uint32_t* bm,
                                  int64_t nq, int k, const ScanShape& sh, uint64_t* partials,
                                  cudaStream_t s) {
    const bool m16 = sh.M == 16 && sh.row_bytes == 16 && sh.tab_words == 64;
    const size_t smem = scan_smem_bytes(sh.tab_words, KP);
    dim3 grid((unsigned)nq, (unsigned)sh.n_chunks);
    cudaError_t e;
    if (m16) {
        e = cudaFuncSetAttribute(k_scan<KP, true>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_scan<KP, true><<<grid, kThreads, smem, s>>>(codes, lut, bm, nq, k, sh, partials);
    } else {
        e = cudaFuncSetAttribute(k_scan<KP, false>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
        if (e != cudaSuccess) return e;
        k_scan<KP, false><<<grid, kThreads, smem, s>>>(codes, lut, bm, nq, k, sh, partials);
    }
    return cudaGetLastError();
}

cudaError_t launch_scan(const uint8_t* codes, const float* lut, const uint32_t* bm, int64_t nq,
                        int k, const ScanShape& sh, uint64_t* partials, cudaStream_t s) {
    if (nq <= 0) return cudaSuccess;
    switch (scan_kp(k)) {
        case 32: return launch_scan_kp<32>(codes, lut, bm, nq, k, sh, partials, s);
        case 64: return launch_scan_kp<64>(codes, lut, bm, nq, k, sh, partials, s);
        case 128: return launch_scan_kp<128>(codes, lut, bm, nq, k, sh, partials, s);
        default: return launch_scan_kp<256>(codes, lut, bm, nq, k, sh, partials, s);
    }
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
