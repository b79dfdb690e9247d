// Exact top-1 dot-product retrieval over a flat key index (Sec. 4.2).
//
// Batched GEMV on the CUDA cores: every warp streams whole key rows with
// 16-byte loads (several rows in flight per warp), dots them with a group of
// up to kQB queries held in shared memory as fp32, and reduces across lanes
// with a fixed butterfly, so a row's score never depends on where the row
// sits: equal rows get equal scores and the lowest row wins a tie. Each
// (score, row) pair is packed into one 64-bit key ordered by score, then by
// lower row; per-CTA maxima go to the workspace and a finalize kernel reduces
// them. A NaN score never enters a key, so it never wins.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_retrieve_status;

constexpr int kThreads = 256;
constexpr int kWarps = kThreads / 32;
constexpr int kQB = 4;        // queries per pass over the index
constexpr int kRowsInFlight = 4;
constexpr int kMaxDim = 4096;

// Monotone map of a non-NaN fp32 score to uint32 (-inf -> 0x007fffff > 0).
__device__ __forceinline__ uint32_t ordered_bits(float s) {
    const uint32_t u = __float_as_uint(s + 0.0f);  // -0 -> +0: equal scores, equal keys
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unordered_float(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}
// Larger key = higher score, then lower row. Key 0 = "no row".
__device__ __forceinline__ unsigned long long make_key(float s, int64_t row) {
    return (static_cast<unsigned long long>(ordered_bits(s)) << 32) |
           static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(row));
}

template <typename T> struct Vec;
template <> struct Vec<__half> { static constexpr int n = 8; };
template <> struct Vec<__nv_bfloat16> { static constexpr int n = 8; };
template <> struct Vec<float> { static constexpr int n = 4; };

template <typename T>
__device__ __forceinline__ void widen(const uint4 &v, float (&f)[Vec<T>::n]) {
    if constexpr (std::is_same<T, float>::value) {
        f[0] = __uint_as_float(v.x);
        f[1] = __uint_as_float(v.y);
        f[2] = __uint_as_float(v.z);
        f[3] = __uint_as_float(v.w);
    } else {
        const uint32_t w[4] = {v.x, v.y, v.z, v.w};
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            if constexpr (std::is_same<T, __half>::value) {
                const __half2 h2 = *reinterpret_cast<const __half2 *>(&w[i]);
                const float2 f2v = __half22float2(h2);
                f[2 * i] = f2v.x;
                f[2 * i + 1] = f2v.y;
            } else {
                f[2 * i] = __uint_as_float(w[i] << 16);
                f[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
            }
        }
    }
}

// partial[blockIdx.x * n_queries + q] = best key of this CTA for query q.
template <typename T>
__global__ void __launch_bounds__(kThreads)
    gemv_top1_kernel(const T *__restrict__ index, int64_t M, int dim, const T *__restrict__ queries,
                     int n_queries, int q0, unsigned long long *__restrict__ partial) {
    constexpr int V = Vec<T>::n;
    extern __shared__ float qs[];  // [kQB][dim]
    __shared__ unsigned long long best[kQB];
    const int nq = min(kQB, n_queries - q0);
    for (int i = threadIdx.x; i < kQB * dim; i += kThreads) {
        const int qq = i / dim, k = i % dim;
        qs[i] = (qq < nq) ? to_f32(queries[static_cast<int64_t>(q0 + qq) * dim + k]) : 0.f;
    }
    if (threadIdx.x < kQB) best[threadIdx.x] = 0ull;
    __syncthreads();

    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int64_t gwarp = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kWarps;
    const int vecs = dim / V;              // 16-byte vectors per row
    unsigned long long mykey[kQB];
#pragma unroll
    for (int qq = 0; qq < kQB; ++qq) mykey[qq] = 0ull;

    for (int64_t r0 = gwarp * kRowsInFlight; r0 < M; r0 += nwarps * kRowsInFlight) {
        float acc[kRowsInFlight][kQB];
#pragma unroll
        for (int r = 0; r < kRowsInFlight; ++r)
#pragma unroll
            for (int qq = 0; qq < kQB; ++qq) acc[r][qq] = 0.f;
        for (int v0 = 0; v0 < vecs; v0 += 32) {
            const int v = v0 + lane;
            uint4 raw[kRowsInFlight];
#pragma unroll
            for (int r = 0; r < kRowsInFlight; ++r) {
                const int64_t row = r0 + r;
                raw[r] = (v < vecs && row < M)
                             ? __ldg(reinterpret_cast<const uint4 *>(index + row * dim) + v)
                             : make_uint4(0, 0, 0, 0);
            }
            if (v < vecs) {
#pragma unroll
                for (int r = 0; r < kRowsInFlight; ++r) {
                    float f[V];
                    widen<T>(raw[r], f);
#pragma unroll
                    for (int qq = 0; qq < kQB; ++qq) {
                        const float *qv = qs + qq * dim + v * V;
#pragma unroll
                        for (int e = 0; e < V; ++e) acc[r][qq] = fmaf(f[e], qv[e], acc[r][qq]);
                    }
                }
            }
        }
#pragma unroll
        for (int r = 0; r < kRowsInFlight; ++r) {
#pragma unroll
            for (int qq = 0; qq < kQB; ++qq) {
                float s = acc[r][qq];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) s += __shfl_xor_sync(0xffffffffu, s, o);
                const int64_t row = r0 + r;
                if (row < M && !isnan(s)) {
                    const unsigned long long key = make_key(s, row);
                    mykey[qq] = key > mykey[qq] ? key : mykey[qq];
                }
            }
        }
    }
    if (lane == 0)
        for (int qq = 0; qq < nq; ++qq) atomicMax(&best[qq], mykey[qq]);
    __syncthreads();
    if (threadIdx.x < nq)
        partial[static_cast<int64_t>(blockIdx.x) * n_queries + q0 + threadIdx.x] = best[threadIdx.x];
}

__global__ void finalize_kernel(const unsigned long long *__restrict__ partial, int n_parts,
                                int n_queries, int64_t *__restrict__ best_idx,
                                float *__restrict__ best_score) {
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= n_queries) return;
    unsigned long long k = 0ull;
    for (int i = 0; i < n_parts; ++i) {
        const unsigned long long v = partial[static_cast<int64_t>(i) * n_queries + q];
        k = v > k ? v : k;
    }
    if (k == 0ull) {
        best_idx[q] = -1;
        if (best_score) best_score[q] = __uint_as_float(0x7fc00000u);
    } else {
        best_idx[q] = static_cast<int64_t>(0xffffffffu - static_cast<uint32_t>(k & 0xffffffffu));
        if (best_score) best_score[q] = unordered_float(static_cast<uint32_t>(k >> 32));
    }
}

int num_sms() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    return sms;
}

int gemv_grid(int64_t M) {
    const int64_t rows_per_cta = static_cast<int64_t>(kWarps) * kRowsInFlight;
    const int64_t need = (M + rows_per_cta - 1) / rows_per_cta;
    const int64_t cap = static_cast<int64_t>(num_sms()) * 4;
    return static_cast<int>(need < 1 ? 1 : (need < cap ? need : cap));
}

template <typename T>
cudaError_t launch_gemv(const RetrieveParams &p, cudaStream_t stream) {
    const int grid = gemv_grid(p.M);
    const size_t smem = static_cast<size_t>(kQB) * p.dim * sizeof(float);
    auto kern = gemv_top1_kernel<T>;
    cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize,
                                         static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    auto *partial = static_cast<unsigned long long *>(p.workspace);
    for (int q0 = 0; q0 < p.n_queries; q0 += kQB) {
        kern<<<grid, kThreads, smem, stream>>>(static_cast<const T *>(p.index), p.M, p.dim,
                                               static_cast<const T *>(p.queries), p.n_queries, q0,
                                               partial);
        e = cudaGetLastError();
        if (e != cudaSuccess) return e;
    }
    finalize_kernel<<<(p.n_queries + 127) / 128, 128, 0, stream>>>(partial, grid, p.n_queries,
                                                                    p.best_idx, p.best_score);
    return cudaGetLastError();
}

}  // namespace

size_t retrieve_workspace_size(int64_t M, int32_t dim, int32_t n_queries) {
    (void)dim;
    if (n_queries <= 0) return 0;
    return static_cast<size_t>(gemv_grid(M)) * n_queries * sizeof(unsigned long long);
}

cudaError_t launch_retrieve(const RetrieveParams &p, cudaStream_t stream) {
    if (p.n_queries == 0) return cudaSuccess;
    if (p.dim > kMaxDim) return cudaErrorInvalidValue;
    switch (p.dtype) {
        case PRECOG_F16: return launch_gemv<__half>(p, stream);
        case PRECOG_BF16: return launch_gemv<__nv_bfloat16>(p, stream);
        default: return launch_gemv<float>(p, stream);
    }
}

cudaError_t retrieve_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_retrieve_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_retrieve_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
