// Exact top-1 dot-product retrieval over a flat key index (Sec. 4.2).
//
// Batched GEMV on the CUDA cores: every warp streams whole key rows with
// 16-byte loads (several rows in flight per warp), dots them with a group of
// up to kQB queries held in registers as fp32, and reduces across lanes with
// a fixed butterfly, so a row's score never depends on where the row sits:
// equal rows get equal scores and the lowest row wins a tie. Each
// (score, row) pair is packed into one 64-bit key ordered by score, then by
// lower row; per-CTA maxima go to the workspace and a finalize kernel reduces
// them. A NaN score never enters a key, so it never wins.
#include <algorithm>
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
constexpr int kMaxVecsPerRow = 512;  // 16 vectors per lane

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

// The CUDA-core kernels take fp32 keys (16-bit keys go to the tensor cores).
template <typename T> struct Vec;
template <> struct Vec<float> { static constexpr int n = 4; };

template <typename T>
__device__ __forceinline__ void widen(const uint4 &v, float (&f)[Vec<T>::n]) {
    static_assert(std::is_same<T, float>::value, "fp32 keys only");
    f[0] = __uint_as_float(v.x);
    f[1] = __uint_as_float(v.y);
    f[2] = __uint_as_float(v.z);
    f[3] = __uint_as_float(v.w);
}

// partial[blockIdx.x * n_queries + q] = best key of this CTA for query q.
// Lane l owns the 16-byte vectors l, l+32, ... of every row (VPL of them) and
// holds the matching query values in registers; RIF rows are loaded before any
// is used, so each lane keeps RIF*VPL 16-byte loads in flight.
template <typename T, int QB, int VPL, int RIF>
__global__ void __launch_bounds__(kThreads)
    gemv_top1_kernel(const T *__restrict__ index, int64_t M, int dim, const T *__restrict__ queries,
                     int n_queries, int q0, unsigned long long *__restrict__ partial) {
    constexpr int V = Vec<T>::n;
    __shared__ unsigned long long best[QB];
    const int nq = min(QB, n_queries - q0);
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int vecs = dim / V;
    float qv[QB][VPL][V];
#pragma unroll
    for (int qq = 0; qq < QB; ++qq)
#pragma unroll
        for (int j = 0; j < VPL; ++j) {
            const int v = lane + 32 * j;
            if (qq < nq && v < vecs) {
                const uint4 raw =
                    __ldg(reinterpret_cast<const uint4 *>(queries + static_cast<int64_t>(q0 + qq) * dim) + v);
                widen<T>(raw, qv[qq][j]);
            } else {
#pragma unroll
                for (int e = 0; e < V; ++e) qv[qq][j][e] = 0.f;
            }
        }
    if (threadIdx.x < QB) best[threadIdx.x] = 0ull;
    __syncthreads();

    const int64_t gwarp = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kWarps;
    unsigned long long mykey[QB];
#pragma unroll
    for (int qq = 0; qq < QB; ++qq) mykey[qq] = 0ull;

    for (int64_t r0 = gwarp * RIF; r0 < M; r0 += nwarps * RIF) {
        uint4 raw[RIF][VPL];
#pragma unroll
        for (int r = 0; r < RIF; ++r)
#pragma unroll
            for (int j = 0; j < VPL; ++j) {
                const int v = lane + 32 * j;
                const int64_t row = r0 + r;
                raw[r][j] = (v < vecs && row < M)
                                ? __ldg(reinterpret_cast<const uint4 *>(index + row * dim) + v)
                                : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
        for (int r = 0; r < RIF; ++r) {
            float acc[QB];
#pragma unroll
            for (int qq = 0; qq < QB; ++qq) acc[qq] = 0.f;
#pragma unroll
            for (int j = 0; j < VPL; ++j) {
                float f[V];
                widen<T>(raw[r][j], f);
#pragma unroll
                for (int qq = 0; qq < QB; ++qq)
#pragma unroll
                    for (int e = 0; e < V; ++e) acc[qq] = fmaf(f[e], qv[qq][j][e], acc[qq]);
            }
            const int64_t row = r0 + r;
#pragma unroll
            for (int qq = 0; qq < QB; ++qq) {
                float sc = acc[qq];
#pragma unroll
                for (int o = 16; o > 0; o >>= 1) sc += __shfl_xor_sync(0xffffffffu, sc, o);
                if (row < M && !isnan(sc)) {
                    const unsigned long long key = make_key(sc, row);
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

__device__ __forceinline__ unsigned long long shfl_xor_u64(unsigned long long v, int o) {
    const uint32_t lo = __shfl_xor_sync(0xffffffffu, static_cast<uint32_t>(v), o);
    const uint32_t hi = __shfl_xor_sync(0xffffffffu, static_cast<uint32_t>(v >> 32), o);
    return (static_cast<unsigned long long>(hi) << 32) | lo;
}

// A shard's key with its row made global, in signed order: flipping the top bit
// maps the unsigned key order onto int64 order, so keys of different shards combine
// by a signed maximum (an all-reduce MAX over int64); "no row" becomes INT64_MIN.
__device__ __forceinline__ int64_t global_key(unsigned long long k, int64_t row_offset) {
    if (k != 0ull) {
        const int64_t row = row_offset + static_cast<int64_t>(0xffffffffu - static_cast<uint32_t>(k & 0xffffffffu));
        k = (k & 0xffffffff00000000ull) | static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(row));
    }
    return static_cast<int64_t>(k ^ 0x8000000000000000ull);
}

__device__ __forceinline__ void write_best(unsigned long long k, int64_t *best_idx, float *best_score, int q) {
    if (k == 0ull) {
        best_idx[q] = -1;
        if (best_score) best_score[q] = __uint_as_float(0x7fc00000u);
    } else {
        best_idx[q] = static_cast<int64_t>(0xffffffffu - static_cast<uint32_t>(k & 0xffffffffu));
        if (best_score) best_score[q] = unordered_float(static_cast<uint32_t>(k >> 32));
    }
}

// One warp per query: each lane takes the maximum over a strided share of the
// per-CTA keys (independent loads, so many are in flight), then a butterfly.
__global__ void finalize_kernel(const unsigned long long *__restrict__ partial, int n_parts,
                                int n_queries, int64_t *__restrict__ best_idx,
                                float *__restrict__ best_score, int64_t row_offset,
                                int64_t *__restrict__ keys_out) {
    const int q = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (q >= n_queries) return;
    unsigned long long k = 0ull;
    for (int i = lane; i < n_parts; i += 32) {
        const unsigned long long v = partial[static_cast<int64_t>(i) * n_queries + q];
        k = v > k ? v : k;
    }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        const unsigned long long v = shfl_xor_u64(k, o);
        k = v > k ? v : k;
    }
    if (lane != 0) return;
    if (keys_out) keys_out[q] = global_key(k, row_offset);
    else write_best(k, best_idx, best_score, q);
}

// Signed-order keys (combined over shards) to rows and scores.
__global__ void decode_keys_kernel(const int64_t *__restrict__ keys, int n, int64_t *__restrict__ best_idx,
                                   float *__restrict__ best_score) {
    const int q = blockIdx.x * blockDim.x + threadIdx.x;
    if (q >= n) return;
    write_best(static_cast<unsigned long long>(keys[q]) ^ 0x8000000000000000ull, best_idx, best_score, q);
}

// ---------------------------------------------------------------------------
// Top-k (k <= kListK) for one query per pass: every warp keeps the kListK best
// packed keys seen so far as a sorted list, held identically by all lanes (the
// butterfly leaves the row's score in every lane), so a row costs one compare
// against the list's last entry unless it enters the list. The warps' lists
// are merged per CTA in shared memory; partial[(cta * Q + q) * kListK + j].
constexpr int kListK = 8;

__device__ __forceinline__ void list_insert(unsigned long long (&l)[kListK], unsigned long long v) {
    if (v <= l[kListK - 1]) return;
#pragma unroll
    for (int j = kListK - 1; j > 0; --j) {
        // shift entries below v down by one; v lands in its sorted slot
        const bool shift = v > l[j - 1];
        l[j] = shift ? l[j - 1] : (v > l[j] ? v : l[j]);
    }
    l[0] = v > l[0] ? v : l[0];
}

template <typename T, int VPL>
__global__ void __launch_bounds__(kThreads)
    gemv_topk_kernel(const T *__restrict__ index, int64_t M, int dim, const T *__restrict__ queries,
                     int n_queries, int q, unsigned long long *__restrict__ partial) {
    constexpr int V = Vec<T>::n;
    constexpr int RIF = 4;
    __shared__ unsigned long long lists[kWarps][kListK];
    const int lane = threadIdx.x & 31;
    const int warp = threadIdx.x >> 5;
    const int vecs = dim / V;
    float qv[VPL][V];
#pragma unroll
    for (int j = 0; j < VPL; ++j) {
        const int v = lane + 32 * j;
        if (v < vecs) {
            const uint4 raw = __ldg(reinterpret_cast<const uint4 *>(queries + static_cast<int64_t>(q) * dim) + v);
            widen<T>(raw, qv[j]);
        } else {
#pragma unroll
            for (int e = 0; e < V; ++e) qv[j][e] = 0.f;
        }
    }
    unsigned long long l[kListK];
#pragma unroll
    for (int j = 0; j < kListK; ++j) l[j] = 0ull;
    const int64_t gwarp = static_cast<int64_t>(blockIdx.x) * kWarps + warp;
    const int64_t nwarps = static_cast<int64_t>(gridDim.x) * kWarps;
    for (int64_t r0 = gwarp * RIF; r0 < M; r0 += nwarps * RIF) {
        uint4 raw[RIF][VPL];
#pragma unroll
        for (int r = 0; r < RIF; ++r)
#pragma unroll
            for (int j = 0; j < VPL; ++j) {
                const int v = lane + 32 * j;
                const int64_t row = r0 + r;
                raw[r][j] = (v < vecs && row < M)
                                ? __ldg(reinterpret_cast<const uint4 *>(index + row * dim) + v)
                                : make_uint4(0, 0, 0, 0);
            }
#pragma unroll
        for (int r = 0; r < RIF; ++r) {
            float acc = 0.f;
#pragma unroll
            for (int j = 0; j < VPL; ++j) {
                float f[V];
                widen<T>(raw[r][j], f);
#pragma unroll
                for (int e = 0; e < V; ++e) acc = fmaf(f[e], qv[j][e], acc);
            }
#pragma unroll
            for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
            const int64_t row = r0 + r;
            // acc is the same in every lane (xor butterfly), so the branch is uniform;
            // most rows fall below the list's last key and skip the insertion
            if (row < M && !isnan(acc)) {
                const unsigned long long key = make_key(acc, row);
                if (key > l[kListK - 1]) list_insert(l, key);
            }
        }
    }
    if (lane == 0)
#pragma unroll
        for (int j = 0; j < kListK; ++j) lists[warp][j] = l[j];
    __syncthreads();
    if (threadIdx.x == 0) {
        unsigned long long m[kListK];
#pragma unroll
        for (int j = 0; j < kListK; ++j) m[j] = lists[0][j];
        for (int w = 1; w < kWarps; ++w)
#pragma unroll
            for (int j = 0; j < kListK; ++j) list_insert(m, lists[w][j]);
#pragma unroll
        for (int j = 0; j < kListK; ++j)
            partial[(static_cast<int64_t>(blockIdx.x) * n_queries + q) * kListK + j] = m[j];
    }
}

// Merge the per-CTA lists of one query into its k best, one warp per query:
// each lane merges a strided share of the CTAs' lists, then five butterfly
// rounds merge the lanes' lists (keys are unique, so both partners of a round
// end with the same list).
__global__ void finalize_topk_kernel(const unsigned long long *__restrict__ partial, int n_parts,
                                     int n_queries, int k, int64_t *__restrict__ best_idx,
                                     float *__restrict__ best_score) {
    const int q = (blockIdx.x * blockDim.x + threadIdx.x) >> 5;
    const int lane = threadIdx.x & 31;
    if (q >= n_queries) return;
    unsigned long long l[kListK];
#pragma unroll
    for (int j = 0; j < kListK; ++j) l[j] = 0ull;
    for (int i = lane; i < n_parts; i += 32)
        for (int j = 0; j < kListK; ++j) {
            const unsigned long long v = partial[(static_cast<int64_t>(i) * n_queries + q) * kListK + j];
            if (v <= l[kListK - 1]) break;   // each part's list is sorted: the rest is smaller
            list_insert(l, v);
        }
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) {
        unsigned long long other[kListK];
#pragma unroll
        for (int j = 0; j < kListK; ++j) other[j] = shfl_xor_u64(l[j], o);
#pragma unroll
        for (int j = 0; j < kListK; ++j) list_insert(l, other[j]);
    }
    if (lane != 0) return;
    for (int j = 0; j < k; ++j) {
        const unsigned long long key = l[j];
        const int64_t o = static_cast<int64_t>(q) * k + j;
        if (key == 0ull) {
            best_idx[o] = -1;
            if (best_score) best_score[o] = __uint_as_float(0x7fc00000u);
        } else {
            best_idx[o] = static_cast<int64_t>(0xffffffffu - static_cast<uint32_t>(key & 0xffffffffu));
            if (best_score) best_score[o] = unordered_float(static_cast<uint32_t>(key >> 32));
        }
    }
}

int num_sms() { return device_sm_count(); }

constexpr int kRowsPerWarpPass = 4;

int gemv_grid(int64_t M) {
    const int64_t rows_per_cta = static_cast<int64_t>(kWarps) * kRowsPerWarpPass;
    const int64_t need = (M + rows_per_cta - 1) / rows_per_cta;
    const int64_t cap = static_cast<int64_t>(num_sms()) * 4;
    return static_cast<int>(need < 1 ? 1 : (need < cap ? need : cap));
}

template <typename T, int QB, int VPL>
cudaError_t launch_gemv_pass(const RetrieveParams &p, int grid, int q0, cudaStream_t stream) {
    constexpr int RIF = QB == 1 ? 4 : 2;
    gemv_top1_kernel<T, QB, VPL, RIF><<<grid, kThreads, 0, stream>>>(
        static_cast<const T *>(p.index), p.M, p.dim, static_cast<const T *>(p.queries), p.n_queries,
        q0, static_cast<unsigned long long *>(p.workspace));
    return cudaGetLastError();
}

template <typename T, int QB>
cudaError_t gemv_pass_vpl(const RetrieveParams &p, int grid, int q0, cudaStream_t stream) {
    const int vecs = p.dim / Vec<T>::n;
    const int vpl = (vecs + 31) / 32;
    if (vpl <= 1) return launch_gemv_pass<T, QB, 1>(p, grid, q0, stream);
    if (vpl <= 2) return launch_gemv_pass<T, QB, 2>(p, grid, q0, stream);
    if (vpl <= 3) return launch_gemv_pass<T, QB, 3>(p, grid, q0, stream);
    if (vpl <= 4) return launch_gemv_pass<T, QB, 4>(p, grid, q0, stream);
    if (vpl <= 8) return launch_gemv_pass<T, QB, 8>(p, grid, q0, stream);
    return launch_gemv_pass<T, QB, 16>(p, grid, q0, stream);
}

template <typename T>
cudaError_t launch_gemv(const RetrieveParams &p, cudaStream_t stream, int grid, uint64_t *launches) {
    cudaError_t e = cudaSuccess;
    if (p.n_queries == 1) {
        e = gemv_pass_vpl<T, 1>(p, grid, 0, stream);
        ++*launches;
    } else {
        for (int q0 = 0; q0 < p.n_queries && e == cudaSuccess; q0 += kQB, ++*launches)
            e = gemv_pass_vpl<T, kQB>(p, grid, q0, stream);
    }
    return e;
}

// 16-bit indexes go to the tensor cores: one pass over the keys for up to 256 queries,
// streamed by TMA; even a single query's pass is a little faster there (0.246 vs 0.266
// ms over 1M x 768 fp16 keys) than a CUDA-core GEMV, which needs a pass per 4 queries.
// fp32 indexes stay on the CUDA cores (the GEMV kernels below are instantiated for fp32
// keys only).
bool use_tc(const RetrieveParams &p) { return p.dtype != PRECOG_F32; }

template <typename T, int VPL>
cudaError_t launch_topk_pass(const RetrieveParams &p, int grid, int q, cudaStream_t stream) {
    gemv_topk_kernel<T, VPL><<<grid, kThreads, 0, stream>>>(
        static_cast<const T *>(p.index), p.M, p.dim, static_cast<const T *>(p.queries), p.n_queries, q,
        static_cast<unsigned long long *>(p.workspace));
    return cudaGetLastError();
}

template <typename T>
cudaError_t launch_gemv_topk(const RetrieveParams &p, cudaStream_t stream, int grid,
                             uint64_t *launches) {
    const int vpl = (p.dim / Vec<T>::n + 31) / 32;
    cudaError_t e = cudaSuccess;
    for (int q = 0; q < p.n_queries && e == cudaSuccess; ++q, ++*launches) {
        if (vpl <= 1) e = launch_topk_pass<T, 1>(p, grid, q, stream);
        else if (vpl <= 2) e = launch_topk_pass<T, 2>(p, grid, q, stream);
        else if (vpl <= 3) e = launch_topk_pass<T, 3>(p, grid, q, stream);
        else if (vpl <= 4) e = launch_topk_pass<T, 4>(p, grid, q, stream);
        else if (vpl <= 8) e = launch_topk_pass<T, 8>(p, grid, q, stream);
        else e = launch_topk_pass<T, 16>(p, grid, q, stream);
    }
    return e;
}

}  // namespace

size_t retrieve_workspace_size(int64_t M, int32_t dim, int32_t n_queries) {
    (void)dim;
    if (n_queries <= 0) return 0;
    const int parts = std::max(gemv_grid(M), retrieve_tc_grid(M, num_sms()));
    return static_cast<size_t>(parts) * n_queries * sizeof(unsigned long long);
}

cudaError_t launch_retrieve(const RetrieveParams &p, cudaStream_t stream) {
    if (p.n_queries == 0) return cudaSuccess;
    const int sz = p.dtype == PRECOG_F32 ? 4 : 2;
    if (p.dim * sz / 16 > kMaxVecsPerRow) return cudaErrorInvalidValue;
    uint64_t launches = 0;
    cudaError_t e = cudaSuccess;
    int parts = 0;  // an empty index has no partial keys: the finalize writes row -1, score NaN
    if (p.M > 0 && use_tc(p)) {
        parts = retrieve_tc_grid(p.M, num_sms());
        e = launch_retrieve_tc(p, parts, stream, &launches);
    } else if (p.M > 0) {
        parts = gemv_grid(p.M);
        e = launch_gemv<float>(p, stream, parts, &launches);
    }
    if (e == cudaSuccess) {
        finalize_kernel<<<(p.n_queries + 3) / 4, 128, 0, stream>>>(
            static_cast<const unsigned long long *>(p.workspace), parts, p.n_queries, p.best_idx,
            p.best_score, p.row_offset, p.keys_out);
        e = cudaGetLastError();
        if (e == cudaSuccess) ++launches;
    }
    count_launches(launches);
    return e;
}

cudaError_t launch_decode_keys(const int64_t *keys, int32_t n, int64_t *best_idx, float *best_score,
                               cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    decode_keys_kernel<<<(n + 127) / 128, 128, 0, stream>>>(keys, n, best_idx, best_score);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

size_t retrieve_topk_workspace_size(int64_t M, int32_t dim, int32_t n_queries) {
    (void)dim;
    if (n_queries <= 0) return 0;
    const int parts = std::max(gemv_grid(M), retrieve_tc_grid(M, num_sms()));
    return static_cast<size_t>(parts) * n_queries * kListK * sizeof(unsigned long long);
}

cudaError_t launch_retrieve_topk(const RetrieveParams &p, int k, cudaStream_t stream) {
    if (p.n_queries == 0) return cudaSuccess;
    const int sz = p.dtype == PRECOG_F32 ? 4 : 2;
    if (p.dim * sz / 16 > kMaxVecsPerRow || k < 1 || k > kListK) return cudaErrorInvalidValue;
    uint64_t launches = 0;
    cudaError_t e = cudaSuccess;
    int parts = 0;  // an empty index has no partial lists: the finalize writes rows -1
    if (p.M > 0 && use_tc(p)) {
        parts = retrieve_tc_grid(p.M, num_sms());
        e = launch_retrieve_tc_topk(p, k, parts, stream, &launches);
    } else if (p.M > 0) {
        parts = gemv_grid(p.M);
        e = launch_gemv_topk<float>(p, stream, parts, &launches);
    }
    if (e == cudaSuccess) {
        finalize_topk_kernel<<<(p.n_queries + 3) / 4, 128, 0, stream>>>(
            static_cast<const unsigned long long *>(p.workspace), parts, p.n_queries, k, p.best_idx,
            p.best_score);
        e = cudaGetLastError();
        if (e == cudaSuccess) ++launches;
    }
    count_launches(launches);
    return e;
}

cudaError_t retrieve_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0, tc = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_retrieve_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    e = cudaMemcpyToSymbol(g_retrieve_status, &zero, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    e = retrieve_tc_status_word_read_clear(&tc);
    *bits |= tc;
    return e;
}

}  // namespace precog
