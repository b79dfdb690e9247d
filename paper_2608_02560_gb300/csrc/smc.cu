// Structured Memory Consolidation primitives (Sec. 5): two-level cluster
// routing (Eqs. smc-domain, smc-sub) and the semantic-state EMA (Eq. smc-ema).
// Session initialisation (Sec. 5.3) injects a semantic state with the
// ordinary prefill, so it needs no kernel of its own.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_smc_status;

constexpr int kRouteWarps = 8;

template <typename T>
__device__ __forceinline__ float dot_warp(const T *__restrict__ a, const T *__restrict__ b, int dim,
                                          int lane) {
    // fixed lane mapping and butterfly: the same two vectors always give the same score
    float acc = 0.f;
    for (int k = lane; k < dim; k += 32) acc = fmaf(to_f32(a[k]), to_f32(b[k]), acc);
#pragma unroll
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    return acc;
}

// One warp per embedding: the best domain prototype, then the best of that
// domain's J[m] sub-cluster prototypes (strict '>': lowest index on ties, NaN
// never wins). slot = m * J_max + j, or -1 when no comparable score exists.
template <typename T>
__global__ void __launch_bounds__(kRouteWarps * 32)
    smc_route_kernel(const T *__restrict__ emb, int64_t n, int dim, const T *__restrict__ dom, int M,
                     const T *__restrict__ sub, int J_max, const int32_t *__restrict__ J,
                     int32_t *__restrict__ out_m, int32_t *__restrict__ out_j,
                     int64_t *__restrict__ out_slot) {
    const int lane = threadIdx.x & 31;
    const int64_t c = static_cast<int64_t>(blockIdx.x) * kRouteWarps + (threadIdx.x >> 5);
    if (c >= n) return;
    const T *e = emb + c * dim;
    float best = -__int_as_float(0x7f800000);
    int m = -1;
    for (int i = 0; i < M; ++i) {
        const float s = dot_warp(e, dom + static_cast<int64_t>(i) * dim, dim, lane);
        if (s > best) {
            best = s;
            m = i;
        }
    }
    int j = -1;
    if (m >= 0) {
        int Jm = J[m];
        if (Jm > J_max || Jm < 0) {
            if (lane == 0) atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
            Jm = 0;
        }
        best = -__int_as_float(0x7f800000);
        for (int i = 0; i < Jm; ++i) {
            const float s = dot_warp(e, sub + (static_cast<int64_t>(m) * J_max + i) * dim, dim, lane);
            if (s > best) {
                best = s;
                j = i;
            }
        }
    }
    if (lane == 0) {
        out_m[c] = m;
        out_j[c] = j;
        if (out_slot) out_slot[c] = (m >= 0 && j >= 0) ? static_cast<int64_t>(m) * J_max + j : -1;
    }
}

// s[slot_c] <- (1 - alpha) s[slot_c] + alpha h_c for c = 0, 1, ... in order,
// one thread per state element; slot -1 deposits nothing.
template <typename TS>
__global__ void smc_consolidate_kernel(float *__restrict__ sem, int64_t n_slots, int64_t elems,
                                       const TS *__restrict__ states, const int64_t *__restrict__ slots,
                                       int64_t n, float alpha) {
    const float keep = 1.f - alpha;
    for (int64_t e = static_cast<int64_t>(blockIdx.x) * blockDim.x + threadIdx.x; e < elems;
         e += static_cast<int64_t>(gridDim.x) * blockDim.x) {
        for (int64_t c = 0; c < n; ++c) {
            const int64_t slot = slots[c];
            if (slot < 0) continue;
            if (slot >= n_slots) {
                if (e == 0) atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
                continue;
            }
            float *s = sem + slot * elems + e;
            *s = keep * *s + alpha * to_f32(states[c * elems + e]);
        }
    }
}

int sm_count() {
    static int sms = 0;
    if (sms == 0) {
        int dev = 0;
        cudaGetDevice(&dev);
        cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
        if (sms <= 0) sms = 1;
    }
    return sms;
}

}  // namespace

cudaError_t launch_smc_route(const void *emb, int dtype, int64_t n, int dim, const void *dom, int M,
                             const void *sub, int J_max, const int32_t *J, int32_t *out_m,
                             int32_t *out_j, int64_t *out_slot, cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((n + kRouteWarps - 1) / kRouteWarps);
    switch (dtype) {
        case PRECOG_F16:
            smc_route_kernel<__half><<<grid, kRouteWarps * 32, 0, stream>>>(
                static_cast<const __half *>(emb), n, dim, static_cast<const __half *>(dom), M,
                static_cast<const __half *>(sub), J_max, J, out_m, out_j, out_slot);
            break;
        case PRECOG_BF16:
            smc_route_kernel<__nv_bfloat16><<<grid, kRouteWarps * 32, 0, stream>>>(
                static_cast<const __nv_bfloat16 *>(emb), n, dim, static_cast<const __nv_bfloat16 *>(dom), M,
                static_cast<const __nv_bfloat16 *>(sub), J_max, J, out_m, out_j, out_slot);
            break;
        default:
            smc_route_kernel<float><<<grid, kRouteWarps * 32, 0, stream>>>(
                static_cast<const float *>(emb), n, dim, static_cast<const float *>(dom), M,
                static_cast<const float *>(sub), J_max, J, out_m, out_j, out_slot);
    }
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

cudaError_t launch_smc_consolidate(float *sem, int64_t n_slots, int64_t elems, const void *states,
                                   int states_dtype, const int64_t *slots, int64_t n, float alpha,
                                   cudaStream_t stream) {
    if (n == 0 || elems == 0) return cudaSuccess;
    const int threads = 256;
    const int64_t want = (elems + threads - 1) / threads;
    const unsigned grid = static_cast<unsigned>(want < sm_count() * 16 ? want : sm_count() * 16);
    if (states_dtype == PRECOG_BF16)
        smc_consolidate_kernel<__nv_bfloat16><<<grid, threads, 0, stream>>>(
            sem, n_slots, elems, static_cast<const __nv_bfloat16 *>(states), slots, n, alpha);
    else
        smc_consolidate_kernel<float><<<grid, threads, 0, stream>>>(
            sem, n_slots, elems, static_cast<const float *>(states), slots, n, alpha);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

cudaError_t smc_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_smc_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_smc_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
