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
// one thread per state element. Deposits go in batches of kU: the batch's
// slots are read once into shared memory (uniform across the block), every
// thread issues the batch's state loads and slot loads together, folds the
// batch in deposit order and stores each touched slot once. When a slot
// repeats inside a batch the fold runs through a per-thread shared-memory
// column so that each repeat starts from the value its predecessor left.
// Slot -1 deposits nothing; a slot >= n_slots is flagged and skipped.
constexpr int kU = 32;
constexpr int kConsThreads = 256;

template <typename TS>
__global__ void __launch_bounds__(kConsThreads, 2)
    smc_consolidate_kernel(float *__restrict__ sem, int64_t n_slots, int64_t elems,
                           const TS *__restrict__ states, const int64_t *__restrict__ slots,
                           int64_t n, float alpha) {
    __shared__ int64_t s_slot[kU];
    __shared__ int64_t s_off[kU];   // slot * elems
    __shared__ int s_prev[kU];      // latest earlier position of the same slot in the batch, or -1
    __shared__ int s_last[kU];      // no later position of the batch has the same slot
    __shared__ int s_dups;
    __shared__ float s_val[kU][kConsThreads];
    const float keep = 1.f - alpha;
    const int tid = threadIdx.x;
    const int64_t e = static_cast<int64_t>(blockIdx.x) * kConsThreads + tid;
    for (int64_t c0 = 0; c0 < n; c0 += kU) {
        __syncthreads();                       // the previous batch is done with s_*
        if (tid < kU) {
            const int64_t c = c0 + tid;
            int64_t sl = c < n ? slots[c] : -1;
            if (sl >= n_slots) {
                if (blockIdx.x == 0) atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
                sl = -1;
            }
            if (sl < -1) sl = -1;
            s_slot[tid] = sl;
            s_off[tid] = sl >= 0 ? sl * elems : 0;
        }
        if (tid == 0) s_dups = 0;
        __syncthreads();
        if (tid < kU) {
            const int64_t sl = s_slot[tid];
            int prev = -1, last = 1;
            if (sl >= 0) {
                for (int i = 0; i < tid; ++i)
                    if (s_slot[i] == sl) prev = i;
                for (int i = tid + 1; i < kU; ++i)
                    if (s_slot[i] == sl) last = 0;
            }
            s_prev[tid] = prev;
            s_last[tid] = last;
            if (prev >= 0) atomicOr(&s_dups, 1);
        }
        __syncthreads();
        if (e >= elems) continue;
        float h[kU], v[kU];
#pragma unroll
        for (int j = 0; j < kU; ++j) {
            h[j] = 0.f;
            v[j] = 0.f;
            if (s_slot[j] >= 0) h[j] = to_f32(states[(c0 + j) * elems + e]);
        }
#pragma unroll
        for (int j = 0; j < kU; ++j)
            if (s_slot[j] >= 0 && s_prev[j] < 0) v[j] = sem[s_off[j] + e];
        if (!s_dups) {
#pragma unroll
            for (int j = 0; j < kU; ++j) v[j] = fmaf(keep, v[j], alpha * h[j]);
        } else {
#pragma unroll
            for (int j = 0; j < kU; ++j) {
                if (s_slot[j] < 0) continue;
                const int pj = s_prev[j];
                const float base = pj >= 0 ? s_val[pj][tid] : v[j];
                v[j] = fmaf(keep, base, alpha * h[j]);
                s_val[j][tid] = v[j];
            }
        }
#pragma unroll
        for (int j = 0; j < kU; ++j)
            if (s_slot[j] >= 0 && s_last[j]) sem[s_off[j] + e] = v[j];
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
    const int64_t blocks = (elems + kConsThreads - 1) / kConsThreads;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const unsigned grid = static_cast<unsigned>(blocks);
    if (states_dtype == PRECOG_BF16)
        smc_consolidate_kernel<__nv_bfloat16><<<grid, kConsThreads, 0, stream>>>(
            sem, n_slots, elems, static_cast<const __nv_bfloat16 *>(states), slots, n, alpha);
    else
        smc_consolidate_kernel<float><<<grid, kConsThreads, 0, stream>>>(
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
