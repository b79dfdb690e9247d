// The direct-update scan with readout (Sec. 3 Eq. 1, y_t = C_t h_t) shaped for
// latency: launches with fewer work items than the GPU has SMs, above all the
// query prefill from an injected state (Sec. 4.2, Eq. 2) at batch 1, where each
// (layer, chunk) is a chain of dependent token steps and throughput does not
// matter. Four threads share a channel, each owning four of its N = 16 states,
// so a token step is short: two exponentials, a 3-multiply power step, four
// packed updates and a 4-lane sum of the partial readouts. CTAs cover 64
// channels (256 threads); tiles of 64 tokens are staged by bulk copies that
// 130 threads issue at once (one x row piece, one dt row piece, the B and C
// tiles), two tiles in flight.
//
// A is the power form (A[d,n] = (n+1) A[d,0] <= 0, verified per CTA before the
// first copies: overlapping the check with them measured 2 us slower): with
// r = 2^(dt * A[d,0] * log2 e), the thread owning states n0..n0+3 forms
// alpha_n0 = 2^((n0+1) * dt * A[d,0] * log2 e) on the SFU and the next three by
// multiplying with r.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_scan_latency_status;

constexpr int kN = 16;
constexpr int kLC = 64;                    // channels per CTA
constexpr int kLG = 4;                     // threads per channel (4 states each)
constexpr int kLThreads = kLC * kLG;
constexpr int kLT = 64;                    // tokens per tile
constexpr int kLStages = 2;
constexpr int kLMaxTopk = 8;
constexpr float kLog2e = 1.4426950408889634f;

template <typename TIn>
struct Tile {
    TIn x[kLT][kLC];
    TIn dt[kLT][kLC];
    TIn B[kLT][kN];
    TIn C[kLT][kN];
};

template <typename TIn>
struct LatSmem {
    Tile<TIn> tile[kLStages];
    uint64_t full[kLStages];
};

// Four consecutive values of a 16-value B or C row as two fp32 pairs.
template <typename TIn>
__device__ __forceinline__ void load4(const TIn *p, f2 &lo, f2 &hi) {
    if constexpr (std::is_same<TIn, float>::value) {
        const float4 v = *reinterpret_cast<const float4 *>(p);
        lo = pack2(v.x, v.y);
        hi = pack2(v.z, v.w);
    } else {
        const uint2 w = *reinterpret_cast<const uint2 *>(p);
        lo = pack2(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u));
        hi = pack2(__uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
    }
}

// Four states from a bank entry (fp32 or bf16), as two fp32 pairs.
__device__ __forceinline__ void load_state4(const void *base, int dtype, int64_t off, f2 &lo, f2 &hi) {
    if (dtype == PRECOG_F32) {
        const float4 v = *reinterpret_cast<const float4 *>(static_cast<const float *>(base) + off);
        lo = pack2(v.x, v.y);
        hi = pack2(v.z, v.w);
    } else {
        const uint2 w = *reinterpret_cast<const uint2 *>(static_cast<const __nv_bfloat16 *>(base) + off);
        lo = pack2(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u));
        hi = pack2(__uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
    }
}

__device__ __forceinline__ void store_state4(void *base, int dtype, int64_t off, f2 lo, f2 hi) {
    float v[4];
    unpack2(lo, v[0], v[1]);
    unpack2(hi, v[2], v[3]);
    if (dtype == PRECOG_F32) {
        *reinterpret_cast<float4 *>(static_cast<float *>(base) + off) = make_float4(v[0], v[1], v[2], v[3]);
    } else {
        __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
        *reinterpret_cast<uint2 *>(static_cast<__nv_bfloat16 *>(base) + off) =
            make_uint2(*reinterpret_cast<uint32_t *>(&a), *reinterpret_cast<uint32_t *>(&b));
    }
}

template <typename TIn, bool HAS_H0>
__global__ void __launch_bounds__(kLThreads)
    scan_latency_kernel(const ScanParams p, const int cblocks) {
    extern __shared__ __align__(128) unsigned char smem_raw[];
    LatSmem<TIn> &sm = *reinterpret_cast<LatSmem<TIn> *>(smem_raw);
    const int tid = threadIdx.x;
    const int c = tid / kLG, g = tid % kLG;
    int64_t item = blockIdx.x;
    const int cb = static_cast<int>(item % cblocks);
    item /= cblocks;
    const int64_t chunk = p.order ? p.order[item % p.n_chunks] : item % p.n_chunks;
    if (chunk < 0 || chunk >= p.n_chunks) {  // an order entry outside the chunks: skipped
        if (threadIdx.x == 0) atomicOr(&g_scan_latency_status, PRECOG_DEV_BAD_INDEX);
        return;
    }
    const int layer = static_cast<int>(item / p.n_chunks);
    const int D = p.D;
    const int d0 = cb * kLC;
    const int d = d0 + c;
    int64_t start, len;
    if (p.use_fixed) {
        start = chunk * p.fixed_len;
        len = p.fixed_len;
    } else {
        start = p.offsets[chunk];
        const int64_t end = p.offsets[chunk + 1];
        if (start < 0 || end < start || end > p.T_tot) {
            if (tid == 0) atomicOr(&g_scan_latency_status, PRECOG_DEV_BAD_OFFSETS);
            return;
        }
        len = end - start;
    }
    const TIn *xl = static_cast<const TIn *>(p.x) + layer * p.ls_xd;
    const TIn *dtl = static_cast<const TIn *>(p.dt) + layer * p.ls_xd;
    const TIn *Bl = static_cast<const TIn *>(p.B) + layer * p.ls_bc;
    const TIn *Cl = static_cast<const TIn *>(p.C) + layer * p.ls_bc;

    // ---- the power statement, verified before anything is staged or written ----
    const float *a = p.A + (static_cast<int64_t>(layer) * D + d) * kN;
    const float a0 = a[0];
    const float4 aq = *reinterpret_cast<const float4 *>(a + 4 * g);   // this thread's 4 values
    const float av[4] = {aq.x, aq.y, aq.z, aq.w};
    bool ok = a0 <= 0.f;
#pragma unroll
    for (int k = 0; k < 4; ++k) {
        const int n = 4 * g + k;
        ok &= av[k] == static_cast<float>(n + 1) * a0;
    }
    const float kpow = a0 * kLog2e;
    const float coef = static_cast<float>(4 * g + 1);

    if (!__syncthreads_and(ok)) {
        if (tid == 0) atomicOr(&g_scan_latency_status, PRECOG_DEV_BAD_A);
        return;
    }

    // ---- staging: every thread arrives on the tile's barrier; 130 of them bring bytes ----
    const int64_t ntiles = (len + kLT - 1) / kLT;
    if (tid == 0) {
        for (int s = 0; s < kLStages; ++s) mbar_init(&sm.full[s], kLThreads);
        fence_barrier_init();
    }
    __syncthreads();
    constexpr uint32_t SZ = sizeof(TIn);
    auto issue = [&](int64_t k) {
        const int s = static_cast<int>(k % kLStages);
        Tile<TIn> &tl = sm.tile[s];
        const int64_t row0 = start + k * kLT;
        const int ntok = static_cast<int>(len - k * kLT < kLT ? len - k * kLT : kLT);
        uint32_t bytes = 0;
        const void *src = nullptr;
        void *dst = nullptr;
        if (tid < ntok) {
            bytes = kLC * SZ;
            src = xl + (row0 + tid) * D + d0;
            dst = &tl.x[tid][0];
        } else if (tid >= kLT && tid < kLT + ntok) {
            bytes = kLC * SZ;
            src = dtl + (row0 + tid - kLT) * D + d0;
            dst = &tl.dt[tid - kLT][0];
        } else if (tid == 2 * kLT) {
            bytes = ntok * kN * SZ;
            src = Bl + row0 * kN;
            dst = &tl.B[0][0];
        } else if (tid == 2 * kLT + 1) {
            bytes = ntok * kN * SZ;
            src = Cl + row0 * kN;
            dst = &tl.C[0][0];
        }
        if (bytes) {
            mbar_arrive_expect_tx(&sm.full[s], bytes);
            bulk_g2s(dst, src, bytes, &sm.full[s]);
        } else {
            mbar_arrive(&sm.full[s]);
        }
    };
    for (int64_t k = 0; k < kLStages && k < ntiles; ++k) issue(k);

    // ---- initial state: the injected bank row, a softmax-weighted sum of rows, or zero ----
    f2 h01 = pack2(0.f, 0.f), h23 = pack2(0.f, 0.f);
    if constexpr (HAS_H0) {
        const int64_t soff = static_cast<int64_t>(p.layer0 + layer) * D * kN + static_cast<int64_t>(d) * kN + 4 * g;
        if (p.topk <= 1) {
            const int64_t row = p.idx ? p.idx[chunk] : chunk;
            if (row >= 0 && row < p.bank_entries) {
                load_state4(p.bank, p.bank_dtype, row * p.L_bank * D * kN + soff, h01, h23);
            } else if (!(p.idx && row == -1) && tid == 0) {
                atomicOr(&g_scan_latency_status, PRECOG_DEV_BAD_INDEX);
            }
        } else {
            // Top-k composition (Sec. 4.4): h_init = sum_j w_j bank[row_j], w = softmax of
            // score / temperature over the valid rows (row -1 or a NaN score: weight 0; a row
            // outside the bank: weight 0 and PRECOG_DEV_BAD_INDEX).
            const int64_t *rows = p.idx + chunk * p.topk;
            const float *sc = p.topk_scores + chunk * p.topk;
            float w[kLMaxTopk];
            float smax = -__int_as_float(0x7f800000);
#pragma unroll
            for (int k = 0; k < kLMaxTopk; ++k) {
                w[k] = -__int_as_float(0x7f800000);
                if (k < p.topk) {
                    const int64_t r = rows[k];
                    const bool in_bank = r >= 0 && r < p.bank_entries;
                    if (!in_bank && r != -1 && tid == 0) atomicOr(&g_scan_latency_status, PRECOG_DEV_BAD_INDEX);
                    const float z = sc[k] * p.inv_temp;
                    if (in_bank && !isnan(z)) {
                        w[k] = z;
                        smax = fmaxf(smax, z);
                    }
                }
            }
            float wsum = 0.f;
#pragma unroll
            for (int k = 0; k < kLMaxTopk; ++k) {
                w[k] = (w[k] == -__int_as_float(0x7f800000)) ? 0.f : ex2((w[k] - smax) * kLog2e);
                wsum += w[k];
            }
#pragma unroll
            for (int k = 0; k < kLMaxTopk; ++k) {
                if (k >= p.topk || w[k] == 0.f) continue;
                const float wk = w[k] / wsum;
                const f2 ww = pack2(wk, wk);
                f2 lo, hi;
                load_state4(p.bank, p.bank_dtype, rows[k] * p.L_bank * D * kN + soff, lo, hi);
                h01 = fma2(ww, lo, h01);
                h23 = fma2(ww, hi, h23);
            }
        }
    }

    // ---- token steps ----
    for (int64_t k = 0; k < ntiles; ++k) {
        const int s = static_cast<int>(k % kLStages);
        const int ntok = static_cast<int>(len - k * kLT < kLT ? len - k * kLT : kLT);
        const bool landed = mbar_wait(&sm.full[s], static_cast<uint32_t>((k / kLStages) & 1));
        if (!__syncthreads_and(landed)) {
            // give up on this chunk: record it, let the copies already issued land, leave
            if (tid == 0) {
                atomicOr(&g_scan_latency_status, PRECOG_DEV_TIMEOUT);
                for (int64_t k2 = k; k2 < k + kLStages && k2 < ntiles; ++k2)
                    mbar_wait(&sm.full[k2 % kLStages], static_cast<uint32_t>((k2 / kLStages) & 1));
            }
            return;
        }
        const Tile<TIn> &tl = sm.tile[s];
        const int64_t yrow = static_cast<int64_t>(layer) * p.T_tot + start + k * kLT;
#pragma unroll 4
        for (int t = 0; t < ntok; ++t) {
            const float dv = to_f32(tl.dt[t][c]);
            const float xv = to_f32(tl.x[t][c]);
            f2 b01, b23, c01, c23;
            load4<TIn>(&tl.B[t][4 * g], b01, b23);
            load4<TIn>(&tl.C[t][4 * g], c01, c23);
            const float lr = dv * kpow;
            const float an = ex2(lr * coef);     // r^(n0+1)
            const float r = ex2(lr);
            const float r2 = r * r;
            const f2 a01 = pack2(an, an * r);
            const f2 a23 = mul2(a01, pack2(r2, r2));
            const float u = dv * xv;
            const f2 uu = pack2(u, u);
            h01 = fma2(a01, h01, mul2(uu, b01));
            h23 = fma2(a23, h23, mul2(uu, b23));
            float y0, y1;
            unpack2(fma2(c23, h23, mul2(c01, h01)), y0, y1);
            float y = y0 + y1;
            y += __shfl_xor_sync(0xffffffffu, y, 1);
            y += __shfl_xor_sync(0xffffffffu, y, 2);
            if (g == 0) {
                const int64_t yo = (yrow + t) * D + d;
                if (p.y_dtype == PRECOG_F32) static_cast<float *>(p.y)[yo] = y;
                else static_cast<__nv_bfloat16 *>(p.y)[yo] = __float2bfloat16_rn(y);
            }
        }
        fence_proxy_async_smem();
        __syncthreads();   // every thread is done with stage s
        if (k + kLStages < ntiles) issue(k + kLStages);
    }

    if (p.states) {
        const int64_t off = ((chunk * p.L_out + p.layer0 + layer) * static_cast<int64_t>(D) + d) * kN + 4 * g;
        store_state4(p.states, p.state_dtype, off, h01, h23);
    }
}

template <typename TIn, bool HAS_H0>
cudaError_t launch_l(const ScanParams &p, cudaStream_t stream) {
    const int cblocks = p.D / kLC;
    const int64_t items = static_cast<int64_t>(p.n_layers) * p.n_chunks * cblocks;
    if (items == 0) return cudaSuccess;
    if (items > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const int smem = static_cast<int>(sizeof(LatSmem<TIn>));
    auto kern = scan_latency_kernel<TIn, HAS_H0>;
    cudaError_t e = ensure_smem(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    kern<<<static_cast<unsigned>(items), kLThreads, smem, stream>>>(p, cblocks);
    e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

}  // namespace

bool scan_latency_eligible(const ScanParams &p) {
    return p.y != nullptr && p.traj == nullptr && p.a_kind == PRECOG_A_POWER && p.N == kN &&
           p.D % kLC == 0 && (p.in_dtype == PRECOG_F32 || p.in_dtype == PRECOG_BF16) && p.topk <= kLMaxTopk;
}

cudaError_t launch_scan_latency(const ScanParams &p, cudaStream_t stream) {
    const bool h0 = p.bank != nullptr;
    if (p.in_dtype == PRECOG_F32) return h0 ? launch_l<float, true>(p, stream) : launch_l<float, false>(p, stream);
    return h0 ? launch_l<__nv_bfloat16, true>(p, stream) : launch_l<__nv_bfloat16, false>(p, stream);
}

cudaError_t scan_latency_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_scan_latency_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_scan_latency_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
