// Selective-SSM scan with final-state capture (corpus encode) and with an
// injected initial state (query prefill) -- Sec. 3 Eq. 1, Sec. 4.2, Eq. 2.
//
// Work decomposition: one CTA per (layer, chunk, slice of DS channels). Each
// thread owns kCPT adjacent channels and keeps their N = 16 fp32 states in
// registers for the whole chunk. The chunk's rows of x and dt (DS channels
// each) and of B (and C) are staged into shared memory kTile tokens at a
// time by the TMA engine (1-D bulk copies completing on an mbarrier), in a
// kStages-deep ring, so the time loop only reads shared memory.
//
// Per token and channel the update is, for the 16 state indices n,
//   h[n] <- alpha_n * h[n] + (dt * x) * B[n],   alpha_n = exp(dt * A[d, n]),
// done as 8 packed fp32x2 multiply + 8 packed fp32x2 FMAs. When A[d, n] is
// (n + 1) * A[d, 0] for every n (checked per CTA), alpha_n = r^(n+1) with
// r = exp(dt * A[d, 0]): one SFU exponential per channel and a packed power
// chain instead of 16 exponentials.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_scan_status;

constexpr int kN = 16;          // state size (N) supported by the kernels
constexpr int kCPT = 2;         // channels per thread
constexpr int kTile = 16;       // tokens per pipeline stage
constexpr int kStages = 4;      // pipeline depth
constexpr int kMaxThreads = 128;
constexpr int kBarBytes = 128;  // barrier area at the start of shared memory
constexpr float kLog2e = 1.4426950408889634f;

__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

struct StageLayout {
    uint32_t xs, dts, bs, cs, bf, cf, bytes;
};

__host__ __device__ inline StageLayout stage_layout(int DS, int sz, bool has_y, bool conv) {
    StageLayout L;
    uint32_t o = 0;
    L.xs = o;
    o += kTile * DS * sz;
    L.dts = o;
    o += kTile * DS * sz;
    L.bs = o;
    o += kTile * kN * sz;
    L.cs = o;
    if (has_y) o += kTile * kN * sz;
    L.bf = o;
    if (conv) o += kTile * kN * 4;
    L.cf = o;
    if (conv && has_y) o += kTile * kN * 4;
    L.bytes = (o + 127u) & ~127u;
    return L;
}

template <typename TIn>
__device__ __forceinline__ void load_pair(const unsigned char *p, float &a, float &b) {
    if constexpr (std::is_same<TIn, float>::value) {
        const float2 v = *reinterpret_cast<const float2 *>(p);
        a = v.x;
        b = v.y;
    } else {
        const __nv_bfloat162 v = *reinterpret_cast<const __nv_bfloat162 *>(p);
        a = __low2float(v);
        b = __high2float(v);
    }
}

__device__ __forceinline__ void store_state16(void *base, int dtype, int64_t elem_off,
                                              const f2 (&h)[8]) {
    float v[16];
#pragma unroll
    for (int i = 0; i < 8; ++i) unpack2(h[i], v[2 * i], v[2 * i + 1]);
    if (dtype == PRECOG_F32) {
        float4 *dst = reinterpret_cast<float4 *>(static_cast<float *>(base) + elem_off);
#pragma unroll
        for (int i = 0; i < 4; ++i)
            dst[i] = make_float4(v[4 * i], v[4 * i + 1], v[4 * i + 2], v[4 * i + 3]);
    } else {
        uint4 *dst = reinterpret_cast<uint4 *>(static_cast<__nv_bfloat16 *>(base) + elem_off);
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            uint32_t w[4];
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                __nv_bfloat162 b2 = __floats2bfloat162_rn(v[8 * i + 2 * k], v[8 * i + 2 * k + 1]);
                w[k] = *reinterpret_cast<uint32_t *>(&b2);
            }
            dst[i] = make_uint4(w[0], w[1], w[2], w[3]);
        }
    }
}

__device__ __forceinline__ void load_state16(const void *base, int dtype, int64_t elem_off,
                                             f2 (&h)[8]) {
    float v[16];
    if (dtype == PRECOG_F32) {
        const float4 *src = reinterpret_cast<const float4 *>(static_cast<const float *>(base) + elem_off);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const float4 q = src[i];
            v[4 * i] = q.x;
            v[4 * i + 1] = q.y;
            v[4 * i + 2] = q.z;
            v[4 * i + 3] = q.w;
        }
    } else {
        const uint4 *src =
            reinterpret_cast<const uint4 *>(static_cast<const __nv_bfloat16 *>(base) + elem_off);
#pragma unroll
        for (int i = 0; i < 2; ++i) {
            const uint4 q = src[i];
            const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
            for (int k = 0; k < 4; ++k) {
                v[8 * i + 2 * k] = __uint_as_float(w[k] << 16);
                v[8 * i + 2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
            }
        }
    }
#pragma unroll
    for (int i = 0; i < 8; ++i) h[i] = pack2(v[2 * i], v[2 * i + 1]);
}

// Roll kTile (or fewer) tokens of one stage through the recurrence.
template <typename TIn, bool HAS_Y, bool POW>
__device__ __forceinline__ void scan_tile(const unsigned char *st, const StageLayout &lay, int DS,
                                          int dl, int ntok, f2 (&h)[kCPT][8],
                                          const float (&kpow)[kCPT], const f2 (&kgen)[kCPT][8],
                                          void *yrow, int y_dtype, int64_t y_stride) {
    constexpr bool CONV = !std::is_same<TIn, float>::value;
    constexpr int sz = sizeof(TIn);
    const float *bsrc = reinterpret_cast<const float *>(st + (CONV ? lay.bf : lay.bs));
    const float *csrc = reinterpret_cast<const float *>(st + (CONV ? lay.cf : lay.cs));
    for (int t = 0; t < ntok; ++t) {
        f2 b[8];
        const ulonglong2 *bv = reinterpret_cast<const ulonglong2 *>(bsrc + t * kN);
#pragma unroll
        for (int i = 0; i < 4; ++i) {
            const ulonglong2 v = bv[i];
            b[2 * i] = v.x;
            b[2 * i + 1] = v.y;
        }
        float xv[kCPT], dv[kCPT];
        load_pair<TIn>(st + lay.xs + (t * DS + dl) * sz, xv[0], xv[1]);
        load_pair<TIn>(st + lay.dts + (t * DS + dl) * sz, dv[0], dv[1]);
        float yv[kCPT];
#pragma unroll
        for (int j = 0; j < kCPT; ++j) {
            const float u = dv[j] * xv[j];
            const f2 uu = pack2(u, u);
            if constexpr (POW) {
                const float r = ex2(dv[j] * kpow[j]);
                const float r2 = r * r;
                f2 aa = pack2(r, r2);
                const f2 rr = pack2(r2, r2);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    if (i) aa = mul2(aa, rr);
                    h[j][i] = fma2(aa, h[j][i], mul2(uu, b[i]));
                }
            } else {
                const f2 dd = pack2(dv[j], dv[j]);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float e0, e1;
                    unpack2(mul2(dd, kgen[j][i]), e0, e1);
                    h[j][i] = fma2(pack2(ex2(e0), ex2(e1)), h[j][i], mul2(uu, b[i]));
                }
            }
            if constexpr (HAS_Y) {
                const ulonglong2 *cv = reinterpret_cast<const ulonglong2 *>(csrc + t * kN);
                f2 acc = 0;
#pragma unroll
                for (int i = 0; i < 4; ++i) {
                    const ulonglong2 c = cv[i];
                    acc = (i == 0) ? mul2(c.x, h[j][0]) : fma2(c.x, h[j][2 * i], acc);
                    acc = fma2(c.y, h[j][2 * i + 1], acc);
                }
                float lo, hi;
                unpack2(acc, lo, hi);
                yv[j] = lo + hi;
            }
        }
        if constexpr (HAS_Y) {
            if (y_dtype == PRECOG_F32) {
                float2 *dst = reinterpret_cast<float2 *>(static_cast<float *>(yrow) + t * y_stride);
                *dst = make_float2(yv[0], yv[1]);
            } else {
                __nv_bfloat162 *dst = reinterpret_cast<__nv_bfloat162 *>(
                    static_cast<__nv_bfloat16 *>(yrow) + t * y_stride);
                *dst = __floats2bfloat162_rn(yv[0], yv[1]);
            }
        }
    }
}

// ---------------------------------------------------------------------------
// Rescaled accumulation (capture without readout, A[d, n] = (n + 1) * a, a <= 0).
// With E_t = 2^(L_t), L_t = sum over the tokens since the last renormalisation
// of dt * (-a * log2 e), the state is h_n = E_t^-(n+1) * G_n and one token adds
//   G_n += (u * E_t^(n+1)) * B_n,     u = dt * x,
// so the per-n decay multiply of the direct update disappears: per token and
// channel one exponential, a packed power chain and 16 FMAs. Whenever some
// lane's L would pass kLmax the whole warp renormalises (h_n = G_n E^-(n+1),
// L = 0), which keeps E^16 <= 2^(16 * kLmax) far from fp32 overflow. A single
// token whose own increment exceeds kLmax is applied directly to h.
constexpr float kLmax = 6.0f;

// p[i] = (r^(2i+1), r^(2i+2)) for i = 0..7
__device__ __forceinline__ void pow_pairs(float r, f2 (&p)[8]) {
    const float r2 = r * r;
    p[0] = pack2(r, r2);
    const f2 rr = pack2(r2, r2);
#pragma unroll
    for (int i = 1; i < 8; ++i) p[i] = mul2(p[i - 1], rr);
}

__device__ __forceinline__ void renormalise(f2 (&g)[8], float &L) {
    f2 p[8];
    pow_pairs(ex2(-L), p);
#pragma unroll
    for (int i = 0; i < 8; ++i) g[i] = mul2(g[i], p[i]);
    L = 0.f;
}

// G_n += u * 2^((n+1) * Ln) * B_n
__device__ __forceinline__ void accumulate(f2 (&g)[8], const f2 (&b)[8], float u, float Ln) {
    const float E = ex2(Ln);
    const float w0 = u * E;
    const float E2 = E * E;
    f2 w = pack2(w0, w0 * E);
    const f2 ee = pack2(E2, E2);
    g[0] = fma2(w, b[0], g[0]);
#pragma unroll
    for (int i = 1; i < 8; ++i) {
        w = mul2(w, ee);
        g[i] = fma2(w, b[i], g[i]);
    }
}

// One token with the window check: renormalise the whole warp when some lane
// would leave [-kLmax, kLmax]; a token whose own increment is outside it is
// applied to h directly (alpha_n = 2^(-(n+1)*Ln)) and contributes nothing to G.
__device__ __forceinline__ void token_checked(f2 (&g)[kCPT][8], float (&L)[kCPT],
                                              const float (&kk)[kCPT], const f2 (&b)[8],
                                              const float (&xv)[kCPT], const float (&dv)[kCPT],
                                              unsigned wmask) {
    float Ln[kCPT], u[kCPT];
    bool need = false;
#pragma unroll
    for (int j = 0; j < kCPT; ++j) {
        Ln[j] = fmaf(dv[j], kk[j], L[j]);
        u[j] = dv[j] * xv[j];
        need |= !(fabsf(Ln[j]) <= kLmax);
    }
    if (__any_sync(wmask, need)) {
#pragma unroll
        for (int j = 0; j < kCPT; ++j) {
            renormalise(g[j], L[j]);
            Ln[j] = dv[j] * kk[j];
            if (!(fabsf(Ln[j]) <= kLmax)) {
                f2 a[8];
                pow_pairs(ex2(-Ln[j]), a);
                const f2 uu = pack2(u[j], u[j]);
#pragma unroll
                for (int i = 0; i < 8; ++i) g[j][i] = fma2(a[i], g[j][i], mul2(uu, b[i]));
                Ln[j] = 0.f;
                u[j] = 0.f;
            }
        }
    }
#pragma unroll
    for (int j = 0; j < kCPT; ++j) {
        accumulate(g[j], b, u[j], Ln[j]);
        L[j] = Ln[j];
    }
}

template <typename TIn>
__device__ __forceinline__ void load_token(const unsigned char *st, const StageLayout &lay,
                                           const float *bsrc, int DS, int dl, int t, f2 (&b)[8],
                                           float (&xv)[kCPT], float (&dv)[kCPT]) {
    constexpr int sz = sizeof(TIn);
    const ulonglong2 *bv = reinterpret_cast<const ulonglong2 *>(bsrc + t * kN);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const ulonglong2 v = bv[i];
        b[2 * i] = v.x;
        b[2 * i + 1] = v.y;
    }
    load_pair<TIn>(st + lay.xs + (t * DS + dl) * sz, xv[0], xv[1]);
    load_pair<TIn>(st + lay.dts + (t * DS + dl) * sz, dv[0], dv[1]);
}

// Tokens go in groups of kGroup: the exponents of the whole group are summed
// first (one serial FMA per token), one warp vote decides whether the group
// stays inside the window, and then the group's accumulations carry no branch,
// so the scheduler can interleave the power chains of its tokens.
constexpr int kGroup = 4;

template <typename TIn>
__device__ __forceinline__ void scan_tile_rescaled(const unsigned char *st, const StageLayout &lay,
                                                   int DS, int dl, int ntok, f2 (&g)[kCPT][8],
                                                   float (&L)[kCPT], const float (&kk)[kCPT],
                                                   unsigned wmask) {
    constexpr bool CONV = !std::is_same<TIn, float>::value;
    constexpr int sz = sizeof(TIn);
    const float *bsrc = reinterpret_cast<const float *>(st + (CONV ? lay.bf : lay.bs));
    int t = 0;
    for (; t + kGroup <= ntok; t += kGroup) {
        float Lk[kGroup][kCPT];
        bool need = false;
#pragma unroll
        for (int k = 0; k < kGroup; ++k) {
            float dv[kCPT], xv[kCPT];
            load_pair<TIn>(st + lay.dts + ((t + k) * DS + dl) * sz, dv[0], dv[1]);
#pragma unroll
            for (int j = 0; j < kCPT; ++j) {
                Lk[k][j] = fmaf(dv[j], kk[j], k ? Lk[k - 1][j] : L[j]);
                need |= !(fabsf(Lk[k][j]) <= kLmax);
            }
            (void)xv;
        }
        if (__any_sync(wmask, need)) {
#pragma unroll 1
            for (int k = 0; k < kGroup; ++k) {
                f2 b[8];
                float xv[kCPT], dv[kCPT];
                load_token<TIn>(st, lay, bsrc, DS, dl, t + k, b, xv, dv);
                token_checked(g, L, kk, b, xv, dv, wmask);
            }
        } else {
#pragma unroll
            for (int k = 0; k < kGroup; ++k) {
                f2 b[8];
                float xv[kCPT], dv[kCPT];
                load_token<TIn>(st, lay, bsrc, DS, dl, t + k, b, xv, dv);
#pragma unroll
                for (int j = 0; j < kCPT; ++j) accumulate(g[j], b, dv[j] * xv[j], Lk[k][j]);
            }
#pragma unroll
            for (int j = 0; j < kCPT; ++j) L[j] = Lk[kGroup - 1][j];
        }
    }
    for (; t < ntok; ++t) {
        f2 b[8];
        float xv[kCPT], dv[kCPT];
        load_token<TIn>(st, lay, bsrc, DS, dl, t, b, xv, dv);
        token_checked(g, L, kk, b, xv, dv, wmask);
    }
}

// Update form of one kernel instantiation. kGeneral: one exponential per
// (d, n). kPower: A[d, n] = (n + 1) * A[d, 0] (the caller states it, every CTA
// verifies it): with readout, the direct update with a packed power chain;
// without readout, the rescaled accumulation above.
enum Mode { kGeneral = 0, kPower = 1 };

template <int MODE, bool HAS_Y> struct Shape {
    static constexpr bool kRescaled = MODE == kPower && !HAS_Y;
    static constexpr int kStagesUsed = kRescaled ? 2 : kStages;
    static constexpr int kMinBlocks = kRescaled ? 4 : 3;
};

template <typename TIn, bool HAS_Y, bool HAS_H0, int MODE>
__global__ void __launch_bounds__(kMaxThreads, (Shape<MODE, HAS_Y>::kMinBlocks))
    scan_kernel(const ScanParams p, const int DS, const int slices) {
    extern __shared__ __align__(128) unsigned char smem[];
    constexpr int sz = sizeof(TIn);
    constexpr bool CONV = !std::is_same<TIn, float>::value;
    constexpr bool RESCALED = Shape<MODE, HAS_Y>::kRescaled;
    constexpr int STAGES = Shape<MODE, HAS_Y>::kStagesUsed;
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    unsigned char *stage0 = smem + kBarBytes;
    const StageLayout lay = stage_layout(DS, sz, HAS_Y, CONV);
    const int tid = threadIdx.x;
    const int nthr = blockDim.x;

    // ---- work item ----
    int64_t item = blockIdx.x;
    const int slice = static_cast<int>(item % slices);
    item /= slices;
    const int64_t chunk = item % p.n_chunks;
    const int layer = static_cast<int>(item / p.n_chunks);
    int64_t start, len;
    if (p.use_fixed) {
        start = chunk * p.fixed_len;
        len = p.fixed_len;
    } else {
        start = p.offsets[chunk];
        const int64_t end = p.offsets[chunk + 1];
        if (start < 0 || end < start || end > p.T_tot) {
            if (tid == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_OFFSETS);
            return;
        }
        len = end - start;
    }
    const int d0 = slice * DS;
    const int dl = tid * kCPT;
    const int D = p.D;
    const TIn *xl = static_cast<const TIn *>(p.x) + layer * p.ls_xd;
    const TIn *dtl = static_cast<const TIn *>(p.dt) + layer * p.ls_xd;
    const TIn *Bl = static_cast<const TIn *>(p.B) + layer * p.ls_bc;
    const TIn *Cl = HAS_Y ? static_cast<const TIn *>(p.C) + layer * p.ls_bc : nullptr;
    const float *Al = p.A + static_cast<int64_t>(layer) * D * kN;

    // ---- coefficients; kPower verifies the structure before any copy is issued ----
    float kpow[kCPT];                      // A[d, 0] * log2 e
    f2 kgen[kCPT][8];                      // (A[d, n] * log2 e) pairs, kGeneral only
#pragma unroll
    for (int j = 0; j < kCPT; ++j) {
        const float *a = Al + static_cast<int64_t>(d0 + dl + j) * kN;
        kpow[j] = a[0] * kLog2e;
        if constexpr (MODE == kGeneral) {
#pragma unroll
            for (int i = 0; i < 8; ++i) kgen[j][i] = pack2(a[2 * i] * kLog2e, a[2 * i + 1] * kLog2e);
        }
    }
    if constexpr (MODE == kPower) {
        bool ok = true;
#pragma unroll
        for (int j = 0; j < kCPT; ++j) {
            const float *a = Al + static_cast<int64_t>(d0 + dl + j) * kN;
            const float a0 = a[0];
            ok &= a0 <= 0.f;
#pragma unroll
            for (int n = 1; n < kN; ++n) ok &= a[n] == static_cast<float>(n + 1) * a0;
        }
        if (!__syncthreads_and(ok)) {
            if (tid == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_A);
            return;
        }
    }

    // ---- pipeline start: barrier init, first STAGES tiles in flight ----
    const int64_t ntiles = (len + kTile - 1) / kTile;
    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) mbar_init(&full[s], 1);
        fence_barrier_init();
    }
    __syncthreads();
    auto issue = [&](int64_t k) {  // thread 0 only
        const int s = static_cast<int>(k % STAGES);
        unsigned char *st = stage0 + s * lay.bytes;
        const int64_t row0 = start + k * kTile;
        const int ntok = static_cast<int>(min64(kTile, len - k * kTile));
        const uint32_t rowb = DS * sz;
        const uint32_t bytes = ntok * rowb * 2 + ntok * kN * sz * (HAS_Y ? 2 : 1);
        mbar_arrive_expect_tx(&full[s], bytes);
        if (DS == D) {
            bulk_g2s(st + lay.xs, xl + row0 * D, ntok * rowb, &full[s]);
            bulk_g2s(st + lay.dts, dtl + row0 * D, ntok * rowb, &full[s]);
        } else {
            for (int r = 0; r < ntok; ++r) {
                bulk_g2s(st + lay.xs + r * rowb, xl + (row0 + r) * D + d0, rowb, &full[s]);
                bulk_g2s(st + lay.dts + r * rowb, dtl + (row0 + r) * D + d0, rowb, &full[s]);
            }
        }
        bulk_g2s(st + lay.bs, Bl + row0 * kN, ntok * kN * sz, &full[s]);
        if (HAS_Y) bulk_g2s(st + lay.cs, Cl + row0 * kN, ntok * kN * sz, &full[s]);
    };
    if (tid == 0)
        for (int64_t k = 0; k < min64(STAGES, ntiles); ++k) issue(k);

    // ---- initial state (overlaps the first copies) ----
    f2 h[kCPT][8];
    bool h0_valid = false;
    int64_t h0_row = 0;
    if constexpr (HAS_H0) {
        h0_row = p.idx ? p.idx[chunk] : chunk;
        h0_valid = h0_row >= 0 && h0_row < p.bank_entries;
        if (!h0_valid && !(p.idx && h0_row == -1) && tid == 0)
            atomicOr(&g_scan_status, PRECOG_DEV_BAD_INDEX);
    }
#pragma unroll
    for (int j = 0; j < kCPT; ++j) {
        if (HAS_H0 && h0_valid) {
            const int64_t off =
                ((h0_row * p.L_bank + p.layer0 + layer) * static_cast<int64_t>(D) + d0 + dl + j) * kN;
            load_state16(p.bank, p.bank_dtype, off, h[j]);
        } else {
#pragma unroll
            for (int i = 0; i < 8; ++i) h[j][i] = 0;
        }
    }
    const unsigned wmask = __activemask();
    float Lw[kCPT], kk[kCPT];
#pragma unroll
    for (int j = 0; j < kCPT; ++j) {
        Lw[j] = 0.f;
        kk[j] = -kpow[j];
    }

    // ---- time loop ----
    void *yrow = nullptr;
    const int64_t y_stride = D;
    if (HAS_Y) {
        const int64_t off = (static_cast<int64_t>(layer) * p.T_tot + start) * D + d0 + dl;
        yrow = (p.y_dtype == PRECOG_F32) ? static_cast<void *>(static_cast<float *>(p.y) + off)
                                         : static_cast<void *>(static_cast<__nv_bfloat16 *>(p.y) + off);
    }
    for (int64_t k = 0; k < ntiles; ++k) {
        const int s = static_cast<int>(k % STAGES);
        const uint32_t par = static_cast<uint32_t>((k / STAGES) & 1);
        unsigned char *st = stage0 + s * lay.bytes;
        const int ntok = static_cast<int>(min64(kTile, len - k * kTile));
        const bool ok = mbar_wait(&full[s], par);
        if (CONV && ok) {
            const TIn *bsrc = reinterpret_cast<const TIn *>(st + lay.bs);
            float *bdst = reinterpret_cast<float *>(st + lay.bf);
            for (int i = tid; i < ntok * kN; i += nthr) bdst[i] = to_f32(bsrc[i]);
            if (HAS_Y) {
                const TIn *csrc = reinterpret_cast<const TIn *>(st + lay.cs);
                float *cdst = reinterpret_cast<float *>(st + lay.cf);
                for (int i = tid; i < ntok * kN; i += nthr) cdst[i] = to_f32(csrc[i]);
            }
        }
        if (!__syncthreads_and(ok)) {
            // Give up on this chunk: record it, let issued copies land, leave.
            if (tid == 0) {
                atomicOr(&g_scan_status, PRECOG_DEV_TIMEOUT);
                for (int64_t kk2 = k; kk2 < min64(k + STAGES, ntiles); ++kk2)
                    mbar_wait(&full[kk2 % STAGES], static_cast<uint32_t>((kk2 / STAGES) & 1));
            }
            return;
        }
        if constexpr (RESCALED) {
            scan_tile_rescaled<TIn>(st, lay, DS, dl, ntok, h, Lw, kk, wmask);
        } else {
            scan_tile<TIn, HAS_Y, MODE == kPower>(st, lay, DS, dl, ntok, h, kpow, kgen, yrow,
                                                 p.y_dtype, y_stride);
        }
        if (HAS_Y) {
            yrow = (p.y_dtype == PRECOG_F32)
                       ? static_cast<void *>(static_cast<float *>(yrow) + kTile * y_stride)
                       : static_cast<void *>(static_cast<__nv_bfloat16 *>(yrow) + kTile * y_stride);
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0 && k + STAGES < ntiles) issue(k + STAGES);
    }

    // ---- state capture ----
    if constexpr (RESCALED) {
#pragma unroll
        for (int j = 0; j < kCPT; ++j) renormalise(h[j], Lw[j]);
    }
    if (p.states) {
#pragma unroll
        for (int j = 0; j < kCPT; ++j) {
            const int64_t off =
                ((chunk * p.L_out + p.layer0 + layer) * static_cast<int64_t>(D) + d0 + dl + j) * kN;
            store_state16(p.states, p.state_dtype, off, h[j]);
        }
    }
}

int pick_slice(int D, int sz) {
    const int cands[] = {256, 128, 64, 32, 16, 8, 4, 2};
    for (int ds : cands)
        if (D % ds == 0 && (ds * sz) % 16 == 0 && ds / kCPT <= kMaxThreads) return ds;
    return 0;
}

template <typename TIn, bool HAS_Y, bool HAS_H0, int MODE>
cudaError_t launch_t(const ScanParams &p, cudaStream_t stream) {
    const int sz = sizeof(TIn);
    const int DS = pick_slice(p.D, sz);
    if (DS == 0) return cudaErrorInvalidValue;
    const int slices = p.D / DS;
    const StageLayout lay = stage_layout(DS, sz, HAS_Y, !std::is_same<TIn, float>::value);
    const size_t smem = kBarBytes + static_cast<size_t>(Shape<MODE, HAS_Y>::kStagesUsed) * lay.bytes;
    const int64_t items = static_cast<int64_t>(p.n_layers) * p.n_chunks * slices;
    if (items == 0) return cudaSuccess;
    if (items > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    auto kern = scan_kernel<TIn, HAS_Y, HAS_H0, MODE>;
    static int smem_set = 0;
    cudaError_t e = ensure_smem(reinterpret_cast<const void *>(kern), &smem_set, static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    kern<<<static_cast<unsigned>(items), DS / kCPT, smem, stream>>>(p, DS, slices);
    e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

template <typename TIn, int MODE>
cudaError_t launch_mode(const ScanParams &p, cudaStream_t stream) {
    const bool has_y = p.y != nullptr;
    const bool has_h0 = p.bank != nullptr;
    if (has_y)
        return has_h0 ? launch_t<TIn, true, true, MODE>(p, stream)
                      : launch_t<TIn, true, false, MODE>(p, stream);
    return has_h0 ? launch_t<TIn, false, true, MODE>(p, stream)
                  : launch_t<TIn, false, false, MODE>(p, stream);
}

template <typename TIn>
cudaError_t launch_in(const ScanParams &p, cudaStream_t stream) {
    return p.a_kind == PRECOG_A_POWER ? launch_mode<TIn, kPower>(p, stream)
                                      : launch_mode<TIn, kGeneral>(p, stream);
}

}  // namespace

cudaError_t launch_scan(const ScanParams &p, cudaStream_t stream) {
    if (p.in_dtype == PRECOG_F32) return launch_in<float>(p, stream);
    return launch_in<__nv_bfloat16>(p, stream);
}

cudaError_t scan_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_scan_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_scan_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
