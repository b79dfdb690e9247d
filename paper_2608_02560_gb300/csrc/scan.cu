// Selective-SSM scan with final-state capture (corpus encode) and with an
// injected initial state (query prefill) -- Sec. 3 Eq. 1, Sec. 4.2, Eq. 2.
//
// Work decomposition: one CTA per (layer, chunk, slice of DS channels). Each
// thread owns CPT adjacent channels and keeps their N = 16 fp32 states in
// registers for the whole chunk. The chunk's rows of x and dt (DS channels
// each) and of B (and C) are staged into shared memory TILE tokens at a time
// by the TMA engine, completing on an mbarrier, in a STAGES-deep ring, so the
// time loop only reads shared memory: a whole-row slice is one contiguous 1-D
// bulk copy per tensor; a narrower slice (rows wider than 512 channels) is one
// tiled tensor-map copy of TILE rows per tensor.
//
// Per token and channel the recurrence is, for the 16 state indices n,
//   h[n] <- alpha_n * h[n] + (dt * x) * B[n],   alpha_n = exp(dt * A[d, n]).
// Three update forms, all in packed fp32x2 arithmetic:
//   kGeneral   one SFU exponential per (d, n);
//   kPower     A[d, n] = (n + 1) * A[d, 0] (stated by the caller, verified per
//              CTA): alpha_n = r^(n+1), r = exp(dt * A[d, 0]), one exponential
//              and a power chain per (t, d); with a readout y the state is
//              updated directly, without one it is accumulated rescaled
//              (see scan_tile_rescaled), which drops the per-n decay multiply.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_scan_status;

// Shape of the rescaled capture kernel (channels per thread, tokens per stage,
// stages, resident blocks per SM for the register budget).
#ifndef PRECOG_RESCALED_CPT
#define PRECOG_RESCALED_CPT 4
#endif
#ifndef PRECOG_RESCALED_TILE
#define PRECOG_RESCALED_TILE 16
#endif
#ifndef PRECOG_RESCALED_STAGES
#define PRECOG_RESCALED_STAGES 2
#endif
#ifndef PRECOG_RESCALED_MINB
#define PRECOG_RESCALED_MINB 6
#endif
// Shape of the direct-update kernels with A stated structured (readout, prefill).
#ifndef PRECOG_DIRECT_CPT
#define PRECOG_DIRECT_CPT 4
#endif
#ifndef PRECOG_DIRECT_TILE
#define PRECOG_DIRECT_TILE 16
#endif
#ifndef PRECOG_DIRECT_STAGES
#define PRECOG_DIRECT_STAGES 2
#endif
#ifndef PRECOG_DIRECT_MINB
#define PRECOG_DIRECT_MINB 5
#endif
#ifndef PRECOG_RESCALED_GROUP
#define PRECOG_RESCALED_GROUP 4
#endif


constexpr int kN = 16;          // state size (N) supported by the kernels
constexpr int kMaxSlice = 256;  // channels per CTA at most (the default slice)
constexpr int kWideSlice = 512; // rows of up to this many channels are staged whole
constexpr int kBarBytes = 128;  // barrier area at the start of shared memory
constexpr float kLog2e = 1.4426950408889634f;
constexpr int kMaxTopk = 8;     // states composed at most by one injection

__device__ __forceinline__ int64_t min64(int64_t a, int64_t b) { return a < b ? a : b; }

enum Mode { kGeneral = 0, kPower = 1 };

// Compile-time shape of one kernel instantiation.
constexpr int kTrajNone = 0, kTrajDirect = 1, kTrajRescaled = 2;

template <typename TIn_, bool HAS_Y_, bool HAS_H0_, int MODE_, int CPT_, int TILE_, int STAGES_,
          int MINB_, int TRAJ_ = kTrajNone, int MAXSLICE_ = kMaxSlice, int FIXDS_ = 0>
struct Cfg {
    using TIn = TIn_;
    // Channel slice known at compile time (0: a launch argument). A constant slice turns
    // the shared-memory row offsets of the time loop into immediates.
    static constexpr int FIXDS = FIXDS_;
    // Widest channel slice of one CTA. Each CTA stages its slice of every token row; a
    // slice narrower than the row turns the row into separate pieces, and HBM serves
    // short scattered pieces far below its streaming rate, so rows up to 512 channels
    // stay whole. MINB counts resident CTAs of kMaxSlice channels (the register budget
    // per thread), whatever the slice.
    static constexpr int MAXSLICE = MAXSLICE_;
    static constexpr int LB_SLICE = FIXDS_ ? FIXDS_ : MAXSLICE_;
    static constexpr int LB_THREADS = LB_SLICE / CPT_;
    static constexpr int LB_BLOCKS = MINB_ * kMaxSlice / LB_SLICE > 0 ? MINB_ * kMaxSlice / LB_SLICE : 1;
    static constexpr bool HAS_Y = HAS_Y_, HAS_H0 = HAS_H0_;
    // keep every stride-th state (K-dial, Sec. 5.2), with the direct or the rescaled update
    static constexpr int TRAJ = TRAJ_;
    static constexpr int MODE = MODE_, CPT = CPT_, TILE = TILE_, STAGES = STAGES_;
    static constexpr bool CONV = !std::is_same<TIn_, float>::value;
    static constexpr int SZ = sizeof(TIn_);
    static constexpr bool RESCALED = MODE_ == kPower && !HAS_Y_ && TRAJ_ != kTrajDirect;
};

// Where the next trajectory state goes: entry index and tokens left until it.
struct TrajCursor {
    int64_t entry;
    int64_t left;
};

// Tensor maps of x and dt for launches whose CTAs take a slice of each row: the tensor is
// viewed as [layer][row][D / inner][inner] (inner = min(slice, 256) channels, the widest
// box dimension), so a box of [1][TILE][slice / inner][inner] is one slice of TILE rows.
struct SliceMaps {
    CUtensorMap x, dt;
    int32_t valid, inner;
};

struct StageLayout {
    uint32_t xs, dts, bs, cs, bf, cf, bytes;
};

__host__ __device__ inline StageLayout stage_layout(int tile, int DS, int sz, bool has_y, bool conv) {
    StageLayout L;
    uint32_t o = 0;
    L.xs = o;
    o += tile * DS * sz;
    L.dts = o;
    o += tile * DS * sz;
    L.bs = o;
    o += tile * kN * sz;
    L.cs = o;
    if (has_y) o += tile * kN * sz;
    L.bf = o;
    if (conv) o += tile * kN * 4;
    L.cf = o;
    if (conv && has_y) o += tile * kN * 4;
    L.bytes = (o + 127u) & ~127u;
    return L;
}

// CPT adjacent channel values of one token row in shared memory; `neg` gets
// the sign bits of the raw values (nonzero if any is negative).
template <typename TIn, int CPT>
__device__ __forceinline__ void load_chan(const unsigned char *p, float (&v)[CPT], uint32_t &neg) {
    if constexpr (std::is_same<TIn, float>::value) {
        if constexpr (CPT == 2) {
            const float2 q = *reinterpret_cast<const float2 *>(p);
            v[0] = q.x;
            v[1] = q.y;
        } else {
            const float4 q = *reinterpret_cast<const float4 *>(p);
            v[0] = q.x;
            v[1] = q.y;
            v[2] = q.z;
            v[3] = q.w;
        }
        uint32_t s = 0;
#pragma unroll
        for (int j = 0; j < CPT; ++j) s |= __float_as_uint(v[j]);
        neg = s & 0x80000000u;
    } else {
        uint32_t w[CPT / 2];
        if constexpr (CPT == 2) {
            w[0] = *reinterpret_cast<const uint32_t *>(p);
        } else {
            const uint2 q = *reinterpret_cast<const uint2 *>(p);
            w[0] = q.x;
            w[1] = q.y;
        }
        uint32_t s = 0;
#pragma unroll
        for (int i = 0; i < CPT / 2; ++i) {
            v[2 * i] = __uint_as_float(w[i] << 16);
            v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
            s |= w[i];
        }
        neg = s & 0x80008000u;
    }
}

__device__ __forceinline__ void load_b(const float *bsrc, int t, f2 (&b)[8]) {
    const ulonglong2 *bv = reinterpret_cast<const ulonglong2 *>(bsrc + t * kN);
#pragma unroll
    for (int i = 0; i < 4; ++i) {
        const ulonglong2 v = bv[i];
        b[2 * i] = v.x;
        b[2 * i + 1] = v.y;
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

// p[i] = (r^(2i+1), r^(2i+2)) for i = 0..7
// (x*x, x*x) as one register pair with both halves computed: two multiplies the
// compiler may not merge, instead of one multiply and a register move.
__device__ __forceinline__ f2 sq_pair(float x) {
    float a, b;
    asm volatile("mul.rn.f32 %0, %1, %1;" : "=f"(a) : "f"(x));
    asm volatile("mul.rn.f32 %0, %1, %1;" : "=f"(b) : "f"(x));
    return pack2(a, b);
}

// pow_pairs for the direct update, whose FMA-heavy pipe the moves of duplicated pairs
// saturate (the rescaled capture keeps the move: there the extra multiplies cost more)
__device__ __forceinline__ void pow_pairs_direct(float r, f2 (&p)[8]) {
    const float r2 = r * r;
    p[0] = pack2(r, r2);
    const f2 rr = sq_pair(r);
#pragma unroll
    for (int i = 1; i < 8; ++i) p[i] = mul2(p[i - 1], rr);
}

__device__ __forceinline__ void pow_pairs(float r, f2 (&p)[8]) {
    const float r2 = r * r;
    p[0] = pack2(r, r2);
    const f2 rr = pack2(r2, r2);
#pragma unroll
    for (int i = 1; i < 8; ++i) p[i] = mul2(p[i - 1], rr);
}

// dt * x of the low (high) bf16 halves of two words, exact in fp32 (a product of two
// 8-bit significands), by the mixed-precision FMA with -0 as addend: no widening.
__device__ __forceinline__ float mul_bf16_lo(uint32_t a, uint32_t b) {
    float d;
    asm("{ .reg .b16 al, ah, bl, bh; mov.b32 {al, ah}, %1; mov.b32 {bl, bh}, %2;"
        " fma.rn.f32.bf16 %0, al, bl, %3; }"
        : "=f"(d) : "r"(a), "r"(b), "f"(-0.0f));
    return d;
}
// The same products as volatile statements (not merged with an equal one).
__device__ __forceinline__ float mul_bf16_lo_v(uint32_t a, uint32_t b) {
    float d;
    asm volatile("{ .reg .b16 al, ah, bl, bh; mov.b32 {al, ah}, %1; mov.b32 {bl, bh}, %2;"
                 " fma.rn.f32.bf16 %0, al, bl, %3; }"
                 : "=f"(d) : "r"(a), "r"(b), "f"(-0.0f));
    return d;
}
__device__ __forceinline__ float mul_bf16_hi_v(uint32_t a, uint32_t b) {
    float d;
    asm volatile("{ .reg .b16 al, ah, bl, bh; mov.b32 {al, ah}, %1; mov.b32 {bl, bh}, %2;"
                 " fma.rn.f32.bf16 %0, ah, bh, %3; }"
                 : "=f"(d) : "r"(a), "r"(b), "f"(-0.0f));
    return d;
}
__device__ __forceinline__ float mul_bf16_hi(uint32_t a, uint32_t b) {
    float d;
    asm("{ .reg .b16 al, ah, bl, bh; mov.b32 {al, ah}, %1; mov.b32 {bl, bh}, %2;"
        " fma.rn.f32.bf16 %0, ah, bh, %3; }"
        : "=f"(d) : "r"(a), "r"(b), "f"(-0.0f));
    return d;
}

template <int CPT>
__device__ __forceinline__ void load_words(const unsigned char *p, uint32_t (&w)[CPT / 2]) {
    if constexpr (CPT == 2) {
        w[0] = *reinterpret_cast<const uint32_t *>(p);
    } else {
        const uint2 q = *reinterpret_cast<const uint2 *>(p);
        w[0] = q.x;
        w[1] = q.y;
    }
}

template <int CPT>
__device__ __forceinline__ void widen_words(const uint32_t (&w)[CPT / 2], float (&v)[CPT]) {
#pragma unroll
    for (int i = 0; i < CPT / 2; ++i) {
        v[2 * i] = __uint_as_float(w[i] << 16);
        v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
}

// ---------------------------------------------------------------------------
// Direct update (any readout): h_n <- alpha_n h_n + u B_n, y = sum_n C_n h_n.
template <class C>
__device__ __forceinline__ void scan_tile_direct(const unsigned char *st, const StageLayout &lay,
                                                 int DS, int dl, int ntok,
                                                 f2 (&h)[C::CPT][8], const float (&kpow)[C::CPT],
                                                 const f2 (&kgen)[C::CPT][8], void *yrow,
                                                 int y_dtype, int64_t y_stride,
                                                 const ScanParams &p, TrajCursor &tc,
                                                 int64_t tok_left, int traj_layer, int dglob) {
    constexpr int CPT = C::CPT;
    const float *bsrc = reinterpret_cast<const float *>(st + (C::CONV ? lay.bf : lay.bs));
    const float *csrc = reinterpret_cast<const float *>(st + (C::CONV ? lay.cf : lay.cs));
    for (int t = 0; t < ntok; ++t) {
        f2 b[8];
        load_b(bsrc, t, b);
        float xv[CPT], dv[CPT], yv[CPT], uv[CPT];
        uint32_t neg;
        f2 uu2[CPT];   // (u, u) pairs of the 16-bit path, both halves computed
        if constexpr (C::CONV) {
            // u = dt * x from the raw bf16 halves (exact), x never widened
            uint32_t xw[CPT / 2], dw[CPT / 2];
            load_words<CPT>(st + lay.xs + (t * DS + dl) * C::SZ, xw);
            load_words<CPT>(st + lay.dts + (t * DS + dl) * C::SZ, dw);
            widen_words<CPT>(dw, dv);
#pragma unroll
            for (int i = 0; i < CPT / 2; ++i) {
                uv[2 * i] = mul_bf16_lo(dw[i], xw[i]);
                uv[2 * i + 1] = mul_bf16_hi(dw[i], xw[i]);
            }
#pragma unroll
            for (int i = 0; i < CPT / 2; ++i) {
                uu2[2 * i] = pack2(mul_bf16_lo_v(dw[i], xw[i]), mul_bf16_lo_v(dw[i], xw[i]));
                uu2[2 * i + 1] = pack2(mul_bf16_hi_v(dw[i], xw[i]), mul_bf16_hi_v(dw[i], xw[i]));
            }
        } else {
            load_chan<typename C::TIn, CPT>(st + lay.xs + (t * DS + dl) * C::SZ, xv, neg);
            load_chan<typename C::TIn, CPT>(st + lay.dts + (t * DS + dl) * C::SZ, dv, neg);
#pragma unroll
            for (int j = 0; j < CPT; ++j) uv[j] = dv[j] * xv[j];
        }
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const float u = uv[j];
            const f2 uu = C::CONV ? uu2[j] : pack2(u, u);
            if constexpr (C::MODE == kPower) {
                f2 a[8];
                pow_pairs_direct(ex2(dv[j] * kpow[j]), a);
#pragma unroll
                for (int i = 0; i < 8; ++i) h[j][i] = fma2(a[i], h[j][i], mul2(uu, b[i]));
            } else {
                const f2 dd = pack2(dv[j], dv[j]);
#pragma unroll
                for (int i = 0; i < 8; ++i) {
                    float e0, e1;
                    unpack2(mul2(dd, kgen[j][i]), e0, e1);
                    h[j][i] = fma2(pack2(ex2(e0), ex2(e1)), h[j][i], mul2(uu, b[i]));
                }
            }
            if constexpr (C::HAS_Y) {
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
        if constexpr (C::HAS_Y) {
            if (y_dtype == PRECOG_F32) {
                float *dst = static_cast<float *>(yrow) + t * y_stride;
                if constexpr (CPT == 2) {
                    *reinterpret_cast<float2 *>(dst) = make_float2(yv[0], yv[1]);
                } else {
                    *reinterpret_cast<float4 *>(dst) = make_float4(yv[0], yv[1], yv[2], yv[3]);
                }
            } else {
                __nv_bfloat16 *dst = static_cast<__nv_bfloat16 *>(yrow) + t * y_stride;
                __nv_bfloat162 p0 = __floats2bfloat162_rn(yv[0], yv[1]);
                if constexpr (CPT == 2) {
                    *reinterpret_cast<__nv_bfloat162 *>(dst) = p0;
                } else {
                    __nv_bfloat162 p1 = __floats2bfloat162_rn(yv[2], yv[3]);
                    *reinterpret_cast<uint2 *>(dst) = make_uint2(
                        *reinterpret_cast<uint32_t *>(&p0), *reinterpret_cast<uint32_t *>(&p1));
                }
            }
        }
        if constexpr (C::TRAJ == kTrajDirect) {
            // after every stride-th token and after the chunk's last token (uniform)
            if (--tc.left == 0 || t + 1 == tok_left) {
#pragma unroll
                for (int j = 0; j < CPT; ++j)
                    store_state16(p.traj, p.traj_dtype,
                                  ((tc.entry * p.L_out + traj_layer) * static_cast<int64_t>(p.D) + dglob + j) *
                                      kN,
                                  h[j]);
                ++tc.entry;
                tc.left = p.traj_stride;
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
// lane's L would leave [-kLmax, kLmax] the whole warp renormalises
// (h_n = G_n E^-(n+1), L = 0), which keeps E^(+-16) within 2^(16 * kLmax),
// far from fp32 overflow and underflow. A single token whose own increment is
// outside the window is applied to h directly.
constexpr float kLmax = 6.0f;

__device__ __forceinline__ void renormalise(f2 (&g)[8], float &L) {
    f2 p[8];
    pow_pairs(ex2(-L), p);
#pragma unroll
    for (int i = 0; i < 8; ++i) g[i] = mul2(g[i], p[i]);
    L = 0.f;
}

// G_n += u * E^(n+1) * B_n
__device__ __forceinline__ void accumulate_e(f2 (&g)[8], const f2 (&b)[8], float u, float E) {
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

// One token with the window check of every lane and channel.
template <int CPT>
__device__ __forceinline__ void token_checked(f2 (&g)[CPT][8], float (&L)[CPT],
                                              const float (&kk)[CPT], const f2 (&b)[8],
                                              const float (&xv)[CPT], const float (&dv)[CPT],
                                              unsigned wmask) {
    float Ln[CPT], u[CPT];
    bool need = false;
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        Ln[j] = fmaf(dv[j], kk[j], L[j]);
        u[j] = dv[j] * xv[j];
        need |= !(fabsf(Ln[j]) <= kLmax);
    }
    if (__any_sync(wmask, need)) {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
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
    for (int j = 0; j < CPT; ++j) {
        accumulate(g[j], b, u[j], Ln[j]);
        L[j] = Ln[j];
    }
}

// Moves the frame of G to the bottom of the window: h_n = G_n E^-(n+1) is re-expressed
// with L = -kLmax, G_n <- G_n 2^-((n+1)(L + kLmax)). With dt >= 0 the exponent then
// climbs through the whole window [-kLmax, kLmax] before the next renormalisation,
// twice as many tokens as a restart from L = 0. The factor of states 8..15 can fall
// below the fp32 range (s = L + kLmax <= 2 kLmax), so they take it in two multiplies,
// 2^-8s first; every factor and every intermediate stays within 2^(+-16 kLmax).
__device__ __forceinline__ void renorm_floor(f2 (&g)[8], float &L) {
    const float r = ex2(-(L + kLmax));
    const float r2 = r * r;
    f2 p[4];
    p[0] = pack2(r, r2);
    const f2 rr = pack2(r2, r2);
#pragma unroll
    for (int i = 1; i < 4; ++i) p[i] = mul2(p[i - 1], rr);
    float r7, r8;
    unpack2(p[3], r7, r8);
    const f2 q = pack2(r8, r8);
#pragma unroll
    for (int i = 0; i < 4; ++i) g[i] = mul2(g[i], p[i]);
#pragma unroll
    for (int i = 4; i < 8; ++i) g[i] = mul2(mul2(g[i], q), p[i - 4]);
    L = -kLmax;
}

// Tokens go in groups of kGroup. The group's exponents are summed first (one
// serial FMA per token and channel). With dt >= 0 they only grow, so checking
// the group's last exponent covers every token in it. One warp vote per group;
// the fast path then carries no branch, so the power chains of the group's
// tokens can interleave. When some lane's exponent would leave the window, the
// warp renormalises every channel to the bottom of the window before the group
// and takes the fast path all the same; only a negative dt anywhere in the group
// (seen from the sign bits) or a group whose own exponent increment exceeds the
// whole window goes through the per-token check.
constexpr int kGroup = PRECOG_RESCALED_GROUP;

template <class C>
__device__ __forceinline__ void scan_tile_rescaled(const unsigned char *st, const StageLayout &lay,
                                                   const float *bsrc, int DS, int dl, int t0, int ntok,
                                                   f2 (&g)[C::CPT][8], float (&L)[C::CPT],
                                                   const float (&kk)[C::CPT], unsigned wmask) {
    constexpr int CPT = C::CPT;
    using TIn = typename C::TIn;
    // 16-bit inputs: dt is kept as raw words across the vote, and u = dt * x is formed
    // from the raw halves
    constexpr bool MIX = C::CONV;
    int t = t0;
    for (; t + kGroup <= ntok; t += kGroup) {
        float dvk[kGroup][CPT], Lk[kGroup][CPT];
        uint32_t dw[kGroup][CPT / 2];
        uint32_t neg = 0;
#pragma unroll
        for (int k = 0; k < kGroup; ++k) {
            if constexpr (MIX) {
                load_words<CPT>(st + lay.dts + ((t + k) * DS + dl) * C::SZ, dw[k]);
                widen_words<CPT>(dw[k], dvk[k]);
#pragma unroll
                for (int i = 0; i < CPT / 2; ++i) neg |= dw[k][i];
            } else {
                uint32_t nk;
                load_chan<TIn, CPT>(st + lay.dts + ((t + k) * DS + dl) * C::SZ, dvk[k], nk);
                neg |= nk;
            }
#pragma unroll
            for (int j = 0; j < CPT; ++j) Lk[k][j] = fmaf(dvk[k][j], kk[j], k ? Lk[k - 1][j] : L[j]);
        }
        if constexpr (MIX) neg &= 0x80008000u;
        bool up = false;
#pragma unroll
        for (int j = 0; j < CPT; ++j) up |= !(Lk[kGroup - 1][j] <= kLmax);
        bool slow = false;
        if (__any_sync(wmask, up || neg != 0)) {
            slow = __any_sync(wmask, neg != 0);
            if (!slow) {
#pragma unroll
                for (int j = 0; j < CPT; ++j) renorm_floor(g[j], L[j]);
                bool up2 = false;
#pragma unroll
                for (int k = 0; k < kGroup; ++k) {
                    if constexpr (MIX) widen_words<CPT>(dw[k], dvk[k]);
#pragma unroll
                    for (int j = 0; j < CPT; ++j) Lk[k][j] = fmaf(dvk[k][j], kk[j], k ? Lk[k - 1][j] : L[j]);
                }
#pragma unroll
                for (int j = 0; j < CPT; ++j) up2 |= !(Lk[kGroup - 1][j] <= kLmax);
                slow = __any_sync(wmask, up2);
            }
        }
        if (slow) {
            // unrolled so that dvk stays in registers (no dynamic indexing)
#pragma unroll
            for (int k = 0; k < kGroup; ++k) {
                f2 b[8];
                float xv[CPT];
                uint32_t nx;
                load_b(bsrc, t + k, b);
                load_chan<TIn, CPT>(st + lay.xs + ((t + k) * DS + dl) * C::SZ, xv, nx);
                if constexpr (MIX) widen_words<CPT>(dw[k], dvk[k]);
                token_checked<CPT>(g, L, kk, b, xv, dvk[k], wmask);
            }
        } else {
            // the group's exponentials first, so that their latency overlaps the rest
            float Ek[kGroup][CPT];
#pragma unroll
            for (int k = 0; k < kGroup; ++k)
#pragma unroll
                for (int j = 0; j < CPT; ++j) Ek[k][j] = ex2(Lk[k][j]);
#pragma unroll
            for (int k = 0; k < kGroup; ++k) {
                f2 b[8];
                load_b(bsrc, t + k, b);
                float u[CPT];
                if constexpr (MIX) {
                    uint32_t xw[CPT / 2];
                    load_words<CPT>(st + lay.xs + ((t + k) * DS + dl) * C::SZ, xw);
#pragma unroll
                    for (int i = 0; i < CPT / 2; ++i) {
                        u[2 * i] = mul_bf16_lo(dw[k][i], xw[i]);
                        u[2 * i + 1] = mul_bf16_hi(dw[k][i], xw[i]);
                    }
                } else {
                    float xv[CPT];
                    uint32_t nx;
                    load_chan<TIn, CPT>(st + lay.xs + ((t + k) * DS + dl) * C::SZ, xv, nx);
#pragma unroll
                    for (int j = 0; j < CPT; ++j) u[j] = dvk[k][j] * xv[j];
                }
#pragma unroll
                for (int j = 0; j < CPT; ++j) accumulate_e(g[j], b, u[j], Ek[k][j]);
            }
#pragma unroll
            for (int j = 0; j < CPT; ++j) L[j] = Lk[kGroup - 1][j];
        }
    }
    for (; t < ntok; ++t) {
        f2 b[8];
        float xv[CPT], dv[CPT];
        uint32_t n0;
        load_b(bsrc, t, b);
        load_chan<TIn, CPT>(st + lay.xs + (t * DS + dl) * C::SZ, xv, n0);
        load_chan<TIn, CPT>(st + lay.dts + (t * DS + dl) * C::SZ, dv, n0);
        token_checked<CPT>(g, L, kk, b, xv, dv, wmask);
    }
}

// ---------------------------------------------------------------------------
template <class C>
__global__ void __launch_bounds__(C::LB_THREADS, C::LB_BLOCKS)
    scan_kernel(const ScanParams p, const int DS_arg, const int slices, const __grid_constant__ SliceMaps maps) {
    using TIn = typename C::TIn;
    const int DS = C::FIXDS ? C::FIXDS : DS_arg;
    constexpr int CPT = C::CPT, TILE = C::TILE, STAGES = C::STAGES, SZ = C::SZ;
    extern __shared__ __align__(128) unsigned char smem[];
    uint64_t *full = reinterpret_cast<uint64_t *>(smem);
    unsigned char *stage0 = smem + kBarBytes;
    const StageLayout lay = stage_layout(TILE, DS, SZ, C::HAS_Y, C::CONV);
    const int tid = threadIdx.x;
    const int nthr = blockDim.x;

    // ---- work item ----
    int64_t item = blockIdx.x;
    const int slice = static_cast<int>(item % slices);
    item /= slices;
    const int64_t chunk = p.order ? p.order[item % p.n_chunks] : item % p.n_chunks;
    if (chunk < 0 || chunk >= p.n_chunks) {  // an order entry outside the chunks: skipped
        if (threadIdx.x == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_INDEX);
        return;
    }
    const int layer = static_cast<int>(item / p.n_chunks);
    // this thread's rows of A first (16 floats each, 16-byte loads): their latency overlaps
    // the chunk's offsets below
    float a_rows[CPT][kN];
    {
        const float *Al0 = p.A + static_cast<int64_t>(layer) * p.D * kN;
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const float4 *a4 = reinterpret_cast<const float4 *>(
                Al0 + static_cast<int64_t>(slice * DS + static_cast<int>(threadIdx.x) * CPT + j) * kN);
#pragma unroll
            for (int q = 0; q < kN / 4; ++q) {
                const float4 v = a4[q];
                a_rows[j][4 * q] = v.x;
                a_rows[j][4 * q + 1] = v.y;
                a_rows[j][4 * q + 2] = v.z;
                a_rows[j][4 * q + 3] = v.w;
            }
        }
    }
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
    TrajCursor tcur{0, 0};
    if constexpr (C::TRAJ) {
        // chunk c keeps ceil(len / stride) states starting at entry traj_offsets[c]
        const int64_t e0 = p.traj_offsets[chunk], e1 = p.traj_offsets[chunk + 1];
        if (e1 - e0 != (len + p.traj_stride - 1) / p.traj_stride) {
            if (tid == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_OFFSETS);
            return;
        }
        tcur.entry = e0;
        tcur.left = p.traj_stride;
    }
    const int d0 = slice * DS;
    const int dl = tid * CPT;
    const int D = p.D;
    const TIn *xl = static_cast<const TIn *>(p.x) + layer * p.ls_xd;
    const TIn *dtl = static_cast<const TIn *>(p.dt) + layer * p.ls_xd;
    const TIn *Bl = static_cast<const TIn *>(p.B) + layer * p.ls_bc;
    const TIn *Cl = C::HAS_Y ? static_cast<const TIn *>(p.C) + layer * p.ls_bc : nullptr;

    // ---- coefficients; kPower verifies the structure (A[d, n] = (n + 1) A[d, 0] <= 0) ----
    float kpow[CPT];      // A[d, 0] * log2 e
    f2 kgen[CPT][8];      // (A[d, n] * log2 e) pairs, kGeneral only
    bool a_ok = true;
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        const float (&a)[kN] = a_rows[j];
        kpow[j] = a[0] * kLog2e;
        if constexpr (C::MODE == kGeneral) {
#pragma unroll
            for (int i = 0; i < 8; ++i) kgen[j][i] = pack2(a[2 * i] * kLog2e, a[2 * i + 1] * kLog2e);
        } else {
            a_ok &= a[0] <= 0.f;
#pragma unroll
            for (int n = 1; n < kN; ++n) a_ok &= a[n] == static_cast<float>(n + 1) * a[0];
        }
    }
    if constexpr (C::MODE == kPower) {
        if (!__syncthreads_and(a_ok)) {
            if (tid == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_A);
            return;
        }
    }

    // ---- pipeline start: barrier init, first STAGES tiles in flight ----
    const int64_t ntiles = (len + TILE - 1) / TILE;
    if (tid == 0) {
        for (int s = 0; s < STAGES; ++s) mbar_init(&full[s], 1);
        fence_barrier_init();
    }
    __syncthreads();
    auto issue = [&](int64_t k) {  // thread 0 only
        const int s = static_cast<int>(k % STAGES);
        unsigned char *st = stage0 + s * lay.bytes;
        const int64_t row0 = start + k * TILE;
        const int ntok = static_cast<int>(min64(TILE, len - k * TILE));
        const uint32_t rowb = DS * SZ;
        const uint32_t bytes = ntok * rowb * 2 + ntok * kN * SZ * (C::HAS_Y ? 2 : 1);
        if (DS == D) {
            mbar_arrive_expect_tx(&full[s], bytes);
            bulk_g2s(st + lay.xs, xl + row0 * D, ntok * rowb, &full[s]);
            bulk_g2s(st + lay.dts, dtl + row0 * D, ntok * rowb, &full[s]);
        } else if (maps.valid) {
            // the slice of TILE rows as one tensor-map copy per tensor (a box always moves
            // TILE rows; rows past the end of the tensor arrive as zeros)
            mbar_arrive_expect_tx(&full[s], bytes + (TILE - ntok) * rowb * 2);
            tma_load_4d(st + lay.xs, &maps.x, 0, d0 / maps.inner, static_cast<int32_t>(row0), layer, &full[s]);
            tma_load_4d(st + lay.dts, &maps.dt, 0, d0 / maps.inner, static_cast<int32_t>(row0), layer, &full[s]);
        } else {
            mbar_arrive_expect_tx(&full[s], bytes);
            for (int r = 0; r < ntok; ++r) {
                bulk_g2s(st + lay.xs + r * rowb, xl + (row0 + r) * D + d0, rowb, &full[s]);
                bulk_g2s(st + lay.dts + r * rowb, dtl + (row0 + r) * D + d0, rowb, &full[s]);
            }
        }
        bulk_g2s(st + lay.bs, Bl + row0 * kN, ntok * kN * SZ, &full[s]);
        if (C::HAS_Y) bulk_g2s(st + lay.cs, Cl + row0 * kN, ntok * kN * SZ, &full[s]);
    };
    if (tid == 0)
        for (int64_t k = 0; k < min64(STAGES, ntiles); ++k) issue(k);

    // ---- initial state (overlaps the first copies) ----
    f2 h[CPT][8];
    bool h0_valid = false;
    int64_t h0_row = 0;
    if constexpr (C::HAS_H0) {
        if (p.topk <= 1) {
            h0_row = p.idx ? p.idx[chunk] : chunk;
            h0_valid = h0_row >= 0 && h0_row < p.bank_entries;
            if (!h0_valid && !(p.idx && h0_row == -1) && tid == 0)
                atomicOr(&g_scan_status, PRECOG_DEV_BAD_INDEX);
        }
    }
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        if (C::HAS_H0 && h0_valid) {
            const int64_t off =
                ((h0_row * p.L_bank + p.layer0 + layer) * static_cast<int64_t>(D) + d0 + dl + j) * kN;
            load_state16(p.bank, p.bank_dtype, off, h[j]);
        } else {
#pragma unroll
            for (int i = 0; i < 8; ++i) h[j][i] = 0;
        }
    }
    if constexpr (C::HAS_H0) {
        if (p.topk > 1) {
            // Top-k composition (Sec. 4.4, Eq. smc-fusion): h_init = sum_j w_j bank[row_j],
            // w = softmax(score / temperature) over the valid rows (row -1 or a NaN score:
            // weight 0; a row outside the bank: weight 0 and PRECOG_DEV_BAD_INDEX).
            const int64_t *rows = p.idx + chunk * p.topk;
            const float *sc = p.topk_scores + chunk * p.topk;
            float w[kMaxTopk];
            float smax = -__int_as_float(0x7f800000);
#pragma unroll
            for (int k = 0; k < kMaxTopk; ++k) {
                w[k] = -__int_as_float(0x7f800000);
                if (k < p.topk) {
                    const int64_t r = rows[k];
                    const bool in_bank = r >= 0 && r < p.bank_entries;
                    if (!in_bank && r != -1 && tid == 0) atomicOr(&g_scan_status, PRECOG_DEV_BAD_INDEX);
                    const float z = sc[k] * p.inv_temp;
                    if (in_bank && !isnan(z)) {
                        w[k] = z;
                        smax = fmaxf(smax, z);
                    }
                }
            }
            float wsum = 0.f;
#pragma unroll
            for (int k = 0; k < kMaxTopk; ++k) {
                w[k] = (w[k] == -__int_as_float(0x7f800000)) ? 0.f : ex2((w[k] - smax) * kLog2e);
                wsum += w[k];
            }
#pragma unroll
            for (int k = 0; k < kMaxTopk; ++k) {
                if (k >= p.topk || w[k] == 0.f) continue;
                const float wk = w[k] / wsum;
                const f2 ww = pack2(wk, wk);
#pragma unroll
                for (int j = 0; j < CPT; ++j) {
                    f2 hk[8];
                    const int64_t off = ((rows[k] * p.L_bank + p.layer0 + layer) * static_cast<int64_t>(D) +
                                         d0 + dl + j) * kN;
                    load_state16(p.bank, p.bank_dtype, off, hk);
#pragma unroll
                    for (int i = 0; i < 8; ++i) h[j][i] = fma2(ww, hk[i], h[j][i]);
                }
            }
        }
    }
    const unsigned wmask = __activemask();
    float Lw[CPT], kk[CPT];
#pragma unroll
    for (int j = 0; j < CPT; ++j) {
        Lw[j] = 0.f;
        kk[j] = -kpow[j];
    }

    // ---- time loop ----
    void *yrow = nullptr;
    const int64_t y_stride = D;
    if (C::HAS_Y) {
        const int64_t off = (static_cast<int64_t>(layer) * p.T_tot + start) * D + d0 + dl;
        yrow = (p.y_dtype == PRECOG_F32) ? static_cast<void *>(static_cast<float *>(p.y) + off)
                                         : static_cast<void *>(static_cast<__nv_bfloat16 *>(p.y) + off);
    }
    for (int64_t k = 0; k < ntiles; ++k) {
        const int s = static_cast<int>(k % STAGES);
        const uint32_t par = static_cast<uint32_t>((k / STAGES) & 1);
        unsigned char *st = stage0 + s * lay.bytes;
        const int ntok = static_cast<int>(min64(TILE, len - k * TILE));
        const bool ok = mbar_wait(&full[s], par);
        if (C::CONV && ok) {
            const TIn *bsrc = reinterpret_cast<const TIn *>(st + lay.bs);
            float *bdst = reinterpret_cast<float *>(st + lay.bf);
            if constexpr (std::is_same<TIn, __nv_bfloat16>::value) {
                // four values per thread and step: one 8-byte read, one 16-byte write
                for (int i = tid * 4; i < ntok * kN; i += nthr * 4) {
                    const uint2 w = *reinterpret_cast<const uint2 *>(bsrc + i);
                    *reinterpret_cast<float4 *>(bdst + i) =
                        make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                                    __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
                }
            } else {
                for (int i = tid; i < ntok * kN; i += nthr) bdst[i] = to_f32(bsrc[i]);
            }
            if (C::HAS_Y) {
                const TIn *csrc = reinterpret_cast<const TIn *>(st + lay.cs);
                float *cdst = reinterpret_cast<float *>(st + lay.cf);
                if constexpr (std::is_same<TIn, __nv_bfloat16>::value) {
                    for (int i = tid * 4; i < ntok * kN; i += nthr * 4) {
                        const uint2 w = *reinterpret_cast<const uint2 *>(csrc + i);
                        *reinterpret_cast<float4 *>(cdst + i) =
                            make_float4(__uint_as_float(w.x << 16), __uint_as_float(w.x & 0xffff0000u),
                                        __uint_as_float(w.y << 16), __uint_as_float(w.y & 0xffff0000u));
                    }
                } else {
                    for (int i = tid; i < ntok * kN; i += nthr) cdst[i] = to_f32(csrc[i]);
                }
            }
        }
        if (!__syncthreads_and(ok)) {
            // Give up on this chunk: record it, let issued copies land, leave.
            if (tid == 0) {
                atomicOr(&g_scan_status, PRECOG_DEV_TIMEOUT);
                for (int64_t k2 = k; k2 < min64(k + STAGES, ntiles); ++k2)
                    mbar_wait(&full[k2 % STAGES], static_cast<uint32_t>((k2 / STAGES) & 1));
            }
            return;
        }
        if constexpr (C::RESCALED && C::TRAJ == kTrajRescaled) {
            // segments end at the trajectory points; there the state is brought back
            // to h (renormalised, L = 0), stored, and the accumulation continues
            int t = 0;
            while (t < ntok) {
                const int seg = static_cast<int>(min64(ntok - t, tcur.left));
                scan_tile_rescaled<C>(st, lay, reinterpret_cast<const float *>(st + (C::CONV ? lay.bf : lay.bs)), DS, dl, t,
                                      t + seg, h, Lw, kk, wmask);
                t += seg;
                tcur.left -= seg;
                if (tcur.left == 0 || k * TILE + t == len) {
#pragma unroll
                    for (int j = 0; j < CPT; ++j) {
                        renormalise(h[j], Lw[j]);
                        store_state16(p.traj, p.traj_dtype,
                                      ((tcur.entry * p.L_out + p.layer0 + layer) * static_cast<int64_t>(D) +
                                       d0 + dl + j) * kN,
                                      h[j]);
                    }
                    ++tcur.entry;
                    tcur.left = p.traj_stride;
                }
            }
        } else if constexpr (C::RESCALED) {
            scan_tile_rescaled<C>(st, lay, reinterpret_cast<const float *>(st + (C::CONV ? lay.bf : lay.bs)), DS, dl, 0,
                                  ntok, h, Lw, kk, wmask);
        } else {
            scan_tile_direct<C>(st, lay, DS, dl, ntok, h, kpow, kgen, yrow, p.y_dtype, y_stride, p, tcur,
                                len - k * TILE, p.layer0 + layer, d0 + dl);
        }
        if (C::HAS_Y) {
            yrow = (p.y_dtype == PRECOG_F32)
                       ? static_cast<void *>(static_cast<float *>(yrow) + TILE * y_stride)
                       : static_cast<void *>(static_cast<__nv_bfloat16 *>(yrow) + TILE * y_stride);
        }
        fence_proxy_async_smem();
        __syncthreads();
        if (tid == 0 && k + STAGES < ntiles) issue(k + STAGES);
    }

    // ---- state capture ----
    if constexpr (C::RESCALED) {
#pragma unroll
        for (int j = 0; j < CPT; ++j) renormalise(h[j], Lw[j]);
    }
    if (p.states) {
#pragma unroll
        for (int j = 0; j < CPT; ++j) {
            const int64_t off =
                ((chunk * p.L_out + p.layer0 + layer) * static_cast<int64_t>(D) + d0 + dl + j) * kN;
            store_state16(p.states, p.state_dtype, off, h[j]);
        }
    }
}

// Widest channel slice (<= maxslice channels, 16-byte rows) that divides D
// into whole threads of CPT channels.
int pick_slice(int D, int sz, int cpt, int maxslice) {
    const int cands[] = {512, 256, 128, 64, 32, 16, 8, 4, 2};
    for (int ds : cands)
        if (ds <= maxslice && D % ds == 0 && (ds * sz) % 16 == 0 && ds % cpt == 0) return ds;
    return 0;
}

// True when a full-width launch would have fewer CTAs than the device has SMs.
bool few_items(const ScanParams &p) {
    const int sms = device_sm_count();
    const int64_t slices = (p.D + kMaxSlice - 1) / kMaxSlice;
    return static_cast<int64_t>(p.n_layers) * p.n_chunks * slices < sms;
}

template <class C>
cudaError_t launch_cfg(const ScanParams &p, cudaStream_t stream) {
    const int DS = C::FIXDS ? (p.D % C::FIXDS == 0 && (C::FIXDS * C::SZ) % 16 == 0 ? C::FIXDS : 0)
                            : pick_slice(p.D, C::SZ, C::CPT, C::MAXSLICE);
    if (DS == 0) return cudaErrorInvalidValue;
    const int slices = p.D / DS;
    const StageLayout lay = stage_layout(C::TILE, DS, C::SZ, C::HAS_Y, C::CONV);
    const size_t smem = kBarBytes + static_cast<size_t>(C::STAGES) * lay.bytes;
    const int64_t items = static_cast<int64_t>(p.n_layers) * p.n_chunks * slices;
    if (items == 0) return cudaSuccess;
    if (items > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    SliceMaps maps{};
    if (DS < p.D) {
        const int inner = DS < 256 ? DS : 256;
        const cuuint64_t rows = static_cast<cuuint64_t>(p.T_tot);
        const cuuint64_t dims[4] = {static_cast<cuuint64_t>(inner), static_cast<cuuint64_t>(p.D / inner), rows,
                                    static_cast<cuuint64_t>(p.n_layers)};
        const cuuint64_t lstride = static_cast<cuuint64_t>(p.n_layers > 1 ? p.ls_xd : rows * p.D) * C::SZ;
        const cuuint64_t strides[3] = {static_cast<cuuint64_t>(inner) * C::SZ, static_cast<cuuint64_t>(p.D) * C::SZ,
                                       lstride};
        const cuuint32_t box[4] = {static_cast<cuuint32_t>(inner), static_cast<cuuint32_t>(DS / inner),
                                   static_cast<cuuint32_t>(C::TILE), 1};
        const CUtensorMapDataType dt = C::SZ == 4 ? CU_TENSOR_MAP_DATA_TYPE_FLOAT32 : CU_TENSOR_MAP_DATA_TYPE_BFLOAT16;
        maps.valid = encode_tiled_map(&maps.x, dt, 4, p.x, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_NONE) &&
                     encode_tiled_map(&maps.dt, dt, 4, p.dt, dims, strides, box, CU_TENSOR_MAP_SWIZZLE_NONE);
        maps.inner = inner;
    }
    auto kern = scan_kernel<C>;
    cudaError_t e = ensure_smem(reinterpret_cast<const void *>(kern), static_cast<int>(smem));
    if (e != cudaSuccess) return e;
    kern<<<static_cast<unsigned>(items), DS / C::CPT, smem, stream>>>(p, DS, slices, maps);
    e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

// Shapes: the rescaled capture kernel (the corpus-encode hot loop) and the
// direct kernels (readout, prefill, general A).
template <typename TIn, bool HAS_Y, bool HAS_H0, int MODE, int TRAJ = kTrajNone>
cudaError_t launch_t(const ScanParams &p, cudaStream_t stream) {
    if constexpr (TRAJ == kTrajRescaled) {
        return launch_cfg<Cfg<TIn, false, false, kPower, PRECOG_RESCALED_CPT, PRECOG_RESCALED_TILE,
                              PRECOG_RESCALED_STAGES, PRECOG_RESCALED_MINB, kTrajRescaled, kWideSlice>>(p, stream);
    } else if constexpr (TRAJ == kTrajDirect) {
        // short strides and general A: the direct update (h is at hand after every token)
        if constexpr (MODE == kPower)
            return launch_cfg<Cfg<TIn, false, false, MODE, PRECOG_DIRECT_CPT, PRECOG_DIRECT_TILE,
                                  PRECOG_DIRECT_STAGES, PRECOG_DIRECT_MINB, kTrajDirect, kWideSlice>>(p, stream);
        else
            return launch_cfg<Cfg<TIn, false, false, MODE, 2, 16, 4, 3, kTrajDirect>>(p, stream);
    } else if constexpr (MODE == kPower && !HAS_Y) {
        // the corpus encode of 256- and 512-channel slices (the paper's layer width, the
        // ragged and wide workloads' slices) gets the slice fixed at compile time
        if constexpr (!HAS_H0 && !std::is_same<TIn, float>::value) {
            const int ds = pick_slice(p.D, sizeof(TIn), PRECOG_RESCALED_CPT, kWideSlice);
            if (ds == 256)
                return launch_cfg<Cfg<TIn, false, false, MODE, PRECOG_RESCALED_CPT, PRECOG_RESCALED_TILE,
                                      PRECOG_RESCALED_STAGES, PRECOG_RESCALED_MINB, kTrajNone, kWideSlice, 256>>(
                    p, stream);
            if (ds == 512)
                return launch_cfg<Cfg<TIn, false, false, MODE, PRECOG_RESCALED_CPT, PRECOG_RESCALED_TILE,
                                      PRECOG_RESCALED_STAGES, PRECOG_RESCALED_MINB, kTrajNone, kWideSlice, 512>>(
                    p, stream);
        }
        return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, PRECOG_RESCALED_CPT, PRECOG_RESCALED_TILE,
                              PRECOG_RESCALED_STAGES, PRECOG_RESCALED_MINB, kTrajNone, kWideSlice>>(p, stream);
    } else {
        if constexpr (MODE == kPower) {
            // Fewer work items than SMs (a single query's prefill: one CTA per layer) is a
            // latency-bound launch: the latency-shaped kernel splits every channel's states
            // over four threads; shapes it does not take run two channels per thread.
            if (few_items(p)) {
                if (scan_latency_eligible(p)) return launch_scan_latency(p, stream);
                return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, 2, 16, 2, 3>>(p, stream);
            }
            if constexpr (!std::is_same<TIn, float>::value) {
                // 16-bit rows: 256- and 512-channel slices fixed at compile time
                const int ds = pick_slice(p.D, sizeof(TIn), PRECOG_DIRECT_CPT, kWideSlice);
                if (ds == 256)
                    return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, PRECOG_DIRECT_CPT, PRECOG_DIRECT_TILE,
                                          PRECOG_DIRECT_STAGES, PRECOG_DIRECT_MINB, kTrajNone, kWideSlice, 256>>(
                        p, stream);
                if (ds == 512)
                    return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, PRECOG_DIRECT_CPT, PRECOG_DIRECT_TILE,
                                          PRECOG_DIRECT_STAGES, PRECOG_DIRECT_MINB, kTrajNone, kWideSlice, 512>>(
                        p, stream);
            }
            return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, PRECOG_DIRECT_CPT, PRECOG_DIRECT_TILE,
                                  PRECOG_DIRECT_STAGES, PRECOG_DIRECT_MINB, kTrajNone, kWideSlice>>(p, stream);
        } else {
            // general A keeps 16 exponent coefficients per channel: 2 channels per thread
            return launch_cfg<Cfg<TIn, HAS_Y, HAS_H0, MODE, 2, 16, 4, 3>>(p, stream);
        }
    }
}

template <typename TIn, int MODE>
cudaError_t launch_mode(const ScanParams &p, cudaStream_t stream) {
    if (p.traj != nullptr) {
        // strides of at least a few token groups amortise the renormalisation at each
        // trajectory point, so they take the rescaled accumulation
        if constexpr (MODE == kPower)
            if (p.traj_stride >= 4 * kGroup) return launch_t<TIn, false, false, MODE, kTrajRescaled>(p, stream);
        return launch_t<TIn, false, false, MODE, kTrajDirect>(p, stream);
    }
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
