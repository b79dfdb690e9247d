// The scan with the complex diagonal A that Eq. 1 prints (A_k = -softplus(a_k)
// + i*pi*k, h in C^N): alpha = exp(dt * A) = e^(dt*A_re) (cos + i sin)(dt*A_im),
// beta = B * x * dt real, y = Re(sum_n C_n h_n). One thread per channel with its
// 16 complex states in registers; blocks of 256 channels (128 with a readout,
// whose update needs more registers) stage tiles of 32 tokens of their x and dt
// row pieces and of the B (C) rows through a 2-stage shared-memory ring by TMA
// bulk copies on mbarriers (one copy per tensor when the block spans the whole
// row). Per-index form: one SFU exponential and one sine/cosine pair per
// (token, channel, state index); the phase dt * A_im is formed exactly as a
// two-float product (fma error term) and reduced to [-pi, pi] by Cody-Waite with
// 2*pi split into two floats before the SFU sine and cosine.
//
// Eq. 1's imaginary part is harmonic (A_im[n] = pi * n). When a block's A has
// A_im[n] == n * A_im[1] exactly and its inputs are 16-bit, the 16 phase
// rotations of a token are the powers z^n of one rotation z = e^(i dt A_im[1])
// (one reduced SFU sine and cosine per token and channel, the exact product error
// folded in), formed by a complex power tree of depth 3 on the FMA pipe; the
// magnitudes stay one exponential per state index (harmonic form). When the real
// part is also of power form (A_re[n] == (n+1) * A_re[0]), alpha_n = m * (m z)^n
// with m = e^(dt A_re[0]) and the magnitudes ride in the same tree (power form); a
// capture without readout accumulates the state rescaled (power form: one power tree
// of the weights and two real FMAs per state index, see renormalise_c; harmonic form:
// the rotation tree and one exponential per index, see renormalise_h). Other A, and
// fp32 inputs, keep the per-index form.
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_scan_complex_status;

constexpr int kN = 16;
constexpr float kLog2e = 1.4426950408889634f;
constexpr float kInv2Pi = 0.15915494309189535f;
constexpr float k2PiHi = 6.28318548202514648f;     // fp32 nearest to 2*pi
constexpr float k2PiLo = -1.7484556000744487e-07f; // 2*pi - k2PiHi

// sin and cos of the phases (th + tl) of two state indices at once. th is the rounded
// product dt * A_im and tl its exact error (an fma), so th + tl is the phase to twice
// fp32 precision; it is reduced by k = rint(th / 2pi) with 2pi split into a float and
// its remainder (Cody-Waite) before the SFU sine and cosine. Packed fp32x2 arithmetic
// halves the issue slots; each lane rounds exactly as the scalar sequence would.
__device__ __forceinline__ void sincos_pair(f2 th, f2 tl, f2 &s, f2 &c) {
    // k = rint(th / 2pi) on the FMA pipe: adding 1.5 * 2^23 rounds to an integer (round to
    // nearest even) for |th / 2pi| < 2^22; subtracting it again is exact. This keeps the
    // rounding off the SFU/conversion pipe, which the exponential, sine and cosine fill.
    const f2 big = pack2(12582912.f, 12582912.f), nbig = pack2(-12582912.f, -12582912.f);
    const f2 one = pack2(1.f, 1.f);
    const f2 k = fma2(fma2(th, pack2(kInv2Pi, kInv2Pi), big), one, nbig);
    f2 r = fma2(k, pack2(-k2PiHi, -k2PiHi), th);
    r = fma2(k, pack2(-k2PiLo, -k2PiLo), r);
    r = fma2(r, one, tl);
    float r0, r1, s0, s1, c0, c1;
    unpack2(r, r0, r1);
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s0) : "f"(r0));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c0) : "f"(r0));
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s1) : "f"(r1));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c1) : "f"(r1));
    s = pack2(s0, s1);
    c = pack2(c0, c1);
}

// (pr, pi) *= (wr, wi) for a pair of complex values held as a real pair and an
// imaginary pair; wr2 = (wr, wr), wi2 = (wi, wi), nwi2 = (-wi, -wi).
__device__ __forceinline__ void cmul_pair(f2 &pr, f2 &pi, f2 wr2, f2 wi2, f2 nwi2, f2 &qr, f2 &qi) {
    qr = fma2(pr, wr2, mul2(pi, nwi2));
    qi = fma2(pr, wi2, mul2(pi, wr2));
}

struct CScalar {
    f2 r, i, ni;   // (re, re), (im, im), (-im, -im)
};
__device__ __forceinline__ CScalar cbroadcast(float re, float im) {
    return CScalar{pack2(re, re), pack2(im, im), pack2(-im, -im)};
}
__device__ __forceinline__ void csquare(float re, float im, float &r2, float &i2) {
    r2 = fmaf(re, re, -im * im);
    i2 = 2.f * re * im;
}

// The eight pairs (w^(2i) p0, w^(2i+1) p0)... of a power tree: pairs[i] = pairs[0] * z2^i with
// z2 = w^2, from z2, z4 = z2^2 and z8 = z4^2 (depth 3: P1 = P0 z2, P2 = P0 z4, P3 = P1 z4,
// P4..P7 = P0..P3 z8).
__device__ __forceinline__ void power_tree(f2 (&pr)[8], f2 (&pi)[8], float z2r, float z2i) {
    float z4r, z4i, z8r, z8i;
    csquare(z2r, z2i, z4r, z4i);
    csquare(z4r, z4i, z8r, z8i);
    const CScalar w2 = cbroadcast(z2r, z2i), w4 = cbroadcast(z4r, z4i), w8 = cbroadcast(z8r, z8i);
    cmul_pair(pr[0], pi[0], w2.r, w2.i, w2.ni, pr[1], pi[1]);
    cmul_pair(pr[0], pi[0], w4.r, w4.i, w4.ni, pr[2], pi[2]);
    cmul_pair(pr[1], pi[1], w4.r, w4.i, w4.ni, pr[3], pi[3]);
#pragma unroll
    for (int j = 0; j < 4; ++j) cmul_pair(pr[j], pi[j], w8.r, w8.i, w8.ni, pr[4 + j], pi[4 + j]);
}

// e^(i (th + tl)) with th = dt * a the rounded product and tl its exact error: the phase
// reduced to [-pi, pi] as in sincos_pair, then the SFU sine and cosine (absolute error
// about 5e-7; the tree forms run only for 16-bit inputs, held to 2e-3).
__device__ __forceinline__ void rotation(float th, float tl, float &c, float &s) {
    const float k = fmaf(fmaf(th, kInv2Pi, 12582912.f), 1.f, -12582912.f);
    float r = fmaf(k, -k2PiHi, th);
    r = fmaf(k, -k2PiLo, r);
    r += tl;
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s) : "f"(r));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c) : "f"(r));
}

// One 16-value B or C row of a staged tile, widened to fp32 (vector shared-memory loads;
// every thread of the block reads the same row, a broadcast).
template <typename TIn>
__device__ __forceinline__ void widen_row(const TIn *row, float (&v)[kN]) {
    constexpr int kVec = static_cast<int>(kN * sizeof(TIn) / 16);
    const uint4 *r = reinterpret_cast<const uint4 *>(row);
#pragma unroll
    for (int i = 0; i < kVec; ++i) {
        const uint4 q = r[i];
        const uint32_t w[4] = {q.x, q.y, q.z, q.w};
#pragma unroll
        for (int k = 0; k < 4; ++k) {
            if constexpr (std::is_same<TIn, float>::value) {
                v[4 * i + k] = __uint_as_float(w[k]);
            } else {
                v[8 * i + 2 * k] = __uint_as_float(w[k] << 16);
                v[8 * i + 2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
            }
        }
    }
}

// ---- rescaled capture (power form, no readout) ----
// With P_n(t) = prod of alpha_n over the tokens since the last renormalisation
// = M^(n+1) Z^n (M = prod m, Z = prod z), the state is h_n = P_n G_n and a token adds
//   G_n += u B_n P_n^-1 = u B_n E^(n+1) R^n,   E = M^-1 = 2^L, R = conj(Z) = e^(-i Phi),
// L and Phi the running sums of dt * (-A_re[0] log2 e) and dt * A_im[1]: the weights
// are one power tree of V = E R per token and channel and the update is two real FMAs
// per state index (6 FP32 lane operations per index instead of the direct update's 9).
// The block renormalises (h_n = P_n G_n, L = Phi = 0) when some lane's L would leave
// [-kLmaxC, kLmaxC] (E^16 stays far inside fp32) and at least every kRenormTokens
// tokens (the rounding of the running phase, which the tree multiplies by n, stays
// below 64 roundings); a token whose own step leaves the window is applied directly.
constexpr float kLmaxC = 6.0f;
constexpr int kRenormTokens = 64;

// Phi + th + tl reduced to [-pi, pi] (Cody-Waite with 2 pi split in two floats; the
// rounding to an integer on the FMA pipe as in sincos_pair).
__device__ __forceinline__ float wrap_phase(float phi, float th, float tl) {
    const float a = (phi + th) + tl;
    const float k = fmaf(fmaf(a, kInv2Pi, 12582912.f), 1.f, -12582912.f);
    const float r = fmaf(k, -k2PiHi, a);
    return fmaf(k, -k2PiLo, r);
}

// The sixteen alpha_n = m^(n+1) z^n of the power form as pairs (real, imaginary):
// (alpha_2i, alpha_2i+1) = (m, m w) (w^2)^i with w = m z, m = 2^(dt A_re[0] log2 e),
// z = e^(i dt A_im[1]).
__device__ __forceinline__ void alpha_power(float dv, float a1, float kre, f2 (&are)[kN / 2],
                                            f2 (&aim)[kN / 2]) {
    const float th = dv * a1;
    float zr, zi;
    rotation(th, fmaf(dv, a1, -th), zr, zi);
    const float m = ex2(dv * kre);
    const float wr = m * zr, wi = m * zi;
    are[0] = pack2(m, m * wr);
    aim[0] = pack2(0.f, m * wi);
    float w2r, w2i;
    csquare(wr, wi, w2r, w2i);
    power_tree(are, aim, w2r, w2i);
}

// h <- alpha h + u B for the sixteen complex states (held as real and imaginary arrays)
__device__ __forceinline__ void update_direct(float (&hr)[kN], float (&hi)[kN], const f2 (&are)[kN / 2],
                                              const f2 (&aim)[kN / 2], f2 uu, const float (&b)[kN]) {
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        const f2 h_r = pack2(hr[2 * i], hr[2 * i + 1]), h_i = pack2(hi[2 * i], hi[2 * i + 1]);
        const f2 nh_i = pack2(-hi[2 * i], -hi[2 * i + 1]);
        const f2 nr = fma2(are[i], h_r, fma2(aim[i], nh_i, mul2(uu, pack2(b[2 * i], b[2 * i + 1]))));
        const f2 ni = fma2(are[i], h_i, mul2(aim[i], h_r));
        unpack2(nr, hr[2 * i], hr[2 * i + 1]);
        unpack2(ni, hi[2 * i], hi[2 * i + 1]);
    }
}

// h_n = M^(n+1) Z^n G_n with M = 2^-L, Z = e^(i phi); afterwards L = phi = 0
__device__ __forceinline__ void renormalise_c(float (&hr)[kN], float (&hi)[kN], float &L, float &phi) {
    const float M = ex2(-L);
    float c, s;
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s) : "f"(phi));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c) : "f"(phi));
    const float vr = M * c, vi = M * s;
    f2 are[kN / 2], aim[kN / 2];
    are[0] = pack2(M, M * vr);
    aim[0] = pack2(0.f, M * vi);
    float v2r, v2i;
    csquare(vr, vi, v2r, v2i);
    power_tree(are, aim, v2r, v2i);
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        const f2 g_r = pack2(hr[2 * i], hr[2 * i + 1]), g_i = pack2(hi[2 * i], hi[2 * i + 1]);
        const f2 ng_i = pack2(-hi[2 * i], -hi[2 * i + 1]);
        const f2 nr = fma2(are[i], g_r, mul2(aim[i], ng_i));
        const f2 ni = fma2(are[i], g_i, mul2(aim[i], g_r));
        unpack2(nr, hr[2 * i], hr[2 * i + 1]);
        unpack2(ni, hi[2 * i], hi[2 * i + 1]);
    }
    L = 0.f;
    phi = 0.f;
}

// G_n += u E^(n+1) R^n B_n with E = 2^L, R = e^(-i phi) (phi in [-pi, pi])
__device__ __forceinline__ void accumulate_c(float (&hr)[kN], float (&hi)[kN], float u, float L, float phi,
                                             const float (&b)[kN]) {
    const float E = ex2(L);
    float c, s;
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s) : "f"(phi));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c) : "f"(phi));
    const float vr = E * c, vi = -(E * s);
    const float ue = u * E;
    f2 wre[kN / 2], wim[kN / 2];
    wre[0] = pack2(ue, ue * vr);
    wim[0] = pack2(0.f, ue * vi);
    float v2r, v2i;
    csquare(vr, vi, v2r, v2i);
    power_tree(wre, wim, v2r, v2i);
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        const f2 bb = pack2(b[2 * i], b[2 * i + 1]);
        const f2 g_r = fma2(wre[i], bb, pack2(hr[2 * i], hr[2 * i + 1]));
        const f2 g_i = fma2(wim[i], bb, pack2(hi[2 * i], hi[2 * i + 1]));
        unpack2(g_r, hr[2 * i], hr[2 * i + 1]);
        unpack2(g_i, hi[2 * i], hi[2 * i + 1]);
    }
}

// ---- rescaled capture, harmonic form (A_im[n] = n A_im[1], any A_re) ----
// Here P_n = 2^(S c_n) Z^n with S the running sum of dt and c_n = A_re[n] log2 e, so a token
// adds u B_n 2^(-S c_n) R^n: the rotations R^n from the power tree seeded with u, one SFU
// exponential per state index for the magnitude, which multiplies B_n once for both the
// real and the imaginary FMA (8 FP32 lane operations per index instead of the direct
// update's 12). The weights' exponents -S c_n stay within [-kExpMaxC, kExpMaxC].
constexpr float kExpMaxC = 96.0f;

// pairs (s0 w^(2i), s0 w^(2i+1)) of the powers of w = (wr, wi), scaled by s0
__device__ __forceinline__ void rot_tree(float s0, float wr, float wi, f2 (&pr)[kN / 2], f2 (&pi)[kN / 2]) {
    pr[0] = pack2(s0, s0 * wr);
    pi[0] = pack2(0.f, s0 * wi);
    float w2r, w2i;
    csquare(wr, wi, w2r, w2i);
    power_tree(pr, pi, w2r, w2i);
}

// alpha_n = 2^(dt c_n) z^n of the harmonic form, z = e^(i dt A_im[1])
__device__ __forceinline__ void alpha_harmonic(float dv, float a1, const f2 (&ar)[kN / 2], f2 (&are)[kN / 2],
                                               f2 (&aim)[kN / 2]) {
    const float th = dv * a1;
    float zr, zi;
    rotation(th, fmaf(dv, a1, -th), zr, zi);
    rot_tree(1.f, zr, zi, are, aim);
    const f2 dd = pack2(dv, dv);
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        float e0, e1;
        unpack2(mul2(dd, ar[i]), e0, e1);
        const f2 mag = pack2(ex2(e0), ex2(e1));
        are[i] = mul2(mag, are[i]);
        aim[i] = mul2(mag, aim[i]);
    }
}

// h_n = 2^(S c_n) Z^n G_n with Z = e^(i phi); afterwards S = phi = 0
__device__ __forceinline__ void renormalise_h(float (&hr)[kN], float (&hi)[kN], const f2 (&ar)[kN / 2],
                                              float &S, float &phi) {
    float c, s;
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s) : "f"(phi));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c) : "f"(phi));
    f2 are[kN / 2], aim[kN / 2];
    rot_tree(1.f, c, s, are, aim);
    const f2 SS = pack2(S, S);
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        float e0, e1;
        unpack2(mul2(SS, ar[i]), e0, e1);
        const f2 mag = pack2(ex2(e0), ex2(e1));
        const f2 pr = mul2(mag, are[i]), pi = mul2(mag, aim[i]);
        const f2 g_r = pack2(hr[2 * i], hr[2 * i + 1]), g_i = pack2(hi[2 * i], hi[2 * i + 1]);
        const f2 ng_i = pack2(-hi[2 * i], -hi[2 * i + 1]);
        const f2 nr = fma2(pr, g_r, mul2(pi, ng_i));
        const f2 ni = fma2(pr, g_i, mul2(pi, g_r));
        unpack2(nr, hr[2 * i], hr[2 * i + 1]);
        unpack2(ni, hi[2 * i], hi[2 * i + 1]);
    }
    S = 0.f;
    phi = 0.f;
}

// G_n += u 2^(-S c_n) R^n B_n with R = e^(-i phi) (phi in [-pi, pi])
__device__ __forceinline__ void accumulate_h(float (&hr)[kN], float (&hi)[kN], const f2 (&ar)[kN / 2],
                                             float u, float S, float phi, const float (&b)[kN]) {
    float c, s;
    asm("sin.approx.ftz.f32 %0, %1;" : "=f"(s) : "f"(phi));
    asm("cos.approx.ftz.f32 %0, %1;" : "=f"(c) : "f"(phi));
    f2 wre[kN / 2], wim[kN / 2];
    rot_tree(u, c, -s, wre, wim);
    const f2 nS = pack2(-S, -S);
#pragma unroll
    for (int i = 0; i < kN / 2; ++i) {
        float e0, e1;
        unpack2(mul2(nS, ar[i]), e0, e1);
        const f2 mb = mul2(pack2(ex2(e0), ex2(e1)), pack2(b[2 * i], b[2 * i + 1]));
        const f2 g_r = fma2(wre[i], mb, pack2(hr[2 * i], hr[2 * i + 1]));
        const f2 g_i = fma2(wim[i], mb, pack2(hi[2 * i], hi[2 * i + 1]));
        unpack2(g_r, hr[2 * i], hr[2 * i + 1]);
        unpack2(g_i, hi[2 * i], hi[2 * i + 1]);
    }
}

constexpr int kCT = 32;     // tokens per staged tile
constexpr int kCS = 2;      // tiles in flight

template <typename TIn, int CB>
struct CTile {
    TIn x[kCT * CB];        // row stride: the block's width W <= CB
    TIn dt[kCT * CB];
    TIn B[kCT * kN];
    TIn C[kCT * kN];
};

template <typename TIn, int CB>
struct CSmem {
    uint64_t full[kCS];
    alignas(128) CTile<TIn, CB> tile[kCS];
    // the current tile's B and C rows widened to fp32 once per block (16-bit inputs)
    alignas(16) float bw[kCT * kN];
    alignas(16) float cw[kCT * kN];
};

// Update forms of a block, from the structure of its A.
constexpr int kFormIndex = 0;     // one exponential and one sine/cosine per state index
constexpr int kFormHarmonic = 1;  // A_im[n] = n A_im[1]: rotations from one sincosf
constexpr int kFormPower = 2;     // and A_re[n] = (n+1) A_re[0]: alpha_n = m (m z)^n

template <bool HAS_Y>
constexpr int block_channels() { return HAS_Y ? 128 : 256; }

template <typename TIn, bool HAS_Y, bool HAS_H0>
__global__ void __launch_bounds__(block_channels<HAS_Y>())
    scan_complex_kernel(const ScanParams p, const int cblocks) {
    constexpr int CB = block_channels<HAS_Y>();
    constexpr int SZ = static_cast<int>(sizeof(TIn));
    extern __shared__ __align__(128) unsigned char smem_raw[];
    CSmem<TIn, CB> &sm = *reinterpret_cast<CSmem<TIn, CB> *>(smem_raw);
    int64_t item = blockIdx.x;
    const int cb = static_cast<int>(item % cblocks);
    item /= cblocks;
    const int64_t chunk = p.order ? p.order[item % p.n_chunks] : item % p.n_chunks;
    if (chunk < 0 || chunk >= p.n_chunks) {  // an order entry outside the chunks: skipped
        if (threadIdx.x == 0) atomicOr(&g_scan_complex_status, PRECOG_DEV_BAD_INDEX);
        return;
    }
    const int layer = static_cast<int>(item / p.n_chunks);
    const int D = p.D;
    const int d0 = cb * CB;
    const int W = D - d0 < CB ? D - d0 : CB;    // channels of this block (a multiple of 16 bytes)
    const int tid = threadIdx.x;
    const bool live = tid < W;
    const int d = d0 + (live ? tid : 0);
    int64_t start, len;
    if (p.use_fixed) {
        start = chunk * p.fixed_len;
        len = p.fixed_len;
    } else {
        start = p.offsets[chunk];
        const int64_t end = p.offsets[chunk + 1];
        if (start < 0 || end < start || end > p.T_tot) {
            if (tid == 0) atomicOr(&g_scan_complex_status, PRECOG_DEV_BAD_OFFSETS);
            return;
        }
        len = end - start;
    }
    const TIn *xl = static_cast<const TIn *>(p.x) + layer * p.ls_xd;
    const TIn *dtl = static_cast<const TIn *>(p.dt) + layer * p.ls_xd;
    const TIn *Bl = static_cast<const TIn *>(p.B) + layer * p.ls_bc;
    const TIn *Cl = HAS_Y ? static_cast<const TIn *>(p.C) + layer * p.ls_bc : nullptr;
    const float2 *Al = reinterpret_cast<const float2 *>(p.A) + (static_cast<int64_t>(layer) * D + d) * kN;

    // ---- staging ring: first tiles in flight while A and the initial state load ----
    const int64_t ntiles = (len + kCT - 1) / kCT;
    if (tid == 0) {
        for (int s = 0; s < kCS; ++s) mbar_init(&sm.full[s], 1);
        fence_barrier_init();
    }
    __syncthreads();
    // warp 0: lane 0 states the tile's bytes, then the lanes copy it (one copy per tensor
    // when the block spans the row, else one row piece per lane and tensor)
    auto issue = [&](int64_t k) {
        const int lane = tid & 31;
        const int s = static_cast<int>(k % kCS);
        CTile<TIn, CB> &tl = sm.tile[s];
        const int64_t row0 = start + k * kCT;
        const int ntok = static_cast<int>(len - k * kCT < kCT ? len - k * kCT : kCT);
        const uint32_t rowb = static_cast<uint32_t>(W * SZ);
        const uint32_t bcb = static_cast<uint32_t>(ntok * kN * SZ);
        if (lane == 0) mbar_arrive_expect_tx(&sm.full[s], 2 * ntok * rowb + (HAS_Y ? 2 : 1) * bcb);
        __syncwarp();
        if (W == D) {
            if (lane == 0) {
                bulk_g2s(tl.x, xl + row0 * D, ntok * rowb, &sm.full[s]);
                bulk_g2s(tl.dt, dtl + row0 * D, ntok * rowb, &sm.full[s]);
            }
        } else if (lane < ntok) {
            bulk_g2s(tl.x + lane * W, xl + (row0 + lane) * D + d0, rowb, &sm.full[s]);
            bulk_g2s(tl.dt + lane * W, dtl + (row0 + lane) * D + d0, rowb, &sm.full[s]);
        }
        if (lane == 0) {
            bulk_g2s(tl.B, Bl + row0 * kN, bcb, &sm.full[s]);
            if (HAS_Y) bulk_g2s(tl.C, Cl + row0 * kN, bcb, &sm.full[s]);
        }
    };
    if (tid < 32)
        for (int64_t k = 0; k < kCS && k < ntiles; ++k) issue(k);

    // state indices in pairs (2i, 2i+1): A_re * log2 e, A_im, -A_im, and the state
    constexpr int kP = kN / 2;
    f2 ar[kP], ai[kP], nai[kP];
    bool harmonic = true, power = true;
    const float a1 = Al[1].y, re0 = Al[0].x;
#pragma unroll
    for (int i = 0; i < kP; ++i) {
        // the pair of complex values 2i, 2i+1 in one 16-byte load
        const float4 q = reinterpret_cast<const float4 *>(Al)[i];
        const float2 q0 = make_float2(q.x, q.y), q1 = make_float2(q.z, q.w);
        ar[i] = pack2(q0.x * kLog2e, q1.x * kLog2e);
        ai[i] = pack2(q0.y, q1.y);
        nai[i] = pack2(-q0.y, -q1.y);
        harmonic &= q0.y == static_cast<float>(2 * i) * a1 && q1.y == static_cast<float>(2 * i + 1) * a1;
        power &= q0.x == static_cast<float>(2 * i + 1) * re0 && q1.x == static_cast<float>(2 * i + 2) * re0;
    }
    // fp32 inputs keep the per-index form: the tree's rounding (about 1e-6 relative per
    // alpha) compounds over long memories past the 1e-5 agreement fp32 inputs are held to.
    const bool tree = !std::is_same<TIn, float>::value && __syncthreads_and(harmonic);
    const int form = tree ? (__syncthreads_and(power) ? kFormPower : kFormHarmonic) : kFormIndex;
    const float kre = re0 * kLog2e;

    float hr[kN], hi[kN];
#pragma unroll
    for (int n = 0; n < kN; ++n) {
        hr[n] = 0.f;
        hi[n] = 0.f;
    }
    if constexpr (HAS_H0) {
        const int64_t row = p.idx ? p.idx[chunk] : chunk;
        if (row >= 0 && row < p.bank_entries) {
            if (live) {
                const int64_t off = ((row * p.L_bank + p.layer0 + layer) * static_cast<int64_t>(D) + d) * kN;
#pragma unroll
                for (int n = 0; n < kN; ++n) {
                    if (p.bank_dtype == PRECOG_F32) {
                        const float2 v = reinterpret_cast<const float2 *>(p.bank)[off + n];
                        hr[n] = v.x;
                        hi[n] = v.y;
                    } else {
                        const __nv_bfloat162 v = reinterpret_cast<const __nv_bfloat162 *>(p.bank)[off + n];
                        hr[n] = __low2float(v);
                        hi[n] = __high2float(v);
                    }
                }
            }
        } else if (!(p.idx && row == -1) && tid == 0) {
            atomicOr(&g_scan_complex_status, PRECOG_DEV_BAD_INDEX);
        }
    }

    // B and C rows of token t as fp32: the block's widened copy for 16-bit inputs
    constexpr bool kWiden = !std::is_same<TIn, float>::value;
    auto b_row = [&](const CTile<TIn, CB> &tl, int t) -> const float * {
        if constexpr (kWiden) return sm.bw + t * kN;
        else return reinterpret_cast<const float *>(tl.B) + t * kN;
    };
    auto c_row = [&](const CTile<TIn, CB> &tl, int t) -> const float * {
        if constexpr (kWiden) return sm.cw + t * kN;
        else return reinterpret_cast<const float *>(tl.C) + t * kN;
    };

    // Runs token(tile, t, k) for every token of the chunk, a staged tile at a time; false
    // when a tile's wait hit its limit (recorded, and the copies already issued landed).
    auto scan_tiles = [&](auto &&token) -> bool {
        for (int64_t k = 0; k < ntiles; ++k) {
            const int s = static_cast<int>(k % kCS);
            const int ntok = static_cast<int>(len - k * kCT < kCT ? len - k * kCT : kCT);
            const bool landed = mbar_wait(&sm.full[s], static_cast<uint32_t>((k / kCS) & 1));
            if constexpr (kWiden) {
                // every thread has seen the tile land; the barrier below publishes the rows
                // (the previous tile's readers finished at the end of its iteration)
                if (landed) {
                    const CTile<TIn, CB> &tw = sm.tile[s];
                    for (int i = tid; i < ntok * kN; i += CB) sm.bw[i] = to_f32(tw.B[i]);
                    if (HAS_Y)
                        for (int i = tid; i < ntok * kN; i += CB) sm.cw[i] = to_f32(tw.C[i]);
                }
            }
            if (!__syncthreads_and(landed)) {
                if (tid == 0) {
                    atomicOr(&g_scan_complex_status, PRECOG_DEV_TIMEOUT);
                    for (int64_t k2 = k; k2 < k + kCS && k2 < ntiles; ++k2)
                        mbar_wait(&sm.full[k2 % kCS], static_cast<uint32_t>((k2 / kCS) & 1));
                }
                return false;
            }
            const CTile<TIn, CB> &tl = sm.tile[s];
            for (int t = 0; t < ntok && live; ++t) token(tl, t, k);
            fence_proxy_async_smem();
            __syncthreads();   // every thread is done with stage s
            if (tid < 32 && k + kCS < ntiles) issue(k + kCS);
        }
        return true;
    };

    if (!HAS_Y && form == kFormPower) {
        // rescaled capture: running exponent and phase, tokens since the last
        // renormalisation (the same count on every lane), the live lanes of this warp
        float Lc = 0.f, phc = 0.f;
        int since = 0;
        const unsigned lmask = __ballot_sync(0xffffffffu, live);
        const bool done = scan_tiles([&](const CTile<TIn, CB> &tl, int t, int64_t) {
            const float xv = to_f32(tl.x[t * W + tid]);
            const float dv = to_f32(tl.dt[t * W + tid]);
            const float u = dv * xv;
            float b[kN];
            widen_row<float>(b_row(tl, t), b);
            const f2 uu = pack2(u, u);
            const float th = dv * a1, tle = fmaf(dv, a1, -th);
            float Ln = fmaf(dv, -kre, Lc);
            float ph = wrap_phase(phc, th, tle);
            bool acc = true;
            if (__any_sync(lmask, !(fabsf(Ln) <= kLmaxC) || since >= kRenormTokens)) {
                renormalise_c(hr, hi, Lc, phc);
                since = 0;
                Ln = dv * -kre;
                ph = wrap_phase(0.f, th, tle);
                if (!(fabsf(Ln) <= kLmaxC)) {
                    f2 are[kP], aim[kP];
                    alpha_power(dv, a1, kre, are, aim);
                    update_direct(hr, hi, are, aim, uu, b);
                    Ln = 0.f;
                    ph = 0.f;
                    acc = false;
                }
            }
            if (acc) accumulate_c(hr, hi, u, Ln, ph, b);
            Lc = Ln;
            phc = ph;
            ++since;
        });
        if (!done) return;
        if (live) renormalise_c(hr, hi, Lc, phc);
    } else if (!HAS_Y && form == kFormHarmonic) {
        // rescaled capture, harmonic form: running sum of dt and phase; the window on the
        // weights' exponents is |S| * max_n |c_n| <= kExpMaxC
        float cmax = 0.f;
#pragma unroll
        for (int i = 0; i < kP; ++i) {
            float c0, c1;
            unpack2(ar[i], c0, c1);
            cmax = fmaxf(cmax, fmaxf(fabsf(c0), fabsf(c1)));
        }
        float Sc = 0.f, phc = 0.f;
        int since = 0;
        const unsigned lmask = __ballot_sync(0xffffffffu, live);
        const bool done = scan_tiles([&](const CTile<TIn, CB> &tl, int t, int64_t) {
            const float xv = to_f32(tl.x[t * W + tid]);
            const float dv = to_f32(tl.dt[t * W + tid]);
            const float u = dv * xv;
            float b[kN];
            widen_row<float>(b_row(tl, t), b);
            const float th = dv * a1, tle = fmaf(dv, a1, -th);
            float Sn = Sc + dv;
            float ph = wrap_phase(phc, th, tle);
            bool acc = true;
            if (__any_sync(lmask, !(fabsf(Sn) * cmax <= kExpMaxC) || since >= kRenormTokens)) {
                renormalise_h(hr, hi, ar, Sc, phc);
                since = 0;
                Sn = dv;
                ph = wrap_phase(0.f, th, tle);
                if (!(fabsf(Sn) * cmax <= kExpMaxC)) {
                    f2 are[kP], aim[kP];
                    alpha_harmonic(dv, a1, ar, are, aim);
                    update_direct(hr, hi, are, aim, pack2(u, u), b);
                    Sn = 0.f;
                    ph = 0.f;
                    acc = false;
                }
            }
            if (acc) accumulate_h(hr, hi, ar, u, Sn, ph, b);
            Sc = Sn;
            phc = ph;
            ++since;
        });
        if (!done) return;
        if (live) renormalise_h(hr, hi, ar, Sc, phc);
    } else {
        const bool done = scan_tiles([&](const CTile<TIn, CB> &tl, int t, int64_t k) {
            const float xv = to_f32(tl.x[t * W + tid]);
            const float dv = to_f32(tl.dt[t * W + tid]);
            const float u = dv * xv;
            float b[kN], cr[kN];
            widen_row<float>(b_row(tl, t), b);
            if constexpr (HAS_Y) widen_row<float>(c_row(tl, t), cr);
            const f2 dd = pack2(dv, dv), uu = pack2(u, u);
            // alpha for the eight pairs of state indices: (re pair, im pair)
            f2 are[kP], aim[kP];
            if (form == kFormIndex) {
#pragma unroll
                for (int i = 0; i < kP; ++i) {
                    float e0, e1;
                    unpack2(mul2(dd, ar[i]), e0, e1);
                    const f2 mag = pack2(ex2(e0), ex2(e1));
                    const f2 th = mul2(dd, ai[i]);
                    const f2 tl2 = fma2(dd, ai[i], mul2(dd, nai[i]));   // exact error of the product
                    f2 sn, cs;
                    sincos_pair(th, tl2, sn, cs);
                    are[i] = mul2(mag, cs);
                    aim[i] = mul2(mag, sn);
                }
            } else if (form == kFormPower) {
                alpha_power(dv, a1, kre, are, aim);
            } else {
                alpha_harmonic(dv, a1, ar, are, aim);
            }
            f2 y2 = pack2(0.f, 0.f);
#pragma unroll
            for (int i = 0; i < kP; ++i) {
                const f2 h_r = pack2(hr[2 * i], hr[2 * i + 1]), h_i = pack2(hi[2 * i], hi[2 * i + 1]);
                const f2 nh_i = pack2(-hi[2 * i], -hi[2 * i + 1]);
                const f2 nr = fma2(are[i], h_r, fma2(aim[i], nh_i, mul2(uu, pack2(b[2 * i], b[2 * i + 1]))));
                const f2 ni = fma2(are[i], h_i, mul2(aim[i], h_r));
                unpack2(nr, hr[2 * i], hr[2 * i + 1]);
                unpack2(ni, hi[2 * i], hi[2 * i + 1]);
                if constexpr (HAS_Y) y2 = fma2(pack2(cr[2 * i], cr[2 * i + 1]), nr, y2);
            }
            if constexpr (HAS_Y) {
                float y0, y1;
                unpack2(y2, y0, y1);
                const float y = y0 + y1;
                const int64_t yo = (static_cast<int64_t>(layer) * p.T_tot + start + k * kCT + t) * D + d;
                if (p.y_dtype == PRECOG_F32) static_cast<float *>(p.y)[yo] = y;
                else static_cast<__nv_bfloat16 *>(p.y)[yo] = __float2bfloat16_rn(y);
            }
        });
        if (!done) return;
    }
    if (p.states && live) {
        const int64_t off = ((chunk * p.L_out + p.layer0 + layer) * static_cast<int64_t>(D) + d) * kN;
#pragma unroll
        for (int n = 0; n < kN; ++n) {
            if (p.state_dtype == PRECOG_F32)
                reinterpret_cast<float2 *>(p.states)[off + n] = make_float2(hr[n], hi[n]);
            else
                reinterpret_cast<__nv_bfloat162 *>(p.states)[off + n] = __floats2bfloat162_rn(hr[n], hi[n]);
        }
    }
}

template <typename TIn, bool HAS_Y, bool HAS_H0>
cudaError_t launch_c(const ScanParams &p, cudaStream_t stream) {
    constexpr int CB = block_channels<HAS_Y>();
    const int cblocks = (p.D + CB - 1) / CB;
    const int64_t items = static_cast<int64_t>(p.n_layers) * p.n_chunks * cblocks;
    if (items == 0) return cudaSuccess;
    if (items > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const int smem = static_cast<int>(sizeof(CSmem<TIn, CB>));
    auto kern = scan_complex_kernel<TIn, HAS_Y, HAS_H0>;
    cudaError_t e = ensure_smem(reinterpret_cast<const void *>(kern), smem);
    if (e != cudaSuccess) return e;
    kern<<<static_cast<unsigned>(items), CB, smem, stream>>>(p, cblocks);
    e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

template <typename TIn>
cudaError_t launch_in(const ScanParams &p, cudaStream_t stream) {
    const bool y = p.y != nullptr, h0 = p.bank != nullptr;
    if (y) return h0 ? launch_c<TIn, true, true>(p, stream) : launch_c<TIn, true, false>(p, stream);
    return h0 ? launch_c<TIn, false, true>(p, stream) : launch_c<TIn, false, false>(p, stream);
}

}  // namespace

cudaError_t launch_scan_complex(const ScanParams &p, cudaStream_t stream) {
    if (p.in_dtype == PRECOG_F32) return launch_in<float>(p, stream);
    return launch_in<__nv_bfloat16>(p, stream);
}

cudaError_t scan_complex_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_scan_complex_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_scan_complex_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
