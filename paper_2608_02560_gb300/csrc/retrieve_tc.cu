// Top-1 (and top-k) retrieval for a batch of queries on the 5th-generation tensor
// cores (Sec. 4.2 query-time retrieval, exact dot product, lowest row on ties).
//
// S = Q K^T is a dense contraction once several queries share a pass over the
// index, so it runs on tcgen05: queries are the A operand, key rows the B operand
// (tiles of 256 rows), dim the K dimension in blocks of 64 (128 bytes,
// 128B-swizzled). The query operand is re-read for every key tile, so the key
// tile is as wide as one MMA allows (N = 256). fp32 accumulators live in tensor
// memory; the score matrix never leaves the SM: thread q of the epilogue owns
// TMEM lane q (one query) and scans its columns (key rows) in increasing order
// with a strict '>', which keeps the lowest row on ties; NaN never compares
// greater.
//
// Two kernels. retrieve_tc_kernel (one CTA per SM) takes a pass of up to 128
// queries, or 256 when the grid does not split into pairs: one query half uses
// 256 TMEM columns and is double-buffered, so the argmax of one tile overlaps the
// MMAs of the next; two halves fill all 512 columns with one buffer. Warp roles
// (320 threads):
//   warp 0  TMA producer: A (queries) and B (key tile) k-blocks into a 3-stage ring
//   warp 1  TMEM owner and MMA issuer (one elected lane)
//   warps 2-5 / 6-9 epilogue of query half 0 / 1: TMEM -> registers -> running
//   (score, row) per query
// retrieve_tc_pair_kernel (clusters of two CTAs, cta_group::2) takes a pass of
// more than 128 queries on SM pairs; its comment below gives the reasons.
// Every wait is bounded; on expiry the CTA flags PRECOG_DEV_TIMEOUT and leaves
// through the same teardown (TMEM freed, issued copies drained).
#include <cuda.h>
#include <cudaTypedefs.h>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_retrieve_status_tc;

constexpr int kBM = 128;          // queries per MMA (one half)
constexpr int kBN = 256;          // key rows per tile
constexpr int kBK = 64;           // dim per k-block (128 bytes of fp16/bf16)
constexpr int kStages = 3;
constexpr int kTopkStride = 8;    // keys per (CTA, query) in the top-k workspace
constexpr int kThreads = 320;     // 2 control warps + 8 epilogue warps
constexpr uint32_t kTmemCols = 512;
constexpr uint32_t kABytes = kBM * kBK * 2;   // one query half per stage
constexpr uint32_t kBBytes = kBN * kBK * 2;

struct Smem {
    // 1024-byte aligned operand tiles (128B swizzle atoms are 8 rows x 128 B)
    uint8_t a[kStages][2][kABytes];
    uint8_t b[kStages][kBBytes];
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint32_t tmem_base;
    uint32_t abort_flag;
    // epilogue scratch: one row of 32 scores per epilogue thread (padded: conflict-free)
    float epi[8 * 32][33];
};

// Shared-memory matrix descriptor: K-major operand, 128B swizzle, rows of 128
// bytes, 8-row groups 1024 bytes apart.
__device__ __forceinline__ uint64_t sw128_desc(const void *tile) {
    const uint32_t addr = smem_u32(tile);
    uint64_t d = 0;
    d |= static_cast<uint64_t>((addr & 0x3ffffu) >> 4);          // start address
    d |= static_cast<uint64_t>(1) << 16;                            // leading byte offset (unused)
    d |= static_cast<uint64_t>(1024 >> 4) << 32;                    // stride byte offset
    d |= static_cast<uint64_t>(1) << 46;                            // descriptor version
    d |= static_cast<uint64_t>(2) << 61;                            // swizzle: 128B
    return d;
}

// Instruction descriptor, kind::f16: fp32 accumulate, A and B of the same
// 16-bit type, both K-major, M = 128, N = 256.
__host__ __device__ constexpr uint32_t idesc_f16(bool bf16) {
    return (1u << 4)                                    // D: f32
           | ((bf16 ? 1u : 0u) << 7)                    // A type
           | ((bf16 ? 1u : 0u) << 10)                   // B type
           | (static_cast<uint32_t>(kBN >> 3) << 17)    // N / 8
           | (static_cast<uint32_t>(kBM >> 4) << 24);   // M / 16
}

__device__ __forceinline__ uint32_t ordered_bits_tc(float s) {
    const uint32_t u = __float_as_uint(s + 0.0f);
    return (u & 0x80000000u) ? ~u : (u | 0x80000000u);
}
__device__ __forceinline__ float unordered_tc(uint32_t k) {
    return __uint_as_float((k & 0x80000000u) ? (k & 0x7fffffffu) : ~k);
}

__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, uint32_t *abort_flag) {
    for (uint32_t i = 0; i < kWaitLimit; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 1023u) == 1023u && *reinterpret_cast<volatile uint32_t *>(abort_flag)) return false;
    }
    atomicOr(&g_retrieve_status_tc, PRECOG_DEV_TIMEOUT);
    *reinterpret_cast<volatile uint32_t *>(abort_flag) = 1u;
    return false;
}
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Smem &sm) {
    return wait_or_abort(bar, parity, &sm.abort_flag);
}

// Sorted insertion into a descending list of packed keys (the smallest drops out).
template <int K>
__device__ __forceinline__ void tc_list_insert(unsigned long long (&l)[K], unsigned long long v) {
#pragma unroll
    for (int j = K - 1; j > 0; --j) {
        const bool shift = v > l[j - 1];
        l[j] = shift ? l[j - 1] : (v > l[j] ? v : l[j]);
    }
    l[0] = v > l[0] ? v : l[0];
}

__device__ __forceinline__ unsigned long long tc_key(float s, int64_t row) {
    return (static_cast<unsigned long long>(ordered_bits_tc(s)) << 32) |
           static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(row));
}

// Running top-1 (LIST = 1) or top-LIST list of one query (one epilogue thread).
template <int LIST>
struct Best {
    float best;   // LIST > 1: the list's last score once it is full
    int64_t row;
    unsigned long long lst[LIST > 1 ? LIST : 1];
    __device__ Best() : best(-INFINITY), row(-1) {
#pragma unroll
        for (int j = 0; j < (LIST > 1 ? LIST : 1); ++j) lst[j] = 0ull;
    }
};

// Fold 32 consecutive scores (key rows rbase ..) into the running result. Fast path:
// the column maximum (NaN ignored). Only when it beats the running best (rare after the
// first tiles) are the columns scanned again in increasing order with a strict '>', so
// the lowest row still wins ties. The re-scan (rare per thread, but a warp takes it
// whenever one of its 32 queries does) marks the columns that beat the running best,
// parks the scores in this thread's scratch row and visits only the marked ones, lowest
// column first: a compact loop keeps the epilogue's code small.
template <int LIST>
__device__ __forceinline__ void fold_columns(const float (&v)[32], int64_t rbase, int64_t M, Best<LIST> &b,
                                             float *scratch) {
    const bool full_cols = rbase + 32 <= M;
    float m = -__int_as_float(0x7f800000);
    if (full_cols) {
#pragma unroll
        for (int j = 0; j < 32; ++j) m = fmaxf(m, v[j]);
    } else {
#pragma unroll
        for (int j = 0; j < 32; ++j)
            if (rbase + j < M) m = fmaxf(m, v[j]);
    }
    if (!(m > b.best)) return;
    uint32_t mask = 0u;
#pragma unroll
    for (int j = 0; j < 32; ++j) {
        const bool in = (full_cols || rbase + j < M) && v[j] > b.best;
        mask |= in ? (1u << j) : 0u;
        scratch[j] = v[j];
    }
    while (mask) {
        const int j = __ffs(static_cast<int>(mask)) - 1;
        mask &= mask - 1u;
        const float val = scratch[j];
        if (!(val > b.best)) continue;
        if constexpr (LIST == 1) {
            b.best = val;
            b.row = rbase + j;
        } else {
            tc_list_insert<LIST>(b.lst, tc_key(val, rbase + j));
            if (b.lst[LIST - 1] != 0ull) b.best = unordered_tc(static_cast<uint32_t>(b.lst[LIST - 1] >> 32));
        }
    }
}

// This CTA's result for query q (absolute index) into partial slot `part`: the packed
// best key (LIST = 1; zero for "no row") or the sorted list padded with zero keys.
template <int LIST>
__device__ __forceinline__ void write_partial(unsigned long long *partial, int64_t part, int n_queries, int q,
                                              const Best<LIST> &b) {
    if constexpr (LIST > 1) {
#pragma unroll
        for (int j = 0; j < kTopkStride; ++j)
            partial[(part * n_queries + q) * kTopkStride + j] = j < LIST ? b.lst[j < LIST ? j : 0] : 0ull;
    } else {
        partial[part * n_queries + q] = b.row >= 0 ? tc_key(b.best, b.row) : 0ull;
    }
}

// LIST = 1: partial[blockIdx.x * n_queries + q0 + q] = packed best key of this CTA.
// LIST > 1: partial[(blockIdx.x * n_queries + q0 + q) * kTopkStride + j] = its LIST best,
// sorted, then zero keys ("no row") up to kTopkStride. A shorter list (the smallest of
// 2, 4, 8 that holds k) raises the running threshold sooner and costs less per insertion.
template <int LIST>
__global__ void __launch_bounds__(kThreads, 1)
    retrieve_tc_kernel(const __grid_constant__ CUtensorMap tmap_q,
                       const __grid_constant__ CUtensorMap tmap_k, int64_t M, int dim,
                       int n_queries, int q0, int nq, int a_rows, bool bf16,
                       unsigned long long *__restrict__ partial) {
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    Smem &sm = *reinterpret_cast<Smem *>(
        (reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const int nhalf = nq > kBM ? 2 : 1;
    // accumulator columns: one query half x 256 keys = 256 columns, so a single half is
    // double-buffered (the argmax of a tile overlaps the next tile's MMAs) and two halves
    // fill all 512 columns with one buffer
    const int nbuf = nhalf == 1 ? 2 : 1;
    const int nkb = (dim + kBK - 1) / kBK;
    const int64_t ntiles = (M + kBN - 1) / kBN;

    if (threadIdx.x == 0) {
        for (int s = 0; s < kStages; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&sm.acc_full[a], 1);
            mbar_init(&sm.acc_empty[a], nhalf * 4 * 32);   // the epilogue threads of the halves in use
        }
        sm.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc(&sm.tmem_base, kTmemCols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ---------------- TMA producer ----------------
        if (lane == 0) {
            uint32_t g = 0;
            bool alive = true;
            for (int64_t tile = blockIdx.x; tile < ntiles && alive; tile += gridDim.x) {
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = g % kStages;
                    const uint32_t use = g / kStages;
                    if (!wait_or_abort(&sm.empty[s], (use & 1u) ^ 1u, sm)) {
                        alive = false;
                        break;
                    }
                    mbar_arrive_expect_tx(&sm.full[s], static_cast<uint32_t>(nhalf * a_rows * kBK * 2) + kBBytes);
                    for (int h = 0; h < nhalf; ++h)
                        tma_load_2d(sm.a[s][h], &tmap_q, kb * kBK, q0 + h * kBM, &sm.full[s]);
                    tma_load_2d(sm.b[s], &tmap_k, kb * kBK, static_cast<int32_t>(tile * kBN),
                                &sm.full[s]);
                }
            }
            // Drain: every issued stage must have landed before the CTA may exit.
            const uint32_t issued = g;
            for (uint32_t g2 = (issued > kStages ? issued - kStages : 0); g2 < issued; ++g2)
                mbar_wait(&sm.full[g2 % kStages], (g2 / kStages) & 1u);
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer ----------------
        if (lane == 0) {
            const uint32_t idesc = idesc_f16(bf16);
            uint32_t g = 0;
            int it = 0;
            bool alive = true;
            for (int64_t tile = blockIdx.x; tile < ntiles && alive; tile += gridDim.x, ++it) {
                const int acc = it % nbuf;
                const uint32_t ause = static_cast<uint32_t>(it / nbuf);
                if (!wait_or_abort(&sm.acc_empty[acc], (ause & 1u) ^ 1u, sm)) break;
                tc_fence_after();
                const uint32_t d0 = tmem + static_cast<uint32_t>(acc * kBN);
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = g % kStages;
                    if (!wait_or_abort(&sm.full[s], (g / kStages) & 1u, sm)) {
                        alive = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t bdesc = sw128_desc(sm.b[s]);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k) {
                        // advancing K by 16 elements = 32 bytes = 2 in the address field
                        for (int h = 0; h < nhalf; ++h)
                            tc_mma_f16(d0 + h * kBN, sw128_desc(sm.a[s][h]) + 2 * k, bdesc + 2 * k,
                                       idesc, kb > 0 || k > 0);
                    }
                    tc_commit(&sm.empty[s]);
                }
                if (alive) tc_commit(&sm.acc_full[acc]);
            }
        }
        __syncwarp();
    } else {
        // ---------------- epilogue: argmax over key rows, per query ----------------
        // Warps 2-5 read query half 0, warps 6-9 half 1: a warp may only read the TMEM
        // lanes of its quarter (warp % 4), and each group covers all four quarters.
        const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31
        const int h = (warp - 2) >> 2;                // query half of this warp
        const int qrow = quarter * 32 + lane;         // query row inside the half
        const int ethr = threadIdx.x - 64;            // scratch row of this epilogue thread
        if (h < nhalf) {
            Best<LIST> b;
            int it = 0;
            for (int64_t tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
                const int acc = it % nbuf;
                // one lane waits, the warp follows its result (tcgen05.ld needs the whole warp)
                bool ok = true;
                if (lane == 0) ok = wait_or_abort(&sm.acc_full[acc], static_cast<uint32_t>(it / nbuf) & 1u, sm);
                ok = __shfl_sync(0xffffffffu, ok, 0);
                if (!ok) break;
                tc_fence_after();
                const int64_t row0 = tile * kBN;
#pragma unroll 1
                for (int c0 = 0; c0 < kBN; c0 += 32) {
                    float v[32];
                    tmem_ld32(tmem + (static_cast<uint32_t>(quarter * 32) << 16) +
                                  static_cast<uint32_t>(acc * kBN + h * kBN + c0),
                              v);
                    fold_columns<LIST>(v, row0 + c0, M, b, sm.epi[ethr]);
                }
                tc_fence_before();
                mbar_arrive(&sm.acc_empty[acc]);
            }
            __syncwarp();
            const int q = h * kBM + qrow;
            if (q < nq) write_partial<LIST>(partial, blockIdx.x, n_queries, q0 + q, b);
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
    }
}

// ---------------------------------------------------------------------------------------
// SM pairs for a pass of more than 128 queries (cta_group::2).
//
// With two 128-query halves on one SM the two accumulators fill all 512 TMEM columns, so
// each tile's MMAs wait for the previous tile's epilogue. A cluster of two CTAs runs one
// M = 256 MMA instead: CTA r stages only its own 128 queries (rows r*128.. of A) and 128
// of the tile's 256 keys (rows r*128.. of B), 32 KB per k-block, and holds the 128 x 256
// scores of its own queries in its own tensor memory. 256 columns per tile leave room for
// two buffers, so the epilogue overlaps the next tile's MMAs again. (Shared-memory traffic
// per multiply-add is unchanged: each SM's B half is read by both tensor cores.)
//
// Roles (both CTAs unless noted): warp 0 TMA producer of this CTA's query and key rows,
// counted on the even CTA's full barrier; warp 1 TMEM allocation (collective over the
// pair) and, in the even CTA only, the MMA issuer; warps 2-5 epilogue over this CTA's
// 128 queries. Barriers: full[s] (even CTA: 64 KB per stage from both CTAs), empty[s]
// (each CTA: the MMAs' multicast commit), acc_full[b] (each CTA: multicast commit) and
// acc_empty[b] (even CTA: one arrival from each of the pair's 8 epilogue warps). Pair p
// takes key tiles p, p + P, ... (P pairs); its CTAs write partial slots 2p (the result)
// and 2p + 1 (no row) for their queries, so the finalize reads as many slots as after
// the single-CTA kernel on the same grid.
constexpr int kPairThreads = 6 * 32;
constexpr uint32_t kPairRows = kBN / 2;                              // key rows per CTA and tile
constexpr uint32_t kPairStageBytes = kABytes + kPairRows * kBK * 2;  // per CTA: 16 KB + 16 KB

template <int LIST>
struct PairSmem {
    static constexpr int kStages = 6;   // 192 KB in flight, as the single-CTA ring
    static constexpr int kScratchRows = 4 * 32;
    uint8_t a[kStages][kABytes];
    uint8_t b[kStages][kPairRows * kBK * 2];
    uint64_t full[kStages];
    uint64_t empty[kStages];
    uint64_t acc_full[2];
    uint64_t acc_empty[2];
    uint32_t tmem_base;
    uint32_t abort_flag;
    float epi[kScratchRows][33];
};

// kind::f16 instruction descriptor of the pair MMA: M = 256 (128 rows per CTA), N = 256.
__host__ __device__ constexpr uint32_t idesc_f16_pair(bool bf16) {
    return (1u << 4) | ((bf16 ? 1u : 0u) << 7) | ((bf16 ? 1u : 0u) << 10) |
           (static_cast<uint32_t>(kBN >> 3) << 17) | (static_cast<uint32_t>((2 * kBM) >> 4) << 24);
}

template <int LIST>
__global__ void __launch_bounds__(kPairThreads, 1)
    retrieve_tc_pair_kernel(const __grid_constant__ CUtensorMap tmap_q,
                            const __grid_constant__ CUtensorMap tmap_k, int64_t M, int dim, int n_queries,
                            int q0, int nq, bool bf16, unsigned long long *__restrict__ partial) {
    using Sm = PairSmem<LIST>;
    constexpr int S = Sm::kStages;
    extern __shared__ __align__(1024) uint8_t smem_raw[];
    Sm &sm = *reinterpret_cast<Sm *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~static_cast<uintptr_t>(1023));
    const int warp = threadIdx.x >> 5;
    const int lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();   // 0: the CTA that issues the MMAs
    const int64_t pair = blockIdx.x >> 1;
    const int64_t npairs = gridDim.x >> 1;
    const int nkb = (dim + kBK - 1) / kBK;
    const int64_t ntiles = (M + kBN - 1) / kBN;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(&sm.acc_full[a], 1);
            mbar_init(&sm.acc_empty[a], 8);
        }
        sm.abort_flag = 0;
        fence_barrier_init();
    }
    if (warp == 1) {
        tmem_alloc_pair(&sm.tmem_base, kTmemCols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    // the even CTA's barriers must be initialised before the peer's copies and arrivals reach them
    cluster_sync_all();
    tc_fence_after();
    const uint32_t tmem = sm.tmem_base;

    if (warp == 0) {
        // ---------------- TMA producer (both CTAs) ----------------
        if (lane == 0) {
            uint32_t g = 0;
            bool alive = true;
            for (int64_t tile = pair; tile < ntiles && alive; tile += npairs) {
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = static_cast<int>(g % S);
                    if (!wait_or_abort(&sm.empty[s], ((g / S) & 1u) ^ 1u, &sm.abort_flag)) {
                        alive = false;
                        break;
                    }
                    if (rank == 0) mbar_arrive_expect_tx(&sm.full[s], 2 * kPairStageBytes);
                    const uint32_t full0 = mapa_shared(&sm.full[s], 0);
                    tma_load_2d_pair(sm.a[s], &tmap_q, kb * kBK, q0 + static_cast<int>(rank) * kBM, full0);
                    tma_load_2d_pair(sm.b[s], &tmap_k, kb * kBK,
                                     static_cast<int32_t>(tile * kBN + rank * kPairRows), full0);
                }
            }
            // Before the CTA may exit: every issued stage landed (the even CTA's full
            // barriers count both CTAs' bytes) and the MMAs released it (their commits
            // reach both CTAs' empty barriers, so none is still on its way here).
            const uint32_t lo = g > static_cast<uint32_t>(S) ? g - S : 0u;
            if (rank == 0)
                for (uint32_t g2 = lo; g2 < g; ++g2) mbar_wait(&sm.full[g2 % S], (g2 / S) & 1u);
            if (alive)
                for (uint32_t g2 = lo; g2 < g; ++g2)
                    if (!wait_or_abort(&sm.empty[g2 % S], (g2 / S) & 1u, &sm.abort_flag)) break;
        }
    } else if (warp == 1) {
        // ---------------- MMA issuer (even CTA) ----------------
        if (rank == 0 && lane == 0) {
            const uint32_t idesc = idesc_f16_pair(bf16);
            uint32_t g = 0;
            int it = 0;
            bool alive = true;
            for (int64_t tile = pair; tile < ntiles && alive; tile += npairs, ++it) {
                const int acc = it & 1;
                if (!wait_or_abort(&sm.acc_empty[acc], (static_cast<uint32_t>(it >> 1) & 1u) ^ 1u, &sm.abort_flag))
                    break;
                tc_fence_after();
                const uint32_t d0 = tmem + static_cast<uint32_t>(acc * kBN);
                for (int kb = 0; kb < nkb; ++kb, ++g) {
                    const int s = static_cast<int>(g % S);
                    if (!wait_or_abort(&sm.full[s], (g / S) & 1u, &sm.abort_flag)) {
                        alive = false;
                        break;
                    }
                    tc_fence_after();
                    const uint64_t adesc = sw128_desc(sm.a[s]);
                    const uint64_t bdesc = sw128_desc(sm.b[s]);
#pragma unroll
                    for (int k = 0; k < kBK / 16; ++k)
                        tc_mma_f16_pair(d0, adesc + 2 * k, bdesc + 2 * k, idesc, kb > 0 || k > 0);
                    tc_commit_pair_mc(&sm.empty[s], static_cast<uint16_t>(0x3));
                }
                if (alive) tc_commit_pair_mc(&sm.acc_full[acc], static_cast<uint16_t>(0x3));
            }
        }
        __syncwarp();
    } else {
        // ---------------- epilogue: this CTA's 128 queries over the tile's 256 keys ----------------
        const int quarter = warp & 3;                 // TMEM lanes 32*quarter .. +31 (warps 2-5)
        const int qrow = quarter * 32 + lane;         // query row inside this CTA's half
        const int ethr = threadIdx.x - 64;
        const uint32_t acc_empty_even0 = mapa_shared(&sm.acc_empty[0], 0);
        const uint32_t acc_empty_even1 = mapa_shared(&sm.acc_empty[1], 0);
        Best<LIST> b;
        int it = 0;
        for (int64_t tile = pair; tile < ntiles; tile += npairs, ++it) {
            const int acc = it & 1;
            bool ok = true;
            if (lane == 0)
                ok = wait_or_abort(&sm.acc_full[acc], static_cast<uint32_t>(it >> 1) & 1u, &sm.abort_flag);
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) break;
            tc_fence_after();
            // column c of the accumulator is key row tile * 256 + c (the even CTA's 128 rows first)
            const int64_t row0 = tile * kBN;
#pragma unroll 1
            for (int c0 = 0; c0 < kBN; c0 += 32) {
                float v[32];
                tmem_ld32(tmem + (static_cast<uint32_t>(quarter * 32) << 16) + static_cast<uint32_t>(acc * kBN + c0),
                          v);
                fold_columns<LIST>(v, row0 + c0, M, b, sm.epi[ethr]);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(acc ? acc_empty_even1 : acc_empty_even0);
        }
        const int q = static_cast<int>(rank) * kBM + qrow;
        if (q < nq) {
            write_partial<LIST>(partial, 2 * pair, n_queries, q0 + q, b);
            write_partial<LIST>(partial, 2 * pair + 1, n_queries, q0 + q, Best<LIST>());
        }
    }

    tc_fence_before();
    __syncthreads();
    // neither CTA leaves (or frees tensor memory) while the other may still reach into it
    cluster_sync_all();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc_pair(tmem, kTmemCols);
    }
}

bool make_map(CUtensorMap *map, const void *base, int64_t rows, int dim, bool bf16, int box_rows) {
    const cuuint64_t gdim[2] = {static_cast<cuuint64_t>(dim), static_cast<cuuint64_t>(rows)};
    const cuuint64_t gstride[1] = {static_cast<cuuint64_t>(dim) * 2};
    const cuuint32_t box[2] = {static_cast<cuuint32_t>(kBK), static_cast<cuuint32_t>(box_rows)};
    return encode_tiled_map(map, bf16 ? CU_TENSOR_MAP_DATA_TYPE_BFLOAT16 : CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2,
                            base, gdim, gstride, box, CU_TENSOR_MAP_SWIZZLE_128B);
}

}  // namespace

using EncodeTiled = PFN_cuTensorMapEncodeTiled_v12000;

bool encode_tiled_map(CUtensorMap *map, CUtensorMapDataType dtype, cuuint32_t rank, const void *base,
                      const cuuint64_t *dims, const cuuint64_t *strides_bytes, const cuuint32_t *box,
                      CUtensorMapSwizzle swizzle) {
    static EncodeTiled fn = [] {
        void *p = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            return reinterpret_cast<EncodeTiled>(p);
        return static_cast<EncodeTiled>(nullptr);
    }();
    if (fn == nullptr) return false;
    const cuuint32_t estride[5] = {1, 1, 1, 1, 1};
    const CUresult r = fn(map, dtype, rank, const_cast<void *>(base), dims, strides_bytes, box, estride,
                          CU_TENSOR_MAP_INTERLEAVE_NONE, swizzle, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                          CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

static_assert(sizeof(Smem) + 1024 <= 227 * 1024, "the ring and scratch must fit one CTA's shared memory");
static_assert(sizeof(PairSmem<1>) + 1024 <= 227 * 1024, "the pair ring must fit one CTA's shared memory");
static_assert(sizeof(PairSmem<8>) + 1024 <= 227 * 1024, "the pair ring and scratch must fit one CTA's shared memory");

size_t retrieve_tc_smem_bytes() { return sizeof(Smem) + 1024; }

int retrieve_tc_grid(int64_t M, int sms) {
    const int64_t ntiles = (M + kBN - 1) / kBN;
    return static_cast<int>(ntiles < 1 ? 1 : (ntiles < sms ? ntiles : sms));
}

// One pass per 256 queries; partial holds LIST packed keys per (CTA, query).
template <int LIST>
cudaError_t launch_tc(const RetrieveParams &p, int grid, cudaStream_t stream, uint64_t *launches) {
    const bool bf16 = p.dtype == PRECOG_BF16;
    CUtensorMap tq, tk;
    // A batch of fewer than 128 queries loads only its rows (rounded up to the 8-row
    // swizzle atom); the rest of the A tile is never read back (its TMEM lanes belong to
    // no query), and copies that are mostly out of bounds are slow.
    const int a_rows = p.n_queries >= kBM ? kBM : ((p.n_queries + 7) & ~7);
    if (!make_map(&tq, p.queries, p.n_queries, p.dim, bf16, a_rows) ||
        !make_map(&tk, p.index, p.M > 0 ? p.M : 1, p.dim, bf16, kBN))
        return cudaErrorInvalidValue;
    const int smem = static_cast<int>(retrieve_tc_smem_bytes());
    cudaError_t e = ensure_smem(reinterpret_cast<const void *>(retrieve_tc_kernel<LIST>), smem);
    if (e != cudaSuccess) return e;
    // Passes of more than 128 queries run on SM pairs when the grid splits into pairs.
    const bool pairs = grid % 2 == 0 && p.n_queries > kBM;
    CUtensorMap tk_pair;
    const int smem_pair = static_cast<int>(sizeof(PairSmem<LIST>) + 1024);
    if (pairs) {
        if (!make_map(&tk_pair, p.index, p.M, p.dim, bf16, static_cast<int>(kPairRows))) return cudaErrorInvalidValue;
        e = ensure_smem(reinterpret_cast<const void *>(retrieve_tc_pair_kernel<LIST>), smem_pair);
        if (e != cudaSuccess) return e;
    }
    unsigned long long *partial = static_cast<unsigned long long *>(p.workspace);
    for (int q0 = 0; q0 < p.n_queries; q0 += 2 * kBM) {
        const int nq = p.n_queries - q0 < 2 * kBM ? p.n_queries - q0 : 2 * kBM;
        if (pairs && nq > kBM) {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3(static_cast<unsigned>(grid));
            cfg.blockDim = dim3(kPairThreads);
            cfg.dynamicSmemBytes = static_cast<size_t>(smem_pair);
            cfg.stream = stream;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeClusterDimension;
            attr[0].val.clusterDim.x = 2;
            attr[0].val.clusterDim.y = 1;
            attr[0].val.clusterDim.z = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            e = cudaLaunchKernelEx(&cfg, retrieve_tc_pair_kernel<LIST>, tq, tk_pair, p.M, p.dim, p.n_queries, q0,
                                   nq, bf16, partial);
        } else {
            retrieve_tc_kernel<LIST><<<grid, kThreads, smem, stream>>>(tq, tk, p.M, p.dim, p.n_queries, q0, nq,
                                                                       a_rows, bf16, partial);
            e = cudaGetLastError();
        }
        if (e != cudaSuccess) return e;
        ++*launches;
    }
    return cudaSuccess;
}

cudaError_t launch_retrieve_tc(const RetrieveParams &p, int grid, cudaStream_t stream,
                               uint64_t *launches) {
    return launch_tc<1>(p, grid, stream, launches);
}

cudaError_t launch_retrieve_tc_topk(const RetrieveParams &p, int k, int grid, cudaStream_t stream,
                                    uint64_t *launches) {
    if (k <= 2) return launch_tc<2>(p, grid, stream, launches);
    if (k <= 4) return launch_tc<4>(p, grid, stream, launches);
    return launch_tc<8>(p, grid, stream, launches);
}

cudaError_t retrieve_tc_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_retrieve_status_tc, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_retrieve_status_tc, &zero, sizeof(uint32_t));
}

}  // namespace precog
