// Top-1 (and top-k) retrieval for a batch of queries on the 5th-generation tensor
// cores (Sec. 4.2 query-time retrieval, exact dot product, lowest row on ties).
//
// S = Q K^T is a dense contraction once several queries share a pass over the
// index, so it runs on tcgen05: queries are the A operand (up to two 128-row
// halves), key rows the B operand (tiles of 256 rows), dim the K dimension in
// blocks of 64 (128 bytes, 128B-swizzled). The kernel is bound by what shared
// memory can be filled with from L2 (about 10 TB/s over the chip), and the
// query operand is re-read for every key tile, so the key tile is as wide as
// one MMA allows (N = 256): 64 KB staged per 64-wide k-block for 2 x 128 x 256
// x 64 multiply-adds. fp32 accumulators live in tensor memory: one query half
// uses 256 columns and is double-buffered, so the argmax of one tile overlaps
// the MMAs of the next; two halves fill all 512 columns with one buffer. The
// score matrix never leaves the SM: thread q of the epilogue owns TMEM lane q
// (one query) and scans its columns (key rows) in increasing order with a
// strict '>', which keeps the lowest row on ties; NaN never compares greater.
//
// Warp roles (one persistent CTA per SM, 320 threads):
//   warp 0  TMA producer: A (queries) and B (key tile) k-blocks into a 3-stage ring
//   warp 1  TMEM owner and MMA issuer (one elected lane)
//   warps 2-5 / 6-9 epilogue of query half 0 / 1: TMEM -> registers -> running
//   (score, row) per query; with two halves the accumulators are single-buffered, so
//   splitting the halves over two groups halves the time the MMAs wait for them
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

__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, Smem &sm) {
    for (uint32_t i = 0; i < kWaitLimit; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 1023u) == 1023u && *reinterpret_cast<volatile uint32_t *>(&sm.abort_flag)) return false;
    }
    atomicOr(&g_retrieve_status_tc, PRECOG_DEV_TIMEOUT);
    *reinterpret_cast<volatile uint32_t *>(&sm.abort_flag) = 1u;
    return false;
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
            float best = -__int_as_float(0x7f800000);
            int64_t best_row = -1;
            unsigned long long lst[LIST > 1 ? LIST : 1];
#pragma unroll
            for (int j = 0; j < (LIST > 1 ? LIST : 1); ++j) lst[j] = 0ull;
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
                    const int64_t rbase = row0 + c0;
                    // Fast path: the column maximum of the 32 values (NaN ignored). Only
                    // when it beats the running best (rare after the first tiles) are the
                    // columns scanned again in increasing order with a strict '>', so the
                    // lowest row still wins ties.
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
                    if (m > best) {
                        // Slow path (rare per thread, but a warp takes it whenever one of
                        // its 32 queries does): mark the columns that beat the running
                        // best, park the scores in this thread's scratch row and visit
                        // only the marked ones, lowest column first. A compact loop keeps
                        // the epilogue's code small.
                        uint32_t mask = 0u;
#pragma unroll
                        for (int j = 0; j < 32; ++j) {
                            const bool in = (full_cols || rbase + j < M) && v[j] > best;
                            mask |= in ? (1u << j) : 0u;
                            sm.epi[ethr][j] = v[j];
                        }
                        while (mask) {
                            const int j = __ffs(static_cast<int>(mask)) - 1;
                            mask &= mask - 1u;
                            const float val = sm.epi[ethr][j];
                            if (!(val > best)) continue;
                            if constexpr (LIST == 1) {
                                best = val;
                                best_row = rbase + j;
                            } else {
                                // best tracks the list's last score
                                tc_list_insert<LIST>(lst, tc_key(val, rbase + j));
                                if (lst[LIST - 1] != 0ull)
                                    best = unordered_tc(static_cast<uint32_t>(lst[LIST - 1] >> 32));
                            }
                        }
                    }
                }
                tc_fence_before();
                mbar_arrive(&sm.acc_empty[acc]);
            }
            __syncwarp();
            const int q = h * kBM + qrow;
            if (LIST > 1 && q < nq) {
#pragma unroll
                for (int j = 0; j < kTopkStride; ++j)
                    partial[(static_cast<int64_t>(blockIdx.x) * n_queries + q0 + q) * kTopkStride + j] =
                        j < LIST ? lst[j < LIST ? j : 0] : 0ull;
            }
            if (LIST == 1 && q < nq) {
                unsigned long long key = 0ull;
                if (best_row >= 0)
                    key = (static_cast<unsigned long long>(ordered_bits_tc(best)) << 32) |
                          static_cast<unsigned long long>(0xffffffffu - static_cast<uint32_t>(best_row));
                partial[static_cast<int64_t>(blockIdx.x) * n_queries + q0 + q] = key;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    if (warp == 1) {
        tc_fence_after();
        tmem_dealloc(tmem, kTmemCols);
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
    for (int q0 = 0; q0 < p.n_queries; q0 += 2 * kBM) {
        const int nq = p.n_queries - q0 < 2 * kBM ? p.n_queries - q0 : 2 * kBM;
        retrieve_tc_kernel<LIST><<<grid, kThreads, smem, stream>>>(
            tq, tk, p.M, p.dim, p.n_queries, q0, nq, a_rows, bf16,
            static_cast<unsigned long long *>(p.workspace));
        e = cudaGetLastError();
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
