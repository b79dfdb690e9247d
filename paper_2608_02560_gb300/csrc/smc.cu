// Structured Memory Consolidation primitives (Sec. 5): two-level cluster
// routing (Eqs. smc-domain, smc-sub) and the semantic-state EMA (Eq. smc-ema).
// Session initialisation (Sec. 5.3) injects a semantic state with the
// ordinary prefill, so it needs no kernel of its own.
#include <climits>
#include <cstdint>
#include <type_traits>

#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_smc_status;

constexpr int kRouteWarps = 8;

constexpr int kRouteP = 8;   // prototypes scored per pass

// acc[p] = <e, protos[p]> for p < count (<= kRouteP prototypes, `stride` elements
// apart). Each lane sums a fixed subset of the coordinates in a fixed order -- 16-byte
// vectors v = lane, lane + 32, ... when VEC, single elements otherwise -- and a fixed
// xor butterfly adds the lanes, so the same two vectors always give the same score
// and every lane holds it. The count prototypes' loads of a vector are in flight
// together.
template <typename T, bool VEC>
__device__ __forceinline__ void dots_warp(const T *__restrict__ e, const T *__restrict__ protos, int64_t stride,
                                          int count, int dim, int lane, float (&acc)[kRouteP]) {
#pragma unroll
    for (int q = 0; q < kRouteP; ++q) acc[q] = 0.f;
    if constexpr (VEC) {
        constexpr int EL = 16 / static_cast<int>(sizeof(T));
        const int nvec = dim / EL;
        for (int v = lane; v < nvec; v += 32) {
            const uint4 ev = *reinterpret_cast<const uint4 *>(e + static_cast<int64_t>(v) * EL);
            uint4 pv[kRouteP];
#pragma unroll
            for (int q = 0; q < kRouteP; ++q)
                if (q < count) pv[q] = *reinterpret_cast<const uint4 *>(protos + q * stride + static_cast<int64_t>(v) * EL);
            const T *ee = reinterpret_cast<const T *>(&ev);
#pragma unroll
            for (int q = 0; q < kRouteP; ++q) {
                if (q >= count) break;
                const T *pp = reinterpret_cast<const T *>(&pv[q]);
#pragma unroll
                for (int k = 0; k < EL; ++k) acc[q] = fmaf(to_f32(ee[k]), to_f32(pp[k]), acc[q]);
            }
        }
    } else {
        for (int k = lane; k < dim; k += 32) {
            const float ek = to_f32(e[k]);
#pragma unroll
            for (int q = 0; q < kRouteP; ++q)
                if (q < count) acc[q] = fmaf(ek, to_f32(protos[q * stride + k]), acc[q]);
        }
    }
#pragma unroll
    for (int q = 0; q < kRouteP; ++q)
#pragma unroll
        for (int o = 16; o > 0; o >>= 1) acc[q] += __shfl_xor_sync(0xffffffffu, acc[q], o);
}

// One warp per embedding: the best domain prototype, then the best of that
// domain's J[m] sub-cluster prototypes (strict '>' in index order: lowest index on
// ties, NaN never wins). slot = m * J_max + j, or -1 when no comparable score exists.
// VEC: rows are whole 16-byte vectors on 16-byte boundaries.
template <typename T, bool VEC>
__global__ void __launch_bounds__(kRouteWarps * 32, 3)
    smc_route_kernel(const T *__restrict__ emb, int64_t n, int dim, const T *__restrict__ dom, int M,
                     const T *__restrict__ sub, int J_max, const int32_t *__restrict__ J,
                     int32_t *__restrict__ out_m, int32_t *__restrict__ out_j,
                     int64_t *__restrict__ out_slot) {
    const int lane = threadIdx.x & 31;
    const int64_t c = static_cast<int64_t>(blockIdx.x) * kRouteWarps + (threadIdx.x >> 5);
    if (c >= n) return;
    const T *e = emb + c * dim;
    float acc[kRouteP];
    float best = -__int_as_float(0x7f800000);
    int m = -1;
    for (int i0 = 0; i0 < M; i0 += kRouteP) {
        const int cnt = M - i0 < kRouteP ? M - i0 : kRouteP;
        dots_warp<T, VEC>(e, dom + static_cast<int64_t>(i0) * dim, dim, cnt, dim, lane, acc);
#pragma unroll
        for (int q = 0; q < kRouteP; ++q)
            if (q < cnt && acc[q] > best) {
                best = acc[q];
                m = i0 + q;
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
        const T *sm_ = sub + static_cast<int64_t>(m) * J_max * dim;
        for (int i0 = 0; i0 < Jm; i0 += kRouteP) {
            const int cnt = Jm - i0 < kRouteP ? Jm - i0 : kRouteP;
            dots_warp<T, VEC>(e, sm_ + static_cast<int64_t>(i0) * dim, dim, cnt, dim, lane, acc);
#pragma unroll
            for (int q = 0; q < kRouteP; ++q)
                if (q < cnt && acc[q] > best) {
                    best = acc[q];
                    j = i0 + q;
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
// one thread per VEC adjacent state elements. Deposits go in batches of kU:
// warp 0 reads a batch's slots and describes it for the whole block (per
// deposit: the slot's offset, the latest earlier deposit of the same slot in
// the batch, whether a later one follows), one batch ahead, with a match-any
// vote instead of pairwise compares. Every thread then issues the batch's
// state loads and first-touch slot loads together, folds the batch in deposit
// order (a repeat inside the batch starts from its predecessor's result, kept
// in a per-thread shared-memory column) and stores each touched slot once.
// Slot -1 deposits nothing; a slot >= n_slots is flagged and skipped.
constexpr int kU = 16;
constexpr int kConsThreads = 128;

struct BatchMeta {
    int64_t off[kU];      // slot * elems (valid deposits)
    int prev[kU];         // latest earlier position of the same slot, or -1
    uint32_t valid;       // bit j: deposit j has a slot
    uint32_t last;        // bit j: no later deposit of the batch has the same slot
    uint32_t dups;        // some deposit repeats an earlier slot of the batch
};

// Lane j < kU of warp 0 reads deposit c0 + j's slot (-1 past the end); the reads
// run two batches ahead of their use so that their latency is hidden.
__device__ __forceinline__ int64_t read_slot(const int64_t *__restrict__ slots, int64_t c0, int64_t n, int lane) {
    const int64_t c = c0 + lane;
    return lane < kU && c < n ? slots[c] : -1;
}

__device__ __forceinline__ void describe_batch(BatchMeta &m, int64_t raw, int64_t n_slots, int64_t elems,
                                               int lane) {
    int64_t sl = INT64_MIN;                       // lanes beyond the batch never match
    if (lane < kU) {
        sl = raw;
        if (sl >= n_slots || sl < -1) {
            atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
            sl = -1;
        }
    }
    const bool valid = lane < kU && sl >= 0;
    const uint32_t same = __match_any_sync(0xffffffffu, sl);
    const uint32_t below = same & ((1u << lane) - 1u);
    const uint32_t above = lane == 31 ? 0u : (same & ~((2u << lane) - 1u));
    const int prev = valid && below ? 31 - __clz(below) : -1;
    const uint32_t vmask = __ballot_sync(0xffffffffu, valid);
    const uint32_t lmask = __ballot_sync(0xffffffffu, valid && above == 0u);
    const uint32_t dmask = __ballot_sync(0xffffffffu, prev >= 0);
    if (lane < kU) {
        m.off[lane] = valid ? sl * elems : 0;
        m.prev[lane] = prev;
    }
    if (lane == 0) {
        m.valid = vmask;
        m.last = lmask;
        m.dups = dmask != 0u;
    }
}

template <typename TS, int VEC>
__device__ __forceinline__ void load_state_vec(const TS *p, float (&h)[VEC]) {
    if constexpr (VEC == 1) {
        h[0] = to_f32(p[0]);
    } else if constexpr (std::is_same<TS, float>::value) {
        const float2 v = *reinterpret_cast<const float2 *>(p);
        h[0] = v.x;
        h[1] = v.y;
    } else {
        const uint32_t w = *reinterpret_cast<const uint32_t *>(p);
        h[0] = __uint_as_float(w << 16);
        h[1] = __uint_as_float(w & 0xffff0000u);
    }
}

template <int VEC>
__device__ __forceinline__ void load_sem(const float *p, float (&v)[VEC]) {
    if constexpr (VEC == 1) {
        v[0] = p[0];
    } else {
        const float2 q = *reinterpret_cast<const float2 *>(p);
        v[0] = q.x;
        v[1] = q.y;
    }
}

template <int VEC>
__device__ __forceinline__ void store_sem(float *p, const float (&v)[VEC]) {
    if constexpr (VEC == 1) p[0] = v[0];
    else *reinterpret_cast<float2 *>(p) = make_float2(v[0], v[1]);
}

template <typename TS, int VEC>
__global__ void __launch_bounds__(kConsThreads)
    smc_consolidate_kernel(float *__restrict__ sem, int64_t n_slots, int64_t elems,
                           const TS *__restrict__ states, const int64_t *__restrict__ slots,
                           int64_t n, float alpha) {
    __shared__ BatchMeta s_meta[2];
    __shared__ float s_val[kU][VEC][kConsThreads];
    const float keep = 1.f - alpha;
    const int tid = threadIdx.x, lane = tid & 31;
    const int64_t e = (static_cast<int64_t>(blockIdx.x) * kConsThreads + tid) * VEC;
    const bool mine = e < elems;
    const int64_t nbatch = (n + kU - 1) / kU;
    // The deposits' states do not depend on the semantic table, so each batch's state
    // loads are issued one batch ahead (every deposit that exists, slot or not).
    auto load_states = [&](int64_t c0, float (&h)[kU][VEC]) {
#pragma unroll
        for (int j = 0; j < kU; ++j) {
#pragma unroll
            for (int i = 0; i < VEC; ++i) h[j][i] = 0.f;
            if (mine && c0 + j < n) load_state_vec<TS, VEC>(states + (c0 + j) * elems + e, h[j]);
        }
    };
    float h[kU][VEC];
    load_states(0, h);
    int64_t raw_next = 0;
    if (tid < 32) {
        const int64_t raw0 = read_slot(slots, 0, n, lane);
        raw_next = read_slot(slots, kU, n, lane);
        describe_batch(s_meta[0], raw0, n_slots, elems, lane);
    }
    __syncthreads();
    for (int64_t b = 0; b < nbatch; ++b) {
        const BatchMeta &m = s_meta[b & 1];
        const int64_t c0 = b * kU;
        float v[kU][VEC];
        if (mine) {
            // first touch of each slot in this batch: after the previous batch's stores
            // (same thread, program order)
#pragma unroll
            for (int j = 0; j < kU; ++j) {
#pragma unroll
                for (int i = 0; i < VEC; ++i) v[j][i] = 0.f;
                if ((m.valid >> j & 1u) && m.prev[j] < 0) load_sem<VEC>(sem + m.off[j] + e, v[j]);
            }
        }
        float hn[kU][VEC];
        load_states(c0 + kU, hn);
        // the next batch's description overlaps this batch's loads
        if (tid < 32 && b + 1 < nbatch) {
            const int64_t raw = raw_next;
            raw_next = read_slot(slots, c0 + 2 * kU, n, lane);
            describe_batch(s_meta[(b + 1) & 1], raw, n_slots, elems, lane);
        }
        if (mine) {
            if (!m.dups) {
#pragma unroll
                for (int j = 0; j < kU; ++j)
#pragma unroll
                    for (int i = 0; i < VEC; ++i) v[j][i] = fmaf(keep, v[j][i], alpha * h[j][i]);
            } else {
#pragma unroll
                for (int j = 0; j < kU; ++j) {
                    if (!(m.valid >> j & 1u)) continue;
                    const int pj = m.prev[j];
#pragma unroll
                    for (int i = 0; i < VEC; ++i) {
                        const float base = pj >= 0 ? s_val[pj][i][tid] : v[j][i];
                        v[j][i] = fmaf(keep, base, alpha * h[j][i]);
                        s_val[j][i][tid] = v[j][i];
                    }
                }
            }
#pragma unroll
            for (int j = 0; j < kU; ++j)
                if (m.last >> j & 1u) store_sem<VEC>(sem + m.off[j] + e, v[j]);
        }
#pragma unroll
        for (int j = 0; j < kU; ++j)
#pragma unroll
            for (int i = 0; i < VEC; ++i) h[j][i] = hn[j][i];
        __syncthreads();   // the next batch's description is complete; this one may be rewritten
    }
}

// The same fold with one CTA per (slot, range of elements), for tables of few
// slots: the CTA gathers its slot's deposits in deposit order (ballots over the
// slot ids, kGather at a time), then streams their states with several deposits'
// loads in flight, keeping its elements' semantic values in registers from the
// first deposit to the last: each state element is read once and each semantic
// element read and written once.
constexpr int kSlotThreads = 256;
constexpr int kSlotItems = 4;                    // element groups of VEC per thread
constexpr int kGather = 4 * kSlotThreads;        // slot ids examined per gathering pass
constexpr int kFoldAhead = 4;                    // deposits whose loads are in flight together

template <typename TS, int VEC>
__global__ void __launch_bounds__(kSlotThreads)
    smc_consolidate_slot_kernel(float *__restrict__ sem, int64_t n_slots, int64_t elems,
                                const TS *__restrict__ states, const int64_t *__restrict__ slots,
                                int64_t n, float alpha) {
    __shared__ int32_t s_list[kGather];
    __shared__ int s_warp[kSlotThreads / 32];
    __shared__ int s_total;
    const int64_t slot = blockIdx.y;
    const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
    const float keep = 1.f - alpha;
    const bool flagger = blockIdx.x == 0 && blockIdx.y == 0;
    int64_t e[kSlotItems];
    float v[kSlotItems][VEC];
#pragma unroll
    for (int i = 0; i < kSlotItems; ++i) {
        e[i] = ((static_cast<int64_t>(blockIdx.x) * kSlotItems + i) * kSlotThreads + tid) * VEC;
        if (e[i] < elems) load_sem<VEC>(sem + slot * elems + e[i], v[i]);
    }
    for (int64_t c0 = 0; c0 < n; c0 += kGather) {
        int64_t sl[4];
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const int64_t c = c0 + r * kSlotThreads + tid;
            sl[r] = c < n ? slots[c] : -1;
            if (flagger && (sl[r] >= n_slots || sl[r] < -1)) atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
        }
        if (tid == 0) s_total = 0;
        __syncthreads();
#pragma unroll
        for (int r = 0; r < 4; ++r) {
            const bool hit = sl[r] == slot;
            const uint32_t ball = __ballot_sync(0xffffffffu, hit);
            if (lane == 0) s_warp[warp] = __popc(ball);
            __syncthreads();
            int base = s_total;
            for (int w = 0; w < warp; ++w) base += s_warp[w];
            if (hit) s_list[base + __popc(ball & ((1u << lane) - 1u))] = static_cast<int32_t>(r * kSlotThreads + tid);
            __syncthreads();
            if (tid == 0)
                for (int w = 0; w < kSlotThreads / 32; ++w) s_total += s_warp[w];
            __syncthreads();
        }
        const int m = s_total;
        for (int j0 = 0; j0 < m; j0 += kFoldAhead) {
            float h[kFoldAhead][kSlotItems][VEC];
#pragma unroll
            for (int q = 0; q < kFoldAhead; ++q) {
                const int j = j0 + q;
                const int64_t c = j < m ? c0 + s_list[j] : 0;
#pragma unroll
                for (int i = 0; i < kSlotItems; ++i) {
#pragma unroll
                    for (int k = 0; k < VEC; ++k) h[q][i][k] = 0.f;
                    if (j < m && e[i] < elems) load_state_vec<TS, VEC>(states + c * elems + e[i], h[q][i]);
                }
            }
#pragma unroll
            for (int q = 0; q < kFoldAhead; ++q) {
                if (j0 + q >= m) break;
#pragma unroll
                for (int i = 0; i < kSlotItems; ++i)
#pragma unroll
                    for (int k = 0; k < VEC; ++k) v[i][k] = fmaf(keep, v[i][k], alpha * h[q][i][k]);
            }
        }
        __syncthreads();   // s_list is rebuilt by the next pass
    }
#pragma unroll
    for (int i = 0; i < kSlotItems; ++i)
        if (e[i] < elems) store_sem<VEC>(sem + slot * elems + e[i], v[i]);
}

// The per-slot fold with the states streamed through shared memory by the TMA
// engine. A persistent CTA takes a contiguous run of (slot, element range)
// tiles. Its producer warp streams the slot ids through a ring of kIdRing
// chunks of kIdChunk ids (bulk copies kIdRing chunks ahead, so that finding
// the deposits does not wait on one round trip per chunk), matches them in
// deposit order and, for each deposit of the tile's slot, queues one bulk copy
// of that deposit's range of elements into a ring of kRing stages; the
// kBulkConsumers consumer threads fold every stage into the range's semantic
// values, which stay in registers for the whole tile. A stage tagged
// kTagTileEnd carries no data and closes the tile: its values are stored and
// the next tile's loaded while the ring keeps streaming. Each state element
// crosses HBM once, each semantic element is read and written once.
constexpr int kBulkConsumers = 256;
constexpr int kBulkThreads = kBulkConsumers + 32;
constexpr int kStageBytes = 16384;
constexpr int kRing = 6;
constexpr int kChunksPerThread = kStageBytes / 16 / kBulkConsumers;
constexpr int kIdChunk = 256;
constexpr int kIdRing = 6;
constexpr int32_t kTagData = 1;
constexpr int32_t kTagTileEnd = 2;
static_assert(kChunksPerThread * 16 * kBulkConsumers == kStageBytes, "stage = whole 16-byte chunks");
static_assert(kIdChunk % 32 == 0, "whole warps of ids");

struct BulkSmem {
    unsigned char ring[kRing][kStageBytes];
    int64_t ids[kIdRing][kIdChunk];
    uint64_t full[kRing];
    uint64_t empty[kRing];
    uint64_t idfull[kIdRing];
    int32_t tag[kRing];
    int32_t abort;
};

// Bounded wait that also gives up once another role of the CTA has given up.
__device__ __forceinline__ bool wait_or_abort(uint64_t *bar, uint32_t parity, const volatile int32_t *abort) {
    for (uint32_t i = 0; i < kWaitLimit; ++i) {
        if (mbar_try_wait(bar, parity)) return true;
        if ((i & 255u) == 255u && *abort) return false;
    }
    return false;
}

// Producer: claim stage g (wait until the consumers released its previous
// use), tag it and start its copy (src == nullptr: a tile-end marker).
// Warp-uniform result; false when the wait ran out or the CTA gave up.
__device__ __forceinline__ bool produce_stage(BulkSmem &sm, uint32_t g, int lane, const void *src,
                                              uint32_t bytes) {
    const int s = static_cast<int>(g % kRing);
    int ok = 1;
    if (lane == 0) {
        ok = wait_or_abort(&sm.empty[s], ((g / kRing) & 1u) ^ 1u, &sm.abort);
        if (ok) {
            sm.tag[s] = src ? kTagData : kTagTileEnd;
            if (src) {
                mbar_arrive_expect_tx(&sm.full[s], bytes);
                bulk_g2s(sm.ring[s], src, bytes, &sm.full[s]);
            } else {
                mbar_arrive(&sm.full[s]);
            }
        }
    }
    return __shfl_sync(0xffffffffu, ok, 0) != 0;
}

// Producer lane 0: start id chunk k of the scan (ids [k * kIdChunk, ...)), the u-th
// chunk of the CTA, into id stage u % kIdRing. An odd count leaves its last id to a
// plain load (bulk sizes are multiples of 16).
__device__ __forceinline__ void issue_ids(BulkSmem &sm, const int64_t *__restrict__ slots, int64_t n, int64_t k,
                                          int64_t u) {
    const int s = static_cast<int>(u % kIdRing);
    const int64_t c0 = k * kIdChunk;
    const int64_t cnt = n - c0 < kIdChunk ? n - c0 : kIdChunk;
    const uint32_t bytes = static_cast<uint32_t>((cnt & ~static_cast<int64_t>(1)) * 8);
    if (bytes == 0) {
        mbar_arrive(&sm.idfull[s]);
    } else {
        mbar_arrive_expect_tx(&sm.idfull[s], bytes);
        bulk_g2s(sm.ids[s], slots + c0, bytes, &sm.idfull[s]);
    }
}

template <typename TS>
__global__ void __launch_bounds__(kBulkThreads, 2)
    smc_consolidate_bulk_kernel(float *__restrict__ sem, int64_t n_slots, int64_t elems,
                                const TS *__restrict__ states, const int64_t *__restrict__ slots,
                                int64_t n, float alpha, int64_t ntiles, int64_t per_cta) {
    constexpr int CH = 16 / static_cast<int>(sizeof(TS));          // state elements per 16-byte chunk
    constexpr int64_t R = kStageBytes / static_cast<int64_t>(sizeof(TS));  // elements per tile
    extern __shared__ __align__(16) unsigned char smem_raw[];
    BulkSmem &sm = *reinterpret_cast<BulkSmem *>(smem_raw);
    const int tid = threadIdx.x, warp = tid >> 5, lane = tid & 31;
    const int64_t nranges = (elems + R - 1) / R;
    const int64_t t_begin = static_cast<int64_t>(blockIdx.x) * per_cta;
    const int64_t t_end = t_begin + per_cta < ntiles ? t_begin + per_cta : ntiles;
    if (tid == 0) {
        for (int s = 0; s < kRing; ++s) {
            mbar_init(&sm.full[s], 1);
            mbar_init(&sm.empty[s], kBulkConsumers / 32);
        }
        for (int s = 0; s < kIdRing; ++s) mbar_init(&sm.idfull[s], 1);
        sm.abort = 0;
        fence_barrier_init();
    }
    __syncthreads();

    if (warp == kBulkConsumers / 32) {
        // ---- producer warp ----
        uint32_t g = 0;        // ring stages produced
        int64_t kid = 0;       // id chunks consumed (all tiles)
        int64_t kid_issued = 0;
        bool ok = true;
        const int64_t nchunks = (n + kIdChunk - 1) / kIdChunk;
        for (int64_t t = t_begin; t < t_end && ok; ++t) {
            const int64_t slot = t / nranges;
            const int64_t e0 = (t % nranges) * R;
            const int64_t rlen = elems - e0 < R ? elems - e0 : R;
            const uint32_t bytes = static_cast<uint32_t>(rlen * static_cast<int64_t>(sizeof(TS)));
            const TS *src = states + e0;
            const bool flagger = t == 0;
            const int64_t base = kid;
            const int64_t first = nchunks < kIdRing ? nchunks : kIdRing;
            if (lane == 0) {
                fence_proxy_async_smem();   // the previous tile's reads of the id stages precede their refill
                for (int64_t k = 0; k < first; ++k) issue_ids(sm, slots, n, k, base + k);
            }
            kid_issued = base + first;
            for (int64_t k = 0; k < nchunks && ok; ++k, ++kid) {
                const int is = static_cast<int>(kid % kIdRing);
                int waited = 1;
                if (lane == 0) waited = wait_or_abort(&sm.idfull[is], static_cast<uint32_t>((kid / kIdRing) & 1), &sm.abort);
                if (__shfl_sync(0xffffffffu, waited, 0) == 0) {
                    ok = false;
                    break;
                }
                const int64_t c0 = k * kIdChunk;
                const int64_t cnt = n - c0 < kIdChunk ? n - c0 : kIdChunk;
                const int64_t cnt_even = cnt & ~static_cast<int64_t>(1);
#pragma unroll
                for (int p = 0; p < kIdChunk / 32; ++p) {
                    const int j = p * 32 + lane;
                    const int64_t id = j < cnt_even ? sm.ids[is][j] : (j < cnt ? slots[c0 + j] : -1);
                    if (flagger && (id >= n_slots || id < -1)) atomicOr(&g_smc_status, PRECOG_DEV_BAD_INDEX);
                    uint32_t ball = __ballot_sync(0xffffffffu, id == slot);
                    while (ball != 0u && ok) {
                        const int jj = __ffs(static_cast<int>(ball)) - 1;
                        ball &= ball - 1u;
                        ok = produce_stage(sm, g, lane, src + (c0 + p * 32 + jj) * elems, bytes);
                        if (ok) ++g;
                    }
                }
                __syncwarp();
                if (ok && k + kIdRing < nchunks) {
                    if (lane == 0) {
                        fence_proxy_async_smem();   // the warp's reads of this id stage precede its refill
                        issue_ids(sm, slots, n, k + kIdRing, base + k + kIdRing);
                    }
                    ++kid_issued;
                }
            }
            if (ok) {
                ok = produce_stage(sm, g, lane, nullptr, 0);
                if (ok) ++g;
            }
        }
        if (!ok && lane == 0) {
            // Give up: record it, stop the consumers, let the issued copies land.
            atomicOr(&g_smc_status, PRECOG_DEV_TIMEOUT);
            *static_cast<volatile int32_t *>(&sm.abort) = 1;
            for (uint32_t g2 = g > kRing ? g - kRing : 0; g2 < g; ++g2)
                mbar_wait(&sm.full[g2 % kRing], (g2 / kRing) & 1u);
            for (int64_t u = kid; u < kid_issued; ++u)
                mbar_wait(&sm.idfull[u % kIdRing], static_cast<uint32_t>((u / kIdRing) & 1));
        }
        return;
    }

    // ---- consumer warps ----
    const float keep = 1.f - alpha;
    uint32_t g = 0;
    for (int64_t t = t_begin; t < t_end; ++t) {
        const int64_t slot = t / nranges;
        const int64_t e0 = (t % nranges) * R;
        const int64_t rlen = elems - e0 < R ? elems - e0 : R;
        float *srow = sem + slot * elems + e0;
        float v[kChunksPerThread][CH];
        bool have[kChunksPerThread];
#pragma unroll
        for (int i = 0; i < kChunksPerThread; ++i) {
            const int64_t q = static_cast<int64_t>(i) * kBulkConsumers + tid;
            have[i] = q * CH < rlen;
#pragma unroll
            for (int k = 0; k < CH; k += 4) {
                float4 f = make_float4(0.f, 0.f, 0.f, 0.f);
                if (have[i]) f = *reinterpret_cast<const float4 *>(srow + q * CH + k);
                v[i][k] = f.x;
                v[i][k + 1] = f.y;
                v[i][k + 2] = f.z;
                v[i][k + 3] = f.w;
            }
        }
        bool touched = false;
        while (true) {
            const int s = static_cast<int>(g % kRing);
            if (!wait_or_abort(&sm.full[s], (g / kRing) & 1u, &sm.abort)) {
                if (lane == 0) atomicOr(&g_smc_status, PRECOG_DEV_TIMEOUT);
                *static_cast<volatile int32_t *>(&sm.abort) = 1;
                return;
            }
            const int32_t tag = sm.tag[s];
            if (tag == kTagData) {
#pragma unroll
                for (int i = 0; i < kChunksPerThread; ++i) {
                    if (!have[i]) continue;
                    const uint4 raw = *reinterpret_cast<const uint4 *>(
                        sm.ring[s] + (static_cast<int>(i) * kBulkConsumers + tid) * 16);
                    float h[CH];
                    if constexpr (std::is_same<TS, float>::value) {
                        h[0] = __uint_as_float(raw.x);
                        h[1] = __uint_as_float(raw.y);
                        h[2] = __uint_as_float(raw.z);
                        h[3] = __uint_as_float(raw.w);
                    } else {
                        const uint32_t w[4] = {raw.x, raw.y, raw.z, raw.w};
#pragma unroll
                        for (int k = 0; k < 4; ++k) {
                            h[2 * k] = __uint_as_float(w[k] << 16);
                            h[2 * k + 1] = __uint_as_float(w[k] & 0xffff0000u);
                        }
                    }
#pragma unroll
                    for (int k = 0; k < CH; ++k) v[i][k] = fmaf(keep, v[i][k], alpha * h[k]);
                }
                touched = true;
            }
            __syncwarp();
            if (lane == 0) mbar_arrive(&sm.empty[s]);
            ++g;
            if (tag != kTagData) break;
        }
        if (touched) {
#pragma unroll
            for (int i = 0; i < kChunksPerThread; ++i) {
                if (!have[i]) continue;
                const int64_t q = static_cast<int64_t>(i) * kBulkConsumers + tid;
#pragma unroll
                for (int k = 0; k < CH; k += 4)
                    *reinterpret_cast<float4 *>(srow + q * CH + k) =
                        make_float4(v[i][k], v[i][k + 1], v[i][k + 2], v[i][k + 3]);
            }
        }
    }
}

}  // namespace

template <typename T>
void launch_route_t(const void *emb, int64_t n, int dim, const void *dom, int M, const void *sub, int J_max,
                    const int32_t *J, int32_t *out_m, int32_t *out_j, int64_t *out_slot, unsigned grid,
                    cudaStream_t stream) {
    const auto *e = static_cast<const T *>(emb);
    const auto *d = static_cast<const T *>(dom);
    const auto *s = static_cast<const T *>(sub);
    const auto a16 = [](const void *ptr) { return reinterpret_cast<uintptr_t>(ptr) % 16 == 0; };
    const bool vec = (static_cast<int64_t>(dim) * static_cast<int64_t>(sizeof(T))) % 16 == 0 && a16(emb) &&
                     a16(dom) && a16(sub);
    if (vec)
        smc_route_kernel<T, true><<<grid, kRouteWarps * 32, 0, stream>>>(e, n, dim, d, M, s, J_max, J, out_m,
                                                                        out_j, out_slot);
    else
        smc_route_kernel<T, false><<<grid, kRouteWarps * 32, 0, stream>>>(e, n, dim, d, M, s, J_max, J, out_m,
                                                                         out_j, out_slot);
}

cudaError_t launch_smc_route(const void *emb, int dtype, int64_t n, int dim, const void *dom, int M,
                             const void *sub, int J_max, const int32_t *J, int32_t *out_m,
                             int32_t *out_j, int64_t *out_slot, cudaStream_t stream) {
    if (n == 0) return cudaSuccess;
    const unsigned grid = static_cast<unsigned>((n + kRouteWarps - 1) / kRouteWarps);
    switch (dtype) {
        case PRECOG_F16:
            launch_route_t<__half>(emb, n, dim, dom, M, sub, J_max, J, out_m, out_j, out_slot, grid, stream);
            break;
        case PRECOG_BF16:
            launch_route_t<__nv_bfloat16>(emb, n, dim, dom, M, sub, J_max, J, out_m, out_j, out_slot, grid, stream);
            break;
        default:
            launch_route_t<float>(emb, n, dim, dom, M, sub, J_max, J, out_m, out_j, out_slot, grid, stream);
    }
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

cudaError_t launch_smc_consolidate(float *sem, int64_t n_slots, int64_t elems, const void *states,
                                   int states_dtype, const int64_t *slots, int64_t n, float alpha,
                                   cudaStream_t stream) {
    if (n == 0 || elems == 0) return cudaSuccess;
    // pairs of elements when every row start stays 8-byte (fp32) / 4-byte (bf16) aligned
    const bool pairs = elems % 2 == 0;
    const int vec = pairs ? 2 : 1;
    const int64_t blocks = (elems / vec + kConsThreads - 1) / kConsThreads;
    if (blocks > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
    const unsigned grid = static_cast<unsigned>(blocks);
    // Few slots: CTAs per (slot, element range). Each tile reads all n slot ids (from
    // L2): n_slots / 2048 of its state bytes with 16 KB ranges, so it pays up to 256
    // slots. Rows of whole 16-byte chunks stream through the TMA ring; other rows take
    // the register per-slot kernel (whose 2048-element ranges read n_slots / 512).
    const int64_t chunk = states_dtype == PRECOG_BF16 ? 8 : 4;
    if (n_slots >= 1 && n_slots <= 256 && elems % chunk == 0 && reinterpret_cast<uintptr_t>(slots) % 16 == 0) {
        const int64_t range = kStageBytes / (states_dtype == PRECOG_BF16 ? 2 : 4);
        const int64_t ntiles = n_slots * ((elems + range - 1) / range);
        const int64_t resident = 2 * static_cast<int64_t>(device_sm_count());
        const int64_t per_cta = (ntiles + resident - 1) / resident;
        const int64_t blocks2 = (ntiles + per_cta - 1) / per_cta;
        if (blocks2 > 0x7fffffffLL) return cudaErrorInvalidConfiguration;
        const int smem = static_cast<int>(sizeof(BulkSmem));
        cudaError_t e;
        if (states_dtype == PRECOG_BF16) {
            e = ensure_smem(reinterpret_cast<const void *>(smc_consolidate_bulk_kernel<__nv_bfloat16>), smem);
            if (e != cudaSuccess) return e;
            smc_consolidate_bulk_kernel<__nv_bfloat16><<<static_cast<unsigned>(blocks2), kBulkThreads, smem, stream>>>(
                sem, n_slots, elems, static_cast<const __nv_bfloat16 *>(states), slots, n, alpha, ntiles, per_cta);
        } else {
            e = ensure_smem(reinterpret_cast<const void *>(smc_consolidate_bulk_kernel<float>), smem);
            if (e != cudaSuccess) return e;
            smc_consolidate_bulk_kernel<float><<<static_cast<unsigned>(blocks2), kBulkThreads, smem, stream>>>(
                sem, n_slots, elems, static_cast<const float *>(states), slots, n, alpha, ntiles, per_cta);
        }
        e = cudaGetLastError();
        if (e == cudaSuccess) count_launches(1);
        return e;
    }
    if (n_slots >= 1 && n_slots <= 256) {
        const int64_t per_cta = static_cast<int64_t>(kSlotThreads) * kSlotItems * vec;
        const dim3 g2(static_cast<unsigned>((elems + per_cta - 1) / per_cta), static_cast<unsigned>(n_slots));
        if (states_dtype == PRECOG_BF16) {
            const auto *st = static_cast<const __nv_bfloat16 *>(states);
            if (pairs) smc_consolidate_slot_kernel<__nv_bfloat16, 2><<<g2, kSlotThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
            else smc_consolidate_slot_kernel<__nv_bfloat16, 1><<<g2, kSlotThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
        } else {
            const auto *st = static_cast<const float *>(states);
            if (pairs) smc_consolidate_slot_kernel<float, 2><<<g2, kSlotThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
            else smc_consolidate_slot_kernel<float, 1><<<g2, kSlotThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
        }
        cudaError_t e = cudaGetLastError();
        if (e == cudaSuccess) count_launches(1);
        return e;
    }
    if (states_dtype == PRECOG_BF16) {
        const auto *st = static_cast<const __nv_bfloat16 *>(states);
        if (pairs) smc_consolidate_kernel<__nv_bfloat16, 2><<<grid, kConsThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
        else smc_consolidate_kernel<__nv_bfloat16, 1><<<grid, kConsThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
    } else {
        const auto *st = static_cast<const float *>(states);
        if (pairs) smc_consolidate_kernel<float, 2><<<grid, kConsThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
        else smc_consolidate_kernel<float, 1><<<grid, kConsThreads, 0, stream>>>(sem, n_slots, elems, st, slots, n, alpha);
    }
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
