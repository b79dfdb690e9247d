/*
 * precog.h -- C ABI of the PRECOG hot path on one GB300 GPU (sm_103a).
 *
 * PRECOG (Sec. 4 of "Structured Memory for Edge Language Models: Persistent
 * Context and Corpus Retrieval via O(1) SSM State Injection") pre-encodes
 * corpus chunks into the final hidden state of a selective SSM (offline
 * indexing, Sec. 4.2), retrieves the best-matching chunk for a query by
 * embedding similarity, injects that chunk's state as the recurrence's initial
 * condition (Eq. 2) and prefills only the query tokens from it. Theorem 1
 * guarantees this equals scanning [chunk; query] from the zero state.
 *
 * Conventions shared by every call
 *   - All data pointers are DEVICE pointers owned by the caller; the library
 *     allocates nothing. Each must be 16-byte aligned.
 *   - `stream` is a cudaStream_t passed as void* (NULL = legacy default
 *     stream). Every call only enqueues work on it and returns; results are
 *     ready when the stream reaches that point.
 *   - Argument errors are detected on the host before anything is enqueued;
 *     the call then returns PRECOG_ERR_INVALID_ARG or PRECOG_ERR_UNSUPPORTED and
 *     leaves every output untouched. precog_last_error() describes the cause.
 *   - Errors that only the device can see (a bad chunk offset, an out-of-range
 *     bank row, a pipeline wait that gave up) are recorded in a device status
 *     word instead of faulting; precog_device_status() reports and clears it.
 *   - Floating point: the recurrence and every accumulation run in fp32.
 *   - No call raises a C++ exception or aborts across this boundary.
 */
#ifndef PRECOG_H_
#define PRECOG_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

#define PRECOG_ABI_VERSION 1

typedef enum precog_status {
    PRECOG_OK = 0,
    PRECOG_ERR_INVALID_ARG = 1,  /* a pointer, size or layout argument is invalid */
    PRECOG_ERR_UNSUPPORTED = 2,  /* valid, but outside what the kernels implement */
    PRECOG_ERR_CUDA = 3,         /* a CUDA runtime call or a launch failed */
    PRECOG_ERR_TIMEOUT = 4,      /* a bounded device-side wait gave up */
    PRECOG_ERR_DEVICE = 5        /* the device flagged bad offsets, bank rows, slots or A */
} precog_status;
/* Status 5 reports what only the device can see (precog_device_status: bad offsets, a
 * bank row or slot outside its table, a false PRECOG_A_POWER statement). A retrieval
 * with no comparable score (an empty index, or every score NaN) is not an error: it
 * returns PRECOG_OK with row -1 and score NaN, a well-defined "no context" result that
 * injects the zero state. There is no separate numeric-failure status. */

typedef enum precog_dtype {
    PRECOG_F32 = 0,
    PRECOG_BF16 = 1,
    PRECOG_F16 = 2
} precog_dtype;

/* Structure of the diagonal state matrix A (see precog_scan_inputs). */
typedef enum precog_a_kind {
    PRECOG_A_GENERAL = 0,  /* any A: one exponential per (channel, state index) */
    PRECOG_A_POWER = 1,    /* A[d,n] == (n+1)*A[d,0] exactly and A[d,0] <= 0 */
    PRECOG_A_COMPLEX = 2   /* complex A: see precog_scan_inputs */
} precog_a_kind;

/* Device status bits reported by precog_device_status(). */
#define PRECOG_DEV_BAD_OFFSETS 0x1u  /* offsets not non-decreasing or beyond T_tot */
#define PRECOG_DEV_BAD_INDEX 0x2u    /* a bank row index outside [-1, bank_entries), or a
                                        chunk order entry outside [0, n_chunks) */
#define PRECOG_DEV_TIMEOUT 0x4u      /* an mbarrier wait hit its iteration limit */
#define PRECOG_DEV_BAD_A 0x8u        /* a_kind == PRECOG_A_POWER but A is not */

/*
 * Inputs of the selective-SSM scan for L layers (Sec. 3, Eq. 1).
 *
 * Per layer l, channel d, state index n and token row t:
 *   alpha = exp(dt[t,d] * A[d,n])     (A < 0: the stable reading of Eq. 1)
 *   h[d,n] <- alpha * h[d,n] + B[t,n] * x[t,d] * dt[t,d]
 *   y[t,d]  = sum_n C[t,n] * h[d,n]   (readout of the updated state)
 * dt is per (token, channel) and B, C per (token, state index), shared across
 * channels: the input-dependent timescale and projections of a selective SSM
 * ("dt and B are functions of the current token only", Sec. 3).
 *
 * Layout (row-major, element strides):
 *   x, dt : layer l at  x + l*layer_stride_xd, each block [T_tot][D]
 *   B, C  : layer l at  B + l*layer_stride_bc, each block [T_tot][N]
 *   A     : [L][D][N] fp32, always dense
 * x, dt, B, C share `in_dtype` (PRECOG_F32 or PRECOG_BF16). C may be NULL
 * when no readout is requested. Strides are in elements and must keep every
 * layer block 16-byte aligned; they may be 0 when n_layers == 1.
 * Requirements: N == 16; D >= 1 with D*sizeof(in_dtype) a multiple of 16.
 * x, dt and B (and C) may be NULL only when there are no token rows.
 *
 * a_kind selects the update form. PRECOG_A_GENERAL accepts any A and takes
 * one exponential per (d, n). PRECOG_A_POWER is the caller's statement that
 * A[d,n] == (n+1)*A[d,0] exactly with A[d,0] <= 0 (e.g. A[d,n] = -(n+1)), so
 * that alpha_n = r^(n+1) with r = exp(dt*A[d,0]): one exponential per (t, d).
 * The kernel verifies the statement per block of channels; where it is false
 * nothing is written for that block and PRECOG_DEV_BAD_A is flagged.
 *
 * PRECOG_A_COMPLEX selects the complex diagonal A that Eq. 1 prints
 * (A_k = -softplus(a_k) + i*pi*k) with a complex state h in C^N: A points to
 * [L][D][N] pairs (re, im) of fp32 (torch.complex64 layout); alpha =
 * exp(dt*A) is complex, B and C stay real, y = Re(sum_n C[t,n] h[d,n]);
 * states and banks hold (re, im) pairs per state index, [..][D][N][2]
 * (complex64 for F32 state dtype, bf16 pairs for BF16). Accepted by
 * precog_encode_chunks and precog_prefill_from_state (and k = 1 composition).
 */
typedef struct precog_scan_inputs {
    int32_t n_layers;
    int32_t D;
    int32_t N;
    int32_t in_dtype;          /* precog_dtype */
    int32_t a_kind;            /* precog_a_kind */
    int32_t reserved;          /* must be 0 */
    const void *x;
    const void *dt;
    const void *B;
    const void *C;
    const float *A;
    int64_t layer_stride_xd;
    int64_t layer_stride_bc;
} precog_scan_inputs;

/*
 * precog_encode_chunks -- offline indexing (Sec. 4.2): scan every chunk of a
 * ragged batch from the zero state (Appendix B.1) through L layers and capture
 * each chunk's final per-layer state h(c) = S(0, c) (Theorem 1 notation).
 *
 *   in          scan inputs, L = in->n_layers layers, T_tot token rows each
 *   d_offsets   device int64 [n_chunks+1]: chunk c owns rows
 *               d_offsets[c] .. d_offsets[c+1]-1 of every layer; must be
 *               non-decreasing with d_offsets[n_chunks] <= T_tot (checked on
 *               the device: a bad chunk is skipped and flags
 *               PRECOG_DEV_BAD_OFFSETS). A zero-length chunk captures zeros.
 *   states_out  device [n_chunks][L_total][D][N] in state_dtype (F32 or BF16,
 *               rounded to nearest even once, at capture); the call writes
 *               layers layer0 .. layer0+L-1 and nothing else. May be NULL
 *               when y_out is given.
 *   y_out       device [L][T_tot][D] in y_dtype (F32 or BF16): readout after
 *               every token (used to check Theorem 1), or NULL for capture
 *               only. Rows outside every chunk are left untouched.
 * Returns PRECOG_OK once the work is enqueued.
 */
precog_status precog_encode_chunks(const precog_scan_inputs *in, const int64_t *d_offsets,
                                   int64_t n_chunks, int64_t T_tot, void *states_out,
                                   int32_t state_dtype, int32_t layer0, int32_t L_total,
                                   void *y_out, int32_t y_dtype, void *stream);

/*
 * precog_encode_chunks_ordered -- precog_encode_chunks with the order in which
 * chunks are taken up (Sec. 4.2: chunks are independent, so any order gives the
 * same states). With ragged chunks the last chunks to start decide when the
 * launch ends; a caller that knows the lengths (it built d_offsets) can pass
 * them longest first, so the short ones fill the tail.
 *
 *   d_order   device int64 [n_chunks]: work item i encodes chunk d_order[i],
 *             and its state (and y rows) are written at that chunk's own index.
 *             Meant to be a permutation of 0 .. n_chunks-1 (not verified: a
 *             repeated chunk is written twice with the same result, a missing one
 *             is not written). An entry outside [0, n_chunks) is skipped and
 *             flags PRECOG_DEV_BAD_INDEX. NULL returns PRECOG_ERR_INVALID_ARG.
 * Other arguments, layouts and errors as precog_encode_chunks.
 */
precog_status precog_encode_chunks_ordered(const precog_scan_inputs *in, const int64_t *d_offsets,
                                           int64_t n_chunks, int64_t T_tot, const int64_t *d_order,
                                           void *states_out, int32_t state_dtype, int32_t layer0,
                                           int32_t L_total, void *y_out, int32_t y_dtype, void *stream);

/*
 * precog_encode_trajectory -- the K-dial state trajectory of SMC (Sec. 5.2,
 * Eq. smc-trajectory): scan every chunk from the zero state like
 * precog_encode_chunks and keep the state after every `stride`-th token and
 * after the chunk's last token. Chunk c keeps K_c = ceil(len_c / stride)
 * states (K = N_c / k in the paper; stride 1 keeps every state, stride >=
 * len_c keeps only the final, PRECOG state). Uses the direct update.
 *   d_entry_offsets  device int64 [n_chunks+1]: prefix sums of K_c; a chunk
 *                    whose count disagrees with its length is skipped and
 *                    flags PRECOG_DEV_BAD_OFFSETS
 *   traj_out         device [d_entry_offsets[n_chunks]][L_total][D][N] in
 *                    traj_dtype (F32 or BF16); entry d_entry_offsets[c] + j is
 *                    the state after token min((j+1)*stride, len_c) of chunk c,
 *                    written for layers layer0 .. layer0+L-1
 * Other arguments as precog_encode_chunks.
 */
precog_status precog_encode_trajectory(const precog_scan_inputs *in, const int64_t *d_offsets,
                                       int64_t n_chunks, int64_t T_tot, int64_t stride,
                                       const int64_t *d_entry_offsets, void *traj_out,
                                       int32_t traj_dtype, int32_t layer0, int32_t L_total,
                                       void *stream);

/*
 * precog_retrieve -- query-time retrieval (Sec. 4.2): for every query q the
 * row i* of the key index with the highest dot product <query_q, key_i>
 * (unit-norm keys and queries make this the cosine similarity of the paper).
 * Exact top-1, not an approximate index. Scores accumulate in fp32 from the
 * stored values; ties go to the lowest row; a NaN score never wins; if no row
 * has a comparable score (M == 0, or every score NaN) the result is index -1 and
 * score NaN, and the call still returns PRECOG_OK.
 *
 *   index          device [M][dim] keys in index_dtype (F16, BF16 or F32)
 *   queries        device [n_queries][dim], same dtype as the index
 *   d_best_idx     device int64 [n_queries] (written)
 *   d_best_score   device fp32 [n_queries] (written), or NULL
 *   workspace      device scratch of at least
 *                  precog_retrieve_workspace_size(M, dim, n_queries) bytes;
 *                  contents on entry are ignored and clobbered
 * Requirements: 0 <= M < 2^31 - 1; dim >= 1 with dim*sizeof(dtype) a
 * multiple of 16; n_queries >= 0.
 */
precog_status precog_retrieve(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                              const void *queries, int32_t n_queries, int64_t *d_best_idx,
                              float *d_best_score, void *workspace, size_t workspace_bytes,
                              void *stream);

/* Bytes of device workspace precog_retrieve needs for these sizes. */
size_t precog_retrieve_workspace_size(int64_t M, int32_t dim, int32_t n_queries);

/*
 * precog_retrieve_noalloc -- precog_retrieve for callers that cannot allocate
 * device memory when they retrieve (a serving loop that must never call
 * cudaMalloc, which may synchronise the device; code that runs inside someone
 * else's memory pool). The paper has no counterpart: this is a property of the
 * library, not of the method. Same arguments and results as precog_retrieve,
 * without the workspace: the partial keys go to a fixed 2 MiB array compiled
 * into the library, which every GPU that loads the library holds until exit.
 *   - Allocates nothing and calls no allocating routine.
 *   - The first call in a CUDA context looks up that array's device address in
 *     that context (once per context, with the context current; a reset device
 *     or another context of the same device gets its own lookup); make that
 *     first call before any stream capture.
 *   - Calls whose sizes need more than the 2 MiB (keys = precog_retrieve
 *     workspace bytes / 8; about 430 queries per call at any M on a 152-SM GPU)
 *     return PRECOG_ERR_UNSUPPORTED without launching anything.
 *   - All calls share the array and nothing in it needs to start at zero; two
 *     calls that overlap on the GPU (different streams, or different host
 *     threads without ordering) race on it and may return wrong rows.
 */
precog_status precog_retrieve_noalloc(const void *index, int32_t index_dtype, int64_t M,
                                      int32_t dim, const void *queries, int32_t n_queries,
                                      int64_t *d_best_idx, float *d_best_score, void *stream);

/*
 * precog_prefill_from_state -- state injection and query prefill (Sec. 4.2,
 * Eq. 2): for every query q and layer l, h_init[l] <- bank[row_q][layer0+l],
 * then scan the query's T_q tokens from h_init, producing y_t for every query
 * token and the updated state. By Theorem 1 this equals scanning
 * [chunk; query] from the zero state.
 *
 *   in           scan inputs with T_tot = n_queries*T_q rows per layer: query
 *                q owns rows q*T_q .. q*T_q+T_q-1; C is required when y_out
 *                is given
 *   bank         device [bank_entries][L_bank][D][N] in bank_dtype (F32/BF16)
 *   d_idx        device int64 [n_queries]: bank row injected for query q
 *                (e.g. precog_retrieve's d_best_idx, read on the device with
 *                no host round trip). -1 injects the zero state (no context).
 *                Other rows outside [0, bank_entries) also inject zeros and
 *                flag PRECOG_DEV_BAD_INDEX. NULL means row q for query q.
 *   layer0       first bank layer used; layers layer0 .. layer0+L-1 must be
 *                < L_bank
 *   y_out        device [L][n_queries*T_q][D] in y_dtype, or NULL
 *   state_out    device [n_queries][L_bank][D][N] in state_dtype (layers
 *                layer0 .. layer0+L-1 written), or NULL
 */
precog_status precog_prefill_from_state(const precog_scan_inputs *in, int32_t n_queries,
                                        int32_t T_q, const void *bank, int32_t bank_dtype,
                                        int64_t bank_entries, int32_t L_bank, int32_t layer0,
                                        const int64_t *d_idx, void *y_out, int32_t y_dtype,
                                        void *state_out, int32_t state_dtype, void *stream);

/*
 * precog_retrieve_topk -- the k best rows per query (1 <= k <= 8), best first:
 * the top-k retrieval of Sec. 4.2 (k = 3 by default in the paper) that feeds
 * the softmax-weighted composition of Sec. 4.4 and Eq. smc-fusion. Same
 * scoring and tie rule as precog_retrieve (ties to the lower row, NaN never
 * selected); missing entries (fewer than k comparable rows) are row -1 with
 * score NaN.
 *   d_idx    device int64 [n_queries][k] (written)
 *   d_score  device fp32 [n_queries][k] (written), or NULL
 *   workspace at least precog_retrieve_topk_workspace_size(M, dim, n_queries)
 */
precog_status precog_retrieve_topk(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                                   const void *queries, int32_t n_queries, int32_t k,
                                   int64_t *d_idx, float *d_score, void *workspace,
                                   size_t workspace_bytes, void *stream);

/* Bytes of device workspace precog_retrieve_topk needs for these sizes (any k). */
size_t precog_retrieve_topk_workspace_size(int64_t M, int32_t dim, int32_t n_queries);

/*
 * precog_prefill_composed -- top-k state composition, then prefill: the
 * heuristic multi-chunk extension of Sec. 4.4 (Eq. smc-fusion),
 *   h_init[l] = sum_j w_j bank[row_qj][layer0+l],  w = softmax(score_qj / temperature),
 * over the valid entries of query q (a row of -1 or a NaN score has weight 0;
 * a row outside the bank has weight 0 and flags PRECOG_DEV_BAD_INDEX), then
 * the same prefill as precog_prefill_from_state. Weights and the sum are fp32.
 * Unlike top-1 injection this is not exact in-context equivalence (Theorem 1
 * covers a single chunk only).
 *   k          1..8 entries per query; k == 1 is precog_prefill_from_state
 *   d_idx      device int64 [n_queries][k] rows (e.g. precog_retrieve_topk's)
 *   d_score    device fp32 [n_queries][k] scores (ignored when k == 1)
 *   temperature > 0; the paper's plain softmax of the similarity is 1.0
 * Other arguments as precog_prefill_from_state.
 */
precog_status precog_prefill_composed(const precog_scan_inputs *in, int32_t n_queries, int32_t T_q,
                                      const void *bank, int32_t bank_dtype, int64_t bank_entries,
                                      int32_t L_bank, int32_t layer0, int32_t k,
                                      const int64_t *d_idx, const float *d_score, float temperature,
                                      void *y_out, int32_t y_dtype, void *state_out,
                                      int32_t state_dtype, void *stream);

/*
 * precog_retrieve_keys -- precog_retrieve over one shard of an index whose rows are
 * partitioned (e.g. across ranks): the shard holds rows row_offset .. row_offset+M-1
 * of the whole index. For every query it writes one 64-bit key of its best row,
 *   key = ((ordered bits of the fp32 score) << 32 | (2^32 - 1 - global row)) XOR 2^63,
 * so that keys compare as signed int64 by score, then lower row ("no comparable row"
 * is INT64_MIN). The signed maximum of the shards' keys (an all-reduce MAX over
 * int64) is the key of the exact top-1 of the whole index, ties to the lowest global
 * row, as precog_retrieve would return on the whole index; precog_decode_keys turns
 * keys into rows and scores. This is the exchange step of row-sharded retrieval.
 *   d_keys       device int64 [n_queries] (written)
 *   row_offset   >= 0, with row_offset + M <= 2^32 - 1
 * Other arguments and requirements as precog_retrieve (same workspace size).
 */
precog_status precog_retrieve_keys(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                                   const void *queries, int32_t n_queries, int64_t row_offset,
                                   int64_t *d_keys, void *workspace, size_t workspace_bytes,
                                   void *stream);

/*
 * precog_decode_keys -- rows and scores of keys from precog_retrieve_keys (after
 * combining shards): d_best_idx[q] = global row or -1, d_best_score[q] = score or NaN
 * (d_best_score may be NULL).
 */
precog_status precog_decode_keys(const int64_t *d_keys, int32_t n_queries, int64_t *d_best_idx,
                                 float *d_best_score, void *stream);

/*
 * precog_smc_route -- two-level cluster routing of Structured Memory
 * Consolidation (Sec. 5.1, Eqs. smc-domain and smc-sub): for every embedding e
 * (a chunk's or an opening utterance's text embedding)
 *   m* = argmax_m <e, p_m>,   j* = argmax_{j < J[m*]} <e, q_{m*, j}>,
 * dot products accumulated in fp32 with a fixed order; ties go to the lower
 * index; NaN never wins; -1 when nothing is comparable.
 *   embeddings   device [n][dim]; domain_protos device [M][dim];
 *                sub_protos device [M][J_max][dim]; all of `dtype` (F16/BF16/F32)
 *   d_J          device int32 [M]: sub-clusters in use per domain (<= J_max;
 *                larger values flag PRECOG_DEV_BAD_INDEX and route to none)
 *   d_domain, d_sub  device int32 [n] (written)
 *   d_slot       device int64 [n]: m* * J_max + j*, the row of the semantic-
 *                state table (or -1); may be NULL
 */
precog_status precog_smc_route(const void *embeddings, int32_t dtype, int64_t n, int32_t dim,
                               const void *domain_protos, int32_t M, const void *sub_protos,
                               int32_t J_max, const int32_t *d_J, int32_t *d_domain, int32_t *d_sub,
                               int64_t *d_slot, void *stream);

/*
 * precog_smc_consolidate -- semantic consolidation (Sec. 5.3, Eq. smc-ema): for
 * c = 0, 1, ..., n-1 in order, s[slot_c] <- (1 - alpha) s[slot_c] + alpha h_c,
 * in fp32. A slot of -1 (a forgetting candidate) deposits nothing; a slot
 * outside [0, n_slots) deposits nothing and flags PRECOG_DEV_BAD_INDEX.
 *   semantic     device fp32 [n_slots][state_elems], updated in place (e.g. the
 *                [slots][L][D][N] semantic-state table; inject a row with
 *                precog_prefill_from_state for O(1) session initialisation)
 *   states       device [n][state_elems] in states_dtype (F32 or BF16), e.g. the
 *                chunks' K = 1 states from precog_encode_chunks
 *   d_slots      device int64 [n], e.g. precog_smc_route's d_slot
 *   alpha        in (0, 1]
 * semantic and states must be 16-byte aligned (else PRECOG_ERR_INVALID_ARG).
 * Each element's deposits are applied in deposit order, so the result does not
 * depend on how the work is split.
 */
precog_status precog_smc_consolidate(float *semantic, int64_t n_slots, int64_t state_elems,
                                     const void *states, int32_t states_dtype, const int64_t *d_slots,
                                     int64_t n, float alpha, void *stream);

/*
 * precog_selftest_wait_timeout -- diagnostic; the paper has no counterpart.
 * Every kernel here that waits on copies (TMA completion on an mbarrier) gives
 * the wait an iteration limit: when it runs out, the kernel sets
 * PRECOG_DEV_TIMEOUT in its device status word and returns, so a lost copy
 * becomes an error status instead of a hung GPU. This call exercises that path
 * on purpose: one warp waits, for `iterations` try-wait rounds (1 .. 2^20), on
 * an mbarrier that nothing arrives on, records PRECOG_DEV_TIMEOUT and returns.
 * The next precog_device_status on the stream reports PRECOG_ERR_TIMEOUT with
 * that bit (and clears it); the context stays usable. Asynchronous on `stream`.
 */
precog_status precog_selftest_wait_timeout(uint32_t iterations, void *stream);

/*
 * precog_device_status -- synchronise `stream`, then report and clear the
 * device status word shared by all calls on this device. *bits_out receives
 * the PRECOG_DEV_* bits seen since the last clear. Returns PRECOG_OK when no
 * bit was set, PRECOG_ERR_TIMEOUT when PRECOG_DEV_TIMEOUT was set, otherwise
 * PRECOG_ERR_DEVICE; PRECOG_ERR_CUDA if the synchronisation itself failed.
 */
precog_status precog_device_status(void *stream, uint32_t *bits_out);

/* Human-readable name of a status code (static storage). */
const char *precog_status_string(int32_t status);

/* Detail of the last error returned on the calling thread ("" if none). */
const char *precog_last_error(void);

/* PRECOG_ABI_VERSION of the loaded library. */
int32_t precog_abi_version(void);

/* Number of CUDA kernels this library has launched in this process (all
 * devices, all threads); callers difference it around a region of work. */
uint64_t precog_launch_count(void);

#ifdef __cplusplus
}
#endif

#endif /* PRECOG_H_ */
