// Host-side interfaces between the C ABI (api.cu) and the kernel files.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda.h>
#include <cuda_runtime.h>

namespace precog {

// One scan launch: L layers x n_chunks chunks x channel slices, each work item
// a CTA that rolls the recurrence over one chunk for one slice of channels.
struct ScanParams {
    // inputs
    const void *x, *dt, *B, *C;
    const float *A;
    int64_t ls_xd, ls_bc;     // layer strides in elements
    int32_t n_layers, D, N;
    int32_t in_dtype;         // precog_dtype
    int32_t a_kind;           // precog_a_kind
    int64_t T_tot;            // rows per layer
    // chunking: use_fixed -> chunk c is rows [c*fixed_len, (c+1)*fixed_len),
    // else rows [offsets[c], offsets[c+1])
    const int64_t *offsets;
    int64_t n_chunks;
    // processing order: work item i takes chunk order[i] (nullptr: chunk i); results are
    // written at the chunk's own index, so any permutation gives the same outputs
    const int64_t *order = nullptr;
    int32_t use_fixed;
    int32_t fixed_len;
    // initial state (prefill); bank == nullptr -> zero state
    const void *bank;
    int32_t bank_dtype;
    int64_t bank_entries;
    const int64_t *idx;       // nullptr -> row = chunk; [n_chunks][topk] when topk > 1
    int32_t topk;             // rows composed per chunk (<= 1: plain injection)
    const float *topk_scores; // [n_chunks][topk] retrieval scores (topk > 1)
    float inv_temp;           // 1 / softmax temperature
    int32_t L_bank;           // layers per bank entry
    // outputs
    void *states;             // [n_chunks][L_out][D][N] or nullptr
    int32_t state_dtype;
    int32_t L_out;            // layers per output entry
    int32_t layer0;           // first layer of the bank / output entries
    void *y;                  // [L][T_tot][D] or nullptr
    int32_t y_dtype;
    // trajectory (K-dial): states after every traj_stride-th token and the last
    void *traj;               // [entries][L_out][D][N] or nullptr
    int32_t traj_dtype;
    int64_t traj_stride;
    const int64_t *traj_offsets;  // [n_chunks+1] first entry of each chunk
};

// Bounded-wait self-test (selftest.cu).
cudaError_t launch_wait_timeout(uint32_t limit, cudaStream_t stream);
cudaError_t selftest_status_word_read_clear(uint32_t *bits);

// SM count of the current device (cached per device; 1 if it cannot be read).
int device_sm_count();

// cuTensorMapEncodeTiled through the runtime's driver entry point (no link against
// libcuda); false if the entry point is missing or the driver rejects the map.
bool encode_tiled_map(CUtensorMap *map, CUtensorMapDataType dtype, cuuint32_t rank, const void *base,
                      const cuuint64_t *dims, const cuuint64_t *strides_bytes, const cuuint32_t *box,
                      CUtensorMapSwizzle swizzle);

// Kernel launches made by this library since the process started.
void count_launches(uint64_t n);

// Raise a kernel's dynamic shared-memory limit once per device (a host-side
// attribute, not a stream operation, so later calls stay graph-capturable).
cudaError_t ensure_smem(const void *kernel, int bytes);

cudaError_t launch_scan(const ScanParams &p, cudaStream_t stream);

// Latency-shaped direct scan with readout (scan_latency.cu): power-form A, D a
// multiple of 64; scan.cu routes launches with fewer work items than SMs to it.
bool scan_latency_eligible(const ScanParams &p);
cudaError_t launch_scan_latency(const ScanParams &p, cudaStream_t stream);
cudaError_t scan_latency_status_word_read_clear(uint32_t *bits);
cudaError_t scan_status_word_read_clear(uint32_t *bits);

struct RetrieveParams {
    const void *index;
    int32_t dtype;
    int64_t M;
    int32_t dim;
    const void *queries;
    int32_t n_queries;
    int64_t *best_idx;
    float *best_score;
    void *workspace;
    size_t workspace_bytes;
    // shard mode (precog_retrieve_keys): rows are row_offset + local row, and the result
    // is one signed-order key per query in keys_out instead of best_idx / best_score
    int64_t row_offset = 0;
    int64_t *keys_out = nullptr;
};

size_t retrieve_workspace_size(int64_t M, int32_t dim, int32_t n_queries);
cudaError_t launch_decode_keys(const int64_t *keys, int32_t n, int64_t *best_idx, float *best_score,
                               cudaStream_t stream);

// Tensor-core path (retrieve_tc.cu): fp16/bf16 index, batches of queries.
size_t retrieve_tc_smem_bytes();
int retrieve_tc_grid(int64_t M, int sms);
cudaError_t launch_retrieve_tc(const RetrieveParams &p, int grid, cudaStream_t stream,
                               uint64_t *launches);
cudaError_t retrieve_tc_status_word_read_clear(uint32_t *bits);

// Top-k retrieval (k <= 8): partial lists of 8 packed keys per (part, query).
size_t retrieve_topk_workspace_size(int64_t M, int32_t dim, int32_t n_queries);
cudaError_t launch_retrieve_topk(const RetrieveParams &p, int k, cudaStream_t stream);
cudaError_t launch_retrieve_tc_topk(const RetrieveParams &p, int k, int grid, cudaStream_t stream,
                                    uint64_t *launches);
cudaError_t launch_retrieve(const RetrieveParams &p, cudaStream_t stream);
cudaError_t retrieve_status_word_read_clear(uint32_t *bits);

// Complex diagonal A (scan_complex.cu): A is [L][D][N] (re, im) pairs, states
// [..][D][N] (re, im) pairs.
cudaError_t launch_scan_complex(const ScanParams &p, cudaStream_t stream);
cudaError_t scan_complex_status_word_read_clear(uint32_t *bits);

// SMC primitives (smc.cu)
cudaError_t launch_smc_route(const void *emb, int dtype, int64_t n, int dim, const void *dom, int M,
                             const void *sub, int J_max, const int32_t *J, int32_t *out_m,
                             int32_t *out_j, int64_t *out_slot, cudaStream_t stream);
cudaError_t launch_smc_consolidate(float *sem, int64_t n_slots, int64_t elems, const void *states,
                                   int states_dtype, const int64_t *slots, int64_t n, float alpha,
                                   cudaStream_t stream);
cudaError_t smc_status_word_read_clear(uint32_t *bits);

}  // namespace precog
