// C ABI of the PRECOG hot path: argument validation, dispatch to the
// kernels, status codes. Nothing here allocates device memory.
#include <atomic>
#include <cstdarg>
#include <map>
#include <mutex>
#include <utility>
#include <cstdio>
#include <cstring>

#include "../../include/precog.h"
#include "internal.h"

namespace {

thread_local char g_last_error[512] = "";

precog_status fail(precog_status s, const char *fmt, ...) {
    va_list ap;
    va_start(ap, fmt);
    vsnprintf(g_last_error, sizeof(g_last_error), fmt, ap);
    va_end(ap);
    return s;
}

precog_status ok() {
    g_last_error[0] = '\0';
    return PRECOG_OK;
}

precog_status cuda_fail(cudaError_t e, const char *what) {
    return fail(PRECOG_ERR_CUDA, "%s: %s", what, cudaGetErrorString(e));
}

bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }

int dtype_size(int32_t dt) {
    switch (dt) {
        case PRECOG_F32: return 4;
        case PRECOG_BF16: return 2;
        case PRECOG_F16: return 2;
        default: return 0;
    }
}

bool state_dtype_ok(int32_t dt) { return dt == PRECOG_F32 || dt == PRECOG_BF16; }

// Checks shared by encode and prefill. rows = T_tot per layer.
precog_status check_scan_inputs(const precog_scan_inputs *in, int64_t rows, bool need_C) {
    if (in == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "scan inputs pointer is NULL");
    if (in->n_layers < 1) return fail(PRECOG_ERR_INVALID_ARG, "n_layers must be >= 1");
    if (in->N != 16) return fail(PRECOG_ERR_UNSUPPORTED, "N=%d: only N=16 is implemented", in->N);
    if (in->D < 1) return fail(PRECOG_ERR_INVALID_ARG, "D must be >= 1");
    if (in->a_kind != PRECOG_A_GENERAL && in->a_kind != PRECOG_A_POWER &&
        in->a_kind != PRECOG_A_COMPLEX)
        return fail(PRECOG_ERR_INVALID_ARG, "a_kind must be PRECOG_A_GENERAL, _POWER or _COMPLEX");
    if (in->in_dtype != PRECOG_F32 && in->in_dtype != PRECOG_BF16)
        return fail(PRECOG_ERR_UNSUPPORTED, "in_dtype must be PRECOG_F32 or PRECOG_BF16");
    const int sz = dtype_size(in->in_dtype);
    if ((static_cast<int64_t>(in->D) * sz) % 16 != 0)
        return fail(PRECOG_ERR_UNSUPPORTED, "D*sizeof(in_dtype) must be a multiple of 16");
    if (in->A == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "A must be non-NULL");
    if (rows > 0 && (in->x == nullptr || in->dt == nullptr || in->B == nullptr))
        return fail(PRECOG_ERR_INVALID_ARG, "x, dt and B must be non-NULL");
    if (rows > 0 && need_C && in->C == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "C is required when y_out is given");
    if (!aligned16(in->x) || !aligned16(in->dt) || !aligned16(in->B) || !aligned16(in->A) ||
        (in->C && !aligned16(in->C)))
        return fail(PRECOG_ERR_INVALID_ARG, "input pointers must be 16-byte aligned");
    if (in->n_layers > 1) {
        if (in->layer_stride_xd < rows * in->D || in->layer_stride_bc < rows * in->N)
            return fail(PRECOG_ERR_INVALID_ARG, "layer strides smaller than one layer block");
        if ((in->layer_stride_xd * sz) % 16 != 0 || (in->layer_stride_bc * sz) % 16 != 0)
            return fail(PRECOG_ERR_INVALID_ARG, "layer strides must keep 16-byte alignment");
    }
    return PRECOG_OK;
}

precog::ScanParams base_params(const precog_scan_inputs *in, int64_t rows) {
    precog::ScanParams p;
    std::memset(&p, 0, sizeof(p));
    p.x = in->x;
    p.dt = in->dt;
    p.B = in->B;
    p.C = in->C;
    p.A = in->A;
    p.ls_xd = in->n_layers > 1 ? in->layer_stride_xd : 0;
    p.ls_bc = in->n_layers > 1 ? in->layer_stride_bc : 0;
    p.n_layers = in->n_layers;
    p.D = in->D;
    p.N = in->N;
    p.in_dtype = in->in_dtype;
    p.a_kind = in->a_kind;
    p.T_tot = rows;
    return p;
}

std::atomic<uint64_t> g_launches{0};
std::mutex g_attr_mutex;
// dynamic shared-memory limit already set, per (kernel, device): the attribute is per device
std::map<std::pair<const void *, int>, int> g_smem_attr;

}  // namespace

namespace precog {

void count_launches(uint64_t n) { g_launches.fetch_add(n, std::memory_order_relaxed); }

int device_sm_count() {
    constexpr int kMaxDevices = 64;
    static std::atomic<int> cache[kMaxDevices];
    int dev = 0;
    if (cudaGetDevice(&dev) != cudaSuccess || dev < 0) return 1;
    if (dev < kMaxDevices) {
        const int c = cache[dev].load(std::memory_order_relaxed);
        if (c > 0) return c;
    }
    int n = 0;
    if (cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev) != cudaSuccess || n <= 0) return 1;
    if (dev < kMaxDevices) cache[dev].store(n, std::memory_order_relaxed);
    return n;
}

cudaError_t ensure_smem(const void *kernel, int bytes) {
    int dev = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e != cudaSuccess) return e;
    std::lock_guard<std::mutex> lock(g_attr_mutex);
    int &cached = g_smem_attr[std::make_pair(kernel, dev)];
    if (cached >= bytes) return cudaSuccess;
    e = cudaFuncSetAttribute(kernel, cudaFuncAttributeMaxDynamicSharedMemorySize, bytes);
    if (e == cudaSuccess) cached = bytes;
    return e;
}

}  // namespace precog

namespace {

precog_status encode_chunks(const precog_scan_inputs *in, const int64_t *d_offsets, int64_t n_chunks,
                            int64_t T_tot, void *states_out, int32_t state_dtype, int32_t layer0,
                            int32_t L_total, void *y_out, int32_t y_dtype, const int64_t *d_order,
                            void *stream) {
    if (T_tot < 0) return fail(PRECOG_ERR_INVALID_ARG, "T_tot must be >= 0");
    precog_status s = check_scan_inputs(in, T_tot, y_out != nullptr);
    if (s != PRECOG_OK) return s;
    if (n_chunks < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_chunks must be >= 0");
    if (d_offsets == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "d_offsets is NULL");
    if (states_out == nullptr && y_out == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "states_out and y_out are both NULL: nothing to do");
    if (states_out) {
        if (!state_dtype_ok(state_dtype))
            return fail(PRECOG_ERR_UNSUPPORTED, "state_dtype must be PRECOG_F32 or PRECOG_BF16");
        if (!aligned16(states_out)) return fail(PRECOG_ERR_INVALID_ARG, "states_out not 16-byte aligned");
        if (layer0 < 0 || L_total < 1 || layer0 + in->n_layers > L_total)
            return fail(PRECOG_ERR_INVALID_ARG, "layers [layer0, layer0+n_layers) exceed L_total");
    }
    if (y_out) {
        if (!state_dtype_ok(y_dtype))
            return fail(PRECOG_ERR_UNSUPPORTED, "y_dtype must be PRECOG_F32 or PRECOG_BF16");
        if (!aligned16(y_out)) return fail(PRECOG_ERR_INVALID_ARG, "y_out not 16-byte aligned");
    }
    if (n_chunks == 0) return ok();
    precog::ScanParams p = base_params(in, T_tot);
    p.offsets = d_offsets;
    p.order = d_order;
    p.n_chunks = n_chunks;
    p.states = states_out;
    p.state_dtype = state_dtype;
    p.L_out = L_total;
    p.layer0 = states_out ? layer0 : 0;
    p.y = y_out;
    p.y_dtype = y_dtype;
    cudaError_t e = in->a_kind == PRECOG_A_COMPLEX
                        ? precog::launch_scan_complex(p, static_cast<cudaStream_t>(stream))
                        : precog::launch_scan(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "scan launch");
    return ok();
}

}  // namespace

extern "C" {

precog_status precog_encode_chunks(const precog_scan_inputs *in, const int64_t *d_offsets,
                                   int64_t n_chunks, int64_t T_tot, void *states_out,
                                   int32_t state_dtype, int32_t layer0, int32_t L_total,
                                   void *y_out, int32_t y_dtype, void *stream) {
    return encode_chunks(in, d_offsets, n_chunks, T_tot, states_out, state_dtype, layer0, L_total, y_out,
                         y_dtype, nullptr, stream);
}

precog_status precog_encode_chunks_ordered(const precog_scan_inputs *in, const int64_t *d_offsets,
                                           int64_t n_chunks, int64_t T_tot, const int64_t *d_order,
                                           void *states_out, int32_t state_dtype, int32_t layer0,
                                           int32_t L_total, void *y_out, int32_t y_dtype, void *stream) {
    if (d_order == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "d_order is NULL");
    return encode_chunks(in, d_offsets, n_chunks, T_tot, states_out, state_dtype, layer0, L_total, y_out,
                         y_dtype, d_order, stream);
}

precog_status precog_prefill_from_state(const precog_scan_inputs *in, int32_t n_queries,
                                        int32_t T_q, const void *bank, int32_t bank_dtype,
                                        int64_t bank_entries, int32_t L_bank, int32_t layer0,
                                        const int64_t *d_idx, void *y_out, int32_t y_dtype,
                                        void *state_out, int32_t state_dtype, void *stream) {
    if (n_queries < 0 || T_q < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries and T_q must be >= 0");
    const int64_t rows = static_cast<int64_t>(n_queries) * T_q;
    precog_status s = check_scan_inputs(in, rows, y_out != nullptr);
    if (s != PRECOG_OK) return s;
    if (bank == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "bank is NULL");
    if (!state_dtype_ok(bank_dtype))
        return fail(PRECOG_ERR_UNSUPPORTED, "bank_dtype must be PRECOG_F32 or PRECOG_BF16");
    if (!aligned16(bank)) return fail(PRECOG_ERR_INVALID_ARG, "bank not 16-byte aligned");
    if (bank_entries < 0) return fail(PRECOG_ERR_INVALID_ARG, "bank_entries must be >= 0");
    if (L_bank < 1 || layer0 < 0 || layer0 + in->n_layers > L_bank)
        return fail(PRECOG_ERR_INVALID_ARG, "layers [layer0, layer0+n_layers) exceed L_bank");
    if (d_idx == nullptr && bank_entries < n_queries)
        return fail(PRECOG_ERR_INVALID_ARG, "d_idx is NULL but bank has fewer rows than queries");
    if (y_out == nullptr && state_out == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "y_out and state_out are both NULL: nothing to do");
    if (y_out && (!state_dtype_ok(y_dtype) || !aligned16(y_out)))
        return fail(PRECOG_ERR_INVALID_ARG, "y_out must be 16-byte aligned F32 or BF16");
    if (state_out && (!state_dtype_ok(state_dtype) || !aligned16(state_out)))
        return fail(PRECOG_ERR_INVALID_ARG, "state_out must be 16-byte aligned F32 or BF16");
    if (n_queries == 0) return ok();
    precog::ScanParams p = base_params(in, rows);
    p.n_chunks = n_queries;
    p.use_fixed = 1;
    p.fixed_len = T_q;
    p.bank = bank;
    p.bank_dtype = bank_dtype;
    p.bank_entries = bank_entries;
    p.idx = d_idx;
    p.L_bank = L_bank;
    p.states = state_out;
    p.state_dtype = state_dtype;
    p.L_out = L_bank;
    p.layer0 = layer0;
    p.y = y_out;
    p.y_dtype = y_dtype;
    cudaError_t e = in->a_kind == PRECOG_A_COMPLEX
                        ? precog::launch_scan_complex(p, static_cast<cudaStream_t>(stream))
                        : precog::launch_scan(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "prefill launch");
    return ok();
}

precog_status precog_encode_trajectory(const precog_scan_inputs *in, const int64_t *d_offsets,
                                       int64_t n_chunks, int64_t T_tot, int64_t stride,
                                       const int64_t *d_entry_offsets, void *traj_out,
                                       int32_t traj_dtype, int32_t layer0, int32_t L_total,
                                       void *stream) {
    if (T_tot < 0) return fail(PRECOG_ERR_INVALID_ARG, "T_tot must be >= 0");
    precog_status s = check_scan_inputs(in, T_tot, false);
    if (s != PRECOG_OK) return s;
    if (n_chunks < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_chunks must be >= 0");
    if (stride < 1) return fail(PRECOG_ERR_INVALID_ARG, "stride must be >= 1");
    if (in->a_kind == PRECOG_A_COMPLEX)
        return fail(PRECOG_ERR_UNSUPPORTED, "trajectories of a complex-A scan are not implemented");
    if (d_offsets == nullptr || d_entry_offsets == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "d_offsets and d_entry_offsets must be non-NULL");
    if (traj_out == nullptr || !state_dtype_ok(traj_dtype) || !aligned16(traj_out))
        return fail(PRECOG_ERR_INVALID_ARG, "traj_out must be a 16-byte aligned F32 or BF16 array");
    if (layer0 < 0 || L_total < 1 || layer0 + in->n_layers > L_total)
        return fail(PRECOG_ERR_INVALID_ARG, "layers [layer0, layer0+n_layers) exceed L_total");
    if (n_chunks == 0) return ok();
    precog::ScanParams p = base_params(in, T_tot);
    p.offsets = d_offsets;
    p.n_chunks = n_chunks;
    p.L_out = L_total;
    p.layer0 = layer0;
    p.traj = traj_out;
    p.traj_dtype = traj_dtype;
    p.traj_stride = stride;
    p.traj_offsets = d_entry_offsets;
    cudaError_t e = precog::launch_scan(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "trajectory launch");
    return ok();
}

precog_status precog_prefill_composed(const precog_scan_inputs *in, int32_t n_queries, int32_t T_q,
                                     const void *bank, int32_t bank_dtype, int64_t bank_entries,
                                     int32_t L_bank, int32_t layer0, int32_t k,
                                     const int64_t *d_idx, const float *d_score, float temperature,
                                     void *y_out, int32_t y_dtype, void *state_out,
                                     int32_t state_dtype, void *stream) {
    if (k < 1 || k > 8) return fail(PRECOG_ERR_UNSUPPORTED, "k must be in [1, 8]");
    if (d_idx == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "d_idx is NULL");
    if (in != nullptr && in->a_kind == PRECOG_A_COMPLEX && k > 1)
        return fail(PRECOG_ERR_UNSUPPORTED, "composition of complex states is not implemented");
    if (k > 1 && d_score == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "d_score is NULL");
    if (!(temperature > 0.f)) return fail(PRECOG_ERR_INVALID_ARG, "temperature must be > 0");
    if (k == 1)
        return precog_prefill_from_state(in, n_queries, T_q, bank, bank_dtype, bank_entries, L_bank,
                                         layer0, d_idx, y_out, y_dtype, state_out, state_dtype, stream);
    if (n_queries < 0 || T_q < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries and T_q must be >= 0");
    const int64_t rows = static_cast<int64_t>(n_queries) * T_q;
    precog_status s = check_scan_inputs(in, rows, y_out != nullptr);
    if (s != PRECOG_OK) return s;
    if (bank == nullptr || !state_dtype_ok(bank_dtype) || !aligned16(bank))
        return fail(PRECOG_ERR_INVALID_ARG, "bank must be a 16-byte aligned F32 or BF16 array");
    if (bank_entries < 0) return fail(PRECOG_ERR_INVALID_ARG, "bank_entries must be >= 0");
    if (L_bank < 1 || layer0 < 0 || layer0 + in->n_layers > L_bank)
        return fail(PRECOG_ERR_INVALID_ARG, "layers [layer0, layer0+n_layers) exceed L_bank");
    if (y_out == nullptr && state_out == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "y_out and state_out are both NULL: nothing to do");
    if (y_out && (!state_dtype_ok(y_dtype) || !aligned16(y_out)))
        return fail(PRECOG_ERR_INVALID_ARG, "y_out must be 16-byte aligned F32 or BF16");
    if (state_out && (!state_dtype_ok(state_dtype) || !aligned16(state_out)))
        return fail(PRECOG_ERR_INVALID_ARG, "state_out must be 16-byte aligned F32 or BF16");
    if (n_queries == 0) return ok();
    precog::ScanParams p = base_params(in, rows);
    p.n_chunks = n_queries;
    p.use_fixed = 1;
    p.fixed_len = T_q;
    p.bank = bank;
    p.bank_dtype = bank_dtype;
    p.bank_entries = bank_entries;
    p.idx = d_idx;
    p.topk = k;
    p.topk_scores = d_score;
    p.inv_temp = 1.f / temperature;
    p.L_bank = L_bank;
    p.states = state_out;
    p.state_dtype = state_dtype;
    p.L_out = L_bank;
    p.layer0 = layer0;
    p.y = y_out;
    p.y_dtype = y_dtype;
    cudaError_t e = precog::launch_scan(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "composed prefill launch");
    return ok();
}

size_t precog_retrieve_topk_workspace_size(int64_t M, int32_t dim, int32_t n_queries) {
    if (M < 0 || dim < 1 || n_queries < 0) return 0;
    return precog::retrieve_topk_workspace_size(M, dim, n_queries);
}

precog_status precog_retrieve_topk(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                                   const void *queries, int32_t n_queries, int32_t k,
                                   int64_t *d_idx, float *d_score, void *workspace,
                                   size_t workspace_bytes, void *stream) {
    if (k < 1 || k > 8) return fail(PRECOG_ERR_UNSUPPORTED, "k must be in [1, 8]");
    const int sz = dtype_size(index_dtype);
    if (sz == 0) return fail(PRECOG_ERR_UNSUPPORTED, "index_dtype must be F16, BF16 or F32");
    if (M < 0) return fail(PRECOG_ERR_INVALID_ARG, "M must be >= 0");
    if (M >= 0x7fffffffLL) return fail(PRECOG_ERR_UNSUPPORTED, "M must be below 2^31-1");
    if (dim < 1) return fail(PRECOG_ERR_INVALID_ARG, "dim must be >= 1");
    if ((static_cast<int64_t>(dim) * sz) % 16 != 0)
        return fail(PRECOG_ERR_UNSUPPORTED, "dim*sizeof(dtype) must be a multiple of 16");
    if (static_cast<int64_t>(dim) * sz > 8192)
        return fail(PRECOG_ERR_UNSUPPORTED, "rows longer than 8 KiB (dim*sizeof(dtype)) are not implemented");
    if (n_queries < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries must be >= 0");
    if (n_queries == 0) return ok();
    if ((M > 0 && index == nullptr) || queries == nullptr || d_idx == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "index, queries and d_idx must be non-NULL");
    if ((index && !aligned16(index)) || !aligned16(queries))
        return fail(PRECOG_ERR_INVALID_ARG, "index and queries must be 16-byte aligned");
    const size_t need = precog::retrieve_topk_workspace_size(M, dim, n_queries);
    if (workspace_bytes < need || (need > 0 && (workspace == nullptr || !aligned16(workspace))))
        return fail(PRECOG_ERR_INVALID_ARG, "workspace too small or misaligned (%zu bytes needed)", need);
    precog::RetrieveParams p;
    p.index = index;
    p.dtype = index_dtype;
    p.M = M;
    p.dim = dim;
    p.queries = queries;
    p.n_queries = n_queries;
    p.best_idx = d_idx;
    p.best_score = d_score;
    p.workspace = workspace;
    p.workspace_bytes = workspace_bytes;
    cudaError_t e = precog::launch_retrieve_topk(p, k, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "top-k retrieve launch");
    return ok();
}

size_t precog_retrieve_workspace_size(int64_t M, int32_t dim, int32_t n_queries) {
    if (M < 0 || dim < 1 || n_queries < 0) return 0;
    return precog::retrieve_workspace_size(M, dim, n_queries);
}

precog_status precog_retrieve(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                              const void *queries, int32_t n_queries, int64_t *d_best_idx,
                              float *d_best_score, void *workspace, size_t workspace_bytes,
                              void *stream) {
    const int sz = dtype_size(index_dtype);
    if (sz == 0) return fail(PRECOG_ERR_UNSUPPORTED, "index_dtype must be F16, BF16 or F32");
    if (M < 0) return fail(PRECOG_ERR_INVALID_ARG, "M must be >= 0");
    if (M >= 0x7fffffffLL) return fail(PRECOG_ERR_UNSUPPORTED, "M must be below 2^31-1");
    if (dim < 1) return fail(PRECOG_ERR_INVALID_ARG, "dim must be >= 1");
    if ((static_cast<int64_t>(dim) * sz) % 16 != 0)
        return fail(PRECOG_ERR_UNSUPPORTED, "dim*sizeof(dtype) must be a multiple of 16");
    if (static_cast<int64_t>(dim) * sz > 8192)
        return fail(PRECOG_ERR_UNSUPPORTED, "rows longer than 8 KiB (dim*sizeof(dtype)) are not implemented");
    if (n_queries < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries must be >= 0");
    if (n_queries == 0) return ok();
    if ((M > 0 && index == nullptr) || queries == nullptr || d_best_idx == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "index, queries and d_best_idx must be non-NULL");
    if ((index && !aligned16(index)) || !aligned16(queries))
        return fail(PRECOG_ERR_INVALID_ARG, "index and queries must be 16-byte aligned");
    const size_t need = precog::retrieve_workspace_size(M, dim, n_queries);
    if (workspace_bytes < need || (need > 0 && (workspace == nullptr || !aligned16(workspace))))
        return fail(PRECOG_ERR_INVALID_ARG, "workspace too small or misaligned (%zu bytes needed)", need);
    precog::RetrieveParams p;
    p.index = index;
    p.dtype = index_dtype;
    p.M = M;
    p.dim = dim;
    p.queries = queries;
    p.n_queries = n_queries;
    p.best_idx = d_best_idx;
    p.best_score = d_best_score;
    p.workspace = workspace;
    p.workspace_bytes = workspace_bytes;
    cudaError_t e = precog::launch_retrieve(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "retrieve launch");
    return ok();
}

precog_status precog_retrieve_keys(const void *index, int32_t index_dtype, int64_t M, int32_t dim,
                                   const void *queries, int32_t n_queries, int64_t row_offset,
                                   int64_t *d_keys, void *workspace, size_t workspace_bytes,
                                   void *stream) {
    const int sz = dtype_size(index_dtype);
    if (sz == 0) return fail(PRECOG_ERR_UNSUPPORTED, "index_dtype must be F16, BF16 or F32");
    if (M < 0) return fail(PRECOG_ERR_INVALID_ARG, "M must be >= 0");
    if (M >= 0x7fffffffLL) return fail(PRECOG_ERR_UNSUPPORTED, "M must be below 2^31-1");
    if (row_offset < 0 || row_offset + M > 0xffffffffLL)
        return fail(PRECOG_ERR_INVALID_ARG, "need row_offset >= 0 and row_offset + M <= 2^32 - 1");
    if (dim < 1) return fail(PRECOG_ERR_INVALID_ARG, "dim must be >= 1");
    if ((static_cast<int64_t>(dim) * sz) % 16 != 0)
        return fail(PRECOG_ERR_UNSUPPORTED, "dim*sizeof(dtype) must be a multiple of 16");
    if (static_cast<int64_t>(dim) * sz > 8192)
        return fail(PRECOG_ERR_UNSUPPORTED, "rows longer than 8 KiB (dim*sizeof(dtype)) are not implemented");
    if (n_queries < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries must be >= 0");
    if (n_queries == 0) return ok();
    if ((M > 0 && index == nullptr) || queries == nullptr || d_keys == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "index, queries and d_keys must be non-NULL");
    if ((index && !aligned16(index)) || !aligned16(queries))
        return fail(PRECOG_ERR_INVALID_ARG, "index and queries must be 16-byte aligned");
    const size_t need = precog::retrieve_workspace_size(M, dim, n_queries);
    if (workspace_bytes < need || (need > 0 && (workspace == nullptr || !aligned16(workspace))))
        return fail(PRECOG_ERR_INVALID_ARG, "workspace too small or misaligned (%zu bytes needed)", need);
    precog::RetrieveParams p;
    p.index = index;
    p.dtype = index_dtype;
    p.M = M;
    p.dim = dim;
    p.queries = queries;
    p.n_queries = n_queries;
    p.best_idx = nullptr;
    p.best_score = nullptr;
    p.workspace = workspace;
    p.workspace_bytes = workspace_bytes;
    p.row_offset = row_offset;
    p.keys_out = d_keys;
    cudaError_t e = precog::launch_retrieve(p, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "retrieve launch");
    return ok();
}

precog_status precog_decode_keys(const int64_t *d_keys, int32_t n_queries, int64_t *d_best_idx,
                                 float *d_best_score, void *stream) {
    if (n_queries < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries must be >= 0");
    if (n_queries == 0) return ok();
    if (d_keys == nullptr || d_best_idx == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "d_keys and d_best_idx must be non-NULL");
    cudaError_t e = precog::launch_decode_keys(d_keys, n_queries, d_best_idx, d_best_score,
                                               static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "decode launch");
    return ok();
}

precog_status precog_smc_route(const void *embeddings, int32_t dtype, int64_t n, int32_t dim,
                               const void *domain_protos, int32_t M, const void *sub_protos,
                               int32_t J_max, const int32_t *d_J, int32_t *d_domain, int32_t *d_sub,
                               int64_t *d_slot, void *stream) {
    if (dtype_size(dtype) == 0) return fail(PRECOG_ERR_UNSUPPORTED, "dtype must be F16, BF16 or F32");
    if (n < 0 || dim < 1 || M < 0 || J_max < 0)
        return fail(PRECOG_ERR_INVALID_ARG, "n, M, J_max must be >= 0 and dim >= 1");
    if (n == 0) return ok();
    if (n > 0x7fffffffLL * 8) return fail(PRECOG_ERR_UNSUPPORTED, "too many embeddings");
    if (embeddings == nullptr || d_domain == nullptr || d_sub == nullptr ||
        (M > 0 && (domain_protos == nullptr || d_J == nullptr)) ||
        (M > 0 && J_max > 0 && sub_protos == nullptr))
        return fail(PRECOG_ERR_INVALID_ARG, "a required pointer is NULL");
    cudaError_t e = precog::launch_smc_route(embeddings, dtype, n, dim, domain_protos, M, sub_protos,
                                             J_max, d_J, d_domain, d_sub, d_slot,
                                             static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "smc route launch");
    return ok();
}

precog_status precog_smc_consolidate(float *semantic, int64_t n_slots, int64_t state_elems,
                                     const void *states, int32_t states_dtype, const int64_t *d_slots,
                                     int64_t n, float alpha, void *stream) {
    if (!state_dtype_ok(states_dtype)) return fail(PRECOG_ERR_UNSUPPORTED, "states_dtype must be F32 or BF16");
    if (n_slots < 0 || state_elems < 0 || n < 0)
        return fail(PRECOG_ERR_INVALID_ARG, "sizes must be >= 0");
    if (!(alpha > 0.f && alpha <= 1.f)) return fail(PRECOG_ERR_INVALID_ARG, "alpha must be in (0, 1]");
    if (n == 0 || state_elems == 0) return ok();
    if (semantic == nullptr || states == nullptr || d_slots == nullptr)
        return fail(PRECOG_ERR_INVALID_ARG, "semantic, states and d_slots must be non-NULL");
    if (!aligned16(semantic) || !aligned16(states))
        return fail(PRECOG_ERR_INVALID_ARG, "semantic and states must be 16-byte aligned");
    cudaError_t e = precog::launch_smc_consolidate(semantic, n_slots, state_elems, states, states_dtype,
                                                   d_slots, n, alpha, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "smc consolidate launch");
    return ok();
}

precog_status precog_selftest_wait_timeout(uint32_t iterations, void *stream) {
    if (iterations < 1 || iterations > (1u << 20))
        return fail(PRECOG_ERR_INVALID_ARG, "iterations must be in [1, 2^20]");
    cudaError_t e = precog::launch_wait_timeout(iterations, static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "self-test launch");
    return ok();
}

precog_status precog_device_status(void *stream, uint32_t *bits_out) {
    if (bits_out == nullptr) return fail(PRECOG_ERR_INVALID_ARG, "bits_out is NULL");
    *bits_out = 0;
    cudaError_t e = cudaStreamSynchronize(static_cast<cudaStream_t>(stream));
    if (e != cudaSuccess) return cuda_fail(e, "stream synchronize");
    uint32_t a = 0, b = 0;
    e = precog::scan_status_word_read_clear(&a);
    if (e != cudaSuccess) return cuda_fail(e, "read scan status");
    e = precog::retrieve_status_word_read_clear(&b);
    if (e != cudaSuccess) return cuda_fail(e, "read retrieve status");
    uint32_t c = 0, z = 0;
    e = precog::smc_status_word_read_clear(&c);
    if (e != cudaSuccess) return cuda_fail(e, "read smc status");
    e = precog::scan_complex_status_word_read_clear(&z);
    if (e != cudaSuccess) return cuda_fail(e, "read complex scan status");
    uint32_t w = 0;
    e = precog::selftest_status_word_read_clear(&w);
    if (e != cudaSuccess) return cuda_fail(e, "read self-test status");
    uint32_t l = 0;
    e = precog::scan_latency_status_word_read_clear(&l);
    if (e != cudaSuccess) return cuda_fail(e, "read latency scan status");
    *bits_out = a | b | c | z | w | l;
    if (*bits_out == 0) return ok();
    if (*bits_out & PRECOG_DEV_TIMEOUT)
        return fail(PRECOG_ERR_TIMEOUT, "a device-side wait gave up (bits 0x%x)", *bits_out);
    return fail(PRECOG_ERR_DEVICE, "device flagged invalid offsets, bank rows or A (bits 0x%x)", *bits_out);
}

const char *precog_status_string(int32_t status) {
    switch (status) {
        case PRECOG_OK: return "PRECOG_OK";
        case PRECOG_ERR_INVALID_ARG: return "PRECOG_ERR_INVALID_ARG";
        case PRECOG_ERR_UNSUPPORTED: return "PRECOG_ERR_UNSUPPORTED";
        case PRECOG_ERR_CUDA: return "PRECOG_ERR_CUDA";
        case PRECOG_ERR_TIMEOUT: return "PRECOG_ERR_TIMEOUT";
        case PRECOG_ERR_DEVICE: return "PRECOG_ERR_DEVICE";
        default: return "PRECOG_UNKNOWN_STATUS";
    }
}

const char *precog_last_error(void) { return g_last_error; }

int32_t precog_abi_version(void) { return PRECOG_ABI_VERSION; }

uint64_t precog_launch_count(void) { return g_launches.load(std::memory_order_relaxed); }

}  // extern "C"

// ---------------------------------------------------------------------------
// Retrieval without a caller workspace.
//
// Some callers cannot allocate device memory at the moment they retrieve: a
// real-time serving loop that must not call cudaMalloc (it can synchronise the
// device and stall every stream), code running inside a memory pool owned by
// someone else, or a host whose allocator is not the CUDA one. For them the
// partial (score, row) keys of precog_retrieve live in a fixed array compiled
// into this library instead of a workspace they would have to provide.
namespace {

// 262,144 packed keys = 2 MiB, held on every GPU that loads this library until
// the process exits. Enough for about 430 queries per call at any index size on
// a 152-SM GPU (keys needed = scratch partitions x n_queries).
constexpr size_t kNoallocKeys = 262144;
static __device__ __align__(256) unsigned long long g_noalloc_scratch[kNoallocKeys];

// The array's device address belongs to one CUDA context: after cudaDeviceReset, or
// when a caller makes another context of the same device current, it is another
// address. So the address is looked up once per context (keyed by the driver's unique
// context id), not once per device number.
using CtxGetCurrentFn = CUresult (*)(CUcontext *);
using CtxGetIdFn = CUresult (*)(CUcontext, unsigned long long *);

template <typename F>
F driver_fn(const char *name) {
    void *p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion(name, &p, 12000, cudaEnableDefault, &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
        return reinterpret_cast<F>(p);
    return nullptr;
}

// Unique id of the calling thread's current context; false if there is none yet or the
// driver cannot tell.
bool current_context_id(unsigned long long *id) {
    static const CtxGetCurrentFn get_current = driver_fn<CtxGetCurrentFn>("cuCtxGetCurrent");
    static const CtxGetIdFn get_id = driver_fn<CtxGetIdFn>("cuCtxGetId");
    if (get_current == nullptr || get_id == nullptr) return false;
    CUcontext ctx = nullptr;
    if (get_current(&ctx) != CUDA_SUCCESS || ctx == nullptr) return false;
    return get_id(ctx, id) == CUDA_SUCCESS;
}

struct NoallocSlot {
    unsigned long long ctx_id;
    void *ptr;
};
constexpr int kNoallocSlots = 64;
std::mutex g_noalloc_mutex;
NoallocSlot g_noalloc_slots[kNoallocSlots];
int g_noalloc_filled = 0, g_noalloc_next = 0;

// Device address of the scratch in the current context. The first call in a context
// asks the runtime (cudaGetSymbolAddress, a host-side lookup that allocates nothing);
// later calls in that context reuse the answer. Without context ids every call asks.
precog_status noalloc_scratch(void **ptr) {
    unsigned long long id = 0;
    bool have_id = current_context_id(&id);
    if (have_id) {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        for (int i = 0; i < g_noalloc_filled; ++i)
            if (g_noalloc_slots[i].ctx_id == id) {
                *ptr = g_noalloc_slots[i].ptr;
                return PRECOG_OK;
            }
    }
    void *p = nullptr;
    const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
    if (e != cudaSuccess) return cuda_fail(e, "cudaGetSymbolAddress(scratch)");
    if (!have_id) have_id = current_context_id(&id);   // the lookup may have created the context
    if (have_id) {
        std::lock_guard<std::mutex> lock(g_noalloc_mutex);
        g_noalloc_slots[g_noalloc_next] = NoallocSlot{id, p};
        g_noalloc_next = (g_noalloc_next + 1) % kNoallocSlots;
        if (g_noalloc_filled < kNoallocSlots) ++g_noalloc_filled;
    }
    *ptr = p;
    return PRECOG_OK;
}

}  // namespace

extern "C" {

precog_status precog_retrieve_noalloc(const void *index, int32_t index_dtype, int64_t M,
                                      int32_t dim, const void *queries, int32_t n_queries,
                                      int64_t *d_best_idx, float *d_best_score, void *stream) {
    if (n_queries < 0) return fail(PRECOG_ERR_INVALID_ARG, "n_queries must be >= 0");
    if (M < 0 || dim < 1) return fail(PRECOG_ERR_INVALID_ARG, "M must be >= 0 and dim >= 1");
    const size_t need = precog::retrieve_workspace_size(M, dim, n_queries);
    if (need > sizeof(g_noalloc_scratch))
        return fail(PRECOG_ERR_UNSUPPORTED,
                    "precog_retrieve_noalloc: %d queries need %zu bytes of scratch, more than the "
                    "fixed %zu; use fewer queries per call or precog_retrieve with a workspace",
                    n_queries, need, sizeof(g_noalloc_scratch));
    void *scratch = nullptr;
    precog_status s = noalloc_scratch(&scratch);
    if (s != PRECOG_OK) return s;
    return precog_retrieve(index, index_dtype, M, dim, queries, n_queries, d_best_idx,
                           d_best_score, scratch, sizeof(g_noalloc_scratch), stream);
}

}  // extern "C"
