// Exercise of the failure path every pipelined kernel here relies on: an
// mbarrier wait that runs out of iterations records PRECOG_DEV_TIMEOUT in a
// device status word and returns, instead of trapping or spinning forever.
// The kernel waits on a barrier that nothing arrives on, so the wait always
// runs out; the host then reads the status with precog_device_status and the
// context stays usable. No fault, trap or unbounded wait is involved.
#include "../../include/precog.h"
#include "internal.h"
#include "ptx.cuh"

namespace precog {
namespace {

__device__ uint32_t g_selftest_status;

__global__ void wait_timeout_kernel(uint32_t limit) {
    __shared__ uint64_t bar;
    if (threadIdx.x == 0) {
        mbar_init(&bar, 1);   // expects one arrival that never comes
        fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) {
        bool done = false;
        for (uint32_t i = 0; i < limit && !done; ++i) done = mbar_try_wait(&bar, 0);
        if (!done) atomicOr(&g_selftest_status, PRECOG_DEV_TIMEOUT);
    }
}

}  // namespace

cudaError_t launch_wait_timeout(uint32_t limit, cudaStream_t stream) {
    wait_timeout_kernel<<<1, 32, 0, stream>>>(limit);
    cudaError_t e = cudaGetLastError();
    if (e == cudaSuccess) count_launches(1);
    return e;
}

cudaError_t selftest_status_word_read_clear(uint32_t *bits) {
    uint32_t zero = 0;
    cudaError_t e = cudaMemcpyFromSymbol(bits, g_selftest_status, sizeof(uint32_t));
    if (e != cudaSuccess) return e;
    return cudaMemcpyToSymbol(g_selftest_status, &zero, sizeof(uint32_t));
}

}  // namespace precog
