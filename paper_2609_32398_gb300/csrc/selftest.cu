// do_selftest_wait_limit (declared in include/doloss.h): exercises the
// failure path that every device wait of the library shares.  One thread waits
// on an mbarrier that nothing ever completes; the bounded wait gives up after
// kWaitLimitNs, records kDevTimeout in the workspace status word and returns,
// so the host sees DO_ERR_TIMEOUT from do_device_status and the context stays
// usable.  No trap, no fault, no unbounded loop.
#include <cuda_runtime.h>

#include "dol_internal.cuh"
#include "doloss.h"
#include "tma.cuh"

namespace {

__global__ void wait_limit_kernel(int *status) {
    __shared__ __align__(8) uint64_t bar;
    if (threadIdx.x == 0) {
        dol::mbar_init(&bar, 1);
        dol::fence_barrier_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) dol::mbar_wait(&bar, 0u, status);  // nothing arrives
}

}  // namespace

extern "C" do_status do_selftest_wait_limit(void *workspace, void *stream) {
    if (!workspace || reinterpret_cast<uintptr_t>(workspace) % 256 != 0) return DO_ERR_WORKSPACE;
    wait_limit_kernel<<<1, 32, 0, static_cast<cudaStream_t>(stream)>>>(static_cast<int *>(workspace));
    return cudaGetLastError() == cudaSuccess ? DO_OK : DO_ERR_CUDA;
}
