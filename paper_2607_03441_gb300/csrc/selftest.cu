// selftest.cu -- the failure path every device-side wait of the library
// shares, exercised without a fault: a wait on an mbarrier that nothing will
// complete runs out after the wall-clock limit, records ATTT_ERR_TIMEOUT in
// the per-device status word and returns, and the context stays usable.
#include <cuda_runtime.h>

#include "attt_common.cuh"
#include "attt_host.h"

namespace {

// One mbarrier expecting one arrival that never comes; thread 0 waits on its
// first phase through mbar_wait (the bounded wait of every kernel here).
__global__ void wait_selftest_kernel(int *status) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    if (threadIdx.x == 0) {
        attt::mbar_init(attt::smem_u32(&bar), 1);
        abort_flag = 0;
        attt::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0 && !attt::mbar_wait(attt::smem_u32(&bar), 0u, &abort_flag))
        attt::record_error(status, ATTT_ERR_TIMEOUT);
}

}  // namespace

extern "C" attt_status attt_selftest_wait_timeout(attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    int *status = device_status_word(dev);
    if (!status) return ATTT_ERR_CUDA;
    wait_selftest_kernel<<<1, 32, 0, stream>>>(status);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}
