// selftest.cu -- the failure path every device-side wait of the library
// shares, exercised without a fault: a wait on an mbarrier that nothing will
// complete, and a wait on a global counter that no CTA will raise (the kind
// the LoRA gradient launch uses between its passes), each run out after the
// wall-clock limit and return; the kernel then records ATTT_ERR_TIMEOUT in
// the per-device status word, and the context stays usable.
#include <cuda_runtime.h>

#include "attt_common.cuh"
#include "attt_host.h"

namespace {

// A global counter that nothing writes (zero from module load).
__device__ unsigned int g_never_raised;

// Warp 0 waits on the first phase of an mbarrier expecting one arrival that
// never comes (mbar_wait); warp 1 waits for the counter above to reach 1
// (wait_counter_geq).  ATTT_ERR_TIMEOUT is recorded only if both waits ran
// out and returned.
__global__ void wait_selftest_kernel(int *status) {
    __shared__ __align__(8) uint64_t bar;
    __shared__ int abort_flag;
    __shared__ int timed_out[2];
    if (threadIdx.x == 0) {
        attt::mbar_init(attt::smem_u32(&bar), 1);
        abort_flag = 0;
        timed_out[0] = timed_out[1] = 0;
        attt::fence_mbar_init();
    }
    __syncthreads();
    if (threadIdx.x == 0) timed_out[0] = attt::mbar_wait(attt::smem_u32(&bar), 0u, &abort_flag) ? 0 : 1;
    if (threadIdx.x == 32) timed_out[1] = attt::wait_counter_geq(&g_never_raised, 1u, &abort_flag) ? 0 : 1;
    __syncthreads();
    if (threadIdx.x == 0 && timed_out[0] && timed_out[1]) attt::record_error(status, ATTT_ERR_TIMEOUT);
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
    wait_selftest_kernel<<<1, 64, 0, stream>>>(status);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}
