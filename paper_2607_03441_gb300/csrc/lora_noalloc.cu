// lora_noalloc.cu -- attt_lora_grad_noalloc: the LoRA adapter gradients for
// callers that must not allocate device memory.
//
// Some callers cannot call cudaMalloc: a serving process whose device memory
// is all reserved up front by its own pool (a cudaMalloc there fails or
// fragments the pool), a latency-critical loop that forbids allocator calls
// because cudaMalloc/cudaFree can synchronise the device and stall other
// streams, or a plugin whose host application owns every device allocation.
// For them this entry point runs exactly the same kernels as attt_lora_grad,
// but its scratch is a fixed-size array in the library's own device memory
// (a file-scope static __device__ array) instead of a caller workspace.  The
// caller still passes every input and output buffer.
//
// Set-up: the first call on a device, with that device current, looks up the
// array's device address with cudaGetSymbolAddress (in host code the array's
// name is only a host-side stand-in, never a device address) and caches it.
// The same is done for a static status word that records a timed-out device
// wait of this entry point's kernels; attt_device_status() reports it.  The
// cached addresses hold for the life of the device's context: a call after
// cudaDeviceReset() (which re-creates the module's static arrays) is not
// supported.
#include <mutex>

#include "attt_host.h"

namespace attt {

namespace {

constexpr size_t kScratchBytes = ATTT_LORA_NOALLOC_SCRATCH_BYTES;
constexpr int kMaxDevices = 64;

// Held by every GPU that loads this library, until the process exits.
static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];
static __device__ __align__(256) int g_status[64];

std::mutex g_mu;
void *g_scratch_addr[kMaxDevices];
int *g_status_addr[kMaxDevices];

// Device addresses of the static scratch and status word on device `dev`
// (which must be current).  Looked up once per device.
attt_status setup(int dev, void **scratch, int **status) {
    if (dev < 0 || dev >= kMaxDevices) return ATTT_ERR_UNSUPPORTED;
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_scratch_addr[dev]) {
        void *s = nullptr, *w = nullptr;
        if (cudaGetSymbolAddress(&s, g_scratch) != cudaSuccess) return ATTT_ERR_CUDA;
        if (cudaGetSymbolAddress(&w, g_status) != cudaSuccess) return ATTT_ERR_CUDA;
        g_scratch_addr[dev] = s;
        g_status_addr[dev] = static_cast<int *>(w);
    }
    *scratch = g_scratch_addr[dev];
    *status = g_status_addr[dev];
    return ATTT_OK;
}

}  // namespace

int *noalloc_status_word(int dev) {
    if (dev < 0 || dev >= kMaxDevices) return nullptr;
    std::lock_guard<std::mutex> lk(g_mu);
    return g_status_addr[dev];
}

}  // namespace attt

extern "C" attt_status attt_lora_grad_noalloc(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj,
                                              const attt_bf16 *const *d_dy, const int64_t *dout,
                                              const attt_bf16 *const *d_A, const attt_bf16 *const *d_B, int r,
                                              float scale, float *const *d_dA, float *const *d_dB,
                                              attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    // 0 for an invalid shape (nproj, r, sizes or a null dout array)
    const size_t need = attt_lora_workspace_bytes(L, din, nproj, dout, r);
    if (need == 0) return ATTT_ERR_INVALID_ARG;
    if (need > kScratchBytes) return ATTT_ERR_WORKSPACE;  // larger than the static scratch
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    void *scratch = nullptr;
    int *status = nullptr;
    st = setup(dev, &scratch, &status);
    if (st != ATTT_OK) return st;
    // lora_grad_run zeroes the parts of the scratch that accumulate, so the
    // previous call's contents never leak into this one.
    return lora_grad_run(d_x, L, din, nproj, d_dy, dout, d_A, d_B, r, scale, d_dA, d_dB, scratch, kScratchBytes,
                         status, stream);
}
