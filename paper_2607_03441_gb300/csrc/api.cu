// api.cu -- library-wide host plumbing of libattt: status codes, the device
// check, the per-device status word, tensor-map encoding and the dynamic
// shared-memory opt-in.
#include <cudaTypedefs.h>

#include <atomic>
#include <cstdlib>
#include <cstring>
#include <map>
#include <mutex>
#include <utility>

#include "attt_host.h"

namespace attt {

namespace {

std::mutex g_mu;
std::map<int, int> g_sms;
std::map<int, int *> g_status_words;
std::map<std::pair<const void *, int>, size_t> g_smem_set;
PFN_cuTensorMapEncodeTiled_v12000 g_encode = nullptr;
std::atomic<unsigned long long> g_launches{0};
// The pending injected fault (FaultSite), or -1 before ATTT_FAULT was read.
std::atomic<int> g_fault{-1};

int fault_site(const char *s) {
    if (!s || !*s || strcmp(s, "none") == 0) return FAULT_NONE;
    if (strcmp(s, "alloc") == 0) return FAULT_ALLOC;
    if (strcmp(s, "table_full") == 0) return FAULT_TABLE_FULL;
    return -1;
}

int pending_fault() {
    int f = g_fault.load();
    if (f < 0) {  // first use: the environment's fault, if any
        int env = fault_site(std::getenv("ATTT_FAULT"));
        if (env < 0) env = FAULT_NONE;
        g_fault.compare_exchange_strong(f, env);
        f = g_fault.load();
    }
    return f;
}

PFN_cuTensorMapEncodeTiled_v12000 encode_fn() {
    std::lock_guard<std::mutex> lk(g_mu);
    if (!g_encode) {
        void *fn = nullptr;
        cudaDriverEntryPointQueryResult q;
        if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &fn, 12000, cudaEnableDefault, &q) ==
                cudaSuccess &&
            q == cudaDriverEntryPointSuccess)
            g_encode = reinterpret_cast<PFN_cuTensorMapEncodeTiled_v12000>(fn);
    }
    return g_encode;
}

}  // namespace

void count_launch() { g_launches.fetch_add(1, std::memory_order_relaxed); }

bool fault_take(FaultSite site) {
    int expected = pending_fault();
    return expected == site && g_fault.compare_exchange_strong(expected, FAULT_NONE);
}

attt_status current_device(int *dev) {
    if (cudaGetDevice(dev) != cudaSuccess) return ATTT_ERR_CUDA;
    int major = 0, minor = 0;
    if (cudaDeviceGetAttribute(&major, cudaDevAttrComputeCapabilityMajor, *dev) != cudaSuccess ||
        cudaDeviceGetAttribute(&minor, cudaDevAttrComputeCapabilityMinor, *dev) != cudaSuccess)
        return ATTT_ERR_CUDA;
    // The kernels are compiled for sm_103a only.
    if (major != 10 || minor != 3) return ATTT_ERR_UNSUPPORTED;
    return ATTT_OK;
}

int num_sms(int dev) {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_sms.find(dev);
    if (it != g_sms.end()) return it->second;
    int n = 0;
    cudaDeviceGetAttribute(&n, cudaDevAttrMultiProcessorCount, dev);
    if (n <= 0) n = 1;
    g_sms[dev] = n;
    return n;
}

int *device_status_word(int dev) {
    std::lock_guard<std::mutex> lk(g_mu);
    auto it = g_status_words.find(dev);
    if (it != g_status_words.end()) return it->second;
    int *p = nullptr;
    if (cudaMalloc(&p, 256) != cudaSuccess) return nullptr;
    if (cudaMemset(p, 0, 256) != cudaSuccess) return nullptr;
    g_status_words[dev] = p;
    return p;
}

bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                    uint32_t box_inner, uint32_t box_outer, int swizzle_bytes) {
    auto fn = encode_fn();
    if (!fn) return false;
    if (!aligned16(base) || row_bytes % 16 != 0 || inner == 0 || outer == 0) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    const CUtensorMapSwizzle sw = swizzle_bytes == 128  ? CU_TENSOR_MAP_SWIZZLE_128B
                                  : swizzle_bytes == 64 ? CU_TENSOR_MAP_SWIZZLE_64B
                                                        : CU_TENSOR_MAP_SWIZZLE_NONE;
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_BFLOAT16, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, sw, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool make_tmap_f32(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                   uint32_t box_inner, uint32_t box_outer) {
    auto fn = encode_fn();
    if (!fn) return false;
    if (!aligned16(base) || row_bytes % 16 != 0 || inner == 0 || outer == 0) return false;
    cuuint64_t dims[2] = {inner, outer};
    cuuint64_t strides[1] = {row_bytes};
    cuuint32_t box[2] = {box_inner, box_outer};
    cuuint32_t estr[2] = {1, 1};
    CUresult r = fn(map, CU_TENSOR_MAP_DATA_TYPE_FLOAT32, 2, const_cast<void *>(base), dims, strides, box, estr,
                    CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B, CU_TENSOR_MAP_L2_PROMOTION_L2_256B,
                    CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    return r == CUDA_SUCCESS;
}

bool set_smem_limit(const void *func, size_t bytes, int dev) {
    std::lock_guard<std::mutex> lk(g_mu);
    auto key = std::make_pair(func, dev);
    auto it = g_smem_set.find(key);
    if (it != g_smem_set.end() && it->second >= bytes) return true;
    if (cudaFuncSetAttribute(func, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)bytes) != cudaSuccess)
        return false;
    g_smem_set[key] = bytes;
    return true;
}

}  // namespace attt

extern "C" {

const char *attt_status_string(int status) {
    switch (status) {
        case ATTT_OK: return "ATTT_OK";
        case ATTT_ERR_INVALID_ARG: return "ATTT_ERR_INVALID_ARG";
        case ATTT_ERR_TABLE_FULL: return "ATTT_ERR_TABLE_FULL";
        case ATTT_ERR_TOKEN_RANGE: return "ATTT_ERR_TOKEN_RANGE";
        case ATTT_ERR_TIMEOUT: return "ATTT_ERR_TIMEOUT";
        case ATTT_ERR_WORKSPACE: return "ATTT_ERR_WORKSPACE";
        case ATTT_ERR_CUDA: return "ATTT_ERR_CUDA";
        case ATTT_ERR_UNSUPPORTED: return "ATTT_ERR_UNSUPPORTED";
        case ATTT_ERR_CAPACITY: return "ATTT_ERR_CAPACITY";
        case ATTT_ERR_CHECK: return "ATTT_ERR_CHECK";
        default: return "ATTT_ERR_UNKNOWN";
    }
}

int attt_abi_version(void) { return 100; }

uint64_t attt_kernel_launches(void) { return attt::g_launches.load(std::memory_order_relaxed); }

attt_status attt_device_status(attt_stream stream) {
    int dev;
    attt_status st = attt::current_device(&dev);
    if (st != ATTT_OK) return st;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return ATTT_ERR_CUDA;
    // Both words are read and every one that holds an error is cleared, so a
    // single call drains them; the library-wide word's error is reported first.
    int *words[2] = {attt::device_status_word(dev), attt::noalloc_status_word(dev)};
    if (!words[0]) return ATTT_ERR_CUDA;
    int v = 0;
    for (int *w : words) {
        if (!w) continue;  // attt_lora_grad_noalloc has not been set up on this device
        int x = 0;
        if (cudaMemcpy(&x, w, sizeof x, cudaMemcpyDeviceToHost) != cudaSuccess) return ATTT_ERR_CUDA;
        if (x != 0 && cudaMemset(w, 0, sizeof x) != cudaSuccess) return ATTT_ERR_CUDA;
        if (v == 0) v = x;
    }
    return (attt_status)v;
}

}  // extern "C"

extern "C" attt_status attt_fault_inject(const char *site) {
    const int f = attt::fault_site(site);
    if (f < 0) return ATTT_ERR_INVALID_ARG;
    attt::pending_fault();  // the environment is read first, so this call wins
    attt::g_fault.store(f);
    return ATTT_OK;
}
