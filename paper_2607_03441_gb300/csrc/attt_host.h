// attt_host.h -- host-side helpers shared by the translation units of libattt.
#pragma once

#include <cuda.h>
#include <cuda_runtime.h>
#include <nvtx3/nvToolsExt.h>
#include <stddef.h>
#include <stdint.h>

#include "attt.h"

namespace attt {

// Current device if it is a GB300-class part (compute capability 10.3), else
// ATTT_ERR_UNSUPPORTED / ATTT_ERR_CUDA.
attt_status current_device(int *dev);

// Number of SMs of a device (cached).
int num_sms(int dev);

// Per-device status word used by the contraction kernels (lazily allocated).
int *device_status_word(int dev);

// Encodes a 2-D bf16 tensor map with zero fill for out-of-range elements and
// a shared-memory swizzle of `swizzle_bytes` (128, 64, or 0 for none).
// `inner` is the contiguous extent, `outer` the number of rows, `row_bytes`
// the row pitch.  Returns false if the driver rejects it.
bool make_tmap_bf16(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer,
                    uint64_t row_bytes, uint32_t box_inner, uint32_t box_outer, int swizzle_bytes = 128);

// The same for a 2-D fp32 tensor (128-byte swizzle).
bool make_tmap_f32(CUtensorMap *map, const void *base, uint64_t inner, uint64_t outer, uint64_t row_bytes,
                   uint32_t box_inner, uint32_t box_outer);

// Counts one kernel launch (attt_kernel_launches).
void count_launch();

// Host fault injection (attt_fault_inject, or the ATTT_FAULT environment
// variable read at first use): one pending fault, taken by the first site of
// its kind that asks.
enum FaultSite : int { FAULT_NONE = 0, FAULT_ALLOC = 1, FAULT_TABLE_FULL = 2 };
bool fault_take(FaultSite site);

// Raises the dynamic shared memory limit of `func` once per device.
bool set_smem_limit(const void *func, size_t bytes, int dev);

// Body of attt_lora_grad.  `status` is the device word for timed-out waits
// (nullptr: the per-device status word).
attt_status lora_grad_run(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj, const attt_bf16 *const *d_dy,
                          const int64_t *dout, const attt_bf16 *const *d_A, const attt_bf16 *const *d_B, int r,
                          float scale, float *const *d_dA, float *const *d_dB, void *d_ws, size_t ws_bytes,
                          int *status, cudaStream_t stream);

// Batched n-gram work over E histories (ngram.cu): rows [off[e], off[e+1])
// of d_tokens are episode e's update (off: host array of E + 1 offsets).
attt_status ngram_weights_batch(attt_history *const *hs, int E, const int32_t *d_tokens, const int64_t *off,
                                float w_min, float *d_w, float *d_rowscale, cudaStream_t stream);
attt_status history_insert_batch(attt_history *const *hs, int E, const int32_t *d_tokens, const int64_t *off,
                                 cudaStream_t stream);

// Eq. 10 as attt_weighted_ce_fwd_bwd, with per-row normalisers `row_scale`
// (dh_j = w_j row_scale_j (...); nullptr: 1/L for every row) and the per-row
// NLL lse_j - z_{j,t_j} into `nll` (nullptr: not written) (ce.cu).
attt_status ce_fwd_bwd_run(const attt_bf16 *d_h, const attt_bf16 *d_W, const int32_t *d_tgt, const float *d_w,
                           const float *row_scale, int64_t L, int64_t d, int64_t V, float *d_loss, float *d_dh,
                           float *d_lse, float *d_nll, void *d_ws, size_t ws_bytes, cudaStream_t stream);

// The largest Eq. 10 workspace over every row count up to Lmax (ce.cu).
size_t ce_workspace_bound(int64_t Lmax, int64_t d, int64_t V);

// The adapted projections of E episodes of a batch (lora.cu): episode e owns
// rows [off[e], off[e+1]) of the stacked x [*, din] and dy [*, d] (off: host
// array of E + 1) and slot e of the stacked adapters A16 [E][din][r], B16
// [E][r][d] and gradients dA [E][din][r], dB [E][r][d] (slots of episodes
// without rows are left as they are).  rows_bound >= sum_e round_up(L_e, 8)
// sizes the workspace.  batch_adapter_prep (the current adapters) comes first;
// forward (h bf16 [R, d]), grads and input_grad (dx fp32 [R, din]) then read
// what it wrote.
size_t batch_adapter_workspace(int E, int64_t rows_bound, int64_t din, int64_t d, int r);
attt_status batch_adapter_prep(const attt_bf16 *d_A16, const attt_bf16 *d_B16, int E, int64_t din, int64_t d, int r,
                               int64_t rows_bound, void *d_ws, size_t ws_bytes, cudaStream_t stream);
attt_status batch_forward(const attt_bf16 *d_x, const int64_t *off, int E, const attt_bf16 *d_W0, int64_t din,
                          int64_t d, int r, float scale, attt_bf16 *d_h, int64_t rows_bound, void *d_ws,
                          size_t ws_bytes, cudaStream_t stream);
attt_status batch_grads(const attt_bf16 *d_x, const attt_bf16 *d_dy, const int64_t *off, int E, int64_t din,
                        int64_t d, int r, float scale, float *d_dA, float *d_dB, int64_t rows_bound, void *d_ws,
                        size_t ws_bytes, cudaStream_t stream);
attt_status batch_input_grad(const attt_bf16 *d_dy, const int64_t *off, int E, const attt_bf16 *d_W0, int64_t din,
                             int64_t d, int r, float scale, float *d_dx, int64_t rows_bound, void *d_ws,
                             size_t ws_bytes, cudaStream_t stream);

// Device address of attt_lora_grad_noalloc's static status word on `dev`, or
// nullptr if that entry point has not been set up on the device.
int *noalloc_status_word(int dev);

// A named NVTX range over one C-ABI call, so that a timeline shows which
// call each kernel belongs to (nearly free when no tool is attached).
struct NvtxRange {
    explicit NvtxRange(const char *name) { nvtxRangePushA(name); }
    ~NvtxRange() { nvtxRangePop(); }
    NvtxRange(const NvtxRange &) = delete;
    NvtxRange &operator=(const NvtxRange &) = delete;
};
#define ATTT_NVTX_RANGE() ::attt::NvtxRange attt_nvtx_range_(__func__)

inline bool aligned16(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 15u) == 0; }
inline bool aligned256(const void *p) { return (reinterpret_cast<uintptr_t>(p) & 255u) == 0; }
inline int64_t cdiv(int64_t a, int64_t b) { return (a + b - 1) / b; }
inline int64_t round_up(int64_t a, int64_t b) { return cdiv(a, b) * b; }

// Workspace carving: bump allocator over a caller-provided buffer, 256-byte
// aligned pieces.
struct Carve {
    char *base;
    size_t used;
    template <class T>
    T *take(size_t count) {
        used = (size_t)round_up((int64_t)used, 256);
        T *p = reinterpret_cast<T *>(base ? base + used : nullptr);
        used += count * sizeof(T);
        return p;
    }
};

}  // namespace attt
