// batch.cu -- a batch of concurrent episodes (Sec. 4: 16 episodes run
// concurrently, each with a private adapter and history) updated together:
// Algorithm 1 for every episode of the batch that has update text, in one
// chain on one stream.
//
// One batched update (attt_batch_update), with the episodes' update texts
// stacked row after row (episode e owns rows [off_e, off_e + L_e), L_e = 0
// for an episode without an update this round):
//   w, 1/L_e    one launch over every episode (each against its own history)
//   grad_steps times:
//     h_e = x_e W0 + s (x_e A_e) B_e           one contraction over every row
//                                              (block-diagonal adapter terms)
//     loss_e, dh  Eq. 10 over every row in one call (the LM head is shared),
//                 each row with its own episode's 1/L_e; loss_e from the rows'
//                 NLL in a fixed order
//     dy = bf16(dh)                            one launch
//     dA_e, dB_e                               one grouped launch per pass (16 episodes each)
//     dx_e                                     one contraction over every row (if asked)
//     A, B <- A - lr dA, B - lr dB             one launch over every adapter
//   H_e <- H_e || x_e                          one launch over every history
// The adapters live stacked (A [E][din][r], B [E][r][d]), so the SGD step of
// the whole batch is one launch; an episode without rows gets zero
// gradients, which leave its adapter bit-identical.
#include <cuda_runtime.h>

#include <cmath>
#include <new>
#include <vector>

#include "attt.h"
#include "attt_host.h"

struct attt_batch {
    attt_batch_config cfg;
    const attt_bf16 *W0, *Wlm;
    std::vector<attt_history *> hist;
    float *A32, *B32, *A0, *B0, *dA, *dB;
    attt_bf16 *A16, *B16;
    float *w, *rowscale, *nll, *dh, *loss_scratch;
    attt_bf16 *h, *dy;
    void *ws;   // Eq. 10's workspace
    size_t ws_bytes;
    void *aws;  // the adapted projections' workspace (kept across Eq. 10 within a step)
    size_t aws_bytes;
    // the histories' append of an update runs on this stream beside the update's
    // contractions; the update's own stream waits for it before the call returns
    cudaStream_t side;
    cudaEvent_t ev_weights, ev_append;
};

namespace {


constexpr int kMaxEpisodes = 32;

template <class T>
bool dev_alloc(T **p, size_t count) {
    *p = nullptr;
    if (attt::fault_take(attt::FAULT_ALLOC)) return false;  // an injected allocation failure
    return cudaMalloc(reinterpret_cast<void **>(p), (count > 0 ? count : 1) * sizeof(T)) == cudaSuccess;
}

void free_all(attt_batch *b) {
    for (attt_history *h : b->hist)
        if (h) attt_history_destroy(h);
    void *bufs[] = {b->A32, b->B32, b->A0, b->B0, b->dA, b->dB, b->A16, b->B16, b->w, b->rowscale,
                    b->nll, b->dh, b->loss_scratch, b->h, b->dy, b->ws, b->aws};
    for (void *p : bufs) cudaFree(p);
    if (b->ev_weights) cudaEventDestroy(b->ev_weights);
    if (b->ev_append) cudaEventDestroy(b->ev_append);
    if (b->side) cudaStreamDestroy(b->side);
}

bool config_ok(const attt_batch_config *c) {
    return c && c->episodes >= 1 && c->episodes <= kMaxEpisodes && c->n >= 1 && c->n <= 16 && c->w_min > 0.0f &&
           c->w_min <= 1.0f && c->max_history >= 1 && c->max_history <= 16777214 && c->max_update >= 1 &&
           c->max_update <= c->max_history && c->din >= 8 && c->din % 8 == 0 && c->d >= 8 && c->d % 8 == 0 &&
           c->V >= 1 && c->r >= 1 && c->r <= 64 && std::isfinite(c->scale) && std::isfinite(c->lr) &&
           c->grad_steps >= 1 && c->grad_steps <= 64;
}

struct RowOffsets {
    int64_t off[kMaxEpisodes + 1];  // episode e owns rows [off[e], off[e + 1])
};

// Per-episode losses: loss[e * steps + g] = (1/L_e) sum_{j of e} w_j nll_j,
// one block per episode, summed in a fixed order (0 for an episode without
// rows).
__global__ void __launch_bounds__(256) batch_loss_kernel(const float *__restrict__ w, const float *__restrict__ nll,
                                                         const RowOffsets ro, int steps, int g,
                                                         float *__restrict__ loss) {
    __shared__ float s_part[256];
    const int e = blockIdx.x;
    const int64_t a = ro.off[e], b = ro.off[e + 1];
    float acc = 0.f;
    for (int64_t j = a + threadIdx.x; j < b; j += blockDim.x) acc += w[j] * nll[j];
    s_part[threadIdx.x] = acc;
    __syncthreads();
    for (int o = 128; o > 0; o >>= 1) {
        if (threadIdx.x < o) s_part[threadIdx.x] += s_part[threadIdx.x + o];
        __syncthreads();
    }
    if (threadIdx.x == 0) loss[(int64_t)e * steps + g] = b > a ? s_part[0] * (1.0f / (float)(b - a)) : 0.0f;
}

// The initial adapter into every episode's slot, and its bf16 copies.
attt_status load_adapters(attt_batch *b, int e0, int e1, cudaStream_t s) {
    const attt_batch_config &c = b->cfg;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    for (int e = e0; e < e1; ++e) {
        if (cudaMemcpyAsync(b->A32 + e * nA, b->A0, nA * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
            cudaMemcpyAsync(b->B32 + e * nB, b->B0, nB * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
            return ATTT_ERR_CUDA;
    }
    attt_status st = attt_cast_bf16(b->A32 + e0 * nA, b->A16 + e0 * nA, (int64_t)((e1 - e0) * nA), s);
    if (st != ATTT_OK) return st;
    return attt_cast_bf16(b->B32 + e0 * nB, b->B16 + e0 * nB, (int64_t)((e1 - e0) * nB), s);
}

}  // namespace

extern "C" {

attt_status attt_batch_create(const attt_batch_config *cfg, const attt_bf16 *d_W0, const attt_bf16 *d_Wlm,
                              const float *d_A0, const float *d_B0, attt_batch **out) {
    using namespace attt;
    if (!out) return ATTT_ERR_INVALID_ARG;
    *out = nullptr;
    if (!config_ok(cfg) || !d_W0 || !d_Wlm || !d_A0 || !d_B0 || !aligned16(d_W0) || !aligned16(d_Wlm))
        return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    attt_batch *b = new (std::nothrow) attt_batch{};
    if (!b) return ATTT_ERR_CUDA;
    b->cfg = *cfg;
    b->W0 = d_W0;
    b->Wlm = d_Wlm;
    const attt_batch_config &c = b->cfg;
    const int E = c.episodes;
    const int64_t rows = (int64_t)E * c.max_update;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    // Eq. 10 over up to E max_update rows (its bound taken over every row
    // count, since its vocabulary chunk depends on it); the adapted
    // projections' own workspace for up to E max_update rows
    b->ws_bytes = ce_workspace_bound(rows, c.d, c.V);
    b->aws_bytes = batch_adapter_workspace(E, rows + 8 * E, c.din, c.d, c.r);
    b->hist.assign(E, nullptr);
    bool ok = true;
    for (int e = 0; e < E && ok; ++e) ok = attt_history_create(c.n, c.max_history, &b->hist[e]) == ATTT_OK;
    ok = ok && dev_alloc(&b->A32, E * nA) && dev_alloc(&b->B32, E * nB) && dev_alloc(&b->A0, nA) &&
         dev_alloc(&b->B0, nB) && dev_alloc(&b->dA, E * nA) && dev_alloc(&b->dB, E * nB) &&
         dev_alloc(&b->A16, E * nA) && dev_alloc(&b->B16, E * nB) && dev_alloc(&b->w, (size_t)rows) &&
         dev_alloc(&b->rowscale, (size_t)rows) && dev_alloc(&b->nll, (size_t)rows) &&
         dev_alloc(&b->dh, (size_t)rows * c.d) && dev_alloc(&b->loss_scratch, (size_t)E * c.grad_steps + 1) &&
         dev_alloc(&b->h, (size_t)rows * c.d) && dev_alloc(&b->dy, (size_t)rows * c.d) &&
         dev_alloc(reinterpret_cast<char **>(&b->ws), b->ws_bytes) &&
         dev_alloc(reinterpret_cast<char **>(&b->aws), b->aws_bytes);
    ok = ok && cudaStreamCreateWithFlags(&b->side, cudaStreamNonBlocking) == cudaSuccess &&
         cudaEventCreateWithFlags(&b->ev_weights, cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&b->ev_append, cudaEventDisableTiming) == cudaSuccess;
    if (ok)
        ok = cudaMemcpy(b->A0, d_A0, nA * sizeof(float), cudaMemcpyDeviceToDevice) == cudaSuccess &&
             cudaMemcpy(b->B0, d_B0, nB * sizeof(float), cudaMemcpyDeviceToDevice) == cudaSuccess &&
             load_adapters(b, 0, E, nullptr) == ATTT_OK && cudaDeviceSynchronize() == cudaSuccess;
    if (!ok) {
        free_all(b);
        delete b;
        return ATTT_ERR_CUDA;
    }
    *out = b;
    return ATTT_OK;
}

attt_status attt_batch_destroy(attt_batch *b) {
    if (!b) return ATTT_ERR_INVALID_ARG;
    cudaDeviceSynchronize();
    free_all(b);
    delete b;
    return ATTT_OK;
}

attt_status attt_batch_reset(attt_batch *b, int e, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!b || e < -1 || e >= b->cfg.episodes) return ATTT_ERR_INVALID_ARG;
    const int e0 = e < 0 ? 0 : e, e1 = e < 0 ? b->cfg.episodes : e + 1;
    for (int i = e0; i < e1; ++i) {
        attt_status st = attt_history_reset(b->hist[i], stream);
        if (st != ATTT_OK) return st;
    }
    return load_adapters(b, e0, e1, stream);
}

attt_status attt_batch_update(attt_batch *b, const int32_t *d_tokens, const attt_bf16 *d_x, const int64_t *lens,
                              float *d_losses, float *d_dx, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!b || !lens) return ATTT_ERR_INVALID_ARG;
    const attt_batch_config &c = b->cfg;
    const int E = c.episodes;
    RowOffsets ro{};
    int64_t *off = ro.off;
    off[0] = 0;
    for (int e = 0; e < E; ++e) {
        if (lens[e] < 0 || lens[e] > c.max_update) return ATTT_ERR_INVALID_ARG;
        if (attt_history_length(b->hist[e]) + lens[e] > c.max_history) return ATTT_ERR_CAPACITY;
        off[e + 1] = off[e] + lens[e];
    }
    const int64_t R = off[E];
    if (R == 0) return ATTT_OK;
    if (!d_tokens || !d_x || !aligned16(d_x) || (d_dx && !aligned16(d_dx))) return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    const int64_t rb = (int64_t)E * c.max_update + 8 * E;  // the row bound the adapter workspace was sized for
    float *losses = d_losses ? d_losses : b->loss_scratch;

    st = ngram_weights_batch(b->hist.data(), E, d_tokens, off, c.w_min, b->w, b->rowscale, stream);
    // nothing below reads the tables, so the histories' append (last in
    // Algorithm 1) runs on the side stream beside the update's contractions
    if (st == ATTT_OK) {
        if (cudaEventRecord(b->ev_weights, stream) != cudaSuccess ||
            cudaStreamWaitEvent(b->side, b->ev_weights, 0) != cudaSuccess)
            st = ATTT_ERR_CUDA;
        if (st == ATTT_OK) st = history_insert_batch(b->hist.data(), E, d_tokens, off, b->side);
        if (cudaEventRecord(b->ev_append, b->side) != cudaSuccess && st == ATTT_OK) st = ATTT_ERR_CUDA;
    }
    for (int g = 0; g < c.grad_steps && st == ATTT_OK; ++g) {
        // every episode's current adapter padded and stacked, then h for every row
        st = batch_adapter_prep(b->A16, b->B16, E, c.din, c.d, c.r, rb, b->aws, b->aws_bytes, stream);
        if (st == ATTT_OK)
            st = batch_forward(d_x, off, E, b->W0, c.din, c.d, c.r, c.scale, b->h, rb, b->aws, b->aws_bytes, stream);
        if (st == ATTT_OK)
            st = ce_fwd_bwd_run(b->h, b->Wlm, d_tokens, b->w, b->rowscale, R, c.d, c.V, b->loss_scratch + E * c.grad_steps,
                                b->dh, nullptr, b->nll, b->ws, b->ws_bytes, stream);
        if (st == ATTT_OK) {
            batch_loss_kernel<<<E, 256, 0, stream>>>(b->w, b->nll, ro, c.grad_steps, g, losses);
            count_launch();
            if (cudaGetLastError() != cudaSuccess) st = ATTT_ERR_CUDA;
        }
        if (st == ATTT_OK) st = attt_cast_bf16(b->dh, b->dy, R * c.d, stream);
        if (st == ATTT_OK && (cudaMemsetAsync(b->dA, 0, E * nA * sizeof(float), stream) != cudaSuccess ||
                              cudaMemsetAsync(b->dB, 0, E * nB * sizeof(float), stream) != cudaSuccess))
            st = ATTT_ERR_CUDA;
        // every episode's adapter gradients: one grouped launch per pass
        if (st == ATTT_OK)
            st = batch_grads(d_x, b->dy, off, E, c.din, c.d, c.r, c.scale, b->dA, b->dB, rb, b->aws, b->aws_bytes,
                             stream);
        if (st == ATTT_OK && d_dx)
            st = batch_input_grad(b->dy, off, E, b->W0, c.din, c.d, c.r, c.scale, d_dx + (size_t)g * R * c.din, rb,
                                  b->aws, b->aws_bytes, stream);
        // every adapter of the batch in one step: A as [E din, r], B as [r, E d]
        if (st == ATTT_OK)
            st = attt_lora_step(b->A32, b->B32, b->dA, b->dB, (int64_t)E * c.din, (int64_t)E * c.d, c.r, c.lr, b->A16,
                                b->B16, stream);
    }
    // the update's stream waits for the append (a no-op before the first one)
    if (cudaStreamWaitEvent(stream, b->ev_append, 0) != cudaSuccess && st == ATTT_OK) st = ATTT_ERR_CUDA;
    return st;
}

attt_status attt_batch_read_adapter(const attt_batch *b, int e, float *d_A32, float *d_B32, attt_stream stream) {
    if (!b || e < 0 || e >= b->cfg.episodes || !d_A32 || !d_B32) return ATTT_ERR_INVALID_ARG;
    const size_t nA = (size_t)b->cfg.din * b->cfg.r, nB = (size_t)b->cfg.r * b->cfg.d;
    if (cudaMemcpyAsync(d_A32, b->A32 + e * nA, nA * sizeof(float), cudaMemcpyDeviceToDevice, stream) != cudaSuccess ||
        cudaMemcpyAsync(d_B32, b->B32 + e * nB, nB * sizeof(float), cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    return ATTT_OK;
}

attt_history *attt_batch_history(attt_batch *b, int e) {
    return (b && e >= 0 && e < b->cfg.episodes) ? b->hist[e] : nullptr;
}

}  // extern "C"
