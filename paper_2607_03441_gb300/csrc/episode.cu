// episode.cu -- the in-episode update driver: Algorithm 1 run end to end on
// one stream, with the schedule of Sec. 4 / Appendix C (an update every K
// agent steps, two gradient steps per update, the adapter persisting within
// an episode and reset between episodes).
//
// One update k (attt_episode_update):
//   w = Eq. 9(Eq. 8(x_k, H_k))                        attt_ngram_weights
//   repeat grad_steps times (Eq. 2 / Algorithm 1's gradient step):
//     h  = x W0 + s (x A) B                           attt_lora_forward
//     loss, dh = Eq. 10(h, W_lm, targets x_k, w)      attt_weighted_ce_fwd_bwd
//     dy = bf16(dh)                                   attt_cast_bf16
//     dA, dB = adapter gradients of h                 attt_lora_grad
//     dx = dy W0^T + s (dy B^T) A^T  (if requested)   attt_lora_input_grad
//     A, B <- A - lr dA, B - lr dB                    attt_lora_step
//       (or AdamW, optimizer 1)                       attt_lora_adamw_step
//   H_{k+1} = H_k || x_k                              attt_history_insert
//
// Everything is host code that issues the library's own calls; the episode
// owns its device buffers (allocated once at create) and one workspace that
// the calls share, since they run one after another on the caller's stream
// and the first kernel of each call waits for the previous call to finish.
// Two calls run beside that chain on streams of their own, ordered by events:
// the history append (after the weights) and dx (after dy is written; joined
// before the SGD step), the latter with a workspace of its own.
#include <cuda_runtime.h>

#include <cmath>
#include <cstring>
#include <new>

#include "attt.h"
#include "attt_host.h"

struct attt_episode {
    attt_episode_config cfg;
    const attt_bf16 *W0;   // [din, d] frozen projection (borrowed)
    const attt_bf16 *Wlm;  // [V, d] frozen LM head (borrowed)
    attt_history *hist;
    // adapter: fp32 masters, bf16 copies, initial values, gradients
    float *A32, *B32, *A0, *B0, *dA, *dB;
    float *mA, *vA, *mB, *vB;  // AdamW moments (optimizer 1)
    int adam_t;                // AdamW steps taken
    attt_bf16 *A16, *B16;
    // per-update activations
    float *w, *dh, *losses;
    attt_bf16 *h, *dy, *h_base;
    // pending update text (agent steps since the last update)
    int32_t *pend_tok;
    attt_bf16 *pend_x;
    int64_t pend_len;
    int pend_steps;
    void *ws;
    size_t ws_bytes;
    // Algorithm 1's history append of an update runs on this stream, beside
    // the update's contractions (it only needs the weights to have read the
    // table); the update's own stream waits for it before the call returns.
    cudaStream_t side;
    cudaEvent_t ev_weights, ev_append;
    // dx of a gradient step runs on its own stream with its own workspace,
    // beside the adapter gradients: both read dy and the adapter, neither
    // writes what the other reads, and the step waits for both.
    cudaStream_t side_dx;
    cudaEvent_t ev_dy, ev_dx;
    void *ws_dx;
    size_t ws_dx_bytes;
};

namespace {


template <class T>
bool dev_alloc(T **p, size_t count) {
    *p = nullptr;
    if (attt::fault_take(attt::FAULT_ALLOC)) return false;  // an injected allocation failure
    return cudaMalloc(reinterpret_cast<void **>(p), (count > 0 ? count : 1) * sizeof(T)) == cudaSuccess;
}

void free_all(attt_episode *e) {
    if (e->hist) attt_history_destroy(e->hist);
    void *bufs[] = {e->A32, e->B32, e->A0, e->B0, e->dA, e->dB, e->mA, e->vA, e->mB, e->vB, e->A16, e->B16, e->w,
                    e->dh,  e->losses, e->h, e->dy, e->h_base, e->pend_tok, e->pend_x, e->ws, e->ws_dx};
    for (void *b : bufs) cudaFree(b);
    if (e->ev_weights) cudaEventDestroy(e->ev_weights);
    if (e->ev_append) cudaEventDestroy(e->ev_append);
    if (e->side) cudaStreamDestroy(e->side);
    if (e->ev_dy) cudaEventDestroy(e->ev_dy);
    if (e->ev_dx) cudaEventDestroy(e->ev_dx);
    if (e->side_dx) cudaStreamDestroy(e->side_dx);
}

// H <- H || x on the side stream once the update's weights (enqueued on
// `stream`) have read the table; ev_append marks its end.
attt_status append_beside(attt_episode *e, const int32_t *d_tokens, int64_t L, cudaStream_t stream) {
    if (cudaEventRecord(e->ev_weights, stream) != cudaSuccess ||
        cudaStreamWaitEvent(e->side, e->ev_weights, 0) != cudaSuccess)
        return ATTT_ERR_CUDA;
    const attt_status st = attt_history_insert(e->hist, d_tokens, L, e->side);
    return cudaEventRecord(e->ev_append, e->side) == cudaSuccess ? st : ATTT_ERR_CUDA;
}

bool config_ok(const attt_episode_config *c) {
    return c && c->n >= 1 && c->n <= 16 && c->w_min > 0.0f && c->w_min <= 1.0f && c->max_history >= 0 &&
           c->max_history <= 16777214 && c->max_update >= 1 && c->max_update <= c->max_history &&
           c->din >= 8 && c->din % 8 == 0 && c->d >= 8 && c->d % 8 == 0 && c->V >= 1 && c->r >= 1 && c->r <= 64 &&
           std::isfinite(c->scale) && std::isfinite(c->lr) && c->grad_steps >= 1 && c->grad_steps <= 64 &&
           c->cadence >= 1 &&
           (c->optimizer == 0 || (c->optimizer == 1 && c->beta1 >= 0.0 && c->beta1 < 1.0 && c->beta2 >= 0.0 &&
                                  c->beta2 < 1.0 && c->eps > 0.0 && c->weight_decay >= 0.0));
}

// Workspace that every call of an update of up to max_update tokens fits in.
// The Eq. 10 workspace is not monotone in L (its vocabulary chunk depends on
// L): its bound is the maximum over every L.
size_t workspace_bound(const attt_episode_config &c) {
    size_t ws = 0;
    auto upd = [&](size_t b) { if (b > ws) ws = b; };
    upd(attt::ce_workspace_bound(c.max_update, c.d, c.V));
    const int64_t L = c.max_update;
    upd(attt_lora_workspace_bytes(L, c.din, 1, &c.d, c.r));
    upd(attt_lora_forward_workspace_bytes(L, c.din, c.d, c.r));
    upd(attt_kl_workspace_bytes(L, c.d, c.V));  // grows with L
    return ws;
}

attt_status load_adapter(attt_episode *e, cudaStream_t s) {
    const size_t nA = (size_t)e->cfg.din * e->cfg.r, nB = (size_t)e->cfg.r * e->cfg.d;
    if (cudaMemcpyAsync(e->A32, e->A0, nA * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess ||
        cudaMemcpyAsync(e->B32, e->B0, nB * sizeof(float), cudaMemcpyDeviceToDevice, s) != cudaSuccess)
        return ATTT_ERR_CUDA;
    if (e->cfg.optimizer == 1) {
        e->adam_t = 0;
        if (cudaMemsetAsync(e->mA, 0, nA * sizeof(float), s) != cudaSuccess ||
            cudaMemsetAsync(e->vA, 0, nA * sizeof(float), s) != cudaSuccess ||
            cudaMemsetAsync(e->mB, 0, nB * sizeof(float), s) != cudaSuccess ||
            cudaMemsetAsync(e->vB, 0, nB * sizeof(float), s) != cudaSuccess)
            return ATTT_ERR_CUDA;
    }
    attt_status st = attt_cast_bf16(e->A32, e->A16, (int64_t)nA, s);
    if (st != ATTT_OK) return st;
    return attt_cast_bf16(e->B32, e->B16, (int64_t)nB, s);
}

}  // namespace

extern "C" {

attt_status attt_episode_create(const attt_episode_config *cfg, const attt_bf16 *d_W0, const attt_bf16 *d_Wlm,
                                const float *d_A0, const float *d_B0, attt_episode **out) {
    using namespace attt;
    if (!out) return ATTT_ERR_INVALID_ARG;
    *out = nullptr;
    if (!config_ok(cfg) || !d_W0 || !d_Wlm || !d_A0 || !d_B0 || !aligned16(d_W0) || !aligned16(d_Wlm))
        return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;

    attt_episode *e = new (std::nothrow) attt_episode{};
    if (!e) return ATTT_ERR_CUDA;
    e->cfg = *cfg;
    e->W0 = d_W0;
    e->Wlm = d_Wlm;
    const attt_episode_config &c = e->cfg;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d, Ld = (size_t)c.max_update * c.d;
    e->ws_bytes = workspace_bound(c);
    bool ok = attt_history_create(c.n, c.max_history, &e->hist) == ATTT_OK;
    ok = ok && dev_alloc(&e->A32, nA) && dev_alloc(&e->B32, nB) && dev_alloc(&e->A0, nA) && dev_alloc(&e->B0, nB) &&
         dev_alloc(&e->dA, nA) && dev_alloc(&e->dB, nB) && dev_alloc(&e->A16, nA) && dev_alloc(&e->B16, nB) &&
         dev_alloc(&e->w, (size_t)c.max_update) && dev_alloc(&e->dh, Ld) && dev_alloc(&e->losses, (size_t)c.grad_steps) &&
         dev_alloc(&e->h, Ld) && dev_alloc(&e->dy, Ld) && dev_alloc(&e->h_base, Ld) &&
         dev_alloc(&e->pend_tok, (size_t)c.max_update) &&
         dev_alloc(&e->pend_x, (size_t)c.max_update * c.din) &&
         dev_alloc(reinterpret_cast<char **>(&e->ws), e->ws_bytes);
    e->ws_dx_bytes = attt_lora_input_grad_workspace_bytes(c.max_update, c.din, c.d, c.r);
    ok = ok && dev_alloc(reinterpret_cast<char **>(&e->ws_dx), e->ws_dx_bytes);
    if (ok && c.optimizer == 1)
        ok = dev_alloc(&e->mA, nA) && dev_alloc(&e->vA, nA) && dev_alloc(&e->mB, nB) && dev_alloc(&e->vB, nB);
    ok = ok && cudaStreamCreateWithFlags(&e->side, cudaStreamNonBlocking) == cudaSuccess &&
         cudaEventCreateWithFlags(&e->ev_weights, cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&e->ev_append, cudaEventDisableTiming) == cudaSuccess &&
         cudaStreamCreateWithFlags(&e->side_dx, cudaStreamNonBlocking) == cudaSuccess &&
         cudaEventCreateWithFlags(&e->ev_dy, cudaEventDisableTiming) == cudaSuccess &&
         cudaEventCreateWithFlags(&e->ev_dx, cudaEventDisableTiming) == cudaSuccess;
    if (ok) {
        // The initial adapter is copied once; later resets restore it.
        ok = cudaMemcpy(e->A0, d_A0, nA * sizeof(float), cudaMemcpyDeviceToDevice) == cudaSuccess &&
             cudaMemcpy(e->B0, d_B0, nB * sizeof(float), cudaMemcpyDeviceToDevice) == cudaSuccess &&
             load_adapter(e, nullptr) == ATTT_OK && cudaDeviceSynchronize() == cudaSuccess;
    }
    if (!ok) {
        free_all(e);
        delete e;
        return ATTT_ERR_CUDA;
    }
    *out = e;
    return ATTT_OK;
}

attt_status attt_episode_destroy(attt_episode *e) {
    if (!e) return ATTT_ERR_INVALID_ARG;
    cudaDeviceSynchronize();
    free_all(e);
    delete e;
    return ATTT_OK;
}

attt_status attt_episode_reset(attt_episode *e, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!e) return ATTT_ERR_INVALID_ARG;
    attt_status st = attt_history_reset(e->hist, stream);
    if (st != ATTT_OK) return st;
    e->pend_len = 0;
    e->pend_steps = 0;
    return load_adapter(e, stream);
}

attt_status attt_episode_update(attt_episode *e, const int32_t *d_tokens, const attt_bf16 *d_x, int64_t L,
                                float *d_losses, float *d_dx, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!e || L < 1 || !d_tokens || !d_x || !aligned16(d_x) || (d_dx && !aligned16(d_dx)))
        return ATTT_ERR_INVALID_ARG;
    const attt_episode_config &c = e->cfg;
    if (L > c.max_update) return ATTT_ERR_INVALID_ARG;
    if (attt_history_length(e->hist) + L > c.max_history) return ATTT_ERR_CAPACITY;
    if (d_dx && c.r % 8 != 0) return ATTT_ERR_UNSUPPORTED;
    float *losses = d_losses ? d_losses : e->losses;

    attt_status st = attt_ngram_weights(e->hist, d_tokens, L, c.w_min, e->w, stream);
    // nothing below reads the table, so the append (last in Algorithm 1) runs
    // beside the update's contractions
    if (st == ATTT_OK) st = append_beside(e, d_tokens, L, stream);
    for (int g = 0; g < c.grad_steps && st == ATTT_OK; ++g) {
        st = attt_lora_forward(d_x, e->W0, e->A16, e->B16, L, c.din, c.d, c.r, c.scale, e->h, e->ws, e->ws_bytes,
                               stream);
        if (st == ATTT_OK)
            st = attt_weighted_ce_fwd_bwd(e->h, e->Wlm, d_tokens, e->w, L, c.d, c.V, losses + g, e->dh, nullptr,
                                          e->ws, e->ws_bytes, stream);
        if (st == ATTT_OK) st = attt_cast_bf16(e->dh, e->dy, L * c.d, stream);
        // dx on its own stream once dy is written, beside the adapter gradients
        bool dx_beside = false;
        if (st == ATTT_OK && d_dx) {
            if (cudaEventRecord(e->ev_dy, stream) != cudaSuccess ||
                cudaStreamWaitEvent(e->side_dx, e->ev_dy, 0) != cudaSuccess) {
                st = ATTT_ERR_CUDA;
            } else {
                st = attt_lora_input_grad(e->dy, e->W0, e->A16, e->B16, L, c.din, c.d, c.r, c.scale,
                                          d_dx + (size_t)g * L * c.din, e->ws_dx, e->ws_dx_bytes, e->side_dx);
                dx_beside = true;
                if (cudaEventRecord(e->ev_dx, e->side_dx) != cudaSuccess && st == ATTT_OK) st = ATTT_ERR_CUDA;
            }
        }
        if (st == ATTT_OK) {
            const attt_bf16 *dys[1] = {e->dy}, *As[1] = {e->A16}, *Bs[1] = {e->B16};
            float *dAs[1] = {e->dA}, *dBs[1] = {e->dB};
            st = attt_lora_grad(d_x, L, c.din, 1, dys, &c.d, As, Bs, c.r, c.scale, dAs, dBs, e->ws, e->ws_bytes,
                                stream);
        }
        // the step changes the adapter that dx reads: it waits for dx
        if (dx_beside && cudaStreamWaitEvent(stream, e->ev_dx, 0) != cudaSuccess && st == ATTT_OK)
            st = ATTT_ERR_CUDA;
        if (st == ATTT_OK) {
            if (c.optimizer == 0) {
                st = attt_lora_step(e->A32, e->B32, e->dA, e->dB, c.din, c.d, c.r, c.lr, e->A16, e->B16, stream);
            } else {
                st = attt_lora_adamw_step(e->A32, e->B32, e->dA, e->dB, e->mA, e->vA, e->mB, e->vB, c.din, c.d, c.r,
                                          c.lr, c.beta1, c.beta2, c.eps, c.weight_decay, e->adam_t + 1, e->A16,
                                          e->B16, stream);
                if (st == ATTT_OK) ++e->adam_t;
            }
        }
    }
    // the update's stream waits for the append (a no-op before the first one)
    if (cudaStreamWaitEvent(stream, e->ev_append, 0) != cudaSuccess && st == ATTT_OK) st = ATTT_ERR_CUDA;
    return st;
}

attt_status attt_episode_agent_step(attt_episode *e, const int32_t *d_tokens, const attt_bf16 *d_x, int64_t len,
                                    float *d_losses, float *d_dx, int *updated, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!e || len < 0 || (len > 0 && (!d_tokens || !d_x))) return ATTT_ERR_INVALID_ARG;
    const attt_episode_config &c = e->cfg;
    if (updated) *updated = 0;
    if (e->pend_len + len > c.max_update) return ATTT_ERR_CAPACITY;
    const bool fire = e->pend_steps + 1 >= c.cadence;
    if (fire && e->pend_len + len > 0 && attt_history_length(e->hist) + e->pend_len + len > c.max_history)
        return ATTT_ERR_CAPACITY;
    if (len > 0) {
        if (cudaMemcpyAsync(e->pend_tok + e->pend_len, d_tokens, (size_t)len * sizeof(int32_t),
                            cudaMemcpyDeviceToDevice, stream) != cudaSuccess ||
            cudaMemcpyAsync(e->pend_x + (size_t)e->pend_len * c.din, d_x, (size_t)len * c.din * sizeof(attt_bf16),
                            cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
            return ATTT_ERR_CUDA;
    }
    e->pend_len += len;
    e->pend_steps += 1;
    if (!fire) return ATTT_OK;
    const int64_t L = e->pend_len;
    e->pend_len = 0;
    e->pend_steps = 0;
    if (L == 0) return ATTT_OK;  // K steps without update text: nothing to train on
    attt_status st = attt_episode_update(e, e->pend_tok, e->pend_x, L, d_losses, d_dx, stream);
    if (st == ATTT_OK && updated) *updated = 1;
    return st;
}

attt_status attt_episode_drift(attt_episode *e, const attt_bf16 *d_x, int64_t L, float *d_kl, float *d_kl_mean,
                               attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!e || L < 1 || L > e->cfg.max_update || !d_x || !aligned16(d_x) || (!d_kl && !d_kl_mean))
        return ATTT_ERR_INVALID_ARG;
    const attt_episode_config &c = e->cfg;
    // the adapted model (current adapter) and the base model (no adapter: s = 0)
    attt_status st = attt_lora_forward(d_x, e->W0, e->A16, e->B16, L, c.din, c.d, c.r, c.scale, e->h, e->ws,
                                       e->ws_bytes, stream);
    if (st == ATTT_OK)
        st = attt_lora_forward(d_x, e->W0, e->A16, e->B16, L, c.din, c.d, c.r, 0.0f, e->h_base, e->ws,
                               e->ws_bytes, stream);
    if (st == ATTT_OK)
        st = attt_kl_drift(e->h, e->h_base, e->Wlm, L, c.d, c.V, d_kl, d_kl_mean, e->ws, e->ws_bytes, stream);
    return st;
}

attt_status attt_episode_read_adapter(const attt_episode *e, float *d_A32, float *d_B32, attt_stream stream) {
    if (!e || !d_A32 || !d_B32) return ATTT_ERR_INVALID_ARG;
    const size_t nA = (size_t)e->cfg.din * e->cfg.r, nB = (size_t)e->cfg.r * e->cfg.d;
    if (cudaMemcpyAsync(d_A32, e->A32, nA * sizeof(float), cudaMemcpyDeviceToDevice, stream) != cudaSuccess ||
        cudaMemcpyAsync(d_B32, e->B32, nB * sizeof(float), cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    return ATTT_OK;
}

// Checkpoint layout (host bytes, native endianness): a header, then the
// arrays in this order, each as stored on the device.
struct EpisodeCkptHeader {
    char magic[8];  // "ATTTEPC1"
    attt_episode_config cfg;
    int64_t hist_len, pend_len;
    int32_t pend_steps, adam_t;
};

static size_t ckpt_bytes(const attt_episode *e, int64_t hist_len, int64_t pend_len) {
    const attt_episode_config &c = e->cfg;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    size_t b = sizeof(EpisodeCkptHeader) + (nA + nB) * sizeof(float);
    if (c.optimizer == 1) b += 2 * (nA + nB) * sizeof(float);
    b += (size_t)hist_len * sizeof(int32_t) + (size_t)pend_len * (sizeof(int32_t) + c.din * sizeof(attt_bf16));
    return b;
}

size_t attt_episode_checkpoint_bytes(const attt_episode *e) {
    return e ? ckpt_bytes(e, attt_history_length(e->hist), e->pend_len) : 0;
}

attt_status attt_episode_save(attt_episode *e, void *host_buf, size_t bytes, attt_stream stream) {
    if (!e || !host_buf) return ATTT_ERR_INVALID_ARG;
    const int64_t hl = attt_history_length(e->hist);
    if (bytes < ckpt_bytes(e, hl, e->pend_len)) return ATTT_ERR_INVALID_ARG;
    const attt_episode_config &c = e->cfg;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    char *p = static_cast<char *>(host_buf);
    EpisodeCkptHeader hdr{};
    memcpy(hdr.magic, "ATTTEPC1", 8);
    hdr.cfg = c;
    hdr.hist_len = hl;
    hdr.pend_len = e->pend_len;
    hdr.pend_steps = e->pend_steps;
    hdr.adam_t = e->adam_t;
    memcpy(p, &hdr, sizeof hdr);
    p += sizeof hdr;
    struct Piece { const void *src; size_t n; };
    Piece pieces[] = {{e->A32, nA * sizeof(float)}, {e->B32, nB * sizeof(float)},
                      {c.optimizer == 1 ? e->mA : nullptr, nA * sizeof(float)},
                      {c.optimizer == 1 ? e->vA : nullptr, nA * sizeof(float)},
                      {c.optimizer == 1 ? e->mB : nullptr, nB * sizeof(float)},
                      {c.optimizer == 1 ? e->vB : nullptr, nB * sizeof(float)},
                      {e->pend_tok, (size_t)e->pend_len * sizeof(int32_t)},
                      {e->pend_x, (size_t)e->pend_len * c.din * sizeof(attt_bf16)}};
    for (const Piece &q : pieces) {
        if (!q.src || q.n == 0) continue;
        if (cudaMemcpyAsync(p, q.src, q.n, cudaMemcpyDeviceToHost, stream) != cudaSuccess) return ATTT_ERR_CUDA;
        p += q.n;
    }
    attt_status st = attt_history_save(e->hist, reinterpret_cast<int32_t *>(p), stream);  // synchronises
    if (st != ATTT_OK) return st;
    return cudaStreamSynchronize(stream) == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status attt_episode_load(attt_episode *e, const void *host_buf, size_t bytes, attt_stream stream) {
    if (!e || !host_buf || bytes < sizeof(EpisodeCkptHeader)) return ATTT_ERR_INVALID_ARG;
    EpisodeCkptHeader hdr;
    memcpy(&hdr, host_buf, sizeof hdr);
    const attt_episode_config &c = e->cfg;
    if (memcmp(hdr.magic, "ATTTEPC1", 8) != 0 || memcmp(&hdr.cfg, &c, sizeof c) != 0) return ATTT_ERR_INVALID_ARG;
    if (hdr.hist_len < 0 || hdr.hist_len > c.max_history || hdr.pend_len < 0 || hdr.pend_len > c.max_update ||
        bytes < ckpt_bytes(e, hdr.hist_len, hdr.pend_len))
        return ATTT_ERR_INVALID_ARG;
    const size_t nA = (size_t)c.din * c.r, nB = (size_t)c.r * c.d;
    const char *p = static_cast<const char *>(host_buf) + sizeof hdr;
    struct Piece { void *dst; size_t n; };
    Piece pieces[] = {{e->A32, nA * sizeof(float)}, {e->B32, nB * sizeof(float)},
                      {c.optimizer == 1 ? e->mA : nullptr, nA * sizeof(float)},
                      {c.optimizer == 1 ? e->vA : nullptr, nA * sizeof(float)},
                      {c.optimizer == 1 ? e->mB : nullptr, nB * sizeof(float)},
                      {c.optimizer == 1 ? e->vB : nullptr, nB * sizeof(float)},
                      {e->pend_tok, (size_t)hdr.pend_len * sizeof(int32_t)},
                      {e->pend_x, (size_t)hdr.pend_len * c.din * sizeof(attt_bf16)}};
    for (const Piece &q : pieces) {
        if (!q.dst || q.n == 0) continue;
        if (cudaMemcpyAsync(q.dst, p, q.n, cudaMemcpyHostToDevice, stream) != cudaSuccess) return ATTT_ERR_CUDA;
        p += q.n;
    }
    attt_status st = attt_cast_bf16(e->A32, e->A16, (int64_t)nA, stream);
    if (st == ATTT_OK) st = attt_cast_bf16(e->B32, e->B16, (int64_t)nB, stream);
    if (st == ATTT_OK) st = attt_history_restore(e->hist, reinterpret_cast<const int32_t *>(p), hdr.hist_len, stream);
    if (st != ATTT_OK) return st;
    e->pend_len = hdr.pend_len;
    e->pend_steps = hdr.pend_steps;
    e->adam_t = hdr.adam_t;
    return cudaStreamSynchronize(stream) == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_history *attt_episode_history(attt_episode *e) { return e ? e->hist : nullptr; }

int64_t attt_episode_pending_tokens(const attt_episode *e) { return e ? e->pend_len : -1; }

}  // extern "C"
