// wordset.cu -- Eq. 6 / Eq. 7 of aTTT on the GPU: the word-level Jaccard
// repetition rho(x_k) of an update text against every previous update text
// of the episode, the novelty nu = 1 - rho, and the sequence-level filter
// that skips an update whose novelty falls below tau (Sec. 4, Appendix C).
//
// Design (GB300-first):
//   * every update text is appended to a device byte arena, followed by one
//     space, so every word in the arena ends at a whitespace byte;
//   * one exact word index for the whole episode: open addressing, linear
//     probing, power-of-two capacity >= 2 * the most words the arena can
//     hold, slots of one 64-bit key
//       [63:48] hash tag | [47:32] min(length, 65535) | [31:0] arena position + 1
//     of the word's first occurrence (0 = empty) and a bitmask of the updates
//     whose text contains the word (one bit per update, W 64-bit words).
//     Equality is decided byte by byte in the arena after a tag match;
//   * one launch per update (repetition_kernel): the blocks copy the text into
//     the arena, find and hash its words, dedup them per chunk in shared
//     memory and record them in the index while counting |W(x_k)| and every
//     |W(x_k) & W(x_i)|; the last block to finish forms J_i = |inter| /
//     |union| with one IEEE fp32 division of the integer sizes, rho = max_i
//     J_i (0 for the first update), nu = 1 - rho in fp32 and keep =
//     !(nu < tau): bit-exact with the definition.
#include <cuda_runtime.h>

#include <new>

#include "attt_common.cuh"
#include "attt_host.h"

namespace {

constexpr int kMaxUpdates = 4096;
constexpr int kProbeLimit = 1 << 20;
constexpr int kInsThreads = 256;

__device__ __forceinline__ bool is_space(unsigned int c) {
    // ASCII whitespace: space, tab, LF, VT, FF, CR
    return c == 0x20u || (c >= 0x09u && c <= 0x0Du);
}

__device__ __forceinline__ unsigned long long finalize64(unsigned long long h) {
    h ^= h >> 33;
    h *= 0xff51afd7ed558ccdull;
    h ^= h >> 33;
    h *= 0xc4ceb9fe1a85ec53ull;
    h ^= h >> 33;
    return h;
}

// The episode's texts as one byte sequence: positions below `base` are the
// arena (earlier texts, each followed by a space), [base, base + n) the
// current text (read from the caller's buffer), a space after it.
struct TextView {
    const uint8_t *arena;
    const uint8_t *text;
    int64_t base, n;
    __device__ __forceinline__ unsigned int at(int64_t p) const {
        return p < base ? (unsigned int)arena[p] : (p < base + n ? (unsigned int)text[p - base] : 0x20u);
    }
};

// Two words are equal when their bytes agree up to a whitespace byte that
// ends both at the same offset (every word ends at one).
__device__ __forceinline__ bool word_equal(const TextView &v, int64_t a, int64_t b) {
    for (int64_t i = 0;; ++i) {
        const unsigned int ca = v.at(a + i), cb = v.at(b + i);
        const bool ea = is_space(ca), eb = is_space(cb);
        if (ea || eb) return ea && eb;
        if (ca != cb) return false;
    }
}

struct RepArgs {
    const uint8_t *text;
    int64_t n;
    uint8_t *arena;
    int64_t base;
    int k, W;
    unsigned long long *keys, *masks;
    unsigned long long cap_mask;
    unsigned int *sizes, *inter, *distinct, *ticket;
    int *status;
    float tau;
    float *rho_out, *nu_out;
    int32_t *keep_out;
    int chunk;  // text bytes per block iteration, <= kChunk
};

constexpr int kChunk = 2048;                 // largest text chunk of a block iteration
constexpr int kChunkWords = kChunk / 2 + 1;  // a word start follows whitespace
constexpr int kLocalSlots = 2048;            // block-local word table (>= 2 x kChunkWords)

// Hashes the word at chunk offset `off` (FNV-1a 64 over its bytes, then a
// 64-bit finalizer), drops it if it repeats an earlier word of the chunk
// (block-local table of 64-bit shared-memory keys: hash tag | offset + 1),
// else claims or finds its slot in the episode's index and sets update k's
// bit.  Returns the slot's mask words if this thread set the bit first (it
// owns the word's element of W(x_k)), with the previous value of mask word
// k / 64 in *old; nullptr otherwise.
__device__ __forceinline__ const unsigned long long *record_word(const RepArgs &a, const TextView &v, int64_t c0,
                                                                 uint32_t off, unsigned long long *s_key, int kw,
                                                                 unsigned long long kbit, unsigned long long *old) {
    const int64_t p = a.base + c0 + off;
    unsigned long long h = 0xcbf29ce484222325ull;
    int64_t e = p;
    for (unsigned int ch = v.at(e); !is_space(ch); ch = v.at(++e)) h = (h ^ ch) * 0x100000001b3ull;
    const int64_t len = e - p;
    h = finalize64(h);
    const unsigned long long lkey = (h & 0xFFFFFFFF00000000ull) | (unsigned long long)(off + 1u);
    unsigned int li = (unsigned int)(h >> 20) & (kLocalSlots - 1);
    for (int probe = 0; probe < kLocalSlots; ++probe, li = (li + 1) & (kLocalSlots - 1)) {
        const unsigned long long o = atomicCAS(&s_key[li], 0ull, lkey);
        if (o == 0ull) break;
        if ((o >> 32) == (lkey >> 32) && word_equal(v, a.base + c0 + (int64_t)(o & 0xFFFFFFFFull) - 1, p))
            return nullptr;  // repeats a word of this chunk
    }
    const unsigned long long key = (h & 0xFFFF000000000000ull) |
                                   ((unsigned long long)(len < 0xFFFF ? len : 0xFFFF) << 32) |
                                   (unsigned long long)(p + 1);
    unsigned long long idx = h & a.cap_mask;
    for (int probe = 0; probe < kProbeLimit; ++probe) {
        const unsigned long long k0 = atomicCAS(a.keys + idx, 0ull, key);
        if (k0 == 0ull || ((k0 >> 32) == (key >> 32) &&
                           ATTT_GUARD((int64_t)(k0 & 0xFFFFFFFFull) - 1 < a.base + a.n, a.status) &&
                           word_equal(v, (int64_t)(k0 & 0xFFFFFFFFull) - 1, p))) {
            unsigned long long *m = a.masks + (size_t)idx * a.W;
            *old = atomicOr(m + kw, kbit);
            return (*old & kbit) ? nullptr : m;  // else another block owns it
        }
        idx = (idx + 1) & a.cap_mask;
    }
    atomicCAS(a.status, 0, (int)ATTT_ERR_TABLE_FULL);
    return nullptr;
}

// One update: copies the text into the arena, finds its words, records them
// in the index and counts |W(x_k)| and |W(x_k) & W(x_i)|; the last block to
// finish applies Eq. 6 / Eq. 7 and the filter.
//
// Each block takes chunks of 256 to 2,048 bytes of the text.  Word starts go to a list
// in shared memory; each word goes through record_word (a word repeated
// inside the chunk costs one global probe instead of one per occurrence: Zipf
// text repeats its frequent words many times per chunk).  The owners of
// words of W(x_k) add one to |W(x_k) & W(x_i)| for every earlier update i
// whose bit their mask has: one warp ballot per bit set in any lane, added by
// one lane into a shared-memory histogram per block, flushed once.
__global__ void __launch_bounds__(kInsThreads) repetition_kernel(RepArgs a) {
    extern __shared__ unsigned int s_inter[];  // [k]
    __shared__ unsigned long long s_key[kLocalSlots];
    __shared__ uint32_t s_start[kChunkWords];
    __shared__ unsigned int s_nstart, s_distinct;
    __shared__ float s_max[kInsThreads / 32];
    __shared__ int s_last;
    const TextView v{a.arena, a.text, a.base, a.n};
    for (int i = threadIdx.x; i < a.k; i += blockDim.x) s_inter[i] = 0u;
    if (threadIdx.x == 0) s_distinct = 0u;

    const int kw = a.k >> 6;
    const unsigned long long kbit = 1ull << (a.k & 63);
    for (int64_t c0 = (int64_t)blockIdx.x * a.chunk; c0 < a.n; c0 += (int64_t)gridDim.x * a.chunk) {
        for (int i = threadIdx.x; i < kLocalSlots; i += blockDim.x) s_key[i] = 0ull;
        if (threadIdx.x == 0) s_nstart = 0u;
        __syncthreads();
        const int cn = (int)(a.n - c0 < a.chunk ? a.n - c0 : a.chunk);
        for (int i = threadIdx.x; i < cn; i += blockDim.x) {
            const int64_t off = c0 + i;
            const unsigned int b = a.text[off];
            a.arena[a.base + off] = (uint8_t)b;
            const unsigned int prev = off == 0 ? 0x20u : (unsigned int)a.text[off - 1];
            if (!is_space(b) && is_space(prev)) s_start[atomicAdd(&s_nstart, 1u)] = (uint32_t)i;
        }
        __syncthreads();
        const int ns = (int)s_nstart;
        // rounds of blockDim.x words, so that whole warps reach the counting
        // step together
        for (int w0 = 0; w0 < ns; w0 += blockDim.x) {
            const int w = w0 + threadIdx.x;
            const unsigned long long *m = nullptr;  // this lane's word of x_k, if it owns one
            unsigned long long old = 0ull;
            if (w < ns) m = record_word(a, v, c0, s_start[w], s_key, kw, kbit, &old);
            const bool own = m != nullptr;
            if (own) atomicAdd(&s_distinct, 1u);
            __syncwarp();
            // |W(x_k) & W(x_i)| += number of owned words whose mask has bit i:
            // per mask word, one ballot per bit set in any lane
            for (int j = 0; j <= kw; ++j) {
                const unsigned long long bits = !own ? 0ull : (j == kw ? (old & (kbit - 1ull)) : __ldcg(m + j));
                const unsigned int lo = (unsigned int)bits, hi = (unsigned int)(bits >> 32);
                unsigned int any_lo = __reduce_or_sync(0xffffffffu, lo);
                unsigned int any_hi = __reduce_or_sync(0xffffffffu, hi);
                while (any_lo) {
                    const int b = __ffs((int)any_lo) - 1;
                    any_lo &= any_lo - 1u;
                    const unsigned int c = __popc(__ballot_sync(0xffffffffu, (lo >> b) & 1u));
                    if ((threadIdx.x & 31) == 0) atomicAdd(&s_inter[j * 64 + b], c);
                }
                while (any_hi) {
                    const int b = __ffs((int)any_hi) - 1;
                    any_hi &= any_hi - 1u;
                    const unsigned int c = __popc(__ballot_sync(0xffffffffu, (hi >> b) & 1u));
                    if ((threadIdx.x & 31) == 0) atomicAdd(&s_inter[j * 64 + 32 + b], c);
                }
            }
        }
        __syncthreads();
    }
    __syncthreads();
    for (int i = threadIdx.x; i < a.k; i += blockDim.x)
        if (s_inter[i]) atomicAdd(a.inter + i, s_inter[i]);
    if (threadIdx.x == 0 && s_distinct) atomicAdd(a.distinct, s_distinct);
    __threadfence();
    __syncthreads();
    if (threadIdx.x == 0) s_last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
    __syncthreads();
    if (!s_last) return;
    __threadfence();

    // Eq. 6 / Eq. 7 and the filter; clears the counters for the next update
    const unsigned int dk = __ldcg(a.distinct);
    float best = 0.0f;
    for (int i = threadIdx.x; i < a.k; i += blockDim.x) {
        const unsigned int it = __ldcg(a.inter + i);
        const unsigned int un = dk + a.sizes[i] - it;
        const float j = un ? __fdiv_rn((float)it, (float)un) : 0.0f;
        best = fmaxf(best, j);
        a.inter[i] = 0u;
    }
    for (int o = 16; o > 0; o >>= 1) best = fmaxf(best, __shfl_xor_sync(0xffffffffu, best, o));
    if ((threadIdx.x & 31) == 0) s_max[threadIdx.x >> 5] = best;
    __syncthreads();
    if (threadIdx.x == 0) {
        float rho = 0.0f;
        for (int w = 0; w < kInsThreads / 32; ++w) rho = fmaxf(rho, s_max[w]);
        const float nu = __fsub_rn(1.0f, rho);
        if (a.rho_out) *a.rho_out = rho;
        if (a.nu_out) *a.nu_out = nu;
        if (a.keep_out) *a.keep_out = (nu < a.tau) ? 0 : 1;
        a.sizes[a.k] = dk;
        *a.distinct = 0u;
        *a.ticket = 0u;
        a.arena[a.base + a.n] = 0x20;  // the separator after this text
    }
}

}  // namespace

struct attt_wordsets {
    int max_updates, W, count;
    int64_t arena_cap, len;
    uint8_t *d_arena;
    unsigned long long *d_keys, *d_masks;
    unsigned long long capacity;
    unsigned int *d_sizes, *d_inter, *d_distinct, *d_ticket;
    int *d_status;
};

extern "C" {

attt_status attt_wordsets_create(int max_updates, int64_t max_bytes, attt_wordsets **out) {
    using namespace attt;
    if (!out) return ATTT_ERR_INVALID_ARG;
    *out = nullptr;
    if (max_updates < 1 || max_updates > kMaxUpdates || max_bytes < 0 ||
        max_bytes > (int64_t)0xFFFFFFFEll - max_updates)
        return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    attt_wordsets *s = new (std::nothrow) attt_wordsets{};
    if (!s) return ATTT_ERR_CUDA;
    s->max_updates = max_updates;
    s->W = (max_updates + 63) / 64;
    s->arena_cap = max_bytes + max_updates;  // texts and one separator each
    const unsigned long long words = (unsigned long long)(s->arena_cap / 2 + 1);
    unsigned long long cap = 1024;
    while (cap < 2 * words) cap <<= 1;
    s->capacity = cap;
    bool ok = cudaMalloc(&s->d_arena, (size_t)s->arena_cap) == cudaSuccess &&
              cudaMalloc(&s->d_keys, cap * sizeof(unsigned long long)) == cudaSuccess &&
              cudaMalloc(&s->d_masks, cap * s->W * sizeof(unsigned long long)) == cudaSuccess &&
              cudaMalloc(&s->d_sizes, (size_t)max_updates * sizeof(unsigned int)) == cudaSuccess &&
              cudaMalloc(&s->d_inter, (size_t)max_updates * sizeof(unsigned int)) == cudaSuccess &&
              cudaMalloc(&s->d_distinct, sizeof(unsigned int)) == cudaSuccess &&
              cudaMalloc(&s->d_ticket, sizeof(unsigned int)) == cudaSuccess &&
              cudaMalloc(&s->d_status, sizeof(int)) == cudaSuccess;
    ok = ok && cudaMemset(s->d_keys, 0, cap * sizeof(unsigned long long)) == cudaSuccess &&
         cudaMemset(s->d_masks, 0, cap * s->W * sizeof(unsigned long long)) == cudaSuccess &&
         cudaMemset(s->d_inter, 0, (size_t)max_updates * sizeof(unsigned int)) == cudaSuccess &&
         cudaMemset(s->d_distinct, 0, sizeof(unsigned int)) == cudaSuccess &&
         cudaMemset(s->d_ticket, 0, sizeof(unsigned int)) == cudaSuccess &&
         cudaMemset(s->d_status, 0, sizeof(int)) == cudaSuccess && cudaDeviceSynchronize() == cudaSuccess;
    if (!ok) {
        cudaFree(s->d_arena); cudaFree(s->d_keys); cudaFree(s->d_masks); cudaFree(s->d_sizes);
        cudaFree(s->d_inter); cudaFree(s->d_distinct); cudaFree(s->d_ticket); cudaFree(s->d_status);
        delete s;
        return ATTT_ERR_CUDA;
    }
    *out = s;
    return ATTT_OK;
}

attt_status attt_wordsets_destroy(attt_wordsets *s) {
    if (!s) return ATTT_ERR_INVALID_ARG;
    cudaDeviceSynchronize();
    cudaFree(s->d_arena); cudaFree(s->d_keys); cudaFree(s->d_masks); cudaFree(s->d_sizes);
    cudaFree(s->d_inter); cudaFree(s->d_distinct); cudaFree(s->d_ticket); cudaFree(s->d_status);
    delete s;
    return ATTT_OK;
}

attt_status attt_wordsets_reset(attt_wordsets *s, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!s) return ATTT_ERR_INVALID_ARG;
    if (cudaMemsetAsync(s->d_keys, 0, s->capacity * sizeof(unsigned long long), stream) != cudaSuccess ||
        cudaMemsetAsync(s->d_masks, 0, s->capacity * s->W * sizeof(unsigned long long), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    s->len = 0;
    s->count = 0;
    return ATTT_OK;
}

int attt_wordsets_updates(const attt_wordsets *s) { return s ? s->count : -1; }

attt_status attt_wordsets_status(attt_wordsets *s, attt_stream stream) {
    if (!s) return ATTT_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return ATTT_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, s->d_status, sizeof(int), cudaMemcpyDeviceToHost) != cudaSuccess ||
        cudaMemset(s->d_status, 0, sizeof(int)) != cudaSuccess)
        return ATTT_ERR_CUDA;
    return (attt_status)v;
}

attt_status attt_repetition(attt_wordsets *s, const uint8_t *d_text, int64_t nbytes, float tau, float *d_rho,
                            float *d_nu, int32_t *d_keep, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!s || nbytes < 0 || (nbytes > 0 && !d_text) || !(tau == tau)) return ATTT_ERR_INVALID_ARG;
    if (s->count >= s->max_updates || s->len + nbytes + 1 > s->arena_cap) return ATTT_ERR_CAPACITY;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    RepArgs a{};
    a.text = d_text; a.n = nbytes; a.arena = s->d_arena; a.base = s->len; a.k = s->count; a.W = s->W;
    a.keys = s->d_keys; a.masks = s->d_masks; a.cap_mask = s->capacity - 1;
    a.sizes = s->d_sizes; a.inter = s->d_inter; a.distinct = s->d_distinct; a.ticket = s->d_ticket;
    a.status = s->d_status; a.tau = tau; a.rho_out = d_rho; a.nu_out = d_nu; a.keep_out = d_keep;
    // chunks of 256..2048 bytes: a short text spreads over the SMs (each block
    // then takes its words in one round), a long one keeps whole chunks
    const int64_t sms = num_sms(dev);
    a.chunk = (int)(round_up(cdiv(nbytes, sms), 256) < kChunk ? round_up(cdiv(nbytes, sms), 256) : kChunk);
    if (a.chunk < 256) a.chunk = 256;
    int64_t blocks = cdiv(nbytes, a.chunk);
    if (blocks > sms * 4) blocks = sms * 4;
    if (blocks < 1) blocks = 1;
    repetition_kernel<<<(unsigned)blocks, kInsThreads, (size_t)a.k * sizeof(unsigned int), stream>>>(a);
    count_launch();
    if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    s->count = a.k + 1;
    s->len += nbytes + 1;
    return ATTT_OK;
}

}  // extern "C"
