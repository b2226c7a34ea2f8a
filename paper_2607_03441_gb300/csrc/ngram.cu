// ngram.cu -- Eq. 8 / Eq. 9 of aTTT on the GPU: the episode's token history
// H (a concatenation of earlier update texts, Sec. 3.3), an exact n-gram
// count table over it, and the per-token loss weights of an update.
//
// Table design (GB300-first):
//   * open addressing, linear probing, power-of-two capacity >= 4 * max_tokens
//     (load factor <= 1/4: a new n-gram then takes ~1.4 probes, against ~2.5
//     at 1/2) of 8-byte slots, one 64-bit word each:
//       [63:48] 16-bit hash tag | [47:24] history position + 1 of the
//       n-gram's first occurrence | [23:0] count
//     (0 = empty).  A new n-gram costs one CAS that claims the slot with its
//     count already set; a repeat costs one atomic add on the same word.  The
//     history is therefore limited to 2^24 - 2 tokens (count and position fit
//     24 bits).  Equality is decided by comparing the n tokens in the
//     device-resident history stream (exact, any vocabulary, any n up to 16)
//     after a tag match;
//   * lookups are warp-cooperative: eight lanes load eight consecutive
//     slots of an n-gram's probe run at once and ballots find the empty
//     slots and the tag matches, which the group then checks token by token
//     together (one round trip to the table, one per candidate);
//   * the weights kernel stages the update's tokens for a block in shared
//     memory with coalesced loads, looks up each window once, takes the
//     window max of the counts from shared memory and applies Eq. 9 with an
//     IEEE round-to-nearest division (bit-exact with the definition).
#include <cuda_runtime.h>

#include <new>

#include "attt_common.cuh"
#include "attt_host.h"

namespace attt {

typedef unsigned long long Slot;  // tag16 | pos24 | count24, 0 = empty

constexpr int kMaxN = 16;
constexpr int64_t kMaxHistory = (1ll << 24) - 2;

__device__ __forceinline__ unsigned int slot_tag(unsigned long long hsh) { return (unsigned int)(hsh >> 48); }
__device__ __forceinline__ unsigned int slot_pos(Slot k) { return (unsigned int)((k >> 24) & 0xFFFFFFu) - 1u; }
__device__ __forceinline__ unsigned int slot_count(Slot k) { return (unsigned int)(k & 0xFFFFFFu); }
constexpr int kMaxProbe = 1 << 16;

__device__ __forceinline__ unsigned long long mix64(unsigned long long h) {
    h ^= h >> 33;
    h *= 0xff51afd7ed558ccdull;
    h ^= h >> 33;
    h *= 0xc4ceb9fe1a85ec53ull;
    h ^= h >> 33;
    return h;
}

// Hash of n consecutive tokens: one odd 64-bit multiply per token (each step
// a bijection of the state), then one finalizer so that the low bits (the
// slot) and the top 16 bits (the tag) depend on every token.
__device__ __forceinline__ unsigned long long ngram_hash(const int32_t *t, int n) {
    unsigned long long h = 0x9e3779b97f4a7c15ull * (unsigned long long)(n + 1);
    for (int i = 0; i < n; ++i) h = (h ^ (unsigned long long)(uint32_t)t[i]) * 0xbf58476d1ce4e5b9ull;
    return mix64(h);
}

// Lookups are warp-cooperative: a group of kProbeLanes lanes takes one
// n-gram and loads kProbeLanes consecutive slots of its probe sequence at
// once (one 64-byte window, at most three 32-byte sectors), and ballots give
// the group the empty slots and the tag matches.  The candidates are the
// tag matches before the first empty slot (linear probing places an n-gram
// before any slot that was empty when it was inserted); each is checked by
// the group together, lane j comparing tokens j and j + 8, and one more
// ballot.  A lookup thus costs one round trip to the table and one to the
// history per candidate, however long the probe run.
constexpr int kProbeLanes = 8;

// Count of the n-gram g (n tokens in shared or global memory) with hash hsh,
// for the group of kProbeLanes lanes that holds it; lanes of groups with
// active == false take part in the ballots only.  Every lane of the warp
// calls it (the ballots are over the full warp); the result is returned to
// every lane of the group.
__device__ __forceinline__ unsigned int group_lookup(const Slot *table, unsigned long long mask,
                                                     const int32_t *hist, const int32_t *g, int n,
                                                     unsigned long long hsh, int64_t hist_len, bool active,
                                                     int *status) {
    const int lane = threadIdx.x & 31;
    const int j = lane & (kProbeLanes - 1);
    const int gsh = lane & ~(kProbeLanes - 1);  // first lane of the group, and its ballot shift
    const unsigned int tag = slot_tag(hsh);
    unsigned long long base = hsh & mask;
    unsigned int result = 0u;
    // the n-gram's tokens this lane compares: j and j + 8 (n <= 16)
    const int32_t g0 = (active && j < n) ? g[j] : 0;
    const int32_t g1 = (active && j + kProbeLanes < n) ? g[j + kProbeLanes] : 0;
    for (int round = 0; round < kMaxProbe / kProbeLanes; ++round) {
        if (!__any_sync(0xffffffffu, active)) break;
        const Slot k = active ? __ldcg(table + ((base + j) & mask)) : 0ull;
        const unsigned int empty = (__ballot_sync(0xffffffffu, active && k == 0ull) >> gsh) & 0xFFu;
        const unsigned int hit =
            (__ballot_sync(0xffffffffu, active && k != 0ull && (unsigned int)(k >> 48) == tag) >> gsh) & 0xFFu;
        const int stop = empty ? __ffs(empty) - 1 : kProbeLanes;
        unsigned int cand = hit & ((1u << stop) - 1u);
        bool found = false;
        // the candidates in probe order, one group-wide token compare each
        for (;;) {
            const bool have = cand != 0u;
            if (!__any_sync(0xffffffffu, have)) break;
            const int src = gsh + (have ? __ffs(cand) - 1 : 0);
            const Slot kc = __shfl_sync(0xffffffffu, k, src);
            const int64_t pos = (int64_t)slot_pos(kc);
            bool ok = have && ATTT_GUARD(pos + n <= hist_len, status);
            if (ok && j < n) ok = __ldcg(hist + pos + j) == g0;
            if (ok && j + kProbeLanes < n) ok = __ldcg(hist + pos + j + kProbeLanes) == g1;
            const unsigned int bad = (__ballot_sync(0xffffffffu, have && !ok) >> gsh) & 0xFFu;
            if (have && bad == 0u) {
                result = slot_count(kc);
                found = true;
                cand = 0u;
            } else if (have) {
                cand &= cand - 1u;
            }
        }
        if (active) {
            if (found || empty) active = false;
            else base += kProbeLanes;
        }
    }
    return result;
}

// The history stream during an insert: positions below old_len from the
// stream itself, the appended tokens from the caller's buffer (src; null when
// they are already in the stream), which the insert kernel copies into the
// stream as it goes, so nothing of that launch reads them there.
struct HistTokens {
    const int32_t *hist;
    const int32_t *src;
    int64_t old_len;
    __device__ __forceinline__ int32_t at(int64_t pos) const {
        return (src && pos >= old_len) ? __ldg(src + (pos - old_len)) : hist[pos];
    }
};

__device__ __forceinline__ bool ngram_equal_at(const HistTokens &ht, int64_t pos, const int32_t *g, int n) {
    for (int i = 0; i < n; ++i)
        if (ht.at(pos + i) != g[i]) return false;
    return true;
}

// Inserts one occurrence (at history position p) of the n-gram g with hash
// hsh, starting from the result k of the optimistic claim of slot idx.
__device__ __forceinline__ bool insert_rest(Slot *table, unsigned long long mask, const HistTokens &ht,
                                            const int32_t *g, int n, unsigned long long hsh, Slot claim,
                                            unsigned long long idx, Slot k, int64_t hist_len, int *status) {
    const unsigned int tag = slot_tag(hsh);
    for (int probe = 0; probe < kMaxProbe; ++probe) {
        if (k == 0ull) return true;  // claimed with count 1
        if ((unsigned int)(k >> 48) == tag && ATTT_GUARD((int64_t)slot_pos(k) + n <= hist_len, status) &&
            ngram_equal_at(ht, slot_pos(k), g, n)) {
            atomicAdd(table + idx, 1ull);  // count lives in the low 24 bits
            return true;
        }
        idx = (idx + 1) & mask;
        k = atomicCAS(table + idx, 0ull, claim);
    }
    return false;
}

// kInsPer new n-gram start positions per thread, p = p_begin + blockIdx.x *
// kInsTile + k * blockDim.x + threadIdx.x.  The block's tokens are staged in
// shared memory (coalesced); each thread hashes its n-gram there and makes
// the optimistic claim (atomicCAS of an empty slot with count 1); an occupied
// slot returns its word, which is then compared.  Measured on the 1 M-token
// stress history: 2, 4 or 8 n-grams per thread (their claims in flight
// together) were slower than one (the insert is bound by L2 atomic throughput,
// ~88 G random 64-bit CAS/s measured alone, not by a thread's latency), and a
// load factor of 1/4 instead of 1/2 took it from 42-51 to 32-35 us.
// (Aggregating equal n-grams inside a warp with match_any cost more than the
// atomics it saves on Zipf text, so every occurrence is inserted.)
constexpr int kInsPer = 1;
constexpr int kInsTile = 256 * kInsPer;

// One block of history_insert_kernel's work: new n-gram starts
// p = p_begin + blk * kInsTile + threadIdx.x, p - p_begin < count.
__device__ __forceinline__ void insert_block(const HistTokens &ht, int64_t p_begin, int64_t count, int n,
                                             Slot *table, unsigned long long mask, int *status, int64_t blk) {
    __shared__ int32_t tok[kInsTile + kMaxN];
    const int64_t i0 = blk * kInsTile;
    const int64_t rem = count - i0;
    const int nt = (int)(rem < kInsTile ? rem : kInsTile) + n - 1;  // tokens of this block's n-grams
    for (int t = threadIdx.x; t < nt; t += blockDim.x) tok[t] = ht.at(p_begin + i0 + t);
    __syncthreads();
    unsigned long long hsh[kInsPer], idx[kInsPer];
    Slot claim[kInsPer], k[kInsPer];
#pragma unroll
    for (int q = 0; q < kInsPer; ++q) {
        const int li = q * blockDim.x + threadIdx.x;
        if (i0 + li < count) {
            hsh[q] = ngram_hash(tok + li, n);
            idx[q] = hsh[q] & mask;
            claim[q] = ((unsigned long long)slot_tag(hsh[q]) << 48) |
                       ((unsigned long long)(uint32_t)(p_begin + i0 + li + 1) << 24) | 1ull;
            k[q] = atomicCAS(table + idx[q], 0ull, claim[q]);
        }
    }
#pragma unroll
    for (int q = 0; q < kInsPer; ++q) {
        const int li = q * blockDim.x + threadIdx.x;
        if (i0 + li < count && !insert_rest(table, mask, ht, tok + li, n, hsh[q], claim[q], idx[q], k[q],
                                            p_begin + count + n - 1, status))
            record_error(status, ATTT_ERR_TABLE_FULL);
    }
}

// src (may be null): the appended tokens, new_len - old_len of them, not yet
// in the stream; the launch copies them to hist[old_len, new_len) besides
// inserting (one D2D copy fewer per append).
__global__ void __launch_bounds__(256) history_insert_kernel(int32_t *hist, const int32_t *__restrict__ src,
                                                             int64_t old_len, int64_t new_len, int64_t p_begin,
                                                             int64_t count, int n, Slot *table,
                                                             unsigned long long mask, int *status) {
    if (src) {
        const int64_t stride = (int64_t)gridDim.x * blockDim.x;
        for (int64_t j = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; j < new_len - old_len; j += stride)
            hist[old_len + j] = __ldg(src + j);
    }
    const HistTokens ht{hist, src, src ? old_len : INT64_MAX};
    insert_block(ht, p_begin, count, n, table, mask, status, blockIdx.x);
}

// The histories of a batch of episodes (one per blockIdx.y).
constexpr int kMaxBatch = 32;
struct InsertBatch {
    const int32_t *hist[kMaxBatch];
    Slot *table[kMaxBatch];
    unsigned long long mask[kMaxBatch];
    int *status[kMaxBatch];
    int64_t p_begin[kMaxBatch], count[kMaxBatch];
    int n;
};

__global__ void __launch_bounds__(256) history_insert_batch_kernel(const __grid_constant__ InsertBatch b) {
    const int e = blockIdx.y;
    if ((int64_t)blockIdx.x * kInsTile >= b.count[e]) return;
    const HistTokens ht{b.hist[e], nullptr, INT64_MAX};
    insert_block(ht, b.p_begin[e], b.count[e], b.n, b.table[e], b.mask[e], b.status[e], blockIdx.x);
}

// count(g, H) for m query n-grams stored row-major [m, n], one probe group
// per query.
__global__ void __launch_bounds__(256) history_count_kernel(const int32_t *__restrict__ hist, int64_t hist_len,
                                                            const Slot *table, unsigned long long mask,
                                                            const int32_t *__restrict__ q, int64_t m, int n,
                                                            unsigned int *out, int *status) {
    const int64_t i = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) / kProbeLanes;
    const bool active = i < m;
    const int32_t *g = q + (active ? i : 0) * n;
    const unsigned int c = group_lookup(table, mask, hist, g, n, active ? ngram_hash(g, n) : 0ull, hist_len,
                                        active, status);
    if (active && (threadIdx.x & (kProbeLanes - 1)) == 0) out[i] = c;
}

constexpr int kWTile = 48;                              // positions j per block
constexpr int kWWin = kWTile + kMaxN;                       // candidate windows (at most kWTile + n - 1)
constexpr int kWThreads = kProbeLanes * kWWin;              // one probe group per window

// Eq. 8 then Eq. 9 for positions [j0, j0 + kWTile) of the update.  Each
// window has its own probe group, so a block's critical path is one
// cooperative lookup; the window max and Eq. 9 take one thread per position.
// rowscale (may be null) receives `scale` at every position written.
__device__ __forceinline__ void weights_block(const int32_t *__restrict__ x, int64_t L, int n,
                                              const int32_t *__restrict__ hist, int64_t hist_len, const Slot *table,
                                              unsigned long long mask, float w_min, float *__restrict__ w,
                                              float *__restrict__ rowscale, float scale, int64_t j0) {
    __shared__ int32_t tok[kWTile + 2 * kMaxN];
    __shared__ unsigned int cnt[kWWin];
    // Window starts s that cover some j in the tile: s in [j0-n+1, j0+kWTile-1]
    // clipped to [0, L-n].  Tokens needed: x[s0 .. s1+n-1].
    const int64_t s_lo = j0 - (n - 1);
    const int nwin = kWTile + n - 1;  // candidate windows, indexed by s - s_lo
    // stage tokens x[s_lo .. s_lo + nwin + n - 2] (coalesced)
    const int ntok = nwin + n - 1;
    for (int i = threadIdx.x; i < ntok; i += blockDim.x) {
        const int64_t pos = s_lo + i;
        tok[i] = (pos >= 0 && pos < L) ? __ldg(x + pos) : 0;
    }
    __syncthreads();
    const int i = threadIdx.x / kProbeLanes;  // this lane's window
    const int64_t s = s_lo + i;
    const bool valid = i < nwin && s >= 0 && s + n <= L && hist_len >= n;
    const unsigned long long hsh = valid ? ngram_hash(tok + i, n) : 0ull;
    const unsigned int c = group_lookup(table, mask, hist, tok + (valid ? i : 0), n, hsh, hist_len, valid, nullptr);
    if ((threadIdx.x & (kProbeLanes - 1)) == 0 && i < nwin) cnt[i] = c;
    __syncthreads();
    const int64_t j = j0 + threadIdx.x;
    if (threadIdx.x >= kWTile || j >= L) return;
    // windows covering j: s in [j-n+1, j], i.e. indices [threadIdx.x, threadIdx.x + n - 1];
    // invalid windows (s < 0 or s > L-n) hold count 0, which never changes the max.
    unsigned int f = 0u;
    for (int k = 0; k < n; ++k) f = max(f, cnt[threadIdx.x + k]);
    const float q = __fdiv_rn(1.0f, __fadd_rn(1.0f, __uint2float_rn(f)));
    w[j] = fmaxf(w_min, q);
    if (rowscale) rowscale[j] = scale;
}

__global__ void __launch_bounds__(kWThreads) ngram_weights_kernel(const int32_t *__restrict__ x, int64_t L, int n,
                                                               const int32_t *__restrict__ hist, int64_t hist_len,
                                                               const Slot *table, unsigned long long mask,
                                                               float w_min, float *__restrict__ w) {
    weights_block(x, L, n, hist, hist_len, table, mask, w_min, w, nullptr, 0.0f, (int64_t)blockIdx.x * kWTile);
}

// The updates of a batch of episodes (one per blockIdx.y), each against its
// own history; rowscale[j] = 1 / L_e for every row of episode e.
struct WeightsBatch {
    const int32_t *x[kMaxBatch];
    int64_t L[kMaxBatch];
    const int32_t *hist[kMaxBatch];
    int64_t hist_len[kMaxBatch];
    const Slot *table[kMaxBatch];
    unsigned long long mask[kMaxBatch];
    float *w[kMaxBatch];
    float *rowscale[kMaxBatch];
    float inv_L[kMaxBatch];
    int n;
    float w_min;
};

__global__ void __launch_bounds__(kWThreads) ngram_weights_batch_kernel(const __grid_constant__ WeightsBatch b) {
    const int e = blockIdx.y;
    const int64_t j0 = (int64_t)blockIdx.x * kWTile;
    if (j0 >= b.L[e]) return;
    weights_block(b.x[e], b.L[e], b.n, b.hist[e], b.hist_len[e], b.table[e], b.mask[e], b.w_min, b.w[e],
                  b.rowscale[e], b.inv_L[e], j0);
}

}  // namespace attt

// ---------------------------------------------------------------------------
// C ABI
// ---------------------------------------------------------------------------

struct attt_history {
    int n;
    int device;
    int64_t max_tokens;
    int64_t len;
    int32_t *d_tokens;
    attt::Slot *d_table;
    unsigned long long capacity;
    int *d_status;
};

extern "C" {

attt_status attt_history_create(int n, int64_t max_tokens, attt_history **out) {
    if (!out || n < 1 || n > attt::kMaxN || max_tokens < 0 || max_tokens > attt::kMaxHistory)
        return ATTT_ERR_INVALID_ARG;
    *out = nullptr;
    int dev;
    attt_status st = attt::current_device(&dev);
    if (st != ATTT_OK) return st;
    unsigned long long cap = 1024;
    while (cap < 4ull * (unsigned long long)max_tokens) cap <<= 1;
    attt_history *h = new (std::nothrow) attt_history();
    if (!h) return ATTT_ERR_CUDA;
    h->n = n;
    h->device = dev;
    h->max_tokens = max_tokens;
    h->len = 0;
    h->capacity = cap;
    if (cudaMalloc(&h->d_tokens, (size_t)(max_tokens > 0 ? max_tokens : 1) * sizeof(int32_t)) != cudaSuccess ||
        attt::fault_take(attt::FAULT_ALLOC) ||  // an injected allocation failure
        cudaMalloc(&h->d_table, cap * sizeof(attt::Slot)) != cudaSuccess ||
        cudaMalloc(&h->d_status, 256) != cudaSuccess) {
        cudaFree(h->d_tokens);
        cudaFree(h->d_table);
        cudaFree(h->d_status);
        delete h;
        return ATTT_ERR_CUDA;
    }
    if (cudaMemset(h->d_table, 0, cap * sizeof(attt::Slot)) != cudaSuccess ||
        cudaMemset(h->d_status, 0, 256) != cudaSuccess) {
        cudaFree(h->d_tokens);
        cudaFree(h->d_table);
        cudaFree(h->d_status);
        delete h;
        return ATTT_ERR_CUDA;
    }
    *out = h;
    return ATTT_OK;
}

attt_status attt_history_destroy(attt_history *h) {
    if (!h) return ATTT_ERR_INVALID_ARG;
    int prev = -1;
    cudaGetDevice(&prev);
    cudaSetDevice(h->device);
    cudaDeviceSynchronize();
    cudaFree(h->d_tokens);
    cudaFree(h->d_table);
    cudaFree(h->d_status);
    if (prev >= 0) cudaSetDevice(prev);
    delete h;
    return ATTT_OK;
}

attt_status attt_history_reset(attt_history *h, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!h) return ATTT_ERR_INVALID_ARG;
    if (cudaMemsetAsync(h->d_table, 0, h->capacity * sizeof(attt::Slot), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    h->len = 0;
    return ATTT_OK;
}

int64_t attt_history_length(const attt_history *h) { return h ? h->len : -1; }

int attt_history_ngram(const attt_history *h) { return h ? h->n : -1; }

attt_status attt_history_insert(attt_history *h, const int32_t *d_tokens, int64_t len, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!h || len < 0 || (len > 0 && !d_tokens)) return ATTT_ERR_INVALID_ARG;
    if (len == 0) return ATTT_OK;
    if (h->len + len > h->max_tokens) return ATTT_ERR_CAPACITY;
    const int64_t old_len = h->len;
    const int64_t new_len = h->len + len;
    // New n-grams: every start p whose last token p+n-1 is new, i.e.
    // p in [max(0, old_len - n + 1), new_len - n].
    int64_t p_begin = h->len - (h->n - 1);
    if (p_begin < 0) p_begin = 0;
    const int64_t p_end = new_len - h->n;  // inclusive
    h->len = new_len;
    if (p_end < p_begin)  // no new n-gram: the tokens only
        return cudaMemcpyAsync(h->d_tokens + old_len, d_tokens, (size_t)len * sizeof(int32_t),
                               cudaMemcpyDeviceToDevice, stream) == cudaSuccess
                   ? ATTT_OK
                   : ATTT_ERR_CUDA;
    const int64_t count = p_end - p_begin + 1;
    if (attt::fault_take(attt::FAULT_TABLE_FULL)) {
        // an injected full table: the status word reports it as the kernel would
        // (the tokens are still appended)
        static const int code = ATTT_ERR_TABLE_FULL;
        return cudaMemcpyAsync(h->d_tokens + old_len, d_tokens, (size_t)len * sizeof(int32_t),
                               cudaMemcpyDeviceToDevice, stream) == cudaSuccess &&
                       cudaMemcpyAsync(h->d_status, &code, sizeof code, cudaMemcpyHostToDevice, stream) == cudaSuccess
                   ? ATTT_OK
                   : ATTT_ERR_CUDA;
    }
    const int threads = 256;
    const int64_t blocks = (count + attt::kInsTile - 1) / attt::kInsTile;
    attt::history_insert_kernel<<<(unsigned)blocks, threads, 0, stream>>>(h->d_tokens, d_tokens, old_len, new_len,
                                                                          p_begin, count, h->n, h->d_table,
                                                                          h->capacity - 1, h->d_status);
    attt::count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status attt_history_save(const attt_history *h, int32_t *host_tokens, attt_stream stream) {
    if (!h || (h->len > 0 && !host_tokens)) return ATTT_ERR_INVALID_ARG;
    if (h->len == 0) return ATTT_OK;
    if (cudaMemcpyAsync(host_tokens, h->d_tokens, (size_t)h->len * sizeof(int32_t), cudaMemcpyDeviceToHost,
                        stream) != cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    return ATTT_OK;
}

attt_status attt_history_restore(attt_history *h, const int32_t *host_tokens, int64_t len, attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!h || len < 0 || (len > 0 && !host_tokens)) return ATTT_ERR_INVALID_ARG;
    if (len > h->max_tokens) return ATTT_ERR_CAPACITY;
    attt_status st = attt_history_reset(h, stream);
    if (st != ATTT_OK || len == 0) return st;
    if (cudaMemcpyAsync(h->d_tokens, host_tokens, (size_t)len * sizeof(int32_t), cudaMemcpyHostToDevice, stream) !=
            cudaSuccess ||
        cudaStreamSynchronize(stream) != cudaSuccess)  // the host buffer may go once this returns
        return ATTT_ERR_CUDA;
    // every n-gram of the restored stream, as one insert from an empty history
    h->len = len;
    const int64_t count = len - h->n + 1;
    if (count <= 0) return ATTT_OK;
    attt::history_insert_kernel<<<(unsigned)((count + attt::kInsTile - 1) / attt::kInsTile), 256, 0, stream>>>(
        h->d_tokens, nullptr, len, len, 0, count, h->n, h->d_table, h->capacity - 1, h->d_status);
    attt::count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status attt_history_status(attt_history *h, attt_stream stream) {
    if (!h) return ATTT_ERR_INVALID_ARG;
    if (cudaStreamSynchronize(stream) != cudaSuccess) return ATTT_ERR_CUDA;
    int v = 0;
    if (cudaMemcpy(&v, h->d_status, sizeof v, cudaMemcpyDeviceToHost) != cudaSuccess) return ATTT_ERR_CUDA;
    if (v != 0 && cudaMemset(h->d_status, 0, sizeof v) != cudaSuccess) return ATTT_ERR_CUDA;
    return (attt_status)v;
}

attt_status attt_history_count(const attt_history *h, const int32_t *d_ngrams, int64_t m, uint32_t *d_counts,
                               attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!h || m < 0 || (m > 0 && (!d_ngrams || !d_counts))) return ATTT_ERR_INVALID_ARG;
    if (m == 0) return ATTT_OK;
    const int threads = 256;
    const int64_t per_block = threads / attt::kProbeLanes;
    attt::history_count_kernel<<<(unsigned)((m + per_block - 1) / per_block), threads, 0, stream>>>(
        h->d_tokens, h->len, h->d_table, h->capacity - 1, d_ngrams, m, h->n, d_counts, h->d_status);
    attt::count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // extern "C"

namespace attt {

// Eq. 8 / Eq. 9 weights of E updates (rows [off[e], off[e+1]) of d_tokens,
// against history hs[e]) in one launch; rowscale[j] = 1/L_e (fp32 round to
// nearest of 1.0f / L_e) for every row of episode e.
attt_status ngram_weights_batch(attt_history *const *hs, int E, const int32_t *d_tokens, const int64_t *off,
                                float w_min, float *d_w, float *d_rowscale, cudaStream_t stream) {
    if (E < 1 || E > kMaxBatch || !(w_min > 0.0f) || !(w_min <= 1.0f)) return ATTT_ERR_INVALID_ARG;
    WeightsBatch b{};
    b.n = hs[0]->n;
    b.w_min = w_min;
    int64_t maxL = 0;
    for (int e = 0; e < E; ++e) {
        const attt_history *h = hs[e];
        if (h->n != b.n) return ATTT_ERR_INVALID_ARG;
        const int64_t L = off[e + 1] - off[e];
        b.x[e] = d_tokens + off[e];
        b.L[e] = L;
        b.hist[e] = h->d_tokens;
        b.hist_len[e] = h->len;
        b.table[e] = h->d_table;
        b.mask[e] = h->capacity - 1;
        b.w[e] = d_w + off[e];
        b.rowscale[e] = d_rowscale ? d_rowscale + off[e] : nullptr;
        b.inv_L[e] = L > 0 ? 1.0f / (float)L : 0.0f;
        if (L > maxL) maxL = L;
    }
    if (maxL == 0) return ATTT_OK;
    ngram_weights_batch_kernel<<<dim3((unsigned)cdiv(maxL, kWTile), (unsigned)E), kWThreads, 0, stream>>>(b);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

// Algorithm 1's append for E histories (rows [off[e], off[e+1]) of d_tokens
// to hs[e]): one copy per history, then one insert launch for all.
attt_status history_insert_batch(attt_history *const *hs, int E, const int32_t *d_tokens, const int64_t *off,
                                 cudaStream_t stream) {
    if (E < 1 || E > kMaxBatch) return ATTT_ERR_INVALID_ARG;
    for (int e = 0; e < E; ++e)
        if (hs[e]->len + (off[e + 1] - off[e]) > hs[e]->max_tokens) return ATTT_ERR_CAPACITY;
    InsertBatch b{};
    b.n = hs[0]->n;
    int64_t maxc = 0;
    for (int e = 0; e < E; ++e) {
        attt_history *h = hs[e];
        const int64_t len = off[e + 1] - off[e];
        b.hist[e] = h->d_tokens;
        b.table[e] = h->d_table;
        b.mask[e] = h->capacity - 1;
        b.status[e] = h->d_status;
        b.count[e] = 0;
        if (len == 0) continue;
        if (cudaMemcpyAsync(h->d_tokens + h->len, d_tokens + off[e], (size_t)len * sizeof(int32_t),
                            cudaMemcpyDeviceToDevice, stream) != cudaSuccess)
            return ATTT_ERR_CUDA;
        const int64_t new_len = h->len + len;
        int64_t p_begin = h->len - (h->n - 1);
        if (p_begin < 0) p_begin = 0;
        const int64_t p_end = new_len - h->n;
        h->len = new_len;
        if (p_end >= p_begin) {
            b.p_begin[e] = p_begin;
            b.count[e] = p_end - p_begin + 1;
            if (b.count[e] > maxc) maxc = b.count[e];
        }
    }
    if (maxc == 0) return ATTT_OK;
    history_insert_batch_kernel<<<dim3((unsigned)cdiv(maxc, kInsTile), (unsigned)E), 256, 0, stream>>>(b);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // namespace attt

extern "C" {

attt_status attt_ngram_weights(const attt_history *h, const int32_t *d_tokens, int64_t L, float w_min, float *d_w,
                               attt_stream stream) {
    ATTT_NVTX_RANGE();
    if (!h || L < 0 || (L > 0 && (!d_tokens || !d_w)) || !(w_min > 0.0f) || !(w_min <= 1.0f))
        return ATTT_ERR_INVALID_ARG;
    if (L == 0) return ATTT_OK;
    const int64_t blocks = (L + attt::kWTile - 1) / attt::kWTile;
    attt::ngram_weights_kernel<<<(unsigned)blocks, attt::kWThreads, 0, stream>>>(
        d_tokens, L, h->n, h->d_tokens, h->len, h->d_table, h->capacity - 1, w_min, d_w);
    attt::count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // extern "C"
