/*
 * attt.h -- C ABI of libattt, the GB300 (sm_103a) hot path of the aTTT
 * in-episode update step ("Agentic Test-Time Training", Sec. 3.3,
 * Algorithm 1).
 *
 * One update k of Algorithm 1, in call order:
 *
 *   attt_ngram_weights      Algorithm 1's loop over j: Eq. 8 exposure f_k(j)
 *                           against the history table, then Eq. 9 weights.
 *   attt_weighted_ce_fwd_bwd  Eq. 10 loss and its gradient w.r.t. the final
 *                           hidden states (the input of the frozen LM head).
 *   attt_lora_grad          the adapter gradients of the Eq. 2 / Algorithm 1
 *                           gradient step, given the upstream gradient dy of
 *                           each adapted projection.
 *   attt_lora_step          the Eq. 2 SGD step on the adapter parameters.
 *   attt_lora_forward,      the adapted projection of a chained update (its
 *   attt_lora_input_grad    output feeds the LM head): forward and the
 *                           gradient of its input.
 *   attt_history_insert     Algorithm 1's last line: append x_k to the token
 *                           history H (a concatenation, Sec. 3.3).
 *
 * Conventions shared by every call:
 *   - Pointers named d_* are device pointers on the current CUDA device; the
 *     caller owns them.  The library owns only attt_history objects.
 *   - bf16 tensors are passed as attt_bf16 (the IEEE binary32 upper half).
 *   - Matrices are row-major with the last dimension contiguous.
 *   - Every call is asynchronous on `stream` (a cudaStream_t; NULL = the
 *     legacy default stream).  Argument errors are returned synchronously and
 *     launch nothing.  Errors found on the device set a per-device status
 *     word read by attt_device_status() (or attt_history_status()).
 *   - No call aborts, traps or throws.  Every device-side wait is bounded;
 *     a wait that runs out sets ATTT_ERR_TIMEOUT and the kernel returns.
 *   - Inputs must not alias outputs unless a call says so.
 *   - Calls may run concurrently on different streams when they share no
 *     written buffer: each its own outputs and workspace, and no history or
 *     episode object used by two of them at once (attt_lora_grad_noalloc's
 *     static scratch is one per device: its calls are serialised by the
 *     caller).  Kernel errors of either land in the same status word.
 */
#ifndef ATTT_H
#define ATTT_H

#include <stddef.h>
#include <stdint.h>

#if defined(__GNUC__)
#define ATTT_API __attribute__((visibility("default")))
#else
#define ATTT_API
#endif

#ifdef __cplusplus
extern "C" {
#endif

typedef uint16_t attt_bf16;              /* bf16 bit pattern */
typedef struct CUstream_st *attt_stream; /* same handle as cudaStream_t */

typedef enum attt_status {
    ATTT_OK = 0,
    ATTT_ERR_INVALID_ARG = 1,  /* null/misaligned pointer, bad size or mode    */
    ATTT_ERR_TABLE_FULL = 2,   /* history table probe sequence exhausted       */
    ATTT_ERR_TOKEN_RANGE = 3,  /* a CE target outside [0, V)                   */
    ATTT_ERR_TIMEOUT = 4,      /* a bounded device-side wait ran out           */
    ATTT_ERR_WORKSPACE = 5,    /* workspace missing or smaller than required   */
    ATTT_ERR_CUDA = 6,         /* a CUDA runtime call failed                   */
    ATTT_ERR_UNSUPPORTED = 7,  /* not a GB300-class (sm_103) device, or shape  */
    ATTT_ERR_CAPACITY = 8,     /* history would exceed its max_tokens          */
    ATTT_ERR_CHECK = 9         /* a bounds check of the checked build failed   */
} attt_status;

/* Human-readable name of a status code.  Never NULL. */
ATTT_API const char *attt_status_string(int status);

/* ABI version of this header (major * 100 + minor). */
ATTT_API int attt_abi_version(void);

/* Number of CUDA kernels this library has launched in this process (all
 * devices, all threads).  Host-side counter; copies and memsets issued by the
 * library are not kernels and are not counted. */
ATTT_API uint64_t attt_kernel_launches(void);

/*
 * Reads and clears the device-side status word of the current device after
 * synchronising `stream`.  Returns the first error any kernel of this library
 * recorded since the last read (ATTT_ERR_TIMEOUT, ATTT_ERR_TOKEN_RANGE), or
 * ATTT_ERR_CUDA if the synchronisation itself failed.
 */
ATTT_API attt_status attt_device_status(attt_stream stream);

/*
 * Failure-detection self-test: launches one kernel whose only wait (on an
 * mbarrier that nothing completes) runs out after the library's wall-clock
 * limit of 2 s, as any device-side wait of the library would, so the device
 * status word then reads ATTT_ERR_TIMEOUT (attt_device_status) and the
 * context stays usable.  No fault, trap or hang.  Async on `stream`.
 */
ATTT_API attt_status attt_selftest_wait_timeout(attt_stream stream);

/*
 * Host fault injection, for tests of the error paths: makes one pending
 * fault, taken by the first place of its kind that reaches it --
 *   "alloc"       the next device allocation of a create call fails (the call
 *                 frees what it had allocated and returns ATTT_ERR_CUDA);
 *   "table_full"  the next attt_history_insert that has n-grams to record
 *                 records none and sets ATTT_ERR_TABLE_FULL in the history's
 *                 status word, as a full probe sequence would;
 *   "none"        clears a pending fault.
 * The environment variable ATTT_FAULT=<site> sets one at the library's first
 * use.  ATTT_ERR_INVALID_ARG for another name.  Nothing runs on the GPU.
 */
ATTT_API attt_status attt_fault_inject(const char *site);

/* ------------------------------------------------------------------------ */
/* Token history H (Sec. 3.3: every earlier update's tokens of the episode, */
/* joined end to end) and its exact n-gram count table.                     */
/* ------------------------------------------------------------------------ */

typedef struct attt_history attt_history;

/*
 * Creates an empty history for n-grams of size n (1 <= n <= 16) that can
 * hold up to max_tokens tokens (0 <= max_tokens <= 16,777,214 = 2^24 - 2) on
 * the current device.  The library allocates the token stream (4 B/token)
 * and an exact n-gram count table of 8 B slots, at least four times as many slots
 * as max_tokens.  *out is set on success.  Allocation failure returns
 * ATTT_ERR_CUDA.
 */
ATTT_API attt_status attt_history_create(int n, int64_t max_tokens, attt_history **out);

/* Frees the history and its device memory (synchronises the device). */
ATTT_API attt_status attt_history_destroy(attt_history *h);

/*
 * Empties the history (an episode boundary: the adapter and the history are
 * reset between episodes, Sec. 4 / Appendix C).  Async on `stream`.
 */
ATTT_API attt_status attt_history_reset(attt_history *h, attt_stream stream);

/*
 * Algorithm 1, last line: H <- H || x_k.  Appends `len` tokens (any int32
 * values) from d_tokens and counts every n-gram whose last token is new,
 * including the n-1 n-grams that straddle the old tail and the new tokens,
 * so insert(a); insert(b) equals insert(a||b).  Counts are exact (keys are
 * compared token by token).  Returns ATTT_ERR_CAPACITY, launching nothing,
 * if the history would exceed max_tokens.  A full probe sequence sets
 * ATTT_ERR_TABLE_FULL in the history's status word.
 */
ATTT_API attt_status attt_history_insert(attt_history *h, const int32_t *d_tokens, int64_t len,
                                attt_stream stream);

/*
 * Checkpoint of a history: copies its token stream (attt_history_length
 * tokens, int32) to host_tokens and synchronises `stream`.  The counts need
 * no copy: attt_history_restore rebuilds them exactly from the stream.
 */
ATTT_API attt_status attt_history_save(const attt_history *h, int32_t *host_tokens, attt_stream stream);

/*
 * Empties the history, then makes it the history of the len tokens in
 * host_tokens (as one insert from empty: every count exact, so weights after
 * a save and restore are bit-identical).  Synchronises `stream` once the
 * tokens are on the device.  ATTT_ERR_CAPACITY if len > max_tokens.
 */
ATTT_API attt_status attt_history_restore(attt_history *h, const int32_t *host_tokens, int64_t len,
                                          attt_stream stream);

/* Current history length in tokens (host-side bookkeeping, no sync). */
ATTT_API int64_t attt_history_length(const attt_history *h);

/* n of the history. */
ATTT_API int attt_history_ngram(const attt_history *h);

/*
 * Synchronises `stream`, then reads and clears the history's device status
 * word (ATTT_ERR_TABLE_FULL, ATTT_ERR_TIMEOUT) and returns it.
 */
ATTT_API attt_status attt_history_status(attt_history *h, attt_stream stream);

/*
 * Eq. 8's count(g, H) for `m` n-grams: d_ngrams is [m, n] int32 (row i is one
 * n-gram), d_counts is [m] uint32.  Exact.  Async on `stream`.
 */
ATTT_API attt_status attt_history_count(const attt_history *h, const int32_t *d_ngrams, int64_t m,
                               uint32_t *d_counts, attt_stream stream);

/*
 * Algorithm 1's per-token loop (Eq. 8 then Eq. 9).  For the L tokens of the
 * update x_k in d_tokens (int32 [L]) writes d_w (fp32 [L]):
 *   c_s = count(x[s..s+n-1], H)                 for s = 0 .. L-n
 *   f_j = max{ c_s : max(0, j-n+1) <= s <= min(j, L-n) }   (0 if empty)
 *   w_j = max(w_min, 1.0f / (1.0f + (float)f_j))  -- IEEE fp32 RN divide
 * Bit-exact.  0 < w_min <= 1.  L >= 0 (L = 0 launches nothing).
 * H is not modified; positions of x_k do not count against themselves
 * (count runs over the previous updates only, Eq. 8).
 */
ATTT_API attt_status attt_ngram_weights(const attt_history *h, const int32_t *d_tokens, int64_t L,
                               float w_min, float *d_w, attt_stream stream);

/* ------------------------------------------------------------------------ */
/* Eq. 10: token-weighted next-token cross-entropy through the frozen LM    */
/* head, forward and backward, without materialising the [L, V] logits.     */
/* ------------------------------------------------------------------------ */

/*
 * Workspace bytes attt_weighted_ce_fwd_bwd needs for (L, d, V).
 */
ATTT_API size_t attt_ce_workspace_bytes(int64_t L, int64_t d, int64_t V);

/*
 * The largest attt_ce_workspace_bytes(L, d, V) over 1 <= L <= Lmax: one
 * workspace that serves every update length up to Lmax (the size is not
 * monotone in L, because the vocabulary chunk depends on L).  0 if Lmax < 1.
 * Host-only.
 */
ATTT_API size_t attt_ce_workspace_max_bytes(int64_t Lmax, int64_t d, int64_t V);

/*
 * With h = d_h (bf16 [L, d], row j is the state that predicts target x_j),
 * W = d_W (bf16 [V, d], the frozen LM head), z_j = h_j W^T:
 *   lse_j  = log sum_v exp(z_jv)
 *   *d_loss = (1/L) sum_j w_j (lse_j - z_{j, tgt_j})                 (Eq. 10)
 *   d_dh[j, :] = (w_j / L) (sum_v softmax(z_j)_v W_v - W_{tgt_j})     (fp32)
 * d_tgt int32 [L] in [0, V); d_w fp32 [L] (the Eq. 9 weights); d_lse fp32
 * [L] receives lse_j when not NULL.  No gradient for W (it is frozen; only
 * the adapter trains).  bf16 products, fp32 accumulation.
 * Requirements: L >= 1, V >= 1, d >= 8 and d % 8 == 0, d_h / d_W / d_dh
 * 16-byte aligned, d_ws at least attt_ce_workspace_bytes(L, d, V) bytes and
 * 256-byte aligned.  A target outside [0, V) sets ATTT_ERR_TOKEN_RANGE in the
 * device status word and makes the loss NaN.
 */
ATTT_API attt_status attt_weighted_ce_fwd_bwd(const attt_bf16 *d_h, const attt_bf16 *d_W,
                                     const int32_t *d_tgt, const float *d_w,
                                     int64_t L, int64_t d, int64_t V,
                                     float *d_loss, float *d_dh, float *d_lse,
                                     void *d_ws, size_t ws_bytes, attt_stream stream);

/* ------------------------------------------------------------------------ */
/* LoRA adapter gradients and the SGD step (Eq. 2; Appendix C adapter:       */
/* y = x W0 + s (x A) B with A [din, r], B [r, dout], s = alpha / r).        */
/* ------------------------------------------------------------------------ */

/*
 * Workspace bytes attt_lora_grad needs for `nproj` projections that share one
 * input x of shape [L, din], with output widths dout[0..nproj-1] and rank r.
 */
ATTT_API size_t attt_lora_workspace_bytes(int64_t L, int64_t din, int nproj, const int64_t *dout, int r);

/*
 * For each projection p < nproj sharing the input x = d_x (bf16 [L, din]),
 * with upstream gradient dy_p = d_dy[p] (bf16 [L, dout[p]]), adapter
 * A_p = d_A[p] (bf16 [din, r]) and B_p = d_B[p] (bf16 [r, dout[p]]):
 *   u_p = x A_p,  v_p = dy_p B_p^T                           ([L, r])
 *   d_dB[p] = scale * u_p^T dy_p                              (fp32 [r, dout[p]])
 *   d_dA[p] = scale * x^T v_p                                 (fp32 [din, r])
 * u and v are rounded to bf16 before the second contraction; products are
 * bf16, accumulation fp32.  The arrays d_dy, dout, d_A, d_B, d_dA, d_dB are
 * HOST arrays of nproj entries holding device pointers / sizes.
 * Requirements: 1 <= nproj <= 8, 1 <= r <= 64, L >= 1, din and every dout
 * >= 8 and multiples of 8, all tensor pointers 16-byte aligned, d_ws at least
 * attt_lora_workspace_bytes(...) bytes and 256-byte aligned.
 */
ATTT_API attt_status attt_lora_grad(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj,
                           const attt_bf16 *const *d_dy, const int64_t *dout,
                           const attt_bf16 *const *d_A, const attt_bf16 *const *d_B,
                           int r, float scale,
                           float *const *d_dA, float *const *d_dB,
                           void *d_ws, size_t ws_bytes, attt_stream stream);

/*
 * attt_lora_grad_noalloc -- attt_lora_grad for callers that cannot allocate
 * device memory.  (A deployment variant; the paper has no counterpart.)
 *
 * Who needs it: a process whose device memory is reserved up front by its
 * own pool, where a cudaMalloc would fail or fragment the pool; a latency-
 * critical loop that may not call the allocator because cudaMalloc/cudaFree
 * can synchronise the device; a plugin whose host application owns all
 * device allocations.  This call allocates nothing and calls no allocating
 * routine: its scratch is a static array of ATTT_LORA_NOALLOC_SCRATCH_BYTES
 * (16 MiB) inside the library's device memory, held by every GPU that loads
 * the library until the process exits.
 *
 * Arguments, layouts and results are those of attt_lora_grad without the
 * workspace; the caller still passes every input and output buffer.  A
 * problem whose scratch (attt_lora_workspace_bytes) exceeds 16 MiB returns
 * ATTT_ERR_WORKSPACE and launches nothing.
 *
 * The first call on a device (with that device current) looks up the static
 * array's device address and caches it; make that first call before any
 * stream capture begins.  The cached address belongs to the device's current
 * context: after cudaDeviceReset() the array is re-created, possibly at
 * another address, so calling this entry point after a device reset is not
 * supported.  Every call shares the one array per device and the
 * array keeps the last call's contents (the call clears what must start at
 * zero itself), so calls that overlap on the GPU -- on two streams, or from
 * two host threads -- race and must be serialised by the caller.  A timed-out
 * device wait of this call is reported by attt_device_status().
 */
#define ATTT_LORA_NOALLOC_SCRATCH_BYTES ((size_t)16 << 20)
ATTT_API attt_status attt_lora_grad_noalloc(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj,
                                            const attt_bf16 *const *d_dy, const int64_t *dout,
                                            const attt_bf16 *const *d_A, const attt_bf16 *const *d_B,
                                            int r, float scale,
                                            float *const *d_dA, float *const *d_dB, attt_stream stream);

/*
 * Eq. 2 / Algorithm 1 gradient step (plain SGD, no weight decay):
 *   A32 <- A32 - lr * dA,  B32 <- B32 - lr * dB     (fp32: product, then
 *                                                    difference, no FMA)
 * then refreshes the bf16 copies A16, B16 (round to nearest even) when they
 * are not NULL.  A32/dA/A16 are [din, r]; B32/dB/B16 are [r, dout].
 * Bit-exact with the formula.  In-place on A32 and B32.
 */
ATTT_API attt_status attt_lora_step(float *d_A32, float *d_B32, const float *d_dA, const float *d_dB,
                           int64_t din, int64_t dout, int r, float lr,
                           attt_bf16 *d_A16, attt_bf16 *d_B16, attt_stream stream);

/*
 * AdamW (Adam with decoupled weight decay) as an alternative to the paper's
 * SGD step, on the same adapter layout, with the first and second moments
 * d_mA, d_vA ([din, r]) and d_mB, d_vB ([r, dout]) (fp32, caller-owned,
 * zero before the first step) and `step` = 1 for the first step:
 *   p <- p (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2
 *   p <- p - (lr / (1 - b1^step)) m / (sqrt(v) / sqrt(1 - b2^step) + eps)
 * fp32, every operation rounded on its own, the scalars (1 - lr wd, b1,
 * 1 - b1, b2, 1 - b2, lr / (1 - b1^step), sqrt(1 - b2^step), eps) formed in
 * double from the double settings and rounded once; the bf16 copies are
 * refreshed when not NULL.  0 <= b1, b2 < 1, eps > 0, wd >= 0, step >= 1.
 */
ATTT_API attt_status attt_lora_adamw_step(float *d_A32, float *d_B32, const float *d_dA, const float *d_dB,
                                          float *d_mA, float *d_vA, float *d_mB, float *d_vB, int64_t din,
                                          int64_t dout, int r, float lr, double beta1, double beta2, double eps,
                                          double weight_decay, int step, attt_bf16 *d_A16, attt_bf16 *d_B16,
                                          attt_stream stream);

/* ------------------------------------------------------------------------ */
/* The adapted projection of a chained update: the LoRA-adapted linear map   */
/* y = x W0 + s (x A) B (Appendix C adapter; W0 frozen) whose output is the  */
/* LM head's input h, so that the second gradient step of an update         */
/* (Appendix C: two steps per update) sees the adapter the first one moved. */
/* ------------------------------------------------------------------------ */

/*
 * Workspace bytes attt_lora_forward / attt_lora_input_grad need.
 */
ATTT_API size_t attt_lora_forward_workspace_bytes(int64_t L, int64_t din, int64_t dout, int r);
ATTT_API size_t attt_lora_input_grad_workspace_bytes(int64_t L, int64_t din, int64_t dout, int r);

/*
 * h = x W0 + s (x A) B with x = d_x (bf16 [L, din]), W0 = d_W0 (bf16
 * [din, dout], frozen), A = d_A (bf16 [din, r]), B = d_B (bf16 [r, dout]),
 * s = scale; h = d_h (bf16 [L, dout], round to nearest even).  s (x A) is
 * rounded to bf16 once; products are bf16, sums fp32.  Requirements:
 * L >= 1, din and dout multiples of 8 (>= 8), 1 <= r <= 64, every pointer
 * 16-byte aligned, d_ws at least attt_lora_forward_workspace_bytes(L, din,
 * dout, r) bytes and 256-byte aligned.  Three launches.
 */
ATTT_API attt_status attt_lora_forward(const attt_bf16 *d_x, const attt_bf16 *d_W0, const attt_bf16 *d_A,
                                       const attt_bf16 *d_B, int64_t L, int64_t din, int64_t dout, int r,
                                       float scale, attt_bf16 *d_h, void *d_ws, size_t ws_bytes,
                                       attt_stream stream);

/*
 * The gradient of the projection's input from the gradient dy = d_dy (bf16
 * [L, dout]) of its output:  dx = dy W0^T + s (dy B^T) A^T  (fp32 [L, din]
 * into d_dx).  Shapes and alignment as attt_lora_forward; r must be a
 * multiple of 8 (A is read in place; ATTT_ERR_UNSUPPORTED otherwise).
 * s (dy B^T) is rounded to bf16 once.  Two launches.
 */
ATTT_API attt_status attt_lora_input_grad(const attt_bf16 *d_dy, const attt_bf16 *d_W0, const attt_bf16 *d_A,
                                          const attt_bf16 *d_B, int64_t L, int64_t din, int64_t dout, int r,
                                          float scale, float *d_dx, void *d_ws, size_t ws_bytes,
                                          attt_stream stream);

/*
 * d_dst[i] = bf16(d_src[i]) (round to nearest even) for i < n: the gradient
 * of the LM head's input (fp32 dh of attt_weighted_ce_fwd_bwd) as the bf16
 * upstream gradient dy of the adapted projection in a chained update.
 */
ATTT_API attt_status attt_cast_bf16(const float *d_src, attt_bf16 *d_dst, int64_t n, attt_stream stream);

/* ------------------------------------------------------------------------ */
/* Adapter drift (Sec. 4, Fig. 6): the KL divergence of the adapted model's */
/* next-token distribution from the base model's, through the frozen LM     */
/* head, without the [L, V] logits in HBM.                                  */
/* ------------------------------------------------------------------------ */

/* Workspace bytes attt_kl_drift needs for (L, d, V). */
ATTT_API size_t attt_kl_workspace_bytes(int64_t L, int64_t d, int64_t V);

/*
 * With p_j = softmax(h_p[j] W^T) (the adapted model) and q_j =
 * softmax(h_q[j] W^T) (the base model), h_p = d_hp and h_q = d_hq (bf16
 * [L, d]), W = d_W (bf16 [V, d]):
 *   d_kl[j]    = KL(p_j || q_j) = sum_v p_jv (log p_jv - log q_jv)   (fp32 [L])
 *   *d_kl_mean = (1/L) sum_j KL(p_j || q_j)    (summed in a fixed order)
 * Either output may be NULL (not both).  bf16 products, fp32 accumulation;
 * every logit is computed once (4 L V d FLOPs).  Requirements: L >= 1,
 * V >= 1, d >= 8 and d % 8 == 0, d_hp / d_hq / d_W 16-byte aligned, d_ws at
 * least attt_kl_workspace_bytes(L, d, V) bytes and 256-byte aligned.
 */
ATTT_API attt_status attt_kl_drift(const attt_bf16 *d_hp, const attt_bf16 *d_hq, const attt_bf16 *d_W,
                                   int64_t L, int64_t d, int64_t V, float *d_kl, float *d_kl_mean,
                                   void *d_ws, size_t ws_bytes, attt_stream stream);

/* ------------------------------------------------------------------------ */
/* Update-text repetition (Eq. 6), novelty (Eq. 7) and the sequence-level   */
/* filter of Sec. 4 (skip an update whose novelty is below tau; Appendix C: */
/* tau = 0.5), over the episode's word sets.                                */
/* ------------------------------------------------------------------------ */

typedef struct attt_wordsets attt_wordsets;

/*
 * Creates an empty set of update texts for an episode of up to max_updates
 * (1..4096) updates whose texts total at most max_bytes bytes, on the current
 * device.  The library allocates a byte arena for the texts and an exact word
 * index (hash table of 8 B keys plus one bit per update and word).
 */
ATTT_API attt_status attt_wordsets_create(int max_updates, int64_t max_bytes, attt_wordsets **out);

/* Frees the sets and their device memory (synchronises the device). */
ATTT_API attt_status attt_wordsets_destroy(attt_wordsets *s);

/* Forgets every text (an episode boundary).  Async on `stream`. */
ATTT_API attt_status attt_wordsets_reset(attt_wordsets *s, attt_stream stream);

/*
 * For the update text d_text (nbytes bytes, any values) of update k = the
 * number of texts recorded so far, with W(x) the set of words of x (maximal
 * runs of bytes other than the ASCII whitespace space, tab, LF, VT, FF, CR,
 * compared byte for byte):
 *   J_i   = |W(x_k) & W(x_i)| / |W(x_k) | W(x_i)|   (one fp32 division; 0 when
 *           both sets are empty)
 *   *d_rho  = max_{i<k} J_i  (0 for k = 0)                         (Eq. 6)
 *   *d_nu   = 1 - rho in fp32                                      (Eq. 7)
 *   *d_keep = 0 if nu < tau (the filter skips the update), else 1
 * then records x_k as update k (every candidate text counts for the later
 * ones, kept or not).  Outputs may be NULL.  Bit-exact.  ATTT_ERR_CAPACITY
 * (nothing launched) if max_updates texts are recorded or the texts would
 * exceed max_bytes.  A full probe sequence sets ATTT_ERR_TABLE_FULL in the
 * status word read by attt_wordsets_status.  Async on `stream`.
 */
ATTT_API attt_status attt_repetition(attt_wordsets *s, const uint8_t *d_text, int64_t nbytes, float tau,
                                     float *d_rho, float *d_nu, int32_t *d_keep, attt_stream stream);

/* Number of update texts recorded (host-side bookkeeping, no sync). */
ATTT_API int attt_wordsets_updates(const attt_wordsets *s);

/* Synchronises `stream`, then reads and clears the sets' status word. */
ATTT_API attt_status attt_wordsets_status(attt_wordsets *s, attt_stream stream);

/* ------------------------------------------------------------------------ */
/* The episode: Algorithm 1 run end to end with the schedule of Sec. 4 and  */
/* Appendix C -- an update every K agent steps, two gradient steps per      */
/* update, the adapter persisting within an episode and reset between       */
/* episodes.  The adapted projection's output is the LM head's input.       */
/* ------------------------------------------------------------------------ */

typedef struct attt_episode attt_episode;

typedef struct attt_episode_config {
    int n;               /* n-gram size of Eq. 8 (1..16)                        */
    float w_min;         /* Eq. 9 floor, 0 < w_min <= 1                         */
    int64_t max_history; /* tokens the history may hold over the episode        */
    int64_t max_update;  /* largest update text L (<= max_history)              */
    int64_t din;         /* adapted projection: input width  (multiple of 8)    */
    int64_t d;           /*   output width = LM head input   (multiple of 8)    */
    int64_t V;           /* vocabulary (LM head rows)                           */
    int r;               /* adapter rank, 1..64 (a multiple of 8 for dx)        */
    float scale;         /* s = alpha / r                                       */
    float lr;            /* SGD learning rate of Eq. 2                          */
    int grad_steps;      /* gradient steps per update (Appendix C: 2), 1..64    */
    int cadence;         /* K: agent steps per update (Sec. 4 default 5), >= 1  */
    int optimizer;       /* 0: SGD (Eq. 2, the paper's); 1: AdamW               */
    double beta1, beta2, eps, weight_decay; /* AdamW settings (optimizer 1)     */
} attt_episode_config;

/*
 * Creates an episode on the current device.  d_W0 (bf16 [din, d]) and d_Wlm
 * (bf16 [V, d]) are the frozen projection and LM head: borrowed, they must
 * stay valid and unchanged while the episode lives.  d_A0 (fp32 [din, r]) and
 * d_B0 (fp32 [r, d]) are the adapter's initial value, copied at create and
 * restored by every reset.  The episode allocates its history, adapter,
 * activations and one shared workspace up front (the update path allocates
 * nothing) and synchronises the device once.  *out is set on success.
 */
ATTT_API attt_status attt_episode_create(const attt_episode_config *cfg, const attt_bf16 *d_W0,
                                         const attt_bf16 *d_Wlm, const float *d_A0, const float *d_B0,
                                         attt_episode **out);

/* Frees the episode and everything it allocated (synchronises the device). */
ATTT_API attt_status attt_episode_destroy(attt_episode *e);

/*
 * The episode boundary: the adapter returns to (A0, B0), the history is
 * emptied, pending agent-step text is dropped and AdamW's moments and step
 * count (optimizer 1) return to zero.  Async on `stream`.
 */
ATTT_API attt_status attt_episode_reset(attt_episode *e, attt_stream stream);

/*
 * One update (Algorithm 1) on the update text x_k = d_tokens (int32 [L], the
 * targets of Eq. 10, each in [0, V)) whose rows of the adapted projection's
 * input are d_x (bf16 [L, din]):
 *   w = Eq. 9(Eq. 8(x_k, H))
 *   grad_steps times:  h = x W0 + s (x A) B  (bf16);  loss_g, dh = Eq. 10;
 *     dy = bf16(dh);  dA, dB of h;  dx_g = dy W0^T + s (dy B^T) A^T when d_dx
 *     is not NULL;  A -= lr dA, B -= lr dB
 *   H <- H || x_k
 * d_losses (fp32 [grad_steps]) receives each step's Eq. 10 loss (NULL: kept
 * internally).  d_dx (fp32 [grad_steps, L, din], 16-byte aligned) receives the
 * gradient of each step's projection input, or NULL to skip it.  The caller's
 * buffers must stay valid until the stream reaches the end of the update.
 * 1 <= L <= max_update; ATTT_ERR_CAPACITY (nothing launched) if the history
 * would exceed max_history.  Async on `stream`.
 */
ATTT_API attt_status attt_episode_update(attt_episode *e, const int32_t *d_tokens, const attt_bf16 *d_x, int64_t L,
                                         float *d_losses, float *d_dx, attt_stream stream);

/*
 * One agent step: appends its text (d_tokens int32 [len], d_x bf16 [len, din];
 * len may be 0) to the pending update text.  Every cadence-th call runs
 * attt_episode_update on the text of the last `cadence` steps (if it is not
 * empty), clears it and sets *updated (may be NULL) to 1, else 0.  Text of
 * fewer than `cadence` steps at the end of an episode is not trained on.
 * ATTT_ERR_CAPACITY (nothing launched, nothing appended) if the pending text
 * would exceed max_update or the history max_history.  Async on `stream`.
 */
ATTT_API attt_status attt_episode_agent_step(attt_episode *e, const int32_t *d_tokens, const attt_bf16 *d_x,
                                             int64_t len, float *d_losses, float *d_dx, int *updated,
                                             attt_stream stream);

/*
 * The adapter-drift diagnostic (Sec. 4, Fig. 6) on the projection inputs d_x
 * (bf16 [L, din], 1 <= L <= max_update): attt_kl_drift between the adapted
 * model's hidden states x W0 + s (x A) B (the current adapter) and the base
 * model's x W0 (no adapter), through the LM head; d_kl (fp32 [L]) and / or
 * d_kl_mean (fp32 [1]).  Does not change the episode.  Async on `stream`.
 */
ATTT_API attt_status attt_episode_drift(attt_episode *e, const attt_bf16 *d_x, int64_t L, float *d_kl,
                                        float *d_kl_mean, attt_stream stream);

/* Copies the adapter's fp32 values (A [din, r], B [r, d]) out.  Async. */
ATTT_API attt_status attt_episode_read_adapter(const attt_episode *e, float *d_A32, float *d_B32,
                                               attt_stream stream);

/*
 * Checkpoint and resume of an episode (the adapter persists within an
 * episode, Sec. 4): attt_episode_save writes into host_buf (at least
 * attt_episode_checkpoint_bytes(e) bytes) the configuration, the fp32
 * adapter, AdamW's moments and step count (optimizer 1), the history's token
 * stream and the pending agent-step text, and synchronises `stream`.
 * attt_episode_load restores all of it into an episode created with the same
 * configuration (ATTT_ERR_INVALID_ARG otherwise, or for a buffer that is not
 * such a checkpoint); the episode then continues bit for bit as the saved
 * one would.  The frozen W0, LM head and initial adapter are not saved.
 */
ATTT_API size_t attt_episode_checkpoint_bytes(const attt_episode *e);
ATTT_API attt_status attt_episode_save(attt_episode *e, void *host_buf, size_t bytes, attt_stream stream);
ATTT_API attt_status attt_episode_load(attt_episode *e, const void *host_buf, size_t bytes, attt_stream stream);

/* The episode's history (owned by the episode; do not destroy it). */
ATTT_API attt_history *attt_episode_history(attt_episode *e);

/* Tokens of pending agent-step text not yet trained on. */
ATTT_API int64_t attt_episode_pending_tokens(const attt_episode *e);

/* ------------------------------------------------------------------------ */
/* A batch of concurrent episodes (Sec. 4 runs 16 at once, each with a      */
/* private adapter and history) updated together.                           */
/* ------------------------------------------------------------------------ */

typedef struct attt_batch attt_batch;

typedef struct attt_batch_config {
    int episodes;        /* E, 1..32                                            */
    int n;               /* n-gram size of Eq. 8 (1..16)                        */
    float w_min;         /* Eq. 9 floor                                         */
    int64_t max_history; /* tokens each episode's history may hold              */
    int64_t max_update;  /* largest update text of one episode (<= max_history) */
    int64_t din, d, V;   /* adapted projection [din, d], LM head [V, d]         */
    int r;               /* adapter rank, 1..64                                 */
    float scale, lr;     /* s = alpha / r; SGD rate of Eq. 2                    */
    int grad_steps;      /* gradient steps per update (Appendix C: 2)           */
} attt_batch_config;

/*
 * Creates E episodes on the current device sharing the frozen d_W0 (bf16
 * [din, d]) and d_Wlm (bf16 [V, d]) (borrowed, as for attt_episode_create);
 * every episode's adapter starts at d_A0 (fp32 [din, r]) / d_B0 (fp32 [r, d])
 * (copied).  Everything the updates need is allocated here.
 */
ATTT_API attt_status attt_batch_create(const attt_batch_config *cfg, const attt_bf16 *d_W0, const attt_bf16 *d_Wlm,
                                       const float *d_A0, const float *d_B0, attt_batch **out);

/* Frees the batch and everything it allocated (synchronises the device). */
ATTT_API attt_status attt_batch_destroy(attt_batch *b);

/* Episode boundary for episode e (-1: every episode): its adapter returns to
 * (A0, B0) and its history is emptied.  Async on `stream`. */
ATTT_API attt_status attt_batch_reset(attt_batch *b, int e, attt_stream stream);

/*
 * One update (Algorithm 1, as attt_episode_update) for every episode e with
 * lens[e] > 0 (lens: HOST array of E lengths, 0 <= lens[e] <= max_update; an
 * episode with lens[e] = 0 is left unchanged).  The update texts are stacked:
 * d_tokens (int32 [sum lens]) and d_x (bf16 [sum lens, din]) hold episode 0's
 * rows, then episode 1's, and so on.  d_losses (fp32 [E, grad_steps], or
 * NULL) receives each episode's Eq. 10 loss per step (0 for an episode
 * without rows); d_dx (fp32 [grad_steps, sum lens, din], 16-byte aligned, or
 * NULL) the projection-input gradients.  Eq. 8/9, the dh -> dy cast, the SGD
 * step and the history append each run as one launch for the whole batch,
 * Eq. 10 as one call over every row, the projection forward and dx as one
 * contraction each over every row, and the adapter gradients as one grouped
 * launch per pass (16 episodes per launch).  ATTT_ERR_CAPACITY (nothing
 * launched) if an episode's history
 * would exceed max_history.  Async on `stream`.
 */
ATTT_API attt_status attt_batch_update(attt_batch *b, const int32_t *d_tokens, const attt_bf16 *d_x,
                                       const int64_t *lens, float *d_losses, float *d_dx, attt_stream stream);

/* Copies episode e's adapter (fp32 A [din, r], B [r, d]) out.  Async. */
ATTT_API attt_status attt_batch_read_adapter(const attt_batch *b, int e, float *d_A32, float *d_B32,
                                             attt_stream stream);

/* Episode e's history (owned by the batch). */
ATTT_API attt_history *attt_batch_history(attt_batch *b, int e);

#ifdef __cplusplus
}
#endif

#endif /* ATTT_H */
