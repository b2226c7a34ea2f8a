// kl.cu -- the adapter-drift diagnostic of aTTT (Sec. 4, Fig. 6) on the GPU:
// per row j the KL divergence of the adapted model's next-token distribution
// p_j = softmax(h_p[j] W^T) from the base model's q_j = softmax(h_q[j] W^T),
// through the frozen LM head, without the [L, V] logits in HBM.
//
// One contraction over the whole vocabulary: each CTA's 128-row A tile is 64
// rows of h_p over the same 64 rows of h_q, so one tcgen05 MMA per K step
// gives both z_p = h_p W^T and z_q = h_q W^T for those rows (4 L V d FLOPs:
// each logit once).  The epilogue reduces each (row, 256-column tile) to five
// fp32 numbers: the
// maxima m_p, m_q (log2 units), s_p = sum exp2(z_p log2e - m_p), s_q alike,
// and the cross term x = sum exp2(z_p log2e - m_p) (z_p - z_q).  The reduce
// kernel merges the tiles of a row like an online logsumexp (rescaling s_p and
// x together) and forms
//   KL_j = X_j / S_p,j - (lse_p,j - lse_q,j)
// (= E_p[z_p - z_q] - lse_p + lse_q), every term from fp32 accumulators, then
// the mean over the rows in a fixed order.
#include "gemm_launch.cuh"

namespace attt {

constexpr int kKlBN = 256;  // 256-column tiles (the accumulator double-buffered: 512 TMEM columns)
constexpr int kKlRows = 32;
constexpr int kKlWarps = 8;

struct KlLayout {
    int64_t ntiles, plane, nblk;
    float *part;  // five planes of [ntiles, L]
    float *block_sums;
    unsigned int *ticket;
    size_t bytes;
};

static KlLayout kl_layout(void *ws, int64_t L, int64_t V) {
    KlLayout k{};
    k.ntiles = cdiv(V, kKlBN);
    k.plane = k.ntiles * L;
    k.nblk = cdiv(L, kKlRows);
    Carve cv{static_cast<char *>(ws), 0};
    k.part = cv.take<float>((size_t)(5 * k.plane));
    k.block_sums = cv.take<float>((size_t)k.nblk);
    k.ticket = cv.take<unsigned int>(4);
    k.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return k;
}

// 32 rows per block (lane = row); warp w merges tiles t = w (mod 8) with
// coalesced loads of the planes, then warp 0 merges the warps' results.
// Merge of (m, s, x) with (m2, s2, x2): M = max, s = s 2^(m-M) + s2 2^(m2-M),
// x the same with x, x2.  The last block (ticket) sums the blocks' sums of
// KL_j in block order for the mean.
__global__ void __launch_bounds__(kKlWarps * 32) kl_reduce_kernel(const float *__restrict__ part, int64_t plane,
                                                                 int ntiles, int L, float *kl_rows, float *kl_mean,
                                                                 float *block_sums, unsigned int *ticket) {
    __shared__ float s_v[5][kKlWarps][kKlRows];
    __shared__ bool s_last;
    griddep_wait();
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kKlRows + lane;
    float mp = -INFINITY, sp = 0.f, x = 0.f, mq = -INFINITY, sq = 0.f;
    if (j < L) {
        for (int t = warp; t < ntiles; t += kKlWarps) {
            const int64_t o = (int64_t)t * L + j;
            const float m2 = __ldcg(part + o), s2 = __ldcg(part + plane + o);
            const float n2 = __ldcg(part + 2 * plane + o), r2 = __ldcg(part + 3 * plane + o);
            const float x2 = __ldcg(part + 4 * plane + o);
            const float M = fmaxf(mp, m2);
            const float a = exp2f(mp - M), b = exp2f(m2 - M);  // mp = -inf: a = 0
            sp = sp * a + s2 * b;
            x = x * a + x2 * b;
            mp = M;
            const float N = fmaxf(mq, n2);
            sq = sq * exp2f(mq - N) + r2 * exp2f(n2 - N);
            mq = N;
        }
    }
    s_v[0][warp][lane] = mp;
    s_v[1][warp][lane] = sp;
    s_v[2][warp][lane] = x;
    s_v[3][warp][lane] = mq;
    s_v[4][warp][lane] = sq;
    __syncthreads();
    if (warp == 0) {
        float kl = 0.f;
        if (j < L) {
            for (int w = 1; w < kKlWarps; ++w) {
                const float m2 = s_v[0][w][lane], s2 = s_v[1][w][lane], x2 = s_v[2][w][lane];
                const float n2 = s_v[3][w][lane], r2 = s_v[4][w][lane];
                if (m2 != -INFINITY) {
                    const float M = fmaxf(mp, m2);
                    const float a = exp2f(mp - M), b = exp2f(m2 - M);
                    sp = sp * a + s2 * b;
                    x = x * a + x2 * b;
                    mp = M;
                }
                if (n2 != -INFINITY) {
                    const float N = fmaxf(mq, n2);
                    sq = sq * exp2f(mq - N) + r2 * exp2f(n2 - N);
                    mq = N;
                }
            }
            const float dl = ((mp + log2f(sp)) - (mq + log2f(sq))) * 0.69314718055994531f;
            kl = x / sp - dl;
            if (kl_rows) kl_rows[j] = kl;
        }
        float sum = kl;
        for (int o = 16; o > 0; o >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, o);
        if (lane == 0) {
            block_sums[blockIdx.x] = sum;
            __threadfence();
            s_last = atomicAdd(ticket, 1u) == gridDim.x - 1;
        }
    }
    __syncthreads();
    if (s_last && threadIdx.x == 0) {
        __threadfence();
        float total = 0.f;
        for (unsigned b = 0; b < gridDim.x; ++b) total += __ldcg(block_sums + b);
        if (kl_mean) *kl_mean = total / (float)L;
        *ticket = 0u;
    }
}

}  // namespace attt

extern "C" {

size_t attt_kl_workspace_bytes(int64_t L, int64_t d, int64_t V) {
    if (L <= 0 || V <= 0 || d <= 0) return 0;
    return attt::kl_layout(nullptr, L, V).bytes;
}

attt_status attt_kl_drift(const attt_bf16 *d_hp, const attt_bf16 *d_hq, const attt_bf16 *d_W, int64_t L, int64_t d,
                          int64_t V, float *d_kl, float *d_kl_mean, void *d_ws, size_t ws_bytes,
                          attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!d_hp || !d_hq || !d_W || (!d_kl && !d_kl_mean)) return ATTT_ERR_INVALID_ARG;
    if (L < 1 || V < 1 || d < 8 || d % 8 != 0) return ATTT_ERR_INVALID_ARG;
    if (L > (1ll << 30) || V > (1ll << 30) || d > (1ll << 20)) return ATTT_ERR_UNSUPPORTED;
    if (!aligned16(d_hp) || !aligned16(d_hq) || !aligned16(d_W)) return ATTT_ERR_INVALID_ARG;
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_kl_workspace_bytes(L, d, V)) return ATTT_ERR_WORKSPACE;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    KlLayout k = kl_layout(d_ws, L, V);
    if (cudaMemsetAsync(k.ticket, 0, 4 * sizeof(unsigned int), stream) != cudaSuccess) return ATTT_ERR_CUDA;

    GemmProblem p{};
    p.a = d_hp; p.a_rows_ld = d; p.a_rows = L; p.a_k = d;
    p.a2 = d_hq; p.a2_rows_ld = d; p.a2_rows = L; p.a2_k = d;
    p.b = d_W; p.b_rows_ld = d; p.b_rows = V; p.b_k = d;
    p.M = (int)L; p.N = (int)V; p.K = (int)d; p.BN = kKlBN; p.pair = true;
    EpiParams ep{};
    ep.kl_part = k.part;
    ep.kl_plane = k.plane;
    st = launch_gemm<EPI_KL, false, false>(p, ep, dev, stream);
    if (st != ATTT_OK) return st;

    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)k.nblk);
    cfg.blockDim = dim3(kKlWarps * 32);
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kl_reduce_kernel, (const float *)k.part, (int64_t)k.plane, (int)k.ntiles, (int)L,
                           d_kl, d_kl_mean, k.block_sums, k.ticket) != cudaSuccess)
        return ATTT_ERR_CUDA;
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // extern "C"
