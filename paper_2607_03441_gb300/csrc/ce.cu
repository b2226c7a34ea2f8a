// ce.cu -- Eq. 10 of aTTT on the GPU: the token-weighted next-token CE through
// the frozen LM head, its value and its gradient with respect to the hidden
// states, without ever holding the [L, V] logits in HBM.
//
//   pass 1  tcgen05 contraction z = h W^T over 128 x 256 tiles; the epilogue
//           keeps, per row and vocab tile, the running max and sum of exp
//           (online logsumexp in log2 units) and the target logit.  HBM
//           sees only [V/256, L] (max, sum) pairs.
//   reduce  per row: merge the tile pairs into lse_j, nll_j = lse_j - z_{j,x_j};
//           the weighted mean (1/L) sum_j w_j nll_j is summed in a fixed
//           order (deterministic).
//   pass 2  for each vocab chunk of Vc columns (Vc sized so the chunk's
//           gradient block stays L2-resident): recompute z for the chunk and
//           write G = (w_j/L)(softmax(z_j) - onehot(x_j)) as bf16 (fused
//           epilogue), then dh (+)= G W_chunk with W read MN-major by TMA.
// The LM head gets no gradient (frozen; only the adapter trains).
#include "gemm_launch.cuh"

namespace attt {

constexpr int kCeBN = 256;
constexpr int kFinThreads = 128;

struct CeLayout {
    int64_t nvt, Vc, nblk;
    float2 *part;
    float *ztgt, *lse_tmp, *block_sums;
    unsigned int *ticket;
    __nv_bfloat16 *G;
    size_t bytes;
};

static int64_t ce_chunk(int64_t L, int64_t V) {
    // Gradient block of one chunk: L x Vc bf16, kept near 96 MB.
    int64_t vc = (96ll << 20) / (2 * L);
    vc = (vc / kCeBN) * kCeBN;
    if (vc < 4096) vc = 4096;
    const int64_t vmax = round_up(V, kCeBN);
    if (vc > vmax) vc = vmax;
    return vc;
}

static CeLayout ce_layout(void *ws, int64_t L, int64_t V) {
    CeLayout c{};
    c.nvt = cdiv(V, kCeBN);
    c.Vc = ce_chunk(L, V);
    c.nblk = cdiv(L, kFinThreads);
    Carve cv{static_cast<char *>(ws), 0};
    c.part = cv.take<float2>((size_t)(c.nvt * L));
    c.ztgt = cv.take<float>((size_t)L);
    c.lse_tmp = cv.take<float>((size_t)L);
    c.block_sums = cv.take<float>((size_t)c.nblk);
    c.ticket = cv.take<unsigned int>(4);
    c.G = cv.take<__nv_bfloat16>((size_t)(L * c.Vc));
    c.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return c;
}

__global__ void __launch_bounds__(kFinThreads) ce_finalize_kernel(const float2 *__restrict__ part, int nvt,
                                                                   const float *__restrict__ ztgt,
                                                                   const int32_t *__restrict__ tgt,
                                                                   const float *__restrict__ w, int L, int V,
                                                                   float *__restrict__ lse_out, float inv_L,
                                                                   float *block_sums, unsigned int *ticket,
                                                                   float *loss, int *status) {
    __shared__ float red[kFinThreads / 32];
    __shared__ bool last;
    const int j = blockIdx.x * kFinThreads + threadIdx.x;
    float contrib = 0.f;
    if (j < L) {
        float m = -INFINITY, s = 0.f;
        for (int i = 0; i < nvt; ++i) {
            const float2 p = __ldcg(part + (int64_t)i * L + j);
            if (p.x > m) {
                s = s * exp2f(m - p.x) + p.y;
                m = p.x;
            } else {
                s += p.y * exp2f(p.x - m);
            }
        }
        const float lse = (m + log2f(s)) * 0.69314718055994531f;
        lse_out[j] = lse;
        const int t = tgt[j];
        float nll;
        if (t < 0 || t >= V) {
            record_error(status, ATTT_ERR_TOKEN_RANGE);
            nll = __int_as_float(0x7fc00000);
        } else {
            nll = lse - __ldcg(ztgt + j);
        }
        contrib = w[j] * nll;
    }
    for (int o = 16; o > 0; o >>= 1) contrib += __shfl_xor_sync(0xffffffffu, contrib, o);
    if ((threadIdx.x & 31) == 0) red[threadIdx.x >> 5] = contrib;
    __syncthreads();
    if (threadIdx.x == 0) {
        float b = 0.f;
        for (int i = 0; i < kFinThreads / 32; ++i) b += red[i];
        block_sums[blockIdx.x] = b;
        __threadfence();
        last = atomicAdd(ticket, 1u) == gridDim.x - 1;
    }
    __syncthreads();
    if (last && threadIdx.x == 0) {
        __threadfence();
        float total = 0.f;
        for (unsigned i = 0; i < gridDim.x; ++i) total += __ldcg(block_sums + i);
        *loss = total * inv_L;
        *ticket = 0u;
    }
}

}  // namespace attt

extern "C" {

size_t attt_ce_workspace_bytes(int64_t L, int64_t d, int64_t V) {
    (void)d;
    if (L <= 0 || V <= 0) return 0;
    return attt::ce_layout(nullptr, L, V).bytes;
}

attt_status attt_weighted_ce_fwd_bwd(const attt_bf16 *d_h, const attt_bf16 *d_W, const int32_t *d_tgt,
                                     const float *d_w, int64_t L, int64_t d, int64_t V, float *d_loss,
                                     float *d_dh, float *d_lse, void *d_ws, size_t ws_bytes, attt_stream stream) {
    using namespace attt;
    if (!d_h || !d_W || !d_tgt || !d_w || !d_loss || !d_dh) return ATTT_ERR_INVALID_ARG;
    if (L < 1 || V < 1 || d < 8 || d % 8 != 0) return ATTT_ERR_INVALID_ARG;
    if (L > (1ll << 30) || V > (1ll << 30) || d > (1ll << 20)) return ATTT_ERR_UNSUPPORTED;
    if (!aligned16(d_h) || !aligned16(d_W) || !aligned16(d_dh)) return ATTT_ERR_INVALID_ARG;
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_ce_workspace_bytes(L, d, V)) return ATTT_ERR_WORKSPACE;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    int *status = device_status_word(dev);
    if (!status) return ATTT_ERR_CUDA;

    CeLayout c = ce_layout(d_ws, L, V);
    float *lse = d_lse ? d_lse : c.lse_tmp;
    if (cudaMemsetAsync(c.ticket, 0, sizeof(unsigned int), stream) != cudaSuccess) return ATTT_ERR_CUDA;

    // pass 1: per-tile (max, sum exp) and the target logit
    {
        GemmProblem p{};
        p.a = d_h; p.a_rows_ld = d; p.a_rows = L; p.a_k = d;
        p.b = d_W; p.b_rows_ld = d; p.b_rows = V; p.b_k = d;
        p.M = (int)L; p.N = (int)V; p.K = (int)d; p.BN = kCeBN;
        EpiParams ep{};
        ep.tgt = d_tgt; ep.part = c.part; ep.ztgt = c.ztgt; ep.v0 = 0;
        st = launch_gemm<EPI_CE_STATS, false, false>(p, ep, dev, stream);
        if (st != ATTT_OK) return st;
    }
    ce_finalize_kernel<<<(unsigned)c.nblk, kFinThreads, 0, stream>>>(c.part, (int)c.nvt, c.ztgt, d_tgt, d_w, (int)L,
                                                                     (int)V, lse, 1.0f / (float)L, c.block_sums,
                                                                     c.ticket, d_loss, status);
    count_launch();
    if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;

    // pass 2: per vocab chunk, G = (w/L)(softmax - onehot) then dh += G W_chunk
    for (int64_t v0 = 0, ci = 0; v0 < V; v0 += c.Vc, ++ci) {
        const int64_t Nc = (V - v0 < c.Vc) ? V - v0 : c.Vc;
        {
            GemmProblem p{};
            p.a = d_h; p.a_rows_ld = d; p.a_rows = L; p.a_k = d;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = V; p.b_k = d;
            p.M = (int)L; p.N = (int)Nc; p.K = (int)d; p.BN = kCeBN;
            p.b_n_off = (int)v0;
            EpiParams ep{};
            ep.tgt = d_tgt; ep.lse = lse; ep.w = d_w; ep.inv_L = 1.0f / (float)L; ep.v0 = (int)v0;
            ep.G = c.G; ep.G_ld = c.Vc;
            st = launch_gemm<EPI_CE_GRAD, false, false>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
        {
            GemmProblem p{};
            p.a = c.G; p.a_rows_ld = c.Vc; p.a_rows = L; p.a_k = c.Vc;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = d; p.b_k = V;
            p.M = (int)L; p.N = (int)d; p.K = (int)round_up(Nc, 64); p.BN = kCeBN;
            p.b_k_off = (int)v0;
            EpiParams ep{};
            ep.out = d_dh; ep.out_ld = d; ep.accumulate = ci > 0 ? 1 : 0; ep.alpha = 1.0f;
            st = launch_gemm<EPI_F32_ACC, false, true>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
    }
    return ATTT_OK;
}

}  // extern "C"
