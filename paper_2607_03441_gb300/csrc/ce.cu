// ce.cu -- Eq. 10 of aTTT on the GPU: the token-weighted next-token CE through
// the frozen LM head, its value and its gradient with respect to the hidden
// states, in one sweep over the vocabulary (4*L*V*d tensor FLOPs: each logit
// is computed once), never holding the [L, V] logits in HBM.
//
// For each vocab chunk c of Vc columns (Vc sized so that the chunk's bf16
// block stays L2-resident):
//   GEMM1  z = h W_c^T on 128 x 256 tiles; the epilogue keeps per (row, tile)
//          the max m_t and the sum of exp(z - m_t) (log2 units), writes
//          E = exp(z - m_t) as bf16, and catches the target logit;
//          From the second chunk on, E is written against the running max
//          of the earlier chunks instead of the tile max;
//   chunk  per row: the chunk max, a rewrite of E only where needed (the
//          first chunk, or a row whose max jumped by more than 2^32), and the
//          online-softmax factors of the accumulator's reference A:
//          alpha = exp(A_old - A_new), beta = exp(R_E - A_new);
//   GEMM2  D = E W_c (W read MN-major by TMA); the epilogue folds it into the
//          fp32 accumulator: acc = alpha * acc + beta * D.
// Then per row: lse from the (max, sum) pairs of every tile, the loss
// (1/L) sum_j w_j (lse_j - z_{j,x_j}) summed in a fixed order, and
//   dh_j = (w_j / L) (acc_j exp(M_j - lse_j) - W_{x_j}).
// The LM head gets no gradient (frozen; only the adapter trains).
#include "gemm_launch.cuh"

namespace attt {

constexpr int kCeBN = 256;
constexpr int kCeMaxTiles = 256;  // vocab tiles per chunk at most
constexpr int kFinThreads = 256;
constexpr int kFinRows = 32;
// fp32 partials of 128 x kCeBN (128 KB each) for the tail split of the dh
// contraction: enough for every CTA of a 160-SM part to hold one piece.
constexpr int kCeSplitRegions = 160;

struct CeLayout {
    int64_t nvt, Vc, nblk;
    float2 *part;
    float *ztgt, *lse_tmp, *block_sums;
    float *aref, *mref, *alpha, *beta;
    unsigned int *ticket;       // [4] loss ticket, then [split_regions] tail-split counters
    unsigned int *split_tick;
    int split_regions;
    float *split_ws;
    __nv_bfloat16 *G;
    size_t bytes;
};

// Upper bound of the vocab chunk: the chunk's bf16 gradient block L x Vc is
// kept near 96 MB (L2 is 129 MB).  The workspace is sized for this bound.
static int64_t ce_chunk_max(int64_t L, int64_t V) {
    int64_t vc = (96ll << 20) / (2 * L);
    vc = (vc / kCeBN) * kCeBN;
    if (vc < 4096) vc = 4096;
    if (vc > kCeMaxTiles * kCeBN) vc = kCeMaxTiles * kCeBN;
    const int64_t vmax = round_up(V, kCeBN);
    if (vc > vmax) vc = vmax;
    return vc;
}

// Tile plan for `sms` SMs.  Above 128 rows both contractions run on CTA pairs
// (cta_group::2: 256 x 256 accumulator tiles), else on single CTAs (128 x 256).
// The chunk width Vc (<= the workspace bound) minimises an estimate of the
// time that counts whole waves of tiles (a partial wave costs a full one)
// plus a per-launch cost.
struct CePlan {
    int64_t Vc;
    bool pair;
};

static CePlan ce_plan(int64_t L, int64_t d, int64_t V, int sms) {
    const double rate = 1.0e13;    // bf16 FLOP/s of one SM, order of magnitude
    const double launch = 5.0e-6;  // seconds per launch, ramp-up and tail included
    const bool pair = L > 128;
    const int64_t rows = pair ? 256 : 128;       // accumulator rows per tile
    const int64_t units = pair ? sms / 2 : sms;  // tiles in flight
    const double tile_rate = rate * (pair ? 2.0 : 1.0);
    const int64_t tm = cdiv(L, rows);
    const double w2 = (double)cdiv(tm * cdiv(d, kCeBN), units);
    CePlan best{ce_chunk_max(L, V), pair};
    double best_t = 1e30;
    const int64_t vmax = ce_chunk_max(L, V);
    for (int64_t vc = 4 * kCeBN; vc <= vmax; vc += kCeBN) {
        double t = 0.0;
        for (int64_t v0 = 0; v0 < V; v0 += vc) {
            const int64_t nc = (V - v0 < vc) ? V - v0 : vc;
            const double w1 = (double)cdiv(tm * cdiv(nc, kCeBN), units);
            t += (w1 * d + w2 * round_up(nc, 64)) * 2.0 * rows * kCeBN / tile_rate + 3 * launch;
        }
        if (t < best_t) { best_t = t; best = CePlan{vc, pair}; }
        if (vc == vmax) break;
    }
    return best;
}

static CeLayout ce_layout(void *ws, int64_t L, int64_t d, int64_t V) {
    CeLayout c{};
    // tail split of the dh contraction: at most 4 pieces per tile and 2 CTAs
    // per tile, so 8 regions per tile of the contraction bound the need
    const int64_t rows = L > 128 ? 256 : 128;
    const int64_t t2 = cdiv(L, rows) * cdiv(d, kCeBN);
    c.split_regions = (int)(8 * t2 < kCeSplitRegions ? 8 * t2 : kCeSplitRegions);
    c.nvt = cdiv(V, kCeBN);
    c.Vc = ce_chunk_max(L, V);
    c.nblk = cdiv(L, kFinRows);
    Carve cv{static_cast<char *>(ws), 0};
    c.part = cv.take<float2>((size_t)(c.nvt * L));
    c.ztgt = cv.take<float>((size_t)L);
    c.lse_tmp = cv.take<float>((size_t)L);
    c.block_sums = cv.take<float>((size_t)c.nblk);
    c.aref = cv.take<float>((size_t)L);
    c.mref = cv.take<float>((size_t)L);
    c.alpha = cv.take<float>((size_t)L);
    c.beta = cv.take<float>((size_t)L);
    c.ticket = cv.take<unsigned int>(4 + (size_t)c.split_regions);
    c.split_tick = c.ticket + 4;
    c.split_ws = cv.take<float>((size_t)c.split_regions * 128 * kCeBN);
    c.G = cv.take<__nv_bfloat16>((size_t)(L * c.Vc));
    c.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return c;
}

// Merges two (max, sum) pairs of an online logsumexp in log2 units.
__device__ __forceinline__ void lse_merge(float &m, float &s, float m2, float s2) {
    const float mx = fmaxf(m, m2);
    if (mx == -INFINITY) return;
    s = s * exp2f(m - mx) + s2 * exp2f(m2 - mx);
    m = mx;
}

// One block per kFinRows rows; warp w merges the vocab tiles i = w (mod 8) of
// its 32 rows with coalesced loads of part[i, rows], then warp 0 merges the
// 8 partial pairs per row and forms lse, the target NLL and the weighted sum.
// The last block (atomic ticket) adds the block sums in block order, so the
// loss is deterministic.
__global__ void __launch_bounds__(kFinThreads) ce_finalize_kernel(const float2 *__restrict__ part, int nvt,
                                                                   const float *__restrict__ ztgt,
                                                                   const int32_t *__restrict__ tgt,
                                                                   const float *__restrict__ w, int L, int V,
                                                                   float *__restrict__ lse_out, float inv_L,
                                                                   float *block_sums, unsigned int *ticket,
                                                                   float *loss, int *status) {
    constexpr int kWarps = kFinThreads / 32;
    __shared__ float sm_m[kWarps][kFinRows], sm_s[kWarps][kFinRows];
    __shared__ bool last;
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j = blockIdx.x * kFinRows + lane;
    float m = -INFINITY, s = 0.f;
    if (j < L) {
        for (int i = warp; i < nvt; i += kWarps) {
            const float2 p = __ldcg(part + (int64_t)i * L + j);
            lse_merge(m, s, p.x, p.y);
        }
    }
    sm_m[warp][lane] = m;
    sm_s[warp][lane] = s;
    __syncthreads();
    if (warp == 0) {
        for (int k = 1; k < kWarps; ++k) lse_merge(m, s, sm_m[k][lane], sm_s[k][lane]);
        float contrib = 0.f;
        if (j < L) {
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
        if (lane == 0) {
            block_sums[blockIdx.x] = contrib;
            __threadfence();
            last = atomicAdd(ticket, 1u) == gridDim.x - 1;
        }
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

// Bookkeeping of chunk c, one warp per row j (log2 units throughout):
//   M_c  = max over the chunk's tiles of the tile max m_t;
//   R    = the running max of the earlier chunks (mref; -inf for the first).
//   GEMM1 wrote tile t of E against R, or against m_t when m_t - R >
//   kCeRefJump.  If any tile did (M_c - R > kCeRefJump), the row is rewritten
//   against M_c tile by tile; otherwise it stays against R.  Rp = the
//   reference E now has.
//   acc = alpha * acc + beta * (E W_c) with A_new = max(A_old, Rp),
//   alpha = exp2(A_old - A_new), beta = exp2(Rp - A_new);  mref <- max(R, M_c).
__global__ void __launch_bounds__(256) ce_chunk_kernel(const float2 *__restrict__ part, int tile0, int ntiles, int L,
                                                       __nv_bfloat16 *G, int64_t G_ld, float *aref, float *mref,
                                                       float *alpha, float *beta, int first) {
    const int j = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= L) return;
    float mc = -INFINITY;
    for (int t = lane; t < ntiles; t += 32) mc = fmaxf(mc, __ldcg(&part[(int64_t)(tile0 + t) * L + j].x));
    for (int o = 16; o > 0; o >>= 1) mc = fmaxf(mc, __shfl_xor_sync(0xffffffffu, mc, o));
    const float r = first ? -INFINITY : mref[j];
    uint4 *row = reinterpret_cast<uint4 *>(G + (int64_t)j * G_ld);
    const int per_tile = kCeBN / 8;  // uint4 (8 x bf16) per tile row
    float rp = r;
    if (mc - r > kCeRefJump) {
        rp = mc;
        for (int t = 0; t < ntiles; ++t) {
            const float mt = __ldcg(&part[(int64_t)(tile0 + t) * L + j].x);
            const float sc = (mt - r > kCeRefJump) ? exp2f(mt - mc) : exp2f(r - mc);
            for (int i = lane; i < per_tile; i += 32) {
                uint4 u = row[t * per_tile + i];
                uint32_t *w = reinterpret_cast<uint32_t *>(&u);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162 *>(&w[q]);
                    const float2 v = __bfloat1622float2(b);
                    b = __floats2bfloat162_rn(v.x * sc, v.y * sc);
                    w[q] = *reinterpret_cast<uint32_t *>(&b);
                }
                row[t * per_tile + i] = u;
            }
        }
    }
    if (lane == 0) {
        const float aold = first ? -INFINITY : aref[j];
        const float anew = fmaxf(aold, rp);
        alpha[j] = (aold == -INFINITY) ? 0.f : exp2f(aold - anew);
        beta[j] = exp2f(rp - anew);
        aref[j] = anew;
        mref[j] = fmaxf(r, mc);
    }
}

// dh_j = (w_j / L) (acc_j exp(A_j - lse_j) - W_{x_j}); one block per row.
__global__ void __launch_bounds__(256) ce_fixup_kernel(float *dh, int64_t d, const __nv_bfloat16 *__restrict__ W,
                                                       const int32_t *__restrict__ tgt, const float *__restrict__ w,
                                                       float inv_L, const float *__restrict__ aref,
                                                       const float *__restrict__ lse, int V) {
    const int j = blockIdx.x;
    const int t = tgt[j];
    const float c = w[j] * inv_L;
    const float sc = exp2f(aref[j] - lse[j] * kLog2e);
    float *row = dh + (int64_t)j * d;
    if (t < 0 || t >= V) {
        for (int64_t k = threadIdx.x; k < d; k += blockDim.x) row[k] = __int_as_float(0x7fc00000);
        return;
    }
    const __nv_bfloat16 *wt = W + (int64_t)t * d;
    // d % 8 == 0: 8 columns per step (one 16-byte load of W, two float4 of dh)
    for (int64_t k = (int64_t)threadIdx.x * 8; k < d; k += (int64_t)blockDim.x * 8) {
        const uint4 u = *reinterpret_cast<const uint4 *>(wt + k);
        const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&u);
        float4 *o = reinterpret_cast<float4 *>(row + k);
        float4 a0 = o[0], a1 = o[1];
        const float2 w0 = __bfloat1622float2(b[0]), w1 = __bfloat1622float2(b[1]);
        const float2 w2 = __bfloat1622float2(b[2]), w3 = __bfloat1622float2(b[3]);
        a0.x = c * (a0.x * sc - w0.x); a0.y = c * (a0.y * sc - w0.y);
        a0.z = c * (a0.z * sc - w1.x); a0.w = c * (a0.w * sc - w1.y);
        a1.x = c * (a1.x * sc - w2.x); a1.y = c * (a1.y * sc - w2.y);
        a1.z = c * (a1.z * sc - w3.x); a1.w = c * (a1.w * sc - w3.y);
        o[0] = a0;
        o[1] = a1;
    }
}

}  // namespace attt

extern "C" {

size_t attt_ce_workspace_bytes(int64_t L, int64_t d, int64_t V) {
    if (L <= 0 || V <= 0 || d <= 0) return 0;
    return attt::ce_layout(nullptr, L, d, V).bytes;
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

    CeLayout c = ce_layout(d_ws, L, d, V);
    float *lse = d_lse ? d_lse : c.lse_tmp;
    if (cudaMemsetAsync(c.ticket, 0, sizeof(unsigned int) * (4 + (size_t)c.split_regions), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;

    const CePlan plan = ce_plan(L, d, V, num_sms(dev));
    for (int64_t v0 = 0, ci = 0; v0 < V; v0 += plan.Vc, ++ci) {
        const int64_t Nc = (V - v0 < plan.Vc) ? V - v0 : plan.Vc;
        const int ntiles = (int)cdiv(Nc, kCeBN);
        {   // GEMM1: logits of the chunk -> per-tile stats and E = exp(z - m_t)
            GemmProblem p{};
            p.a = d_h; p.a_rows_ld = d; p.a_rows = L; p.a_k = d;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = V; p.b_k = d;
            p.M = (int)L; p.N = (int)Nc; p.K = (int)d; p.BN = kCeBN; p.pair = plan.pair;
            p.b_n_off = (int)v0;
            EpiParams ep{};
            ep.tgt = d_tgt; ep.part = c.part; ep.tile0 = (int)(v0 / kCeBN); ep.ztgt = c.ztgt; ep.v0 = (int)v0;
            ep.G = c.G; ep.G_ld = c.Vc;
            ep.eref = ci == 0 ? nullptr : c.mref;
            st = launch_gemm<EPI_CE_EXP, false, false>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
        ce_chunk_kernel<<<(unsigned)cdiv(L, 8), 256, 0, stream>>>(c.part, (int)(v0 / kCeBN), ntiles, (int)L, c.G,
                                                                  c.Vc, c.aref, c.mref, c.alpha, c.beta,
                                                                  ci == 0 ? 1 : 0);
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
        {   // GEMM2: acc = alpha * acc + beta * (E W_c)
            GemmProblem p{};
            p.a = c.G; p.a_rows_ld = c.Vc; p.a_rows = L; p.a_k = c.Vc;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = d; p.b_k = V;
            p.M = (int)L; p.N = (int)d; p.K = (int)round_up(Nc, 64); p.BN = kCeBN; p.pair = plan.pair;
            p.b_k_off = (int)v0;
            EpiParams ep{};
            ep.out = d_dh; ep.out_ld = d; ep.accumulate = ci > 0 ? 1 : 0; ep.alpha = 1.0f;
            ep.row_alpha = c.alpha; ep.row_beta = c.beta;
            p.split_ws = c.split_ws; p.split_tick = c.split_tick; p.split_regions = c.split_regions;
            st = launch_gemm<EPI_F32_ACC, false, true>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
    }
    ce_finalize_kernel<<<(unsigned)c.nblk, kFinThreads, 0, stream>>>(c.part, (int)c.nvt, c.ztgt, d_tgt, d_w, (int)L,
                                                                     (int)V, lse, 1.0f / (float)L, c.block_sums,
                                                                     c.ticket, d_loss, status);
    count_launch();
    if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    ce_fixup_kernel<<<(unsigned)L, 256, 0, stream>>>(d_dh, d, reinterpret_cast<const __nv_bfloat16 *>(d_W), d_tgt,
                                                     d_w, 1.0f / (float)L, c.aref, lse, (int)V);
    count_launch();
    if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    return ATTT_OK;
}

}  // extern "C"
