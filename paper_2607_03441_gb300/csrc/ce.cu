// ce.cu -- Eq. 10 of aTTT on the GPU: the token-weighted next-token CE through
// the frozen LM head, its value and its gradient with respect to the hidden
// states, in one sweep over the vocabulary (4*L*V*d tensor FLOPs: each logit
// is computed once), never holding the [L, V] logits in HBM.
//
// First, per row j, a reference R_j: the target logit z_{j,x_j} (log2 units).
// Then for each vocab chunk c of Vc columns:
//   GEMM1  z = h W_c^T; the epilogue keeps per (row, tile) the max m_t and the
//          sum of exp(z - m_t) (log2 units), writes E = exp(z - R) as bf16
//          against the row's reference R (against m_t for a tile whose max
//          exceeds R by more than 2^64), and catches the target logit;
//   chunk  per row: the chunk max, the running (max, sum) of the logsumexp,
//          a rewrite of E where a tile used its own max, the online-softmax
//          factors of the accumulator's reference A, alpha = exp(A_old -
//          A_new), beta = exp(R_E - A_new), and R <- max(R, chunk max);
//   GEMM2  D = E W_c (W read MN-major by TMA); the epilogue folds it into the
//          fp32 accumulator: acc = alpha * acc + beta * D.
// The last chunk's bookkeeping also forms lse_j and the loss
// (1/L) sum_j w_j (lse_j - z_{j,x_j}) (summed in a fixed order) and folds
// the gradient's factors into alpha and beta, so that the last GEMM2 writes
//   dh_j = (w_j / L) (acc_j exp(A_j - lse_j) - W_{x_j})
// directly.  The LM head gets no gradient (frozen; only the adapter trains).
#include "gemm_launch.cuh"

namespace attt {

constexpr int kCeBN = 256;
constexpr int kCeMaxTiles = 256;  // vocab tiles per chunk at most
constexpr int kChunkWarps = 8;  // ce_chunk_kernel: 8 warps, 32 rows (one per lane) per block
constexpr int kChunkRows = 32;
// fp32 partials of 128 x kCeBN (128 KB each) for the tail split of the dh
// contraction: enough for every CTA of a 160-SM part to hold one piece.
constexpr int kCeSplitRegions = 160;
// Bound of the chunk's bf16 block E [L, Vc] in bytes.
constexpr int64_t kCeEBytes = 1024ll << 20;

struct CeLayout {
    int64_t nvt, Vc, nblk;
    float2 *part;
    float *ztgt, *block_sums;
    float *aref, *mref, *lm, *ls, *alpha, *beta, *gamma;
    unsigned int *ticket;       // [4] loss ticket, then [split_regions] tail-split counters
    unsigned int *split_tick;
    int split_regions;
    float *split_ws;
    __nv_bfloat16 *G;
    size_t bytes;
};

// Upper bound of the vocab chunk: the chunk's bf16 block E (L x Vc) is kept
// near kCeEBytes (1 GB), so the workspace stays bounded whatever V is.  Each chunk costs
// about 20 us of launch, ramp and tail on top of its FLOPs, and E is streamed
// once from L2 or HBM either way, so wider chunks are faster up to this bound.
static int64_t ce_chunk_max(int64_t L, int64_t V) {
    int64_t vc = kCeEBytes / (2 * L);
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
    const double launch = 7.0e-6;  // seconds per launch, ramp-up and tail included
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
    c.nblk = cdiv(L, kChunkRows);
    Carve cv{static_cast<char *>(ws), 0};
    c.part = cv.take<float2>((size_t)(c.nvt * L));
    c.ztgt = cv.take<float>((size_t)L);
    c.block_sums = cv.take<float>((size_t)c.nblk);
    c.aref = cv.take<float>((size_t)L);
    c.mref = cv.take<float>((size_t)L);
    c.lm = cv.take<float>((size_t)L);
    c.ls = cv.take<float>((size_t)L);
    c.alpha = cv.take<float>((size_t)L);
    c.beta = cv.take<float>((size_t)L);
    c.gamma = cv.take<float>((size_t)L);
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

// Reference of the first chunk, one warp per row: R_j = z_{j,x_j} log2 e (an
// fp32 dot product), -inf for a target outside [0, V).  Any R_j at or below
// the row max keeps E from overflowing; the target logit sits near the max
// for the tokens a model is trained on, so E rarely needs a rewrite.
__global__ void __launch_bounds__(256) ce_ref_kernel(const __nv_bfloat16 *__restrict__ h,
                                                     const __nv_bfloat16 *__restrict__ W,
                                                     const int32_t *__restrict__ tgt, int L, int64_t d, int V,
                                                     float *__restrict__ mref) {
    griddep_launch_dependents();  // the first logits contraction may start its main loop
    const int j = blockIdx.x * 8 + (threadIdx.x >> 5);
    const int lane = threadIdx.x & 31;
    if (j >= L) return;
    const int t = tgt[j];
    if (t < 0 || t >= V) {
        if (lane == 0) mref[j] = -INFINITY;
        return;
    }
    const __nv_bfloat16 *hr = h + (int64_t)j * d;
    const __nv_bfloat16 *wr = W + (int64_t)t * d;
    float acc = 0.f;
    for (int64_t k = (int64_t)lane * 8; k < d; k += 256) {  // d % 8 == 0: 16-byte loads
        const uint4 a = __ldg(reinterpret_cast<const uint4 *>(hr + k));
        const uint4 b = __ldg(reinterpret_cast<const uint4 *>(wr + k));
        const __nv_bfloat162 *a2 = reinterpret_cast<const __nv_bfloat162 *>(&a);
        const __nv_bfloat162 *b2 = reinterpret_cast<const __nv_bfloat162 *>(&b);
#pragma unroll
        for (int e = 0; e < 4; ++e) {
            const float2 x = __bfloat1622float2(a2[e]), y = __bfloat1622float2(b2[e]);
            acc = fmaf(x.x, y.x, acc);
            acc = fmaf(x.y, y.y, acc);
        }
    }
    for (int o = 16; o > 0; o >>= 1) acc += __shfl_xor_sync(0xffffffffu, acc, o);
    if (lane == 0) mref[j] = acc * kLog2e;
}

struct CeChunkArgs {
    const float2 *part;  // [vocab tiles, L] (max, sum) of every tile (log2 units)
    int tile0, ntiles, L, V;
    __nv_bfloat16 *G;
    int64_t G_ld;
    float *aref, *mref, *lm, *ls, *alpha, *beta, *gamma;
    int first, last;
    // last chunk only
    const float *ztgt;
    const int32_t *tgt;
    const float *w;
    float inv_L;
    const float *row_scale;  // per-row normaliser, or nullptr (inv_L)
    float *lse_out;  // or nullptr
    float *nll_out;  // or nullptr
    float *block_sums;
    unsigned int *ticket;
    float *loss;
    int *status;
};

// Bookkeeping of one chunk, 32 rows per block (lane = row), log2 units:
//   warp k reads the chunk's tiles t = k (mod 8) with coalesced loads of
//   part[t, rows]; per row the chunk max M_c and the chunk's (max, sum) pair,
//   merged into the running pair (lm, ls);
//   R = mref, the reference GEMM1 wrote this chunk's E against.  A tile whose
//   max exceeded R by more than kCeRefJump used its own max, and then
//   (M_c - R > kCeRefJump) the row is rewritten against M_c tile by tile
//   (Rp = M_c); otherwise it stays against R (Rp = R);
//   acc = alpha * acc + beta * (E W_c) with A_new = max(A_old, Rp),
//   alpha = exp2(A_old - A_new), beta = exp2(Rp - A_new);  mref <- max(R, M_c).
// Last chunk: lse = ln 2 (lm + log2 ls); the weighted NLL of the block's rows
// goes to block_sums and the last block (ticket) adds them in block order;
// alpha and beta take the factor (w/L) exp2(A_new - lse log2 e) and gamma =
// w/L, so the last GEMM2 writes dh itself.
__global__ void __launch_bounds__(kChunkWarps * 32) ce_chunk_kernel(const CeChunkArgs a) {
    __shared__ float s_mc[kChunkWarps][kChunkRows], s_m[kChunkWarps][kChunkRows], s_s[kChunkWarps][kChunkRows];
    __shared__ float s_r[kChunkRows], s_mcf[kChunkRows];
    __shared__ int s_rw[kChunkRows];
    __shared__ bool s_last;
    griddep_launch_dependents();
    griddep_wait();  // the chunk's logits contraction has completed
    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const int j0 = blockIdx.x * kChunkRows;
    const int j = j0 + lane;
    const int L = a.L;
    float mc = -INFINITY, m = -INFINITY, s = 0.f;
    if (j < L) {
        for (int t = warp; t < a.ntiles; t += kChunkWarps) {
            const float2 p = __ldcg(a.part + (int64_t)(a.tile0 + t) * L + j);
            mc = fmaxf(mc, p.x);
            lse_merge(m, s, p.x, p.y);
        }
    }
    s_mc[warp][lane] = mc;
    s_m[warp][lane] = m;
    s_s[warp][lane] = s;
    __syncthreads();
    if (warp == 0) {
        for (int k = 1; k < kChunkWarps; ++k) {
            mc = fmaxf(mc, s_mc[k][lane]);
            lse_merge(m, s, s_m[k][lane], s_s[k][lane]);
        }
        int rw = 0;
        float r = 0.f, contrib = 0.f;
        if (j < L) {
            if (!a.first) {  // running pair first, then this chunk's
                float rm = a.lm[j], rs = a.ls[j];
                lse_merge(rm, rs, m, s);
                m = rm;
                s = rs;
            }
            a.lm[j] = m;
            a.ls[j] = s;
            r = a.mref[j];
            rw = (mc - r > kCeRefJump) ? 1 : 0;
            const float rp = rw ? mc : r;
            const float aold = a.first ? -INFINITY : a.aref[j];
            const float anew = fmaxf(aold, rp);
            float al = (aold == -INFINITY) ? 0.f : exp2f(aold - anew);
            float be = exp2f(rp - anew);
            a.aref[j] = anew;
            a.mref[j] = fmaxf(r, mc);
            if (a.last) {
                const float lse2 = m + log2f(s);
                const float lse = lse2 * 0.69314718055994531f;
                if (a.lse_out) a.lse_out[j] = lse;
                const int t = a.tgt[j];
                const float c = a.w[j] * (a.row_scale ? a.row_scale[j] : a.inv_L);
                float nll;
                if (t < 0 || t >= a.V) {
                    record_error(a.status, ATTT_ERR_TOKEN_RANGE);
                    nll = __int_as_float(0x7fc00000);
                    a.gamma[j] = __int_as_float(0x7fc00000);
                } else {
                    nll = lse - __ldcg(a.ztgt + j);
                    a.gamma[j] = c;
                }
                contrib = a.w[j] * nll;
                if (a.nll_out) a.nll_out[j] = nll;
                const float f = c * exp2f(anew - lse2);
                al *= f;
                be *= f;
            }
            a.alpha[j] = al;
            a.beta[j] = be;
        }
        s_rw[lane] = rw;
        s_r[lane] = r;
        s_mcf[lane] = mc;
        if (a.last) {
            for (int o = 16; o > 0; o >>= 1) contrib += __shfl_xor_sync(0xffffffffu, contrib, o);
            if (lane == 0) {
                a.block_sums[blockIdx.x] = contrib;
                __threadfence();
                s_last = atomicAdd(a.ticket, 1u) == gridDim.x - 1;
            }
        }
    }
    __syncthreads();
    // rows whose tiles used their own max: E against M_c, tile by tile
    const int per_tile = kCeBN / 8;  // uint4 (8 x bf16) per tile row
    for (int i = warp; i < kChunkRows; i += kChunkWarps) {
        if (!s_rw[i]) continue;
        const int jr = j0 + i;
        const float r = s_r[i], mcr = s_mcf[i];
        uint4 *row = reinterpret_cast<uint4 *>(a.G + (int64_t)jr * a.G_ld);
        for (int t = 0; t < a.ntiles; ++t) {
            const float mt = __ldcg(&a.part[(int64_t)(a.tile0 + t) * L + jr].x);
            const float sc = (mt - r > kCeRefJump) ? exp2f(mt - mcr) : exp2f(r - mcr);
            for (int q = lane; q < per_tile; q += 32) {
                uint4 u = row[t * per_tile + q];
                uint32_t *wd = reinterpret_cast<uint32_t *>(&u);
#pragma unroll
                for (int e = 0; e < 4; ++e) {
                    __nv_bfloat162 b = *reinterpret_cast<__nv_bfloat162 *>(&wd[e]);
                    const float2 v = __bfloat1622float2(b);
                    b = __floats2bfloat162_rn(v.x * sc, v.y * sc);
                    wd[e] = *reinterpret_cast<uint32_t *>(&b);
                }
                row[t * per_tile + q] = u;
            }
        }
    }
    if (a.last && s_last && threadIdx.x == 0) {
        __threadfence();
        float total = 0.f;
        for (unsigned i = 0; i < gridDim.x; ++i) total += __ldcg(a.block_sums + i);
        *a.loss = total * a.inv_L;
        *a.ticket = 0u;
    }
}

}  // namespace attt

extern "C" {

size_t attt_ce_workspace_bytes(int64_t L, int64_t d, int64_t V) {
    if (L <= 0 || V <= 0 || d <= 0) return 0;
    return attt::ce_layout(nullptr, L, d, V).bytes;
}

}  // extern "C"

namespace attt {

// The largest attt_ce_workspace_bytes(L, d, V) over 1 <= L <= Lmax.  The
// workspace grows with L while the vocabulary chunk Vc stays the same, and Vc
// (a multiple of kCeBN, clamped to [4096, kCeMaxTiles kCeBN] and to V) only
// changes where kCeEBytes / (2 L) crosses a multiple of kCeBN, so the maximum is
// at Lmax or at the last L of one of those ranges.
size_t ce_workspace_bound(int64_t Lmax, int64_t d, int64_t V) {
    if (Lmax < 1) return 0;
    size_t best = attt_ce_workspace_bytes(Lmax, d, V);
    const int64_t budget = kCeEBytes / 2;
    for (int64_t vc = kCeBN; vc <= kCeMaxTiles * kCeBN; vc += kCeBN) {
        const int64_t L = budget / vc;  // the last L whose unclamped chunk is at least vc
        for (int64_t c = L - 1; c <= L + 1; ++c)
            if (c >= 1 && c <= Lmax) {
                const size_t b = attt_ce_workspace_bytes(c, d, V);
                if (b > best) best = b;
            }
    }
    return best;
}

}  // namespace attt

extern "C" {

size_t attt_ce_workspace_max_bytes(int64_t Lmax, int64_t d, int64_t V) {
    if (Lmax < 1 || V <= 0 || d <= 0) return 0;
    return attt::ce_workspace_bound(Lmax, d, V);
}

attt_status attt_weighted_ce_fwd_bwd(const attt_bf16 *d_h, const attt_bf16 *d_W, const int32_t *d_tgt,
                                     const float *d_w, int64_t L, int64_t d, int64_t V, float *d_loss,
                                     float *d_dh, float *d_lse, void *d_ws, size_t ws_bytes, attt_stream stream) {
    ATTT_NVTX_RANGE();
    return attt::ce_fwd_bwd_run(d_h, d_W, d_tgt, d_w, nullptr, L, d, V, d_loss, d_dh, d_lse, nullptr, d_ws, ws_bytes,
                                stream);
}

}  // extern "C"

namespace attt {

attt_status ce_fwd_bwd_run(const attt_bf16 *d_h, const attt_bf16 *d_W, const int32_t *d_tgt, const float *d_w,
                           const float *row_scale, int64_t L, int64_t d, int64_t V, float *d_loss, float *d_dh,
                           float *d_lse, float *d_nll, void *d_ws, size_t ws_bytes, cudaStream_t stream) {
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
    if (cudaMemsetAsync(c.ticket, 0, sizeof(unsigned int) * (4 + (size_t)c.split_regions), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;

    ce_ref_kernel<<<(unsigned)cdiv(L, 8), 256, 0, stream>>>(reinterpret_cast<const __nv_bfloat16 *>(d_h),
                                                            reinterpret_cast<const __nv_bfloat16 *>(d_W), d_tgt,
                                                            (int)L, d, (int)V, c.mref);
    count_launch();
    if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;

    const CePlan plan = ce_plan(L, d, V, num_sms(dev));
    for (int64_t v0 = 0, ci = 0; v0 < V; v0 += plan.Vc, ++ci) {
        const int64_t Nc = (V - v0 < plan.Vc) ? V - v0 : plan.Vc;
        const int ntiles = (int)cdiv(Nc, kCeBN);
        const bool last = v0 + Nc >= V;
        {   // GEMM1: logits of the chunk -> per-tile stats and E = exp(z - R)
            GemmProblem p{};
            p.a = d_h; p.a_rows_ld = d; p.a_rows = L; p.a_k = d;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = V; p.b_k = d;
            p.M = (int)L; p.N = (int)Nc; p.K = (int)d; p.BN = kCeBN; p.pair = plan.pair;
            p.b_n_off = (int)v0;
            p.pdl = true;
            p.operands_ready = true;  // h and W are inputs of the call
            EpiParams ep{};
            ep.tgt = d_tgt; ep.part = c.part; ep.tile0 = (int)(v0 / kCeBN); ep.ztgt = c.ztgt; ep.v0 = (int)v0;
            ep.G = c.G; ep.G_ld = c.Vc;
            ep.eref = c.mref;
            st = launch_gemm<EPI_CE_EXP, false, false>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
        CeChunkArgs ca{};
        ca.part = c.part; ca.tile0 = (int)(v0 / kCeBN); ca.ntiles = ntiles; ca.L = (int)L; ca.V = (int)V;
        ca.G = c.G; ca.G_ld = c.Vc;
        ca.aref = c.aref; ca.mref = c.mref; ca.lm = c.lm; ca.ls = c.ls;
        ca.alpha = c.alpha; ca.beta = c.beta; ca.gamma = c.gamma;
        ca.first = ci == 0 ? 1 : 0; ca.last = last ? 1 : 0;
        ca.ztgt = c.ztgt; ca.tgt = d_tgt; ca.w = d_w; ca.inv_L = 1.0f / (float)L; ca.lse_out = d_lse;
        ca.row_scale = row_scale; ca.nll_out = d_nll;
        ca.block_sums = c.block_sums; ca.ticket = c.ticket; ca.loss = d_loss; ca.status = status;
        {
            cudaLaunchConfig_t cfg = {};
            cfg.gridDim = dim3((unsigned)c.nblk);
            cfg.blockDim = dim3(kChunkWarps * 32);
            cfg.stream = stream;
            cudaLaunchAttribute attr[1];
            attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
            attr[0].val.programmaticStreamSerializationAllowed = 1;
            cfg.attrs = attr;
            cfg.numAttrs = 1;
            if (cudaLaunchKernelEx(&cfg, ce_chunk_kernel, ca) != cudaSuccess) return ATTT_ERR_CUDA;
        }
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
        {   // GEMM2: acc = alpha * acc + beta * (E W_c)
            GemmProblem p{};
            p.a = c.G; p.a_rows_ld = c.Vc; p.a_rows = L; p.a_k = c.Vc;
            p.b = d_W; p.b_rows_ld = d; p.b_rows = d; p.b_k = V;
            p.M = (int)L; p.N = (int)d; p.K = (int)round_up(Nc, 64); p.BN = kCeBN; p.pair = plan.pair;
            p.b_k_off = (int)v0;
            p.pdl = true;  // E may be rewritten by the chunk kernel: the producer waits
            EpiParams ep{};
            ep.out = d_dh; ep.out_ld = d; ep.accumulate = ci > 0 ? 1 : 0; ep.alpha = 1.0f;
            ep.row_alpha = c.alpha; ep.row_beta = c.beta;
            if (last) {  // dh = (w/L) (acc exp(A - lse) - W_target), factors folded by the chunk kernel
                ep.row_gamma = c.gamma; ep.fix_tgt = d_tgt;
                ep.fix_W = reinterpret_cast<const __nv_bfloat16 *>(d_W); ep.fix_ld = d; ep.fix_V = (int)V;
            }
            p.split_ws = c.split_ws; p.split_tick = c.split_tick; p.split_regions = c.split_regions;
            st = launch_gemm<EPI_F32_ACC, false, true>(p, ep, dev, stream);
            if (st != ATTT_OK) return st;
        }
    }
    return ATTT_OK;
}

}  // namespace attt
