// lora.cu -- adapter gradients and the SGD step of the aTTT update (Eq. 2,
// Algorithm 1's gradient step, the LoRA adapter of Appendix C:
// y = x W0 + s (x A) B).
//
// For projections p sharing one input x [L, din]:
//   u   = x [A_0 | A_1 | ...]        one contraction for all p (x read once)
//   v_p = dy_p B_p^T
//   dA  = s x^T [v_0 | v_1 | ...]    one contraction for all p (x read once)
//   dB_p^T = s dy_p^T u_p            (dout on the 128-row side)
// Every contraction puts the long dimension (L, din or dout) on the 128-row
// MMA side and the rank on N, so the tensor core streams x and dy once per
// pass at HBM rate.  Reductions over L (or din/dout) are split across CTAs
// (stream-K, tc_group.cuh) and summed in a fixed order by the piece that
// finishes each tile last; u and v go to bf16 in between.  Three launches per
// call: prep (adapters to K-major), pass 1 (u and every v_p, grouped), pass 2
// (dA and every dB_p, grouped).
//
// The adapted projection itself (for a chained update, where the projection
// feeds the LM head): the forward h = x W0 + s (x A) B and the input gradient
// dx = dy W0^T + s (dy B^T) A^T.  Each is one tcgen05 contraction whose K runs
// over two operand pairs, [x | s u] [W0 ; B] and [dy | s v] [W0^T ; A^T], after
// a skinny grouped launch that forms s u = s x A or s v = s dy B^T in bf16.
#include <cmath>

#include "gemm_launch.cuh"
#include "tc_group.cuh"

namespace attt {

struct LoraLayout {
    int rpad, Nu, BN;
    int64_t Lp;
    __nv_bfloat16 *AT;            // [Nu, din]
    __nv_bfloat16 *BT[kMaxProj];  // [rpad, dout_p]
    __nv_bfloat16 *uT16, *vT16;   // [Nu, Lp] each, contiguous
    int64_t tiles;                // group-wide tiles of the larger pass
    unsigned int *tickets;        // [tiles] arrival counters (both passes)
    float *part;                  // [tiles + kGroupMaxGrid] partial slots of 128 x BN fp32
    size_t bytes;
};

static LoraLayout lora_layout(void *ws, int64_t L, int64_t din, int nproj, const int64_t *dout, int r) {
    LoraLayout c{};
    c.rpad = (int)round_up(r, 16);
    c.Nu = nproj * c.rpad;
    c.BN = c.Nu <= 256 ? c.Nu : 256;
    c.Lp = round_up(L, 8);
    // pass 1: u (L x Nu) and each v_p (L x rpad); pass 2: dA (din x Nu) and each dB_p (dout_p x rpad)
    int64_t t1 = cdiv(L, 128) * cdiv(c.Nu, c.BN), t2 = cdiv(din, 128) * cdiv(c.Nu, c.BN);
    for (int p = 0; p < nproj; ++p) {
        t1 += cdiv(L, 128) * cdiv(c.rpad, c.BN);
        t2 += cdiv(dout[p], 128) * cdiv(c.rpad, c.BN);
    }
    c.tiles = t1 > t2 ? t1 : t2;
    Carve cv{static_cast<char *>(ws), 0};
    c.AT = cv.take<__nv_bfloat16>((size_t)(c.Nu * din));
    for (int p = 0; p < nproj; ++p) c.BT[p] = cv.take<__nv_bfloat16>((size_t)(c.rpad * dout[p]));
    c.uT16 = cv.take<__nv_bfloat16>((size_t)(2 * c.Nu * c.Lp));
    c.vT16 = c.uT16 + (size_t)c.Nu * c.Lp;
    c.tickets = cv.take<unsigned int>((size_t)c.tiles);
    c.part = cv.take<float>((size_t)(c.tiles + kGroupMaxGrid) * 128 * c.BN);
    c.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return c;
}

struct PrepArgs {
    const __nv_bfloat16 *A[kMaxProj];
    const __nv_bfloat16 *B[kMaxProj];
    __nv_bfloat16 *BT[kMaxProj];
    int64_t dout[kMaxProj];
    int nproj, r, rpad;
    int64_t din;
    __nv_bfloat16 *AT;
    unsigned int *tickets;
    int64_t ntickets;
};

// AT[p*rpad + c, i] = A_p[i, c] (zero for c >= r); BT_p[c, o] = B_p[c, o]
// (zero rows for c >= r); and the tile tickets set to zero, block row p of
// the grid doing projection p's share.  The transpose goes through shared
// memory in slabs of 64 rows of A_p: a slab is contiguous in A_p and is read
// as 16-byte vectors, and each thread writes 8 consecutive elements of a row
// of AT as one 16-byte vector (din, dout and every tensor pointer are
// multiples of 8 elements / 16 bytes, and a slab starts at a multiple of 64
// rows).  BT is copied 16 bytes at a time.
constexpr int kPrepRows = 64;

__global__ void __launch_bounds__(256) lora_prep_kernel(PrepArgs a) {
    __shared__ __align__(16) __nv_bfloat16 slab[kPrepRows * 64];  // [row of A_p][column c], r <= 64
    griddep_launch_dependents();  // pass 1 may launch; it waits for this grid before reading AT, BT
    const int p = blockIdx.y;
    const int64_t nslab = (a.din + kPrepRows - 1) / kPrepRows;
    for (int64_t sb = blockIdx.x; sb < nslab; sb += gridDim.x) {
        const int64_t k0 = sb * kPrepRows;
        const int rows = (int)min((int64_t)kPrepRows, a.din - k0);  // a multiple of 8
        const uint4 *src = reinterpret_cast<const uint4 *>(a.A[p] + k0 * a.r);
        uint4 *dst = reinterpret_cast<uint4 *>(slab);
        for (int e = threadIdx.x; e < rows * a.r / 8; e += blockDim.x) dst[e] = src[e];  // slab[kk * r + c]
        __syncthreads();
        const int runs = rows / 8;  // 8-row runs per column of AT
        for (int e = threadIdx.x; e < a.rpad * runs; e += blockDim.x) {
            const int c = e / runs, kk0 = (e - c * runs) * 8;
            __align__(16) __nv_bfloat16 v[8];
#pragma unroll
            for (int t = 0; t < 8; ++t) v[t] = c < a.r ? slab[(kk0 + t) * a.r + c] : __float2bfloat16_rn(0.f);
            *reinterpret_cast<uint4 *>(a.AT + ((int64_t)p * a.rpad + c) * a.din + k0 + kk0) =
                *reinterpret_cast<const uint4 *>(v);
        }
        __syncthreads();
    }
    const int64_t nB8 = (int64_t)a.rpad * a.dout[p] / 8;  // 16-byte vectors of BT_p
    const int64_t rB8 = (int64_t)a.r * a.dout[p] / 8;     // of them copied from B_p (rows c < r)
    const int64_t ztk = (a.ntickets + a.nproj - 1) / a.nproj;  // this row's slice of the tickets
    const int64_t n = nB8 > ztk ? nB8 : ztk;
    const uint4 *b_src = reinterpret_cast<const uint4 *>(a.B[p]);
    uint4 *b_dst = reinterpret_cast<uint4 *>(a.BT[p]);
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        if (i < nB8) b_dst[i] = i < rB8 ? b_src[i] : make_uint4(0u, 0u, 0u, 0u);
        if (i < ztk && p * ztk + i < a.ntickets) a.tickets[p * ztk + i] = 0u;
    }
}

// SGD: p <- p - lr * g (product then difference, both rounded), bf16 refresh.
// One tensor (n elements): four elements per thread step (16-byte loads of p
// and g, a 16-byte store of p, an 8-byte store of the bf16 copy) when every
// pointer allows it, else one.
__device__ __forceinline__ void sgd_range(float *p32, const float *g, __nv_bfloat16 *p16, int64_t n, float lr,
                                          int64_t t0, int64_t stride) {
    const bool vec = ((reinterpret_cast<uintptr_t>(p32) | reinterpret_cast<uintptr_t>(g)) & 15) == 0 &&
                     (reinterpret_cast<uintptr_t>(p16) & 7) == 0;
    const int64_t n4 = vec ? n / 4 : 0;
    for (int64_t i = t0; i < n4; i += stride) {
        const float4 p = reinterpret_cast<const float4 *>(p32)[i];
        const float4 d = reinterpret_cast<const float4 *>(g)[i];
        const float4 v = make_float4(__fsub_rn(p.x, __fmul_rn(lr, d.x)), __fsub_rn(p.y, __fmul_rn(lr, d.y)),
                                     __fsub_rn(p.z, __fmul_rn(lr, d.z)), __fsub_rn(p.w, __fmul_rn(lr, d.w)));
        reinterpret_cast<float4 *>(p32)[i] = v;
        if (p16) {
            __nv_bfloat162 o[2] = {__floats2bfloat162_rn(v.x, v.y), __floats2bfloat162_rn(v.z, v.w)};
            reinterpret_cast<uint2 *>(p16)[i] = *reinterpret_cast<uint2 *>(o);
        }
    }
    for (int64_t i = 4 * n4 + t0; i < n; i += stride) {
        const float v = __fsub_rn(p32[i], __fmul_rn(lr, g[i]));
        p32[i] = v;
        if (p16) p16[i] = __float2bfloat16_rn(v);
    }
}

__global__ void lora_step_kernel(float *A32, const float *dA, __nv_bfloat16 *A16, int64_t nA, float *B32,
                                 const float *dB, __nv_bfloat16 *B16, int64_t nB, float lr) {
    const int64_t t0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x, stride = (int64_t)gridDim.x * blockDim.x;
    sgd_range(A32, dA, A16, nA, lr, t0, stride);
    sgd_range(B32, dB, B16, nB, lr, t0, stride);
}

// AdamW (decoupled weight decay) on the fp32 masters of A and B, with the
// moments m, v (fp32) and the bf16 refresh; every product and sum rounded on
// its own (no FMA):
//   p <- p (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2
//   p <- p - step_size m / (sqrt(v) / bc2_sqrt + eps)
// with step_size = lr / (1 - b1^t) and bc2_sqrt = sqrt(1 - b2^t) from the host.
struct AdamWArgs {
    float *p[2];
    const float *g[2];
    float *m[2], *v[2];
    __nv_bfloat16 *p16[2];
    int64_t n[2];
    float decay, b1, one_b1, b2, one_b2, step_size, bc2_sqrt, eps;
};

__global__ void lora_adamw_kernel(const AdamWArgs a) {
    const int64_t total = a.n[0] + a.n[1];
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < total;
         i += (int64_t)gridDim.x * blockDim.x) {
        const int t = i < a.n[0] ? 0 : 1;
        const int64_t k = t == 0 ? i : i - a.n[0];
        const float g = a.g[t][k];
        const float m = __fadd_rn(__fmul_rn(a.b1, a.m[t][k]), __fmul_rn(a.one_b1, g));
        const float v = __fadd_rn(__fmul_rn(a.b2, a.v[t][k]), __fmul_rn(a.one_b2, __fmul_rn(g, g)));
        a.m[t][k] = m;
        a.v[t][k] = v;
        const float denom = __fadd_rn(__fdiv_rn(__fsqrt_rn(v), a.bc2_sqrt), a.eps);
        const float p = __fsub_rn(__fmul_rn(a.p[t][k], a.decay), __fdiv_rn(__fmul_rn(a.step_size, m), denom));
        a.p[t][k] = p;
        if (a.p16[t]) a.p16[t][k] = __float2bfloat16_rn(p);
    }
}

// dst = bf16(src), round to nearest even; 8 elements per thread per step
// (two 16-byte loads, one 16-byte store) when both are 16-byte aligned.
__global__ void cast_bf16_kernel(const float *__restrict__ src, __nv_bfloat16 *__restrict__ dst, int64_t n) {
    const int64_t stride = (int64_t)gridDim.x * blockDim.x;
    const bool vec = ((reinterpret_cast<uintptr_t>(src) | reinterpret_cast<uintptr_t>(dst)) & 15) == 0;
    const int64_t n8 = vec ? n / 8 : 0;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n8; i += stride) {
        const float4 a = reinterpret_cast<const float4 *>(src)[2 * i];
        const float4 b = reinterpret_cast<const float4 *>(src)[2 * i + 1];
        __nv_bfloat162 o[4] = {__floats2bfloat162_rn(a.x, a.y), __floats2bfloat162_rn(a.z, a.w),
                               __floats2bfloat162_rn(b.x, b.y), __floats2bfloat162_rn(b.z, b.w)};
        reinterpret_cast<uint4 *>(dst)[i] = *reinterpret_cast<uint4 *>(o);
    }
    for (int64_t i = 8 * n8 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += stride)
        dst[i] = __float2bfloat16_rn(src[i]);
}

static unsigned grid_for(int64_t n, int threads, int dev) {
    int64_t b = cdiv(n, threads);
    const int64_t cap = (int64_t)num_sms(dev) * 8;
    if (b > cap) b = cap;
    if (b < 1) b = 1;
    return (unsigned)b;
}

// One problem of a grouped launch (see tc_group.cuh).
struct GroupSpec {
    const void *a;
    int64_t a_rows_ld, a_rows, a_k;  // as GemmProblem
    const void *b;
    int64_t b_rows_ld, b_rows, b_k;
    int M, N, K;
    int b_n_off;
    int out;  // GroupOut
    float alpha;
    int r, rpad;
    int64_t ld;
    float *out32;
    __nv_bfloat16 *out16;
    float *outp[kMaxProj];
};

constexpr int kGroupMinStages = 2;
// Ring stages a grouped launch's shared-memory ring keeps when it can (the
// stage shape: the most K blocks per stage that leaves this many).  Measured
// on GB300 (A/B in one process, the order of the two builds alternating):
// five stages of one K block against two of two took the 32B-class q/k/v
// group from 145.5 to 131.7 us and the o group from 121.5 to 106.6 us.
constexpr int kGroupMinRing = 5;

// Launches every problem of `specs` in one grouped kernel; every CTA streams
// the same number of K stages (stream-K split, tc_group.cuh).
template <bool A_MN, bool B_MN, int NP = kMaxGroup>
static attt_status launch_group(const GroupSpec *specs, int n, int BN, float *part, unsigned int *tickets, int dev,
                                cudaStream_t stream, int *status) {
    if (n < 1 || n > NP || BN < 16 || BN > 256 || BN % 16 != 0) return ATTT_ERR_INVALID_ARG;
    static_assert(!B_MN, "grouped B operands are K-major");
    GroupMaps<NP> maps;
    GroupArgs<NP> g{};
    g.nprob = n;
    g.BN = BN;
    g.part = part;
    g.tickets = tickets;
    // Up to four 64-deep K blocks per stage, so each operand row is fetched in
    // runs of up to 512 bytes (better DRAM locality than one 128-byte piece per
    // row per block), as long as at least two stages fit in shared memory.
    g.kbs = 1;
    g.stages = 0;
    // the most K blocks per stage that leaves at least kGroupMinRing stages
    // (the two producers each keep a few stages in flight), else one block
    for (int kbs = 4; kbs >= 1 && g.stages == 0; kbs /= 2) {
        const size_t per_stage = (size_t)kbs * (kABytes + gemm_b_stage_bytes(BN));
        int st = 8;
        while (st >= 2 && 1024 + st * per_stage + kGroupTBytes + 8 * (2 * st + 5) + 16 > kMaxSmem) --st;
        if (st >= kGroupMinRing || (kbs == 1 && st >= 2)) { g.kbs = kbs; g.stages = st; }
    }
    if (g.stages == 0) return ATTT_ERR_UNSUPPORTED;
    g.tmem_cols = gemm_tmem_cols(BN);
    g.status = status ? status : device_status_word(dev);
    const int sms = num_sms(dev);
    int64_t stages = 0;
    int tiles = 0;
    for (int q = 0; q < n; ++q) {
        const GroupSpec &sp = specs[q];
        if (sp.M <= 0 || sp.N <= 0 || sp.K <= 0) return ATTT_ERR_INVALID_ARG;
        bool ok;
        if (!A_MN)
            ok = make_tmap_bf16(&maps.a[q], sp.a, (uint64_t)sp.a_k, (uint64_t)sp.a_rows, (uint64_t)sp.a_rows_ld * 2,
                                64, 128);
        else
            ok = make_tmap_bf16(&maps.a[q], sp.a, (uint64_t)sp.a_rows, (uint64_t)sp.a_k, (uint64_t)sp.a_rows_ld * 2,
                                64, 64);
        if (!ok) return ATTT_ERR_INVALID_ARG;
        if (!make_tmap_bf16(&maps.b[q], sp.b, (uint64_t)sp.b_k, (uint64_t)sp.b_rows, (uint64_t)sp.b_rows_ld * 2, 64,
                            (uint32_t)BN))
            return ATTT_ERR_INVALID_ARG;
        GroupProblem &pr = g.prob[q];
        pr.M = sp.M;
        pr.N = sp.N;
        pr.tiles_m = (int)cdiv(sp.M, 128);
        pr.tiles_n = (int)cdiv(sp.N, BN);
        pr.kb_total = (int)cdiv(sp.K, 64);
        pr.nst = (int)cdiv(pr.kb_total, g.kbs);
        pr.b_n_off = sp.b_n_off;
        pr.stage_begin = stages;
        pr.tile_begin = tiles;
        pr.out = sp.out;
        pr.alpha = sp.alpha;
        pr.r = sp.r;
        pr.rpad = sp.rpad;
        pr.ld = sp.ld;
        pr.out32 = sp.out32;
        pr.out16 = sp.out16;
        for (int j = 0; j < kMaxProj; ++j) pr.outp[j] = sp.outp[j];
        stages += (int64_t)pr.tiles_m * pr.tiles_n * pr.nst;
        tiles += pr.tiles_m * pr.tiles_n;
    }
    g.total_stages = stages;
    const size_t smem =
        1024 + (size_t)g.stages * g.kbs * (kABytes + gemm_b_stage_bytes(BN)) + kGroupTBytes + 8 * (2 * g.stages + 5) + 16;
    auto kern = tc_gemm_group_kernel<A_MN, B_MN, NP>;
    if (!set_smem_limit(reinterpret_cast<const void *>(kern), smem, dev)) return ATTT_ERR_CUDA;
    // every CTA gets at least kGroupMinStages stages (at least one), so that a
    // tile is not cut into more pieces than its final sum can afford
    int64_t gmax = stages / kGroupMinStages;
    if (gmax < 1) gmax = 1;
    int grid = gmax < sms ? (int)gmax : sms;
    if (grid > kGroupMaxGrid) grid = kGroupMaxGrid;
    // a programmatic dependent of the previous kernel of the call (prep, or pass 1)
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)grid);
    cfg.blockDim = dim3(kGroupThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    if (cudaLaunchKernelEx(&cfg, kern, maps, g) != cudaSuccess) return ATTT_ERR_CUDA;
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status lora_grad_run(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj, const attt_bf16 *const *d_dy,
                          const int64_t *dout, const attt_bf16 *const *d_A, const attt_bf16 *const *d_B, int r,
                          float scale, float *const *d_dA, float *const *d_dB, void *d_ws, size_t ws_bytes,
                          int *status, cudaStream_t stream) {
    if (!d_x || !d_dy || !dout || !d_A || !d_B || !d_dA || !d_dB) return ATTT_ERR_INVALID_ARG;
    if (nproj < 1 || nproj > kMaxProj || r < 1 || r > 64 || L < 1 || din < 8 || din % 8 != 0)
        return ATTT_ERR_INVALID_ARG;
    if (L > (1ll << 30) || din > (1ll << 30)) return ATTT_ERR_UNSUPPORTED;
    if (!aligned16(d_x)) return ATTT_ERR_INVALID_ARG;
    for (int p = 0; p < nproj; ++p) {
        if (!d_dy[p] || !d_A[p] || !d_B[p] || !d_dA[p] || !d_dB[p]) return ATTT_ERR_INVALID_ARG;
        if (dout[p] < 8 || dout[p] % 8 != 0 || dout[p] > (1ll << 30)) return ATTT_ERR_INVALID_ARG;
        if (!aligned16(d_dy[p]) || !aligned16(d_A[p]) || !aligned16(d_B[p])) return ATTT_ERR_INVALID_ARG;
    }
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_lora_workspace_bytes(L, din, nproj, dout, r))
        return ATTT_ERR_WORKSPACE;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;

    LoraLayout c = lora_layout(d_ws, L, din, nproj, dout, r);
    const int BN = c.BN;

    // prep: adapters to K-major (rank padded with zeros), accumulators zeroed
    {
        PrepArgs a{};
        int64_t maxn = cdiv(din, kPrepRows) * 256;  // the transpose slabs (one block each)
        for (int p = 0; p < nproj; ++p) {
            a.A[p] = reinterpret_cast<const __nv_bfloat16 *>(d_A[p]);
            a.B[p] = reinterpret_cast<const __nv_bfloat16 *>(d_B[p]);
            a.BT[p] = c.BT[p];
            a.dout[p] = dout[p];
            if (c.rpad * dout[p] / 8 > maxn) maxn = c.rpad * dout[p] / 8;
        }
        a.nproj = nproj; a.r = r; a.rpad = c.rpad; a.din = din; a.AT = c.AT;
        a.tickets = c.tickets; a.ntickets = c.tiles;
        if (a.ntickets / nproj > maxn) maxn = a.ntickets / nproj + 1;
        dim3 grid(grid_for(maxn, 256, dev), nproj);
        lora_prep_kernel<<<grid, 256, 0, stream>>>(a);
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    }

    // pass 1: u^T = (x AT^T)^T and v_p^T = (dy_p BT_p^T)^T, fp32 sums then bf16
    {
        GroupSpec sp[kMaxGroup];
        int n = 0;
        GroupSpec &u = sp[n++];
        u = GroupSpec{};
        u.a = d_x; u.a_rows_ld = din; u.a_rows = L; u.a_k = din;
        u.b = c.AT; u.b_rows_ld = din; u.b_rows = c.Nu; u.b_k = din;
        u.M = (int)L; u.N = c.Nu; u.K = (int)din;
        u.out = GOUT_T16; u.out16 = c.uT16; u.ld = c.Lp; u.alpha = 1.0f; u.r = c.rpad; u.rpad = c.rpad;
        for (int q = 0; q < nproj; ++q) {
            GroupSpec &v = sp[n++];
            v = GroupSpec{};
            v.a = d_dy[q]; v.a_rows_ld = dout[q]; v.a_rows = L; v.a_k = dout[q];
            v.b = c.BT[q]; v.b_rows_ld = dout[q]; v.b_rows = c.rpad; v.b_k = dout[q];
            v.M = (int)L; v.N = c.rpad; v.K = (int)dout[q];
            v.out = GOUT_T16; v.out16 = c.vT16 + (size_t)q * c.rpad * c.Lp; v.ld = c.Lp; v.alpha = 1.0f;
            v.r = c.rpad; v.rpad = c.rpad;
        }
        st = launch_group<false, false>(sp, n, BN, c.part, c.tickets, dev, stream, status);
        if (st != ATTT_OK) return st;
    }

    // pass 2: dA_p = s x^T v_p (all p at once, x MN-major) and
    //         dB_p^T = s dy_p^T u_p (dy MN-major), stored transposed into dB_p
    {
        GroupSpec sp[kMaxGroup];
        int n = 0;
        GroupSpec &a = sp[n++];
        a = GroupSpec{};
        a.a = d_x; a.a_rows_ld = din; a.a_rows = din; a.a_k = L;
        a.b = c.vT16; a.b_rows_ld = c.Lp; a.b_rows = c.Nu; a.b_k = L;  // padding columns read as zeros
        a.M = (int)din; a.N = c.Nu; a.K = (int)L;
        a.out = GOUT_N32;
        for (int q = 0; q < nproj; ++q) a.outp[q] = d_dA[q];
        a.alpha = scale; a.r = r; a.rpad = c.rpad;
        for (int q = 0; q < nproj; ++q) {
            GroupSpec &b = sp[n++];
            b = GroupSpec{};
            b.a = d_dy[q]; b.a_rows_ld = dout[q]; b.a_rows = dout[q]; b.a_k = L;
            b.b = c.uT16; b.b_rows_ld = c.Lp; b.b_rows = c.Nu; b.b_k = L;
            b.b_n_off = q * c.rpad;
            b.M = (int)dout[q]; b.N = c.rpad; b.K = (int)L;
            b.out = GOUT_T32; b.out32 = d_dB[q]; b.ld = dout[q]; b.alpha = scale; b.r = r; b.rpad = c.rpad;
        }
        st = launch_group<true, false>(sp, n, BN, c.part, c.tickets, dev, stream, status);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}


// ---------------------------------------------------------------------------
// The adapted projections of a batch of episodes (attt_batch_update): each
// episode has its own rows of the stacked x and dy and its own adapter.
//   prep      every episode's A^T and B padded to rpad rows (stacked by
//             episode), and A concatenated along the rank, [din, E rpad];
//   forward   h = [x | S] [W0 ; B_all] over every row in one contraction, S
//             block-diagonal: row j of episode e holds s (x_j A_e) in columns
//             [e rpad, (e + 1) rpad) and zeros elsewhere (a grouped pass with one
//             problem per episode writes the blocks);
//   grads     u, v (pass 1) and dA, dB (pass 2) of up to kGroupEpisodes
//             episodes as the problems of one grouped launch each;
//   dx        [dy | S'] [W0^T ; A_cat^T] in one contraction, S' block-diagonal
//             with s (dy_j B_e^T).
// Every episode's rpad values fall in one 16-deep MMA step of the adapter
// part of K and the other episodes' blocks add exact zeros, so each row's h
// and dx are those of the episode's own call.
// ---------------------------------------------------------------------------

// Split slots of the dx contraction's tail split (as for the CE's dh).
constexpr int kDxSplitRegions = 160;

struct BatchLoraLayout {
    int rpad;
    int64_t Ncat;                   // E rpad
    __nv_bfloat16 *AT, *BT;         // [E rpad, din], [E rpad, d]: episode e's rows at e rpad
    __nv_bfloat16 *ACAT;            // [din, E rpad]
    __nv_bfloat16 *uT, *vT;         // per episode [rpad, Lp_e], laid one after another
    __nv_bfloat16 *S;               // [rows_bound, E rpad] block-diagonal s u or s v
    int64_t tiles;
    unsigned int *tickets;          // [tiles + kDxSplitRegions]
    float *part, *split_ws;
    size_t bytes;
};

// rows_bound: an upper bound of sum_e round_up(L_e, 8) (sizes every buffer)
static BatchLoraLayout batch_lora_layout(void *ws, int E, int64_t rows_bound, int64_t din, int64_t d, int r) {
    BatchLoraLayout c{};
    c.rpad = (int)round_up(r, 16);
    c.Ncat = (int64_t)E * c.rpad;
    const int64_t t1 = 2 * (cdiv(rows_bound, 128) + E), t2 = (int64_t)E * (cdiv(din, 128) + cdiv(d, 128));
    c.tiles = t1 > t2 ? t1 : t2;
    Carve cv{static_cast<char *>(ws), 0};
    c.AT = cv.take<__nv_bfloat16>((size_t)c.Ncat * din);
    c.BT = cv.take<__nv_bfloat16>((size_t)c.Ncat * d);
    c.ACAT = cv.take<__nv_bfloat16>((size_t)din * c.Ncat);
    c.uT = cv.take<__nv_bfloat16>((size_t)c.rpad * rows_bound);
    c.vT = cv.take<__nv_bfloat16>((size_t)c.rpad * rows_bound);
    c.S = cv.take<__nv_bfloat16>((size_t)rows_bound * c.Ncat);
    c.tickets = cv.take<unsigned int>((size_t)(c.tiles + kDxSplitRegions));
    c.part = cv.take<float>((size_t)(c.tiles + kGroupMaxGrid) * 128 * c.rpad);
    c.split_ws = cv.take<float>((size_t)kDxSplitRegions * 128 * 256);
    c.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return c;
}

struct BatchPrepArgs {
    const __nv_bfloat16 *A, *B;  // stacked [E][din][r], [E][r][d]
    __nv_bfloat16 *AT, *BT, *ACAT;
    int r, rpad;
    int64_t din, d, Ncat;
    unsigned int *tickets;
    int64_t ntickets;
};

// For episode e = blockIdx.y of a batch's stacked adapters: AT[e rpad + c, i]
// = A_e[i, c], ACAT[i, e rpad + c] = A_e[i, c], BT[e rpad + c, o] = B_e[c, o]
// (zero for c >= r), and the tickets zeroed (each episode row a slice).
__global__ void __launch_bounds__(256) lora_prep_batch_kernel(BatchPrepArgs a) {
    __shared__ __nv_bfloat16 slab[kPrepRows][64 + 2];
    griddep_launch_dependents();
    const int e = blockIdx.y;
    const __nv_bfloat16 *A = a.A + (int64_t)e * a.din * a.r;
    const __nv_bfloat16 *B = a.B + (int64_t)e * a.r * a.d;
    __nv_bfloat16 *AT = a.AT + (int64_t)e * a.rpad * a.din;
    __nv_bfloat16 *BT = a.BT + (int64_t)e * a.rpad * a.d;
    const int64_t nslab = (a.din + kPrepRows - 1) / kPrepRows;
    for (int64_t sb = blockIdx.x; sb < nslab; sb += gridDim.x) {
        const int64_t k0 = sb * kPrepRows;
        const int rows = (int)min((int64_t)kPrepRows, a.din - k0);
        for (int i = threadIdx.x; i < rows * a.r; i += blockDim.x) {
            const int kk = i / a.r, c = i - kk * a.r;
            slab[kk][c] = A[(k0 + kk) * a.r + c];
        }
        __syncthreads();
        for (int i = threadIdx.x; i < a.rpad * kPrepRows; i += blockDim.x) {
            const int c = i / kPrepRows, kk = i - c * kPrepRows;
            if (kk < rows) AT[(int64_t)c * a.din + k0 + kk] = c < a.r ? slab[kk][c] : __float2bfloat16_rn(0.f);
        }
        for (int i = threadIdx.x; i < rows * a.rpad; i += blockDim.x) {
            const int kk = i / a.rpad, c = i - kk * a.rpad;
            a.ACAT[(k0 + kk) * a.Ncat + (int64_t)e * a.rpad + c] = c < a.r ? slab[kk][c] : __float2bfloat16_rn(0.f);
        }
        __syncthreads();
    }
    const int64_t nB = (int64_t)a.rpad * a.d;
    const int64_t ztk = (a.ntickets + gridDim.y - 1) / gridDim.y;
    const int64_t n = nB > ztk ? nB : ztk;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        if (i < nB) {
            const int c = (int)(i / a.d);
            BT[i] = c < a.r ? B[i] : __float2bfloat16_rn(0.f);
        }
        if (i < ztk && e * ztk + i < a.ntickets) a.tickets[e * ztk + i] = 0u;
    }
}

size_t batch_adapter_workspace(int E, int64_t rows_bound, int64_t din, int64_t d, int r) {
    return batch_lora_layout(nullptr, E, rows_bound, din, d, r).bytes;
}

static attt_status batch_check(int E, int64_t din, int64_t d, int r, int64_t rows_bound, size_t ws_bytes,
                               const void *ws) {
    if (E < 1 || r < 1 || r > 64 || din < 8 || d < 8 || din % 8 || d % 8) return ATTT_ERR_INVALID_ARG;
    if (!ws || !aligned256(ws) || ws_bytes < batch_adapter_workspace(E, rows_bound, din, d, r))
        return ATTT_ERR_WORKSPACE;
    return ATTT_OK;
}

attt_status batch_adapter_prep(const attt_bf16 *d_A16, const attt_bf16 *d_B16, int E, int64_t din, int64_t d, int r,
                               int64_t rows_bound, void *d_ws, size_t ws_bytes, cudaStream_t stream) {
    attt_status st = batch_check(E, din, d, r, rows_bound, ws_bytes, d_ws);
    if (st != ATTT_OK) return st;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    BatchLoraLayout c = batch_lora_layout(d_ws, E, rows_bound, din, d, r);
    BatchPrepArgs a{};
    a.A = reinterpret_cast<const __nv_bfloat16 *>(d_A16);
    a.B = reinterpret_cast<const __nv_bfloat16 *>(d_B16);
    a.AT = c.AT; a.BT = c.BT; a.ACAT = c.ACAT; a.r = r; a.rpad = c.rpad; a.din = din; a.d = d; a.Ncat = c.Ncat;
    a.tickets = c.tickets; a.ntickets = c.tiles + kDxSplitRegions;
    int64_t maxn = cdiv(din, kPrepRows) * 256;
    if (c.rpad * d > maxn) maxn = c.rpad * d;
    if (cdiv(a.ntickets, E) > maxn) maxn = cdiv(a.ntickets, E);
    lora_prep_batch_kernel<<<dim3(grid_for(maxn, 256, dev), (unsigned)E), 256, 0, stream>>>(a);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

// S = block-diagonal alpha (rows_e M_e) for M_e = AT_e (mats = c.AT, K = din,
// src = x) or BT_e (mats = c.BT, K = d, src = dy): zeroed, then one grouped
// launch per kGroupEpisodes episodes writes the diagonal blocks.
static attt_status batch_blockdiag(const BatchLoraLayout &c, const attt_bf16 *src, int64_t K,
                                   const __nv_bfloat16 *mats, const int64_t *off, int E, float alpha, int dev,
                                   cudaStream_t stream) {
    if (cudaMemsetAsync(c.S, 0, (size_t)off[E] * c.Ncat * sizeof(__nv_bfloat16), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    for (int e0 = 0; e0 < E; e0 += kMaxGroupBatch) {
        const int e1 = e0 + kMaxGroupBatch < E ? e0 + kMaxGroupBatch : E;
        GroupSpec sp[kMaxGroupBatch];
        int n = 0;
        for (int e = e0; e < e1; ++e) {
            const int64_t L = off[e + 1] - off[e];
            if (L == 0) continue;
            GroupSpec &u = sp[n++];
            u = GroupSpec{};
            u.a = src + off[e] * K; u.a_rows_ld = K; u.a_rows = L; u.a_k = K;
            u.b = mats + (int64_t)e * c.rpad * K; u.b_rows_ld = K; u.b_rows = c.rpad; u.b_k = K;
            u.M = (int)L; u.N = c.rpad; u.K = (int)K;
            u.out = GOUT_N16; u.out16 = c.S + off[e] * c.Ncat + (int64_t)e * c.rpad; u.ld = c.Ncat;
            u.alpha = alpha; u.r = c.rpad; u.rpad = c.rpad;
        }
        if (n == 0) continue;
        attt_status st = launch_group<false, false, kMaxGroupBatch>(sp, n, c.rpad, c.part, c.tickets, dev, stream,
                                                                    nullptr);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}

attt_status batch_forward(const attt_bf16 *d_x, const int64_t *off, int E, const attt_bf16 *d_W0, int64_t din,
                          int64_t d, int r, float scale, attt_bf16 *d_h, int64_t rows_bound, void *d_ws,
                          size_t ws_bytes, cudaStream_t stream) {
    attt_status st = batch_check(E, din, d, r, rows_bound, ws_bytes, d_ws);
    if (st != ATTT_OK) return st;
    const int64_t R = off[E];
    if (R == 0) return ATTT_OK;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    BatchLoraLayout c = batch_lora_layout(d_ws, E, rows_bound, din, d, r);
    st = batch_blockdiag(c, d_x, din, c.AT, off, E, scale, dev, stream);
    if (st != ATTT_OK) return st;
    // h = [x | S] [W0 ; BT]: W0 [din, d] and the padded B rows [E rpad, d] read MN-major
    GemmProblem p{};
    p.a = d_x; p.a_rows_ld = din; p.a_rows = R; p.a_k = din;
    p.b = d_W0; p.b_rows_ld = d; p.b_rows = d; p.b_k = din;
    p.a2 = c.S; p.a2_rows_ld = c.Ncat; p.a2_rows = R; p.a2_k = c.Ncat;
    p.b2 = c.BT; p.b2_rows_ld = d; p.b2_rows = d; p.b2_k = c.Ncat;
    p.M = (int)R; p.N = (int)d; p.K = (int)din; p.K2 = (int)c.Ncat; p.BN = 256; p.pair = R > 128;
    p.pdl = true;
    EpiParams ep{};
    ep.out16 = reinterpret_cast<__nv_bfloat16 *>(d_h); ep.out_ld = d; ep.alpha = 1.0f;
    return launch_gemm<EPI_BF16, false, true>(p, ep, dev, stream);
}

attt_status batch_grads(const attt_bf16 *d_x, const attt_bf16 *d_dy, const int64_t *off, int E, int64_t din,
                        int64_t d, int r, float scale, float *d_dA, float *d_dB, int64_t rows_bound, void *d_ws,
                        size_t ws_bytes, cudaStream_t stream) {
    attt_status st = batch_check(E, din, d, r, rows_bound, ws_bytes, d_ws);
    if (st != ATTT_OK) return st;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    BatchLoraLayout c = batch_lora_layout(d_ws, E, rows_bound, din, d, r);
    const int BN = c.rpad;
    int64_t toff[kGroupEpisodes] = {0};
    for (int e0 = 0; e0 < E; e0 += kGroupEpisodes) {
        const int e1 = e0 + kGroupEpisodes < E ? e0 + kGroupEpisodes : E;
        int64_t acc = 0;
        for (int e = e0; e < e1; ++e) {
            toff[e - e0] = acc;
            acc += (int64_t)c.rpad * round_up(off[e + 1] - off[e], 8);
        }
        // pass 1: u_e^T = (x_e AT_e^T)^T and v_e^T = (dy_e BT_e^T)^T, bf16
        GroupSpec sp[kMaxGroupBatch];
        int n = 0;
        for (int e = e0; e < e1; ++e) {
            const int64_t L = off[e + 1] - off[e];
            if (L == 0) continue;
            const int64_t Lp = round_up(L, 8);
            GroupSpec &u = sp[n++];
            u = GroupSpec{};
            u.a = d_x + off[e] * din; u.a_rows_ld = din; u.a_rows = L; u.a_k = din;
            u.b = c.AT + (int64_t)e * c.rpad * din; u.b_rows_ld = din; u.b_rows = c.rpad; u.b_k = din;
            u.M = (int)L; u.N = c.rpad; u.K = (int)din;
            u.out = GOUT_T16; u.out16 = c.uT + toff[e - e0]; u.ld = Lp; u.alpha = 1.0f; u.r = c.rpad; u.rpad = c.rpad;
            GroupSpec &v = sp[n++];
            v = GroupSpec{};
            v.a = d_dy + off[e] * d; v.a_rows_ld = d; v.a_rows = L; v.a_k = d;
            v.b = c.BT + (int64_t)e * c.rpad * d; v.b_rows_ld = d; v.b_rows = c.rpad; v.b_k = d;
            v.M = (int)L; v.N = c.rpad; v.K = (int)d;
            v.out = GOUT_T16; v.out16 = c.vT + toff[e - e0]; v.ld = Lp; v.alpha = 1.0f; v.r = c.rpad; v.rpad = c.rpad;
        }
        if (n == 0) continue;
        st = launch_group<false, false, kMaxGroupBatch>(sp, n, BN, c.part, c.tickets, dev, stream, nullptr);
        if (st != ATTT_OK) return st;
        // pass 2: dA_e = s x_e^T v_e (x MN-major), dB_e^T = s dy_e^T u_e (dy MN-major)
        n = 0;
        for (int e = e0; e < e1; ++e) {
            const int64_t L = off[e + 1] - off[e];
            if (L == 0) continue;
            const int64_t Lp = round_up(L, 8);
            GroupSpec &a = sp[n++];
            a = GroupSpec{};
            a.a = d_x + off[e] * din; a.a_rows_ld = din; a.a_rows = din; a.a_k = L;
            a.b = c.vT + toff[e - e0]; a.b_rows_ld = Lp; a.b_rows = c.rpad; a.b_k = L;
            a.M = (int)din; a.N = c.rpad; a.K = (int)L;
            a.out = GOUT_N32; a.outp[0] = d_dA + (int64_t)e * din * r; a.alpha = scale; a.r = r; a.rpad = c.rpad;
            GroupSpec &b = sp[n++];
            b = GroupSpec{};
            b.a = d_dy + off[e] * d; b.a_rows_ld = d; b.a_rows = d; b.a_k = L;
            b.b = c.uT + toff[e - e0]; b.b_rows_ld = Lp; b.b_rows = c.rpad; b.b_k = L;
            b.M = (int)d; b.N = c.rpad; b.K = (int)L;
            b.out = GOUT_T32; b.out32 = d_dB + (int64_t)e * r * d; b.ld = d; b.alpha = scale; b.r = r;
            b.rpad = c.rpad;
        }
        st = launch_group<true, false, kMaxGroupBatch>(sp, n, BN, c.part, c.tickets, dev, stream, nullptr);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}

attt_status batch_input_grad(const attt_bf16 *d_dy, const int64_t *off, int E, const attt_bf16 *d_W0, int64_t din,
                             int64_t d, int r, float scale, float *d_dx, int64_t rows_bound, void *d_ws,
                             size_t ws_bytes, cudaStream_t stream) {
    attt_status st = batch_check(E, din, d, r, rows_bound, ws_bytes, d_ws);
    if (st != ATTT_OK) return st;
    const int64_t R = off[E];
    if (R == 0) return ATTT_OK;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    BatchLoraLayout c = batch_lora_layout(d_ws, E, rows_bound, din, d, r);
    st = batch_blockdiag(c, d_dy, d, c.BT, off, E, scale, dev, stream);
    if (st != ATTT_OK) return st;
    // dx = [dy | S'] [W0^T ; A_cat^T]: W0 [din, d] and A_cat [din, E rpad] read K-major
    GemmProblem p{};
    p.a = d_dy; p.a_rows_ld = d; p.a_rows = R; p.a_k = d;
    p.b = d_W0; p.b_rows_ld = d; p.b_rows = din; p.b_k = d;
    p.a2 = c.S; p.a2_rows_ld = c.Ncat; p.a2_rows = R; p.a2_k = c.Ncat;
    p.b2 = c.ACAT; p.b2_rows_ld = c.Ncat; p.b2_rows = din; p.b2_k = c.Ncat;
    p.M = (int)R; p.N = (int)din; p.K = (int)d; p.K2 = (int)c.Ncat; p.BN = 256; p.pair = R > 128;
    p.pdl = true;
    p.split_ws = c.split_ws; p.split_tick = c.tickets + c.tiles; p.split_regions = kDxSplitRegions;
    EpiParams ep{};
    ep.out = d_dx; ep.out_ld = din; ep.accumulate = 0; ep.alpha = 1.0f;
    return launch_gemm<EPI_F32_ACC, false, false>(p, ep, dev, stream);
}

// ---------------------------------------------------------------------------
// The adapted projection: forward and input gradient
// ---------------------------------------------------------------------------


struct ProjLayout {
    int rpad;
    __nv_bfloat16 *AT, *BT;  // forward: A^T padded [rpad, din]; B padded [rpad, dout] (written by the prep)
    __nv_bfloat16 *s16;      // s u or s v, [L, rpad] bf16 row-major
    unsigned int *tickets;   // the skinny launch's tiles, then the tail split's counters
    float *part;             // the skinny launch's partial slots
    float *split_ws;         // input gradient: tail-split partials
    int64_t tiles;
    size_t bytes;
};

static ProjLayout proj_layout(void *ws, int64_t L, int64_t din, int64_t dout, int r, bool fwd) {
    ProjLayout c{};
    c.rpad = (int)round_up(r, 16);
    c.tiles = cdiv(L, 128);
    Carve cv{static_cast<char *>(ws), 0};
    if (fwd) {
        c.AT = cv.take<__nv_bfloat16>((size_t)(c.rpad * din));
        c.BT = cv.take<__nv_bfloat16>((size_t)(c.rpad * dout));
    }
    c.s16 = cv.take<__nv_bfloat16>((size_t)(L * c.rpad));
    c.tickets = cv.take<unsigned int>((size_t)(c.tiles + kDxSplitRegions));
    c.part = cv.take<float>((size_t)(c.tiles + kGroupMaxGrid) * 128 * c.rpad);
    if (!fwd) c.split_ws = cv.take<float>((size_t)kDxSplitRegions * 128 * 256);
    c.bytes = (size_t)round_up((int64_t)cv.used, 256);
    return c;
}

static attt_status proj_check(const void *a, const void *b, const void *c, const void *d, const void *out,
                              int64_t L, int64_t din, int64_t dout, int r) {
    if (!a || !b || !c || !d || !out) return ATTT_ERR_INVALID_ARG;
    if (L < 1 || din < 8 || dout < 8 || din % 8 != 0 || dout % 8 != 0 || r < 1 || r > 64) return ATTT_ERR_INVALID_ARG;
    if (L > (1ll << 30) || din > (1ll << 30) || dout > (1ll << 30)) return ATTT_ERR_UNSUPPORTED;
    if (!aligned16(a) || !aligned16(b) || !aligned16(c) || !aligned16(d) || !aligned16(out)) return ATTT_ERR_INVALID_ARG;
    return ATTT_OK;
}

}  // namespace attt

extern "C" {

size_t attt_lora_forward_workspace_bytes(int64_t L, int64_t din, int64_t dout, int r) {
    if (L < 1 || din < 1 || dout < 1 || r < 1 || r > 64) return 0;
    return attt::proj_layout(nullptr, L, din, dout, r, true).bytes;
}

size_t attt_lora_input_grad_workspace_bytes(int64_t L, int64_t din, int64_t dout, int r) {
    if (L < 1 || din < 1 || dout < 1 || r < 1 || r > 64) return 0;
    return attt::proj_layout(nullptr, L, din, dout, r, false).bytes;
}

attt_status attt_lora_forward(const attt_bf16 *d_x, const attt_bf16 *d_W0, const attt_bf16 *d_A, const attt_bf16 *d_B,
                              int64_t L, int64_t din, int64_t dout, int r, float scale, attt_bf16 *d_h, void *d_ws,
                              size_t ws_bytes, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    attt_status st = proj_check(d_x, d_W0, d_A, d_B, d_h, L, din, dout, r);
    if (st != ATTT_OK) return st;
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_lora_forward_workspace_bytes(L, din, dout, r))
        return ATTT_ERR_WORKSPACE;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    ProjLayout c = proj_layout(d_ws, L, din, dout, r, true);
    {   // A^T (and B) padded to rpad rows, tickets zeroed
        PrepArgs a{};
        a.A[0] = reinterpret_cast<const __nv_bfloat16 *>(d_A);
        a.B[0] = reinterpret_cast<const __nv_bfloat16 *>(d_B);
        a.BT[0] = c.BT;
        a.dout[0] = dout;
        a.nproj = 1; a.r = r; a.rpad = c.rpad; a.din = din; a.AT = c.AT;
        a.tickets = c.tickets; a.ntickets = c.tiles;
        int64_t maxn = cdiv(din, kPrepRows) * 256;
        if (c.rpad * dout / 8 > maxn) maxn = c.rpad * dout / 8;
        lora_prep_kernel<<<dim3(grid_for(maxn, 256, dev), 1), 256, 0, stream>>>(a);
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    }
    {   // s u = s x A, bf16 [L, rpad]
        GroupSpec u{};
        u.a = d_x; u.a_rows_ld = din; u.a_rows = L; u.a_k = din;
        u.b = c.AT; u.b_rows_ld = din; u.b_rows = c.rpad; u.b_k = din;
        u.M = (int)L; u.N = c.rpad; u.K = (int)din;
        u.out = GOUT_N16; u.out16 = c.s16; u.ld = c.rpad; u.alpha = scale; u.r = c.rpad; u.rpad = c.rpad;
        st = launch_group<false, false>(&u, 1, c.rpad, c.part, c.tickets, dev, stream, nullptr);
        if (st != ATTT_OK) return st;
    }
    {   // h = [x | s u] [W0 ; B]: W0 [din, dout] and B [r, dout] are read MN-major
        GemmProblem p{};
        p.a = d_x; p.a_rows_ld = din; p.a_rows = L; p.a_k = din;
        p.b = d_W0; p.b_rows_ld = dout; p.b_rows = dout; p.b_k = din;
        p.a2 = c.s16; p.a2_rows_ld = c.rpad; p.a2_rows = L; p.a2_k = c.rpad;
        p.b2 = d_B; p.b2_rows_ld = dout; p.b2_rows = dout; p.b2_k = r;
        p.M = (int)L; p.N = (int)dout; p.K = (int)din; p.K2 = c.rpad; p.BN = 256; p.pair = L > 128;
        p.pdl = true;
        EpiParams ep{};
        ep.out16 = reinterpret_cast<__nv_bfloat16 *>(d_h); ep.out_ld = dout; ep.alpha = 1.0f;
        st = launch_gemm<EPI_BF16, false, true>(p, ep, dev, stream);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}

attt_status attt_lora_input_grad(const attt_bf16 *d_dy, const attt_bf16 *d_W0, const attt_bf16 *d_A,
                                 const attt_bf16 *d_B, int64_t L, int64_t din, int64_t dout, int r, float scale,
                                 float *d_dx, void *d_ws, size_t ws_bytes, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    attt_status st = proj_check(d_dy, d_W0, d_A, d_B, d_dx, L, din, dout, r);
    if (st != ATTT_OK) return st;
    if (r % 8 != 0) return ATTT_ERR_UNSUPPORTED;  // A [din, r] is read in place: rows of 16-byte multiples
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_lora_input_grad_workspace_bytes(L, din, dout, r))
        return ATTT_ERR_WORKSPACE;
    int dev;
    st = current_device(&dev);
    if (st != ATTT_OK) return st;
    ProjLayout c = proj_layout(d_ws, L, din, dout, r, false);
    if (cudaMemsetAsync(c.tickets, 0, sizeof(unsigned int) * (size_t)(c.tiles + kDxSplitRegions), stream) !=
        cudaSuccess)
        return ATTT_ERR_CUDA;
    {   // s v = s dy B^T, bf16 [L, rpad]; B [r, dout] is the K-major operand (rows past r read as zeros)
        GroupSpec v{};
        v.a = d_dy; v.a_rows_ld = dout; v.a_rows = L; v.a_k = dout;
        v.b = d_B; v.b_rows_ld = dout; v.b_rows = r; v.b_k = dout;
        v.M = (int)L; v.N = c.rpad; v.K = (int)dout;
        v.out = GOUT_N16; v.out16 = c.s16; v.ld = c.rpad; v.alpha = scale; v.r = c.rpad; v.rpad = c.rpad;
        st = launch_group<false, false>(&v, 1, c.rpad, c.part, c.tickets, dev, stream, nullptr);
        if (st != ATTT_OK) return st;
    }
    {   // dx = [dy | s v] [W0^T ; A^T]: W0 [din, dout] and A [din, r] are read K-major
        GemmProblem p{};
        p.a = d_dy; p.a_rows_ld = dout; p.a_rows = L; p.a_k = dout;
        p.b = d_W0; p.b_rows_ld = dout; p.b_rows = din; p.b_k = dout;
        p.a2 = c.s16; p.a2_rows_ld = c.rpad; p.a2_rows = L; p.a2_k = c.rpad;
        p.b2 = d_A; p.b2_rows_ld = r; p.b2_rows = din; p.b2_k = r;
        p.M = (int)L; p.N = (int)din; p.K = (int)dout; p.K2 = c.rpad; p.BN = 256; p.pair = L > 128;
        p.pdl = true;
        p.split_ws = c.split_ws; p.split_tick = c.tickets + c.tiles; p.split_regions = kDxSplitRegions;
        EpiParams ep{};
        ep.out = d_dx; ep.out_ld = din; ep.accumulate = 0; ep.alpha = 1.0f;
        st = launch_gemm<EPI_F32_ACC, false, false>(p, ep, dev, stream);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}



size_t attt_lora_workspace_bytes(int64_t L, int64_t din, int nproj, const int64_t *dout, int r) {
    if (L < 1 || din < 1 || nproj < 1 || nproj > attt::kMaxProj || !dout || r < 1 || r > 64) return 0;
    return attt::lora_layout(nullptr, L, din, nproj, dout, r).bytes;
}

attt_status attt_lora_grad(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj, const attt_bf16 *const *d_dy,
                           const int64_t *dout, const attt_bf16 *const *d_A, const attt_bf16 *const *d_B, int r,
                           float scale, float *const *d_dA, float *const *d_dB, void *d_ws, size_t ws_bytes,
                           attt_stream stream) {
    ATTT_NVTX_RANGE();
    return attt::lora_grad_run(d_x, L, din, nproj, d_dy, dout, d_A, d_B, r, scale, d_dA, d_dB, d_ws, ws_bytes,
                               nullptr, stream);
}

attt_status attt_lora_step(float *d_A32, float *d_B32, const float *d_dA, const float *d_dB, int64_t din,
                           int64_t dout, int r, float lr, attt_bf16 *d_A16, attt_bf16 *d_B16, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!d_A32 || !d_B32 || !d_dA || !d_dB || din < 1 || dout < 1 || r < 1) return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    const int64_t nA = din * r, nB = (int64_t)r * dout;
    lora_step_kernel<<<grid_for((nA + nB) / 4 + 1, 256, dev), 256, 0, stream>>>(
        d_A32, d_dA, reinterpret_cast<__nv_bfloat16 *>(d_A16), nA, d_B32, d_dB,
        reinterpret_cast<__nv_bfloat16 *>(d_B16), nB, lr);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status attt_lora_adamw_step(float *d_A32, float *d_B32, const float *d_dA, const float *d_dB, float *d_mA,
                                 float *d_vA, float *d_mB, float *d_vB, int64_t din, int64_t dout, int r, float lr,
                                 double beta1, double beta2, double eps, double weight_decay, int step,
                                 attt_bf16 *d_A16, attt_bf16 *d_B16, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (!d_A32 || !d_B32 || !d_dA || !d_dB || !d_mA || !d_vA || !d_mB || !d_vB) return ATTT_ERR_INVALID_ARG;
    if (din < 1 || dout < 1 || r < 1 || step < 1 || !(beta1 >= 0.0 && beta1 < 1.0) || !(beta2 >= 0.0 && beta2 < 1.0) ||
        !(eps > 0.0) || !(weight_decay >= 0.0) || !(lr == lr))
        return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    AdamWArgs a{};
    a.p[0] = d_A32; a.p[1] = d_B32;
    a.g[0] = d_dA; a.g[1] = d_dB;
    a.m[0] = d_mA; a.m[1] = d_mB;
    a.v[0] = d_vA; a.v[1] = d_vB;
    a.p16[0] = reinterpret_cast<__nv_bfloat16 *>(d_A16);
    a.p16[1] = reinterpret_cast<__nv_bfloat16 *>(d_B16);
    a.n[0] = din * r;
    a.n[1] = (int64_t)r * dout;
    // the step's scalars in double, rounded once to fp32
    a.decay = (float)(1.0 - (double)lr * weight_decay);
    a.b1 = (float)beta1; a.one_b1 = (float)(1.0 - beta1);
    a.b2 = (float)beta2; a.one_b2 = (float)(1.0 - beta2);
    a.step_size = (float)((double)lr / (1.0 - std::pow(beta1, (double)step)));
    a.bc2_sqrt = (float)std::sqrt(1.0 - std::pow(beta2, (double)step));
    a.eps = (float)eps;
    lora_adamw_kernel<<<grid_for(a.n[0] + a.n[1], 256, dev), 256, 0, stream>>>(a);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

attt_status attt_cast_bf16(const float *d_src, attt_bf16 *d_dst, int64_t n, attt_stream stream) {
    ATTT_NVTX_RANGE();
    using namespace attt;
    if (n < 0 || (n > 0 && (!d_src || !d_dst))) return ATTT_ERR_INVALID_ARG;
    if (n == 0) return ATTT_OK;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    cast_bf16_kernel<<<grid_for(cdiv(n, 8), 256, dev), 256, 0, stream>>>(
        d_src, reinterpret_cast<__nv_bfloat16 *>(d_dst), n);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // extern "C"
