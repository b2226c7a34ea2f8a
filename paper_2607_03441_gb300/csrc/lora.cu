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
// and merged with fp32 atomics; u and v are rounded to bf16 in between.
#include "gemm_launch.cuh"

namespace attt {

struct LoraLayout {
    int rpad, Nu;
    int64_t Lp;
    __nv_bfloat16 *AT;            // [Nu, din]
    __nv_bfloat16 *BT[kMaxProj];  // [rpad, dout_p]
    float *uT32, *vT32;           // [Nu, Lp] each, contiguous
    __nv_bfloat16 *uT16, *vT16;   // [Nu, Lp] each, contiguous
    size_t bytes;
};

static LoraLayout lora_layout(void *ws, int64_t L, int64_t din, int nproj, const int64_t *dout, int r) {
    LoraLayout c{};
    c.rpad = (int)round_up(r, 16);
    c.Nu = nproj * c.rpad;
    c.Lp = round_up(L, 8);
    Carve cv{static_cast<char *>(ws), 0};
    c.AT = cv.take<__nv_bfloat16>((size_t)(c.Nu * din));
    for (int p = 0; p < nproj; ++p) c.BT[p] = cv.take<__nv_bfloat16>((size_t)(c.rpad * dout[p]));
    c.uT32 = cv.take<float>((size_t)(2 * c.Nu * c.Lp));
    c.vT32 = c.uT32 + (size_t)c.Nu * c.Lp;
    c.uT16 = cv.take<__nv_bfloat16>((size_t)(2 * c.Nu * c.Lp));
    c.vT16 = c.uT16 + (size_t)c.Nu * c.Lp;
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
};

// AT[p*rpad + c, i] = A_p[i, c] (zero for c >= r); BT_p[c, o] = B_p[c, o]
// (zero rows for c >= r).
__global__ void lora_prep_kernel(PrepArgs a) {
    const int p = blockIdx.y;
    const int64_t nA = (int64_t)a.rpad * a.din;
    const int64_t nB = (int64_t)a.rpad * a.dout[p];
    const int64_t n = nA > nB ? nA : nB;
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x) {
        if (i < nA) {
            const int c = (int)(i / a.din);
            const int64_t k = i - (int64_t)c * a.din;
            a.AT[((int64_t)p * a.rpad + c) * a.din + k] =
                c < a.r ? a.A[p][k * a.r + c] : __float2bfloat16_rn(0.f);
        }
        if (i < nB) {
            const int c = (int)(i / a.dout[p]);
            a.BT[p][i] = c < a.r ? a.B[p][i] : __float2bfloat16_rn(0.f);
        }
    }
}

__global__ void f32_to_bf16_kernel(const float *__restrict__ in, __nv_bfloat16 *__restrict__ out, int64_t n) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < n; i += (int64_t)gridDim.x * blockDim.x)
        out[i] = __float2bfloat16_rn(in[i]);
}

// SGD: p <- p - lr * g (product then difference, both rounded), bf16 refresh.
__global__ void lora_step_kernel(float *A32, const float *dA, __nv_bfloat16 *A16, int64_t nA, float *B32,
                                 const float *dB, __nv_bfloat16 *B16, int64_t nB, float lr) {
    for (int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; i < nA + nB;
         i += (int64_t)gridDim.x * blockDim.x) {
        if (i < nA) {
            const float v = __fsub_rn(A32[i], __fmul_rn(lr, dA[i]));
            A32[i] = v;
            if (A16) A16[i] = __float2bfloat16_rn(v);
        } else {
            const int64_t k = i - nA;
            const float v = __fsub_rn(B32[k], __fmul_rn(lr, dB[k]));
            B32[k] = v;
            if (B16) B16[k] = __float2bfloat16_rn(v);
        }
    }
}

static unsigned grid_for(int64_t n, int threads, int dev) {
    int64_t b = cdiv(n, threads);
    const int64_t cap = (int64_t)num_sms(dev) * 8;
    if (b > cap) b = cap;
    if (b < 1) b = 1;
    return (unsigned)b;
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
        if (!aligned16(d_dy[p])) return ATTT_ERR_INVALID_ARG;
    }
    if (!d_ws || !aligned256(d_ws) || ws_bytes < attt_lora_workspace_bytes(L, din, nproj, dout, r))
        return ATTT_ERR_WORKSPACE;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;

    LoraLayout c = lora_layout(d_ws, L, din, nproj, dout, r);
    const int BNu = c.Nu <= 256 ? c.Nu : 256;

    // adapters in K-major, rank padded to a multiple of 16 with zeros
    {
        PrepArgs a{};
        int64_t maxn = c.rpad * din;
        for (int p = 0; p < nproj; ++p) {
            a.A[p] = reinterpret_cast<const __nv_bfloat16 *>(d_A[p]);
            a.B[p] = reinterpret_cast<const __nv_bfloat16 *>(d_B[p]);
            a.BT[p] = c.BT[p];
            a.dout[p] = dout[p];
            if (c.rpad * dout[p] > maxn) maxn = c.rpad * dout[p];
        }
        a.nproj = nproj; a.r = r; a.rpad = c.rpad; a.din = din; a.AT = c.AT;
        dim3 grid(grid_for(maxn, 256, dev), nproj);
        lora_prep_kernel<<<grid, 256, 0, stream>>>(a);
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    }
    if (cudaMemsetAsync(c.uT32, 0, (size_t)2 * c.Nu * c.Lp * sizeof(float), stream) != cudaSuccess)
        return ATTT_ERR_CUDA;
    for (int p = 0; p < nproj; ++p) {
        if (cudaMemsetAsync(d_dA[p], 0, (size_t)din * r * sizeof(float), stream) != cudaSuccess ||
            cudaMemsetAsync(d_dB[p], 0, (size_t)r * dout[p] * sizeof(float), stream) != cudaSuccess)
            return ATTT_ERR_CUDA;
    }

    // pass 1a: u^T = (x AT^T)^T for every projection at once
    {
        GemmProblem p{};
        p.a = d_x; p.a_rows_ld = din; p.a_rows = L; p.a_k = din;
        p.b = c.AT; p.b_rows_ld = din; p.b_rows = c.Nu; p.b_k = din;
        p.M = (int)L; p.N = c.Nu; p.K = (int)din; p.BN = BNu; p.allow_split = true;
        EpiParams ep{};
        ep.out = c.uT32; ep.out_ld = c.Lp; ep.alpha = 1.0f; ep.r = c.rpad; ep.rpad = c.rpad;
        st = launch_gemm<EPI_ATOMIC_T, false, false>(p, ep, dev, stream, status);
        if (st != ATTT_OK) return st;
    }
    // pass 1b: v_p^T = (dy_p B_p^T)^T
    for (int q = 0; q < nproj; ++q) {
        GemmProblem p{};
        p.a = d_dy[q]; p.a_rows_ld = dout[q]; p.a_rows = L; p.a_k = dout[q];
        p.b = c.BT[q]; p.b_rows_ld = dout[q]; p.b_rows = c.rpad; p.b_k = dout[q];
        p.M = (int)L; p.N = c.rpad; p.K = (int)dout[q]; p.BN = c.rpad; p.allow_split = true;
        EpiParams ep{};
        ep.out = c.vT32 + (size_t)q * c.rpad * c.Lp; ep.out_ld = c.Lp; ep.alpha = 1.0f;
        ep.r = c.rpad; ep.rpad = c.rpad;
        st = launch_gemm<EPI_ATOMIC_T, false, false>(p, ep, dev, stream, status);
        if (st != ATTT_OK) return st;
    }
    {
        const int64_t n = (int64_t)2 * c.Nu * c.Lp;
        f32_to_bf16_kernel<<<grid_for(n, 256, dev), 256, 0, stream>>>(c.uT32, c.uT16, n);
        count_launch();
        if (cudaGetLastError() != cudaSuccess) return ATTT_ERR_CUDA;
    }
    // pass 2a: dA_p = s x^T v_p for every projection at once (x MN-major)
    {
        GemmProblem p{};
        p.a = d_x; p.a_rows_ld = din; p.a_rows = din; p.a_k = L;
        p.b = c.vT16; p.b_rows_ld = c.Lp; p.b_rows = c.Nu; p.b_k = c.Lp;
        p.M = (int)din; p.N = c.Nu; p.K = (int)L; p.BN = BNu; p.allow_split = true;
        EpiParams ep{};
        for (int q = 0; q < nproj; ++q) ep.outp[q] = d_dA[q];
        ep.alpha = scale; ep.r = r; ep.rpad = c.rpad;
        st = launch_gemm<EPI_ATOMIC_N, true, false>(p, ep, dev, stream, status);
        if (st != ATTT_OK) return st;
    }
    // pass 2b: dB_p^T = s dy_p^T u_p (dy MN-major), stored transposed into dB_p
    for (int q = 0; q < nproj; ++q) {
        GemmProblem p{};
        p.a = d_dy[q]; p.a_rows_ld = dout[q]; p.a_rows = dout[q]; p.a_k = L;
        p.b = c.uT16; p.b_rows_ld = c.Lp; p.b_rows = c.Nu; p.b_k = c.Lp;
        p.b_n_off = q * c.rpad;
        p.M = (int)dout[q]; p.N = c.rpad; p.K = (int)L; p.BN = c.rpad; p.allow_split = true;
        EpiParams ep{};
        ep.out = d_dB[q]; ep.out_ld = dout[q]; ep.alpha = scale; ep.r = r; ep.rpad = c.rpad;
        st = launch_gemm<EPI_ATOMIC_T, true, false>(p, ep, dev, stream, status);
        if (st != ATTT_OK) return st;
    }
    return ATTT_OK;
}

}  // namespace attt

extern "C" {

size_t attt_lora_workspace_bytes(int64_t L, int64_t din, int nproj, const int64_t *dout, int r) {
    if (L < 1 || din < 1 || nproj < 1 || nproj > attt::kMaxProj || !dout || r < 1 || r > 64) return 0;
    return attt::lora_layout(nullptr, L, din, nproj, dout, r).bytes;
}

attt_status attt_lora_grad(const attt_bf16 *d_x, int64_t L, int64_t din, int nproj, const attt_bf16 *const *d_dy,
                           const int64_t *dout, const attt_bf16 *const *d_A, const attt_bf16 *const *d_B, int r,
                           float scale, float *const *d_dA, float *const *d_dB, void *d_ws, size_t ws_bytes,
                           attt_stream stream) {
    return attt::lora_grad_run(d_x, L, din, nproj, d_dy, dout, d_A, d_B, r, scale, d_dA, d_dB, d_ws, ws_bytes,
                               nullptr, stream);
}

attt_status attt_lora_step(float *d_A32, float *d_B32, const float *d_dA, const float *d_dB, int64_t din,
                           int64_t dout, int r, float lr, attt_bf16 *d_A16, attt_bf16 *d_B16, attt_stream stream) {
    using namespace attt;
    if (!d_A32 || !d_B32 || !d_dA || !d_dB || din < 1 || dout < 1 || r < 1) return ATTT_ERR_INVALID_ARG;
    int dev;
    attt_status st = current_device(&dev);
    if (st != ATTT_OK) return st;
    const int64_t nA = din * r, nB = (int64_t)r * dout;
    lora_step_kernel<<<grid_for(nA + nB, 256, dev), 256, 0, stream>>>(
        d_A32, d_dA, reinterpret_cast<__nv_bfloat16 *>(d_A16), nA, d_B32, d_dB,
        reinterpret_cast<__nv_bfloat16 *>(d_B16), nB, lr);
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // extern "C"
