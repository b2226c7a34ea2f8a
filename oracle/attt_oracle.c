/*
 * attt_oracle.c -- plain, slow CPU oracle for the aTTT update step.
 *
 * TEST INFRASTRUCTURE ONLY.  Nothing on the product path may call, link or
 * load this file; only the tests, the smoke check and the CPU baseline leg and
 * reference arm of the benchmark do.  It shares no code, header, table or helper with the CUDA
 * library under paper_2607_03441_gb300/csrc.
 *
 * What it computes (aTTT, "Agentic Test-Time Training", Sec. 3.3):
 *
 *   Eq. 8   f_k(j) = max over the n-grams g of x_k that contain position j of
 *           count(g, H_k), where H_k is the concatenation of every earlier
 *           update's tokens and count() counts every start position
 *           (overlapping occurrences count; an empty max is 0).
 *   Eq. 9   w_{k,j} = max(w_min, 1 / (1 + f_k(j)))  -- one IEEE fp32
 *           round-to-nearest division, then the floor.
 *   Eq. 10  L = (1/L) * sum_j w_j * CE(x_j, z_j), CE = lse(z_j) - z_{j,x_j},
 *           z_j = h_j W^T (the LM head).  Row j of h predicts target x_j.
 *   Eq. 2 / Algorithm 1 (the gradient step): the gradient of Eq. 10 w.r.t.
 *           the hidden state, dh_j = (w_j/L) (sum_v p_jv W_v - W_{x_j}),
 *           and the LoRA adapter gradients of y = x W0 + s (x A) B:
 *           dB = s (xA)^T dy,  dA = s x^T (dy B^T);
 *           then plain SGD  theta <- theta - lr * grad  on fp32 masters and a
 *           round-to-nearest-even refresh of the bf16 copies.
 *   For an update chained through the adapted projection (its output is the
 *           LM head's input): the forward h = x W0 + s (x A) B and the input
 *           gradient dx = dy W0^T + s (dy B^T) A^T.
 *
 * Floating point: all sums in fp64 over the bf16 inputs exactly as stored;
 * Eq. 9 and the SGD step in fp32 exactly as the formulas read (this file is
 * compiled with -ffp-contract=off so that a*b+c is never fused).
 *
 * Parity pins live in tests/test_oracle_*.py: a hand-worked Eq. 8-9 example,
 * brute force on tiny inputs, two independent counters, finite differences,
 * torch CPU cross_entropy / autograd, closed forms and invariants.
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#ifdef _OPENMP
#include <omp.h>
#endif

/* bf16 storage (the upper 16 bits of an IEEE binary32) -> exact double. */
static double bf16_value(uint16_t b)
{
    uint32_t u = ((uint32_t)b) << 16;
    float f;
    memcpy(&f, &u, sizeof f);
    return (double)f;
}

int oracle_num_threads(void)
{
#ifdef _OPENMP
    return omp_get_max_threads();
#else
    return 1;
#endif
}

void oracle_set_num_threads(int t)
{
#ifdef _OPENMP
    if (t > 0) omp_set_num_threads(t);
#else
    (void)t;
#endif
}

/* ------------------------------------------------------------------------ */
/* Eq. 8: count(g, H)                                                        */
/* ------------------------------------------------------------------------ */

/* Naive scan: every start position p in [0, |H|-n] whose n tokens equal g. */
int64_t oracle_count_naive(const int32_t *H, int64_t nH, const int32_t *g, int n)
{
    int64_t c = 0;
    for (int64_t p = 0; p + n <= nH; ++p) {
        int eq = 1;
        for (int i = 0; i < n; ++i) {
            if (H[p + i] != g[i]) { eq = 0; break; }
        }
        c += eq;
    }
    return c;
}

/* Eq. 8 with the naive counter: exposure f[j] for j in [0, L). */
void oracle_exposure_naive(const int32_t *H, int64_t nH, const int32_t *x, int64_t L,
                           int n, int64_t *f)
{
    for (int64_t j = 0; j < L; ++j) f[j] = 0;
    /* Every n-gram of x starting at s covers positions s..s+n-1. */
    for (int64_t s = 0; s + n <= L; ++s) {
        int64_t c = oracle_count_naive(H, nH, x + s, n);
        for (int64_t j = s; j < s + n; ++j)
            if (c > f[j]) f[j] = c;
    }
}

/* Second, independent counter: sort the start positions of H by their n-gram
 * (lexicographic), then count a query by two binary searches. */
static const int32_t *g_sort_H;
static int g_sort_n;

static int cmp_ngram_at(const int32_t *a, const int32_t *b, int n)
{
    for (int i = 0; i < n; ++i) {
        if (a[i] < b[i]) return -1;
        if (a[i] > b[i]) return 1;
    }
    return 0;
}

static int cmp_start(const void *pa, const void *pb)
{
    int64_t a = *(const int64_t *)pa, b = *(const int64_t *)pb;
    int c = cmp_ngram_at(g_sort_H + a, g_sort_H + b, g_sort_n);
    if (c) return c;
    return (a < b) ? -1 : (a > b);
}

void oracle_exposure_sorted(const int32_t *H, int64_t nH, const int32_t *x, int64_t L,
                            int n, int64_t *f)
{
    for (int64_t j = 0; j < L; ++j) f[j] = 0;
    int64_t m = nH - n + 1;
    if (m <= 0 || L < n) return;
    int64_t *idx = (int64_t *)malloc((size_t)m * sizeof(int64_t));
    for (int64_t p = 0; p < m; ++p) idx[p] = p;
    g_sort_H = H;
    g_sort_n = n;
    qsort(idx, (size_t)m, sizeof(int64_t), cmp_start);
    for (int64_t s = 0; s + n <= L; ++s) {
        const int32_t *g = x + s;
        int64_t lo = 0, hi = m; /* first start whose n-gram >= g */
        while (lo < hi) {
            int64_t mid = lo + (hi - lo) / 2;
            if (cmp_ngram_at(H + idx[mid], g, n) < 0) lo = mid + 1; else hi = mid;
        }
        int64_t first = lo;
        hi = m; /* first start whose n-gram > g */
        while (lo < hi) {
            int64_t mid = lo + (hi - lo) / 2;
            if (cmp_ngram_at(H + idx[mid], g, n) <= 0) lo = mid + 1; else hi = mid;
        }
        int64_t c = lo - first;
        for (int64_t j = s; j < s + n; ++j)
            if (c > f[j]) f[j] = c;
    }
    free(idx);
}

/* Eq. 9: w = max(w_min, 1/(1+f)) in fp32, IEEE round-to-nearest divide. */
void oracle_weights_from_exposure(const int64_t *f, int64_t L, float w_min, float *w)
{
    for (int64_t j = 0; j < L; ++j) {
        volatile float denom = 1.0f + (float)f[j];
        volatile float q = 1.0f / denom;
        w[j] = (q > w_min) ? q : w_min;
    }
}

/* ------------------------------------------------------------------------ */
/* Eq. 10 and its gradient w.r.t. the hidden state                          */
/* ------------------------------------------------------------------------ */

/*
 * For each requested row j (rows[i], i < nrows):
 *   z_jv   = sum_k h_jk W_vk                              (fp64)
 *   lse_j  = m + log sum_v exp(z_jv - m),  m = max_v z_jv
 *   nll_j  = lse_j - z_{j, tgt_j}
 *   dh_jk  = (w_j / L) (sum_v exp(z_jv - lse_j) W_vk - W_{tgt_j, k})   (if dh)
 * h is [L, d] and W is [V, d], both bf16, row-major.  Outputs are indexed by
 * i (the position in rows[]), dh is [nrows, d].
 */
void oracle_ce_rows(const uint16_t *h, const uint16_t *W, const int32_t *tgt, const float *w,
                    int64_t L, int64_t d, int64_t V, const int64_t *rows, int64_t nrows,
                    double *lse, double *nll, double *dh)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t i = 0; i < nrows; ++i) {
        int64_t j = rows[i];
        double *hj = (double *)malloc((size_t)d * sizeof(double));
        double *z = (double *)malloc((size_t)V * sizeof(double));
        for (int64_t k = 0; k < d; ++k) hj[k] = bf16_value(h[j * d + k]);
        double m = -INFINITY;
        for (int64_t v = 0; v < V; ++v) {
            const uint16_t *Wv = W + v * d;
            double acc = 0.0;
            for (int64_t k = 0; k < d; ++k) acc += hj[k] * bf16_value(Wv[k]);
            z[v] = acc;
            if (acc > m) m = acc;
        }
        double se = 0.0;
        for (int64_t v = 0; v < V; ++v) se += exp(z[v] - m);
        double l = m + log(se);
        lse[i] = l;
        nll[i] = l - z[tgt[j]];
        if (dh) {
            double c = (double)w[j] / (double)L;
            double *out = dh + i * d;
            for (int64_t k = 0; k < d; ++k) out[k] = 0.0;
            for (int64_t v = 0; v < V; ++v) {
                double p = exp(z[v] - l);
                const uint16_t *Wv = W + v * d;
                for (int64_t k = 0; k < d; ++k) out[k] += p * bf16_value(Wv[k]);
            }
            const uint16_t *Wt = W + (int64_t)tgt[j] * d;
            for (int64_t k = 0; k < d; ++k) out[k] = c * (out[k] - bf16_value(Wt[k]));
        }
        free(z);
        free(hj);
    }
}

/* Eq. 10 over every row: returns the loss, fills lse[L] and nll[L] and, if
 * dh is given, dh[L, d]. */
double oracle_ce_loss(const uint16_t *h, const uint16_t *W, const int32_t *tgt, const float *w,
                      int64_t L, int64_t d, int64_t V, double *lse, double *nll, double *dh)
{
    int64_t *rows = (int64_t *)malloc((size_t)(L > 0 ? L : 1) * sizeof(int64_t));
    for (int64_t j = 0; j < L; ++j) rows[j] = j;
    oracle_ce_rows(h, W, tgt, w, L, d, V, rows, L, lse, nll, dh);
    free(rows);
    double s = 0.0;
    for (int64_t j = 0; j < L; ++j) s += (double)w[j] * nll[j];
    return L > 0 ? s / (double)L : 0.0;
}

/* ------------------------------------------------------------------------ */
/* LoRA adapter gradients (Appendix C adapter; y = x W0 + s (x A) B)        */
/* ------------------------------------------------------------------------ */

/*
 * x [L, din], dy [L, dout], A [din, r], B [r, dout] (bf16, row-major).
 *   u  = x A            [L, r]
 *   v  = dy B^T         [L, r]
 *   dB = s u^T dy       [r, dout]
 *   dA = s x^T v        [din, r]
 * Outputs fp64.
 */
void oracle_lora_grad(const uint16_t *x, const uint16_t *dy, const uint16_t *A, const uint16_t *B,
                      int64_t L, int64_t din, int64_t dout, int r, double s,
                      double *dA, double *dB)
{
    double *u = (double *)calloc((size_t)(L * r > 0 ? L * r : 1), sizeof(double));
    double *v = (double *)calloc((size_t)(L * r > 0 ? L * r : 1), sizeof(double));
#pragma omp parallel for schedule(static)
    for (int64_t l = 0; l < L; ++l) {
        for (int c = 0; c < r; ++c) {
            double a = 0.0;
            for (int64_t i = 0; i < din; ++i) a += bf16_value(x[l * din + i]) * bf16_value(A[i * r + c]);
            u[l * r + c] = a;
            double b = 0.0;
            for (int64_t o = 0; o < dout; ++o) b += bf16_value(dy[l * dout + o]) * bf16_value(B[(int64_t)c * dout + o]);
            v[l * r + c] = b;
        }
    }
#pragma omp parallel for schedule(static)
    for (int64_t o = 0; o < dout; ++o) {
        for (int c = 0; c < r; ++c) {
            double a = 0.0;
            for (int64_t l = 0; l < L; ++l) a += u[l * r + c] * bf16_value(dy[l * dout + o]);
            dB[(int64_t)c * dout + o] = s * a;
        }
    }
#pragma omp parallel for schedule(static)
    for (int64_t i = 0; i < din; ++i) {
        for (int c = 0; c < r; ++c) {
            double a = 0.0;
            for (int64_t l = 0; l < L; ++l) a += bf16_value(x[l * din + i]) * v[l * r + c];
            dA[i * r + c] = s * a;
        }
    }
    free(u);
    free(v);
}

/* ------------------------------------------------------------------------ */
/* The adapted projection of a chained update (Appendix C adapter)          */
/* ------------------------------------------------------------------------ */

/*
 * x [L, din], W0 [din, dout], A [din, r], B [r, dout] (bf16, row-major):
 *   h = x W0 + s (x A) B        [L, dout], fp64
 */
void oracle_lora_forward(const uint16_t *x, const uint16_t *W0, const uint16_t *A, const uint16_t *B,
                         int64_t L, int64_t din, int64_t dout, int r, double s, double *h)
{
#pragma omp parallel
    {
        double *u = (double *)calloc((size_t)(r > 0 ? r : 1), sizeof(double));
#pragma omp for schedule(static)
        for (int64_t l = 0; l < L; ++l) {
            for (int c = 0; c < r; ++c) {
                double a = 0.0;
                for (int64_t i = 0; i < din; ++i) a += bf16_value(x[l * din + i]) * bf16_value(A[i * r + c]);
                u[c] = a;
            }
            for (int64_t o = 0; o < dout; ++o) {
                double a = 0.0;
                for (int64_t i = 0; i < din; ++i) a += bf16_value(x[l * din + i]) * bf16_value(W0[i * dout + o]);
                double b = 0.0;
                for (int c = 0; c < r; ++c) b += u[c] * bf16_value(B[(int64_t)c * dout + o]);
                h[l * dout + o] = a + s * b;
            }
        }
        free(u);
    }
}

/*
 * The gradient of the projection's input, dy [L, dout] being the gradient of
 * its output:  dx = dy W0^T + s (dy B^T) A^T        [L, din], fp64
 */
void oracle_lora_input_grad(const uint16_t *dy, const uint16_t *W0, const uint16_t *A, const uint16_t *B,
                            int64_t L, int64_t din, int64_t dout, int r, double s, double *dx)
{
#pragma omp parallel
    {
        double *v = (double *)calloc((size_t)(r > 0 ? r : 1), sizeof(double));
#pragma omp for schedule(static)
        for (int64_t l = 0; l < L; ++l) {
            for (int c = 0; c < r; ++c) {
                double a = 0.0;
                for (int64_t o = 0; o < dout; ++o) a += bf16_value(dy[l * dout + o]) * bf16_value(B[(int64_t)c * dout + o]);
                v[c] = a;
            }
            for (int64_t i = 0; i < din; ++i) {
                double a = 0.0;
                for (int64_t o = 0; o < dout; ++o) a += bf16_value(dy[l * dout + o]) * bf16_value(W0[i * dout + o]);
                double b = 0.0;
                for (int c = 0; c < r; ++c) b += v[c] * bf16_value(A[i * r + c]);
                dx[l * din + i] = a + s * b;
            }
        }
        free(v);
    }
}

/*
 * Adapter drift (Sec. 4, Fig. 6): per row j, the KL divergence of the
 * adapted model's next-token distribution p_j = softmax(h_p[j] W^T) from the
 * base model's q_j = softmax(h_q[j] W^T):
 *   KL_j = sum_v p_jv (log p_jv - log q_jv)
 * with log p_jv = z_p,jv - lse_p,j (fp64 logits over the bf16 inputs).
 */
void oracle_kl_rows(const uint16_t *hp, const uint16_t *hq, const uint16_t *W, int64_t d, int64_t V,
                    const int64_t *rows, int64_t nrows, double *kl)
{
#pragma omp parallel for schedule(dynamic, 1)
    for (int64_t i = 0; i < nrows; ++i) {
        int64_t j = rows[i];
        double *a = (double *)malloc((size_t)d * sizeof(double));
        double *b = (double *)malloc((size_t)d * sizeof(double));
        double *zp = (double *)malloc((size_t)V * sizeof(double));
        double *zq = (double *)malloc((size_t)V * sizeof(double));
        for (int64_t k = 0; k < d; ++k) {
            a[k] = bf16_value(hp[j * d + k]);
            b[k] = bf16_value(hq[j * d + k]);
        }
        double mp = -INFINITY, mq = -INFINITY;
        for (int64_t v = 0; v < V; ++v) {
            const uint16_t *Wv = W + v * d;
            double sp = 0.0, sq = 0.0;
            for (int64_t k = 0; k < d; ++k) {
                double wv = bf16_value(Wv[k]);
                sp += a[k] * wv;
                sq += b[k] * wv;
            }
            zp[v] = sp;
            zq[v] = sq;
            if (sp > mp) mp = sp;
            if (sq > mq) mq = sq;
        }
        double ep = 0.0, eq = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            ep += exp(zp[v] - mp);
            eq += exp(zq[v] - mq);
        }
        double lp = mp + log(ep), lq = mq + log(eq);
        double acc = 0.0;
        for (int64_t v = 0; v < V; ++v) {
            double logp = zp[v] - lp, logq = zq[v] - lq;
            acc += exp(logp) * (logp - logq);
        }
        kl[i] = acc;
        free(zq);
        free(zp);
        free(b);
        free(a);
    }
}

/* ------------------------------------------------------------------------ */
/* Eq. 2 / Algorithm 1: the SGD step on the fp32 adapter masters            */
/* ------------------------------------------------------------------------ */

/* p <- p - lr * g, in fp32, multiply then subtract (no fused multiply-add). */
void oracle_sgd_step(float *p, const float *g, int64_t n, float lr)
{
    for (int64_t i = 0; i < n; ++i) {
        volatile float step = lr * g[i];
        p[i] = p[i] - step;
    }
}

/* fp32 -> bf16 round-to-nearest-even, NaN kept quiet. */
void oracle_to_bf16(const float *p, uint16_t *out, int64_t n)
{
    for (int64_t i = 0; i < n; ++i) {
        uint32_t u;
        memcpy(&u, &p[i], sizeof u);
        if ((u & 0x7f800000u) == 0x7f800000u && (u & 0x007fffffu)) {
            out[i] = (uint16_t)((u >> 16) | 0x0040u);
            continue;
        }
        uint32_t lsb = (u >> 16) & 1u;
        u += 0x7fffu + lsb;
        out[i] = (uint16_t)(u >> 16);
    }
}
