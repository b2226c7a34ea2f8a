// tc_gemm.cuh -- the tcgen05 contraction engine shared by the Eq. 10 CE
// kernels and the LoRA adapter-gradient kernels.
//
// D[M x N] = A[M x K] * B[N x K]^T with bf16 operands and fp32 accumulation.
// K may run over two operand pairs, D = A B^T + A2 B2^T (the K blocks of A2 /
// B2 follow those of A / B; both pairs share the operand majors).
//   * one CTA per SM, persistent over output tiles of 128 x BN (BN <= 256);
//   * warp 0: TMA producer (one thread) filling a ring of `stages` shared-
//     memory stages of 64-deep K blocks, 128-byte swizzled;
//   * warp 1: allocates TMEM and issues tcgen05.mma (one thread), four
//     M128 x N(BN) x K16 MMAs per stage, into one of two TMEM accumulators;
//   * warps 2-5: epilogue, one accumulator row per thread (tcgen05.ld
//     32x32b), overlapping the next tile's MMAs through the second
//     accumulator.  The epilogue kinds fuse the work that follows the
//     contraction so that nothing of size [M x N] goes back to HBM unless it
//     is the result itself.
// An operand is K-major (K contiguous in memory: a row-major [rows, K] matrix)
// or MN-major (rows contiguous: a row-major [K, rows] matrix); both are
// loaded by TMA with the 128-byte swizzle that tcgen05 reads natively.
// Tiles past M, N or K are zero-filled by TMA and masked in the epilogue.
// When the tiles do not fill the last wave, the tiles of that wave may be
// cut into K pieces spread over the idle SMs (EPI_F32_ACC): each piece
// stores an fp32 partial and the last piece to arrive sums them in piece
// order, so the result does not depend on which piece finishes last.
#pragma once

#include "attt_common.cuh"

namespace attt {

enum EpiKind : int {
    EPI_CE_EXP = 0,    // per (row, vocab tile): max m, E = exp(z - m) as bf16, sum of E, target logit
    EPI_F32_ACC = 2,   // out[m, n] = (acc ? alpha_m out[m, n] : 0) + beta_m acc [- gamma_m W[t_m, n]]  (fp32)
    EPI_BF16 = 5,      // out16[m, n] = bf16(alpha * acc)  (row-major, through TMA boxes)
    EPI_KL = 6,        // A tile = 64 rows of A over the same 64 rows of A2: per (row, tile) max, sum of exp, cross term
};

constexpr int kMaxProj = 8;

struct EpiParams {
    // CE
    const int32_t *tgt;  // [M] target ids
    float2 *part;        // [vocab tiles, M] (max, sum of exp) in log2 units
    int tile0;           // vocab tile index of column 0 of this launch
    float *ztgt;         // [M] target logit
    const float *eref;   // [M] reference (log2 units) E is written against; nullptr: the tile max
    int v0;              // vocab id of column 0 of this launch
    __nv_bfloat16 *G;    // [M, G_ld]
    int64_t G_ld;
    // fp32 outputs
    float *out;
    int64_t out_ld;
    int accumulate;
    float alpha;
    const float *row_alpha;  // [M] or nullptr (1)
    const float *row_beta;   // [M] or nullptr (1)
    const float *row_gamma;  // [M] or nullptr (no W term)
    const int32_t *fix_tgt;  // [M] row of fix_W each output row subtracts (clamped into [0, fix_V))
    const __nv_bfloat16 *fix_W;
    int64_t fix_ld;
    int fix_V;
    __nv_bfloat16 *out16;    // EPI_BF16 output, row pitch out_ld
    // EPI_KL: five planes of [tiles, M] fp32 (m_p, s_p, m_q, s_q, x), kl_plane apart
    float *kl_part;
    int64_t kl_plane;
};

struct GemmArgs {
    int M, N;
    int BN, stages;
    int tiles_m, tiles_n, splits;
    int kb_per_split, kb_total;
    int a_m_off, a_k_off;  // coordinate offsets into A's tensor map
    int b_n_off, b_k_off;  // coordinate offsets into B's tensor map
    uint32_t tmem_cols;
    uint32_t e_stage_bytes;  // shared-memory staging of the TMA-stored epilogue output, else 0
    // Programmatic dependent launch: the A/B operands were complete before the
    // previous grid in the stream started, so the producer need not wait for it
    // (the epilogue always does).
    int operands_ready;
    int kb_split;  // K blocks of the first operand pair; later ones come from A2 / B2
    int *status;
    EpiParams ep;
    // Tail split (tc_gemm_kernel / tc_gemm_pair_kernel): tiles [0, whole_tiles)
    // run whole; every later tile runs as tail_s K pieces.
    int whole_tiles, tail_s;
    float *split_ws;           // [tail tile][piece][CTA rank] fp32 partials of 128 x BN, column-quad major
    unsigned int *split_tick;  // [tail tile][CTA rank] arrival counters; 0 between launches
};

constexpr uint32_t kABytes = 128 * 64 * 2;  // one A stage: 128 rows x 64 bf16
constexpr int kGemmThreads = 192;
// The pair kernel runs a second TMA producer warp (warp 6): the two take
// alternate stages (one issuing thread keeps about one stage in flight).
constexpr int kGemmPairThreads = 224;

__host__ __device__ inline uint32_t gemm_b_stage_bytes(int BN) { return (uint32_t)BN * 128u; }

// EPI_CE_EXP stages E through shared memory: per epilogue warp two buffers of
// 32 rows x 32 bf16 (64-byte swizzle), written out by TMA stores.
constexpr uint32_t kEStageBytes = 4 * 2 * 32 * 64;

__host__ __device__ inline size_t gemm_smem_bytes(int BN, int stages, uint32_t extra = 0) {
    return 1024 + (size_t)stages * (kABytes + gemm_b_stage_bytes(BN)) + extra + 8 * (2 * stages + 5) + 16;
}

// EPI_KL hands z_q from the warps holding it to the warps holding z_p through
// shared memory: per warp pair two buffers of 32 columns x 32 rows fp32.
constexpr uint32_t kKlXBytes = 2 * 2 * 32 * 32 * 4;

// One 32 x 32 bf16 block of E (this warp's 32 rows, 32 columns from x) to
// global memory through the warp's staging buffer `chunk & 1`: lane = row,
// 16-byte pieces placed as the 64-byte swizzle expects (piece q of row r at
// q ^ ((r >> 1) & 3)), so the 8 lanes of each quarter-warp hit distinct banks.
// Lane 0 owns the bulk group; before a buffer is refilled, the store that used
// it two blocks ago has finished reading it.
__device__ __forceinline__ void e_block_store(const CUtensorMap *tm, uint32_t sbuf, int chunk, int lane,
                                              const uint32_t (&pk)[16], int x, int y) {
    const uint32_t buf = sbuf + (uint32_t)(chunk & 1) * 2048u;
    if (lane == 0) bulk_wait_read<1>();
    __syncwarp();
    const uint32_t rowp = buf + (uint32_t)lane * 64u;
    const uint32_t sw = ((uint32_t)lane >> 1) & 3u;
#pragma unroll
    for (uint32_t q = 0; q < 4; ++q)
        st_shared_v4(rowp + ((q ^ sw) << 4), pk[4 * q], pk[4 * q + 1], pk[4 * q + 2], pk[4 * q + 3]);
    fence_proxy_async_smem();
    __syncwarp();
    if (lane == 0) {
        tma_store_2d(tm, buf, x, y);
        bulk_commit();
    }
}

// One unit of work of tc_gemm_kernel / tc_gemm_pair_kernel: an output tile
// (m fastest) and its K-block range; piece >= 0 marks a K piece of tail tile
// `tail`.  `tiles_m` counts row tiles of the kernel's accumulator height.
struct Work {
    int tm, tn, kb0, kb1, piece, tail;
};

__device__ __forceinline__ Work work_item(const GemmArgs &g, int w, int tiles_m) {
    Work k;
    int t = w;
    k.piece = -1;
    k.tail = -1;
    k.kb0 = 0;
    k.kb1 = g.kb_total;
    if (w >= g.whole_tiles) {
        const int j = w - g.whole_tiles;
        k.tail = j / g.tail_s;
        k.piece = j - k.tail * g.tail_s;
        t = g.whole_tiles + k.tail;
        k.kb0 = (int)((int64_t)g.kb_total * k.piece / g.tail_s);
        k.kb1 = (int)((int64_t)g.kb_total * (k.piece + 1) / g.tail_s);
    }
    k.tn = t / tiles_m;
    k.tm = t - k.tn * tiles_m;
    return k;
}

__device__ __forceinline__ int work_count(const GemmArgs &g, int tiles_m) {
    return g.whole_tiles + (tiles_m * g.tiles_n - g.whole_tiles) * g.tail_s;
}

constexpr float kLog2e = 1.4426950408889634f;

// A CE tile whose max exceeds the row reference by more than kCeRefJump
// (log2 units) writes E against its own max instead, so E <= 2^64.  The dh
// contraction of a chunk sums at most 2^16 such terms times |W|, and the fp32
// accumulator holds that for |W| up to 2^40.
constexpr float kCeRefJump = 64.f;

// Per-row terms of EPI_F32_ACC for output row gm: ra, rb and, when the
// epilogue subtracts gamma_m W[t_m, :], gamma and that row of W.
struct AccRow {
    float ra, rb, gam;
    const __nv_bfloat16 *wrow;
};

__device__ __forceinline__ AccRow acc_row(const EpiParams &ep, int gm, bool rv) {
    AccRow a{1.f, 1.f, 0.f, nullptr};
    if (rv) {
        if (ep.row_alpha) a.ra = __ldg(ep.row_alpha + gm);
        if (ep.row_beta) a.rb = __ldg(ep.row_beta + gm);
        if (ep.row_gamma) {
            a.gam = __ldg(ep.row_gamma + gm);
            int t = __ldg(ep.fix_tgt + gm);
            if (t < 0 || t >= ep.fix_V) t = 0;
            a.wrow = ep.fix_W + (int64_t)t * ep.fix_ld;
        }
    }
    return a;
}

// ---------------------------------------------------------------------------
// Epilogues.  Every thread owns accumulator row `row` of the tile; all 32
// lanes of a warp execute the TMEM loads together even when their row is
// past M (the loads are warp-collective); only stores are predicated.
// ---------------------------------------------------------------------------

// EPI_F32_ACC goes through TMA too: per epilogue warp two 32 x 32 fp32 boxes
// (128-byte swizzle) and one mbarrier each, after the 8 boxes.
constexpr uint32_t kF32StageBytes = 4 * 2 * 4096 + 64;

struct F32Stage {
    uint32_t buf0;  // this warp's box 0 (box 1 at +4096)
    uint32_t bar0;  // its mbarrier 0 (1 at +8)
    uint32_t ec;    // boxes handled so far: box ec & 1, load parity (ec >> 1) & 1
};

// TMA load of the old outputs of one box into box `slot`, once the store that
// last used it has read it (lane 0 owns the bulk group and the barrier).
__device__ __forceinline__ void f32_box_load(const CUtensorMap *tm, const F32Stage &st, uint32_t slot, int lane,
                                             int x, int y) {
    if (lane == 0) {
        bulk_wait_read<0>();
        const uint32_t bar = st.bar0 + 8u * slot;
        mbar_arrive_expect_tx(bar, 4096u);
        tma_load_2d(st.buf0 + 4096u * slot, tm, bar, x, y);
    }
}

// EPI_F32_ACC for this warp's 32 rows (from y; lane = row), box by box over
// the tile's columns [n_base, n_end): out = (accumulate ? ra out : 0) + rb v
// - gam W[t, :], where src(c, v) gives the lane's accumulator values of
// columns n_base + c .. + 31.  The old outputs of the next box load while this
// one is combined in shared memory; each box goes back by a TMA store (rows
// past M and columns past N are clipped by the tensor map).
template <class Src>
__device__ __forceinline__ void f32_tile_store(const GemmArgs &g, const CUtensorMap *tm, F32Stage &st, int lane,
                                               int y, const AccRow &a, int n_base, int n_end,
                                               volatile int *abort_flag, Src &&src) {
    const EpiParams &ep = g.ep;
    if (y >= g.M) return;  // every row of this warp lies past M (warp-uniform)
    const int nch = min(g.BN, n_end - n_base + 31) >> 5;
    if (ep.accumulate) f32_box_load(tm, st, st.ec & 1u, lane, n_base, y);
    for (int k = 0; k < nch; ++k, ++st.ec) {
        const uint32_t slot = st.ec & 1u;
        const uint32_t buf = st.buf0 + 4096u * slot;
        const int x = n_base + 32 * k;
        if (ep.accumulate && k + 1 < nch) f32_box_load(tm, st, slot ^ 1u, lane, x + 32, y);
        float v[32];
        src(32 * k, v);
        float w[32];
        if (a.wrow) {
            if (x + 32 <= n_end) {
                const uint4 *wp = reinterpret_cast<const uint4 *>(a.wrow + x);
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const uint4 u = __ldg(wp + q);
                    const __nv_bfloat162 *b = reinterpret_cast<const __nv_bfloat162 *>(&u);
#pragma unroll
                    for (int e = 0; e < 4; ++e) {
                        const float2 f = __bfloat1622float2(b[e]);
                        w[8 * q + 2 * e] = f.x;
                        w[8 * q + 2 * e + 1] = f.y;
                    }
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; ++i) w[i] = (x + i < n_end) ? __bfloat162float(a.wrow[x + i]) : 0.f;
            }
        }
        if (ep.accumulate) {
            if (!mbar_wait(st.bar0 + 8u * slot, (st.ec >> 1) & 1u, abort_flag)) record_error(g.status, ATTT_ERR_TIMEOUT);
        } else if (lane == 0) {
            bulk_wait_read<1>();  // the store two boxes back has read this box
        }
        __syncwarp();
        const uint32_t rowp = buf + (uint32_t)lane * 128u;
#pragma unroll
        for (uint32_t q = 0; q < 8; ++q) {
            const uint32_t ad = rowp + ((q ^ ((uint32_t)lane & 7u)) << 4);
            float4 o = make_float4(a.rb * v[4 * q], a.rb * v[4 * q + 1], a.rb * v[4 * q + 2], a.rb * v[4 * q + 3]);
            if (ep.accumulate) {
                const float4 p = ld_shared_f4(ad);
                o.x = fmaf(a.ra, p.x, o.x); o.y = fmaf(a.ra, p.y, o.y);
                o.z = fmaf(a.ra, p.z, o.z); o.w = fmaf(a.ra, p.w, o.w);
            }
            if (a.wrow) {
                o.x = fmaf(-a.gam, w[4 * q], o.x); o.y = fmaf(-a.gam, w[4 * q + 1], o.y);
                o.z = fmaf(-a.gam, w[4 * q + 2], o.z); o.w = fmaf(-a.gam, w[4 * q + 3], o.w);
            }
            st_shared_f4(ad, o);
        }
        fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) {
            tma_store_2d(tm, buf, x, y);
            bulk_commit();
        }
    }
}

// EPI_BF16 for this warp's 32 rows (from y; lane = row): out16 = bf16(alpha
// acc) for the tile's columns [n_base, n_end), box by box through the warp's
// staging buffers; the running box count `ec` picks the buffer.
__device__ __forceinline__ void bf16_tile_store(const GemmArgs &g, const CUtensorMap *tm, uint32_t sE, uint32_t &ec,
                                                int lane, int y, int n_base, int n_end, uint32_t taddr) {
    if (y >= g.M) return;  // every row of this warp lies past M (warp-uniform)
    for (int c = 0; c < g.BN; c += 32) {
        if (n_base + c >= n_end) break;
        float v[32];
        tmem_ld_x32(taddr + (uint32_t)c, v);
        uint32_t pk[16];
#pragma unroll
        for (int i = 0; i < 32; i += 2) {
            __nv_bfloat162 b = __floats2bfloat162_rn(g.ep.alpha * v[i], g.ep.alpha * v[i + 1]);
            pk[i / 2] = *reinterpret_cast<uint32_t *>(&b);
        }
        e_block_store(tm, sE, (int)(ec++), lane, pk, n_base + c, y);
    }
}

// tmE / sE: the E tensor map and this warp's staging buffers (EPI_CE_EXP).
template <int EPI>
__device__ __forceinline__ void epilogue_tile(const GemmArgs &g, int gm_base, int tn, int row, uint32_t taddr,
                                              const CUtensorMap *tmE = nullptr, uint32_t sE = 0) {
    const int gm = gm_base + row;
    const bool rv = gm < g.M;
    const int n_base = tn * g.BN;
    // Columns this tile owns: [n_base, n_tile) within the tile, [n_base, n_end)
    // within the problem.  TMEM is read in chunks of 32 (or 16) columns, so a
    // chunk may run past the tile when BN is not a multiple of it; nothing
    // past n_tile is ever stored (it belongs to the next tile).
    const int n_tile = n_base + g.BN;
    const int n_end = min(g.N, n_tile);
    const EpiParams &ep = g.ep;

    if constexpr (EPI == EPI_CE_EXP) {
        // One pass over the tile's columns against the row reference R
        // (log2 units): E = exp2(z2 - R) rounded to bf16 into the gradient
        // block (columns past N as zeros), the tile max m, the sum of the
        // unrounded exp2(z2 - R) and the target logit.  The pair stored is
        // (m, sum of exp2(z2 - m)).  A row whose tile max exceeds R by more
        // than kCeRefJump (or has no reference) takes a second pass that
        // writes E = exp2(z2 - m) instead; that pass is warp-wide because TMEM
        // loads are.
        const int t = rv ? __ldg(ep.tgt + gm) - ep.v0 : -1;
        const float R = (ep.eref && rv) ? __ldg(ep.eref + gm) : -INFINITY;
        const int lane = row & 31, y = gm - lane;
        float mx = -INFINITY, zt = 0.f, sr = 0.f;
        bool hit = false;
        for (int c = 0; c < g.BN; c += 32) {
            float v[32];
            tmem_ld_x32(taddr + (uint32_t)c, v);
            const int col0 = n_base + c;
            const int tc = t - col0;
            uint32_t pk[16];
            if (col0 + 32 <= n_end) {
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                    const float z0 = v[i] * kLog2e, z1 = v[i + 1] * kLog2e;
                    mx = fmaxf(mx, fmaxf(z0, z1));
                    if (tc == i) { zt = v[i]; hit = true; }
                    if (tc == i + 1) { zt = v[i + 1]; hit = true; }
                    const float e0 = exp2f(z0 - R), e1 = exp2f(z1 - R);
                    sr += e0 + e1;
                    __nv_bfloat162 b = __floats2bfloat162_rn(e0, e1);
                    pk[i / 2] = *reinterpret_cast<uint32_t *>(&b);
                }
            } else {
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                    float e0 = 0.f, e1 = 0.f;
                    if (col0 + i < n_end) {
                        const float z0 = v[i] * kLog2e;
                        mx = fmaxf(mx, z0);
                        if (tc == i) { zt = v[i]; hit = true; }
                        e0 = exp2f(z0 - R);
                    }
                    if (col0 + i + 1 < n_end) {
                        const float z1 = v[i + 1] * kLog2e;
                        mx = fmaxf(mx, z1);
                        if (tc == i + 1) { zt = v[i + 1]; hit = true; }
                        e1 = exp2f(z1 - R);
                    }
                    sr += e0 + e1;
                    __nv_bfloat162 b = __floats2bfloat162_rn(e0, e1);
                    pk[i / 2] = *reinterpret_cast<uint32_t *>(&b);
                }
            }
            // zeros past N (inside the tile) are stored too: the dh
            // contraction reads whole 64-column K blocks; rows past M are
            // clipped by the tensor map
            e_block_store(tmE, sE, c >> 5, lane, pk, col0, y);
        }
        const bool own = rv && !(mx - R <= kCeRefJump);
        float sm;
        if (!own) {
            // sum against m from the sum against R; when R - m >= 100 every
            // term against R may have underflowed, and such a tile is below
            // 2^-92 of the row's sum (R is at most the row max)
            const float dd = R - mx;
            sm = (dd < 100.f) ? sr * exp2f(dd) : (sr > 0.f ? exp2f(log2f(sr) + dd) : 1.f);
        }
        if (__any_sync(0xffffffffu, own)) {
            // the warp's blocks again, after the first pass's stores have
            // landed: rows against their own max, the others as before
            if (lane == 0) bulk_wait<0>();
            __syncwarp();
            float so = 0.f;
            for (int c = 0; c < g.BN; c += 32) {
                float v[32];
                tmem_ld_x32(taddr + (uint32_t)c, v);
                const int col0 = n_base + c;
                uint32_t pk[16];
#pragma unroll
                for (int i = 0; i < 32; i += 2) {
                    float e0 = 0.f, e1 = 0.f;
                    if (col0 + i < n_end) e0 = own ? exp2f(fmaf(v[i], kLog2e, -mx)) : exp2f(v[i] * kLog2e - R);
                    if (col0 + i + 1 < n_end)
                        e1 = own ? exp2f(fmaf(v[i + 1], kLog2e, -mx)) : exp2f(v[i + 1] * kLog2e - R);
                    so += e0 + e1;
                    __nv_bfloat162 b = __floats2bfloat162_rn(e0, e1);
                    pk[i / 2] = *reinterpret_cast<uint32_t *>(&b);
                }
                e_block_store(tmE, sE, c >> 5, lane, pk, col0, y);
            }
            if (own) sm = so;
        }
        if (rv) {
            ep.part[(int64_t)(ep.tile0 + tn) * g.M + gm] = make_float2(mx, sm);
            if (hit) ep.ztgt[gm] = zt;
        }
    }
}

// EPI_KL.  The CTA's 128 accumulator rows are 64 rows of z_p = h_p W^T
// (TMEM lanes 0-63: warp quarters 0, 1) over the same 64 rows of z_q =
// h_q W^T (lanes 64-127: quarters 2, 3), so quarter q and quarter q + 2 hold
// one row's two logit sets.  Each warp takes its rows' max over the tile's
// columns; then, 32 columns at a time, the z_q warp adds its exp2(z log2e -
// m_q) and hands the chunk to its partner through shared memory (column-major,
// so both sides are conflict-free; two buffers, one 64-thread named barrier
// per chunk), and the z_p warp adds exp2(z_p log2e - m_p) and the cross term
// x = sum exp2(z_p log2e - m_p) (z_p - z_q).  All from fp32 accumulators.
// `ck` counts the chunks handed over so far (the buffer parity).
__device__ __forceinline__ void epilogue_kl(const GemmArgs &g, int gm_base, int tn, int q, int lane, uint32_t taddr,
                                            float *xbuf, uint32_t &ck) {
    const bool isp = q < 2;
    const int gm = gm_base + (q & 1) * 32 + lane;
    const int n_base = tn * g.BN;
    const int nv = min(g.N, n_base + g.BN) - n_base;  // valid columns of the tile
    const uint32_t bar = 2u + (uint32_t)(q & 1);
    float *const pair_buf = xbuf + (q & 1) * 2 * 32 * 32;
    float mx = -INFINITY;
    for (int c = 0; c < g.BN; c += 32) {
        float v[32];
        tmem_ld_x32(taddr + (uint32_t)c, v);
#pragma unroll
        for (int i = 0; i < 32; ++i)
            if (c + i < nv) mx = fmaxf(mx, v[i]);
    }
    const float m2 = mx * kLog2e;
    float sm = 0.f, x = 0.f;
    for (int c = 0; c < g.BN; c += 32, ++ck) {
        float v[32];
        tmem_ld_x32(taddr + (uint32_t)c, v);
        float *buf = pair_buf + (ck & 1u) * 32 * 32;
        if (!isp) {
#pragma unroll
            for (int i = 0; i < 32; ++i) {
                if (c + i < nv) sm += exp2f(fmaf(v[i], kLog2e, -m2));
                buf[i * 32 + lane] = v[i];
            }
        }
        named_barrier_sync(bar, 64);
        if (isp) {
#pragma unroll
            for (int i = 0; i < 32; ++i)
                if (c + i < nv) {
                    const float e = exp2f(fmaf(v[i], kLog2e, -m2));
                    sm += e;
                    x = fmaf(e, v[i] - buf[i * 32 + lane], x);
                }
        }
    }
    const EpiParams &ep = g.ep;
    const int64_t o = (int64_t)(ep.tile0 + tn) * g.M + gm, P = ep.kl_plane;
    if (gm < g.M && ATTT_GUARD(o < P, g.status)) {
        if (isp) {
            ep.kl_part[o] = m2;
            ep.kl_part[P + o] = sm;
            ep.kl_part[4 * P + o] = x;
        } else {
            ep.kl_part[2 * P + o] = m2;
            ep.kl_part[3 * P + o] = sm;
        }
    }
}

// EPI_F32_ACC for K piece k.piece of tail tile k.tail, on the 128 accumulator
// rows this CTA holds (CTA `rank` of `nranks`).  The four epilogue warps store
// the piece's partial (column-quad major: a warp writes 512 contiguous bytes
// per store), then one thread takes a ticket; the piece that arrives last
// forms the sum P_0 + P_1 + ... in piece order, its own term read back from
// TMEM, and applies the epilogue to it.  BN is a multiple of 32.
__device__ __forceinline__ void epilogue_piece_f32_acc(const GemmArgs &g, const Work &k, int gm_base, int rank,
                                                      int nranks, int row, uint32_t taddr, const CUtensorMap *tm,
                                                      F32Stage &st, volatile int *abort_flag) {
    const int BN = g.BN;
    const size_t region = (size_t)128 * (size_t)BN;
    const size_t slot0 = (size_t)k.tail * (size_t)g.tail_s;
    float4 *mine = reinterpret_cast<float4 *>(g.split_ws + ((slot0 + k.piece) * nranks + rank) * region) + row;
    for (int c = 0; c < BN; c += 32) {
        float v[32];
        tmem_ld_x32(taddr + (uint32_t)c, v);
#pragma unroll
        for (int q = 0; q < 8; ++q)
            __stcg(mine + (size_t)(c / 4 + q) * 128, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
    }
    __threadfence();
    named_barrier_sync(1, 128);
    int last = 0;
    if (row == 0) {
        unsigned int *tk = g.split_tick + (size_t)k.tail * nranks + rank;
        last = atomicAdd(tk, 1u) == (unsigned int)(g.tail_s - 1) ? 1 : 0;
        if (last) atomicExch(tk, 0u);  // every piece has arrived: ready for the next launch
        __threadfence();
    }
    if (!named_barrier_or(1, 128, last)) return;

    const int gm = gm_base + row;
    const int n_base = k.tn * BN;
    const AccRow a = acc_row(g.ep, gm, gm < g.M);
    f32_tile_store(g, tm, st, row & 31, gm - (row & 31), a, n_base, min(g.N, n_base + BN), abort_flag,
                   [&](int c, float(&sm)[32]) {
                       for (int j = 0; j < g.tail_s; ++j) {
                           float v[32];
                           if (j == k.piece) {
                               tmem_ld_x32(taddr + (uint32_t)c, v);
                           } else {
                               const float4 *src = reinterpret_cast<const float4 *>(
                                                       g.split_ws + ((slot0 + j) * nranks + rank) * region) +
                                                   row;
#pragma unroll
                               for (int q = 0; q < 8; ++q) {
                                   const float4 p = __ldcg(src + (size_t)(c / 4 + q) * 128);
                                   v[4 * q] = p.x; v[4 * q + 1] = p.y; v[4 * q + 2] = p.z; v[4 * q + 3] = p.w;
                               }
                           }
#pragma unroll
                           for (int i = 0; i < 32; ++i) sm[i] = (j == 0) ? v[i] : sm[i] + v[i];
                       }
                   });
}

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------

template <int EPI, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kGemmThreads, 1)
    tc_gemm_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmA2,
                   const __grid_constant__ CUtensorMap tmB2, const GemmArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = g.stages;
    const uint32_t b_bytes = gemm_b_stage_bytes(g.BN);
    uint8_t *sA = smem;
    uint8_t *sB = smem + (size_t)S * kABytes;
    uint8_t *sE = sB + (size_t)S * b_bytes;  // 1024-byte aligned: b_bytes is a multiple of 2048
    uint64_t *bars = reinterpret_cast<uint64_t *>(sE + g.e_stage_bytes);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = smem_u32(bars + S);
    const uint32_t tfull0 = smem_u32(bars + 2 * S);
    const uint32_t tempty0 = smem_u32(bars + 2 * S + 2);
    const uint32_t drain0 = smem_u32(bars + 2 * S + 4);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * S + 5);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull0 + 8 * a, 1);
            mbar_init(tempty0 + 8 * a, 4);
        }
        griddep_launch_dependents();
        mbar_init(drain0, 1);
        if (EPI == EPI_F32_ACC)
            for (int b = 0; b < 8; ++b) mbar_init(smem_u32(sE) + 32768u + 8u * b, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        if (g.kb_split < g.kb_total) {
            tma_prefetch_desc(&tmA2);
            tma_prefetch_desc(&tmB2);
        }
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), g.tmem_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    const int nwork = work_count(g, g.tiles_m);

    if (warp == 0) {
        if (lane == 0) {
            // ---------------- TMA producer ----------------
            if (!g.operands_ready) griddep_wait();
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;  // per stage: last issue pending?
            bool ok = true;
            for (int w = blockIdx.x; w < nwork && ok; w += gridDim.x) {
                const Work wi = work_item(g, w, g.tiles_m);
                const int tm = wi.tm, tn = wi.tn;
                for (int kb = wi.kb0; kb < wi.kb1; ++kb) {
                    if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) { ok = false; break; }
                    const uint32_t fb = full0 + 8 * stage;
                    mbar_arrive_expect_tx(fb, kABytes + b_bytes);
                    const uint32_t a_dst = smem_u32(sA + (size_t)stage * kABytes);
                    const uint32_t b_dst = smem_u32(sB + (size_t)stage * b_bytes);
                    // K block kb of the first pair, or K block kb - kb_split of the second
                    const bool sec = kb >= g.kb_split;
                    const CUtensorMap *pa = sec ? &tmA2 : &tmA;
                    const CUtensorMap *pb = sec ? &tmB2 : &tmB;
                    const int ka = sec ? (kb - g.kb_split) * 64 : g.a_k_off + kb * 64;
                    const int kbk = sec ? (kb - g.kb_split) * 64 : g.b_k_off + kb * 64;
                    const int am = (sec ? 0 : g.a_m_off) + tm * 128;
                    const int bn = (sec ? 0 : g.b_n_off) + tn * g.BN;
                    if (!A_MN) {
                        tma_load_2d(a_dst, pa, fb, ka, am);
                    } else {
                        tma_load_2d(a_dst, pa, fb, am, ka);
                        tma_load_2d(a_dst + 8192, pa, fb, am + 64, ka);
                    }
                    if (!B_MN) {
                        tma_load_2d(b_dst, pb, fb, kbk, bn);
                    } else {
                        for (int b = 0; b < g.BN / 64; ++b) tma_load_2d(b_dst + 8192 * b, pb, fb, bn + 64 * b, kbk);
                    }
                    issued_mask |= 1u << stage;
                    issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
                // Let every load already issued land before the CTA retires (a wait
                // of its own, bounded, that the raised abort flag does not cut short).
                volatile int no_abort = 0;
                for (int s = 0; s < S; ++s)
                    if (issued_mask & (1u << s))
                        (void)mbar_wait(full0 + 8 * s, (issued_parity >> s) & 1u, &no_abort);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            // ---------------- MMA issuer ----------------
            const uint32_t idesc = idesc_bf16_f32((uint32_t)g.BN, A_MN, B_MN);
            int stage = 0;
            uint32_t phase = 0;
            int it = 0;
            bool ok = true;
            for (int w = blockIdx.x; w < nwork && ok; w += gridDim.x, ++it) {
                const Work wi = work_item(g, w, g.tiles_m);
                const int kb0 = wi.kb0, kb1 = wi.kb1;
                const int acc = it & 1;
                if (!mbar_wait(tempty0 + 8 * acc, (((uint32_t)it >> 1) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * g.BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(sA + (size_t)stage * kABytes);
                    const uint32_t b_addr = smem_u32(sB + (size_t)stage * b_bytes);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t ad = A_MN ? smem_desc_sw128(a_addr + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? smem_desc_sw128(b_addr + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(b_addr + kk * 32, 16, 1024);
                        umma_bf16(d_tmem, ad, bd, idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(empty0 + 8 * stage);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                umma_commit(tfull0 + 8 * acc);
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
            }
            // Drain: every MMA issued by this thread completes before TMEM is
            // freed (bounded wait; on the normal path they are long done).
            umma_commit(drain0);
            volatile int no_abort = 0;
            if (!mbar_wait(drain0, 0u, &no_abort)) record_error(g.status, ATTT_ERR_TIMEOUT);
        }
    } else {
        // ---------------- epilogue (warps 2..5) ----------------
        griddep_wait();  // what the epilogue reads or overwrites may come from the previous grid
        const int q = warp & 3;
        const int row = q * 32 + lane;
        F32Stage fst{smem_u32(sE) + (uint32_t)q * 8192u, smem_u32(sE) + 32768u + (uint32_t)q * 16u, 0u};
        uint32_t bec = 0;  // EPI_BF16 boxes stored by this warp
        int it = 0;
        for (int w = blockIdx.x; w < nwork; w += gridDim.x, ++it) {
            const Work wi = work_item(g, w, g.tiles_m);
            const int acc = it & 1;
            const uint32_t par = ((uint32_t)it >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull0 + 8 * acc, par, abort_flag) ? 1 : 0;
            // one decision for all four epilogue warps
            ok = named_barrier_and(1, 128, __shfl_sync(0xffffffffu, ok, 0));
            if (!ok) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
            (void)mbar_try_wait(tfull0 + 8 * acc, par);  // per-thread acquire of the completed phase
            tc_fence_after();
            const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * g.BN);
            if constexpr (EPI == EPI_F32_ACC) {
                if (wi.piece >= 0) {
                    epilogue_piece_f32_acc(g, wi, wi.tm * 128, 0, 1, row, taddr, &tmC, fst, abort_flag);
                } else {
                    const int gm = wi.tm * 128 + row;
                    const int n_base = wi.tn * g.BN;
                    f32_tile_store(g, &tmC, fst, lane, gm - lane, acc_row(g.ep, gm, gm < g.M), n_base,
                                   min(g.N, n_base + g.BN), abort_flag,
                                   [&](int c, float(&v)[32]) { tmem_ld_x32(taddr + (uint32_t)c, v); });
                }
            } else if constexpr (EPI == EPI_BF16) {
                const int gm = wi.tm * 128 + row;
                bf16_tile_store(g, &tmC, smem_u32(sE) + (uint32_t)q * 4096u, bec, lane, gm - lane, wi.tn * g.BN,
                                min(g.N, (wi.tn + 1) * g.BN), taddr);
            } else {
                epilogue_tile<EPI>(g, wi.tm * 128, wi.tn, row, taddr, &tmC, smem_u32(sE) + (uint32_t)q * 4096u);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
        }
        // every TMA store of the epilogue has landed before the CTA retires
        if constexpr (EPI == EPI_CE_EXP || EPI == EPI_F32_ACC || EPI == EPI_BF16) {
            if (lane == 0) bulk_wait<0>();
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem_base, g.tmem_cols);
}

// ---------------------------------------------------------------------------
// The CTA-pair kernel: one 256 x BN accumulator tile per cluster of 2 CTAs
// (tcgen05 cta_group::2).  Each CTA holds 128 rows of A and BN/2 rows of B
// per stage and 128 rows of the accumulator; the even CTA issues the MMAs,
// which read both CTAs' shared memory, and multicasts its commits to both
// CTAs.  Both CTAs' TMA loads complete on the even CTA's stage barrier; both
// CTAs' epilogues release the accumulator to the even CTA.  Per SM this moves
// a third less shared-memory traffic per FLOP than the single-CTA kernel.
// ---------------------------------------------------------------------------

template <int EPI, bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kGemmPairThreads, 1)
    tc_gemm_pair_kernel(const __grid_constant__ CUtensorMap tmA, const __grid_constant__ CUtensorMap tmB,
                   const __grid_constant__ CUtensorMap tmC, const __grid_constant__ CUtensorMap tmA2,
                   const __grid_constant__ CUtensorMap tmB2, const GemmArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = g.stages;
    const int BNh = g.BN / 2;  // B rows held by this CTA
    const uint32_t b_bytes = gemm_b_stage_bytes(BNh);
    static_assert(EPI != EPI_KL || (!A_MN && !B_MN), "EPI_KL: K-major operands");
    constexpr uint32_t a_bytes = kABytes;
    uint8_t *sA = smem;
    uint8_t *sB = smem + (size_t)S * a_bytes;
    uint8_t *sE = sB + (size_t)S * b_bytes;  // 1024-byte aligned: b_bytes is a multiple of 2048
    uint64_t *bars = reinterpret_cast<uint64_t *>(sE + g.e_stage_bytes);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = smem_u32(bars + S);
    const uint32_t tfull0 = smem_u32(bars + 2 * S);
    const uint32_t tempty0 = smem_u32(bars + 2 * S + 2);
    const uint32_t drain0 = smem_u32(bars + 2 * S + 4);
    uint32_t *tmem_slot = reinterpret_cast<uint32_t *>(bars + 2 * S + 5);
    volatile int *abort_flag = reinterpret_cast<volatile int *>(tmem_slot + 1);

    const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
    const uint32_t rank = cluster_ctarank();
    const bool leader = rank == 0;

    if (threadIdx.x == 0) {
        for (int s = 0; s < S; ++s) {
            mbar_init(full0 + 8 * s, 1);
            mbar_init(empty0 + 8 * s, 1);
        }
        for (int a = 0; a < 2; ++a) {
            mbar_init(tfull0 + 8 * a, 1);
            mbar_init(tempty0 + 8 * a, 8);
        }
        griddep_launch_dependents();
        mbar_init(drain0, 1);
        if (EPI == EPI_F32_ACC)
            for (int b = 0; b < 8; ++b) mbar_init(smem_u32(sE) + 32768u + 8u * b, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&tmA);
        tma_prefetch_desc(&tmB);
        if (g.kb_split < g.kb_total) {
            tma_prefetch_desc(&tmA2);
            tma_prefetch_desc(&tmB2);
        }
    }
    cluster_sync();  // both CTAs' barriers exist before any cross-CTA signal
    if (warp == 1) {
        tmem_alloc_pair(smem_u32(tmem_slot), g.tmem_cols);
        tmem_relinquish_pair();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    const int tiles_m2 = (g.tiles_m + 1) / 2;
    const int nwork = work_count(g, tiles_m2);
    const int cid = blockIdx.x >> 1, ncl = gridDim.x >> 1;
    const uint32_t lead_full0 = mapa_shared(full0, 0);
    const uint32_t lead_tempty0 = mapa_shared(tempty0, 0);

    if (warp == 0 || warp == 6) {
        if (lane == 0) {
            // ---------------- TMA producers (both CTAs; warp 0 even, warp 6 odd stages) ----------------
            if (!g.operands_ready) griddep_wait();
            const uint32_t pid = warp == 0 ? 0u : 1u;  // this producer's stages: pos % 2 == pid
            uint32_t pos = 0;
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;  // leader: stages whose bytes it expects
            bool ok = true;
            for (int w = cid; w < nwork && ok; w += ncl) {
                const Work wi = work_item(g, w, tiles_m2);
                // EPI_KL: 64 rows of A and the same 64 rows of A2 per CTA
                const int arow0 = EPI == EPI_KL ? wi.tm * 128 + 64 * (int)rank : wi.tm * 256 + 128 * (int)rank;
                const int brow0 = wi.tn * g.BN + BNh * (int)rank;
                for (int kb = wi.kb0; kb < wi.kb1; ++kb) {
                    if (((pos++) & 1u) != pid) {
                        if (++stage == S) { stage = 0; phase ^= 1u; }
                        continue;
                    }
                    if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) { ok = false; break; }
                    if (leader) {
                        mbar_arrive_expect_tx(full0 + 8 * stage, 2u * (a_bytes + b_bytes));
                        issued_mask |= 1u << stage;
                        issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    }
                    const uint32_t fb = lead_full0 + 8 * stage;
                    const uint32_t a_dst = smem_u32(sA + (size_t)stage * a_bytes);
                    const uint32_t b_dst = smem_u32(sB + (size_t)stage * b_bytes);
                    // K block kb of the first pair, or K block kb - kb_split of the second
                    const bool sec = kb >= g.kb_split;
                    const CUtensorMap *pa = sec ? &tmA2 : &tmA;
                    const CUtensorMap *pb = sec ? &tmB2 : &tmB;
                    const int ka = sec ? (kb - g.kb_split) * 64 : g.a_k_off + kb * 64;
                    const int kbk = sec ? (kb - g.kb_split) * 64 : g.b_k_off + kb * 64;
                    const int arow = (sec ? 0 : g.a_m_off) + arow0;
                    const int brow = (sec ? 0 : g.b_n_off) + brow0;
                    if constexpr (EPI == EPI_KL) {
                        tma_load_2d_pair(a_dst, &tmA, fb, ka, arow0);          // rows 0-63: h_p
                        tma_load_2d_pair(a_dst + 8192, &tmA2, fb, ka, arow0);  // rows 64-127: h_q
                    } else if (!A_MN) {
                        tma_load_2d_pair(a_dst, pa, fb, ka, arow);
                    } else {
                        tma_load_2d_pair(a_dst, pa, fb, arow, ka);
                        tma_load_2d_pair(a_dst + 8192, pa, fb, arow + 64, ka);
                    }
                    if (!B_MN) {
                        tma_load_2d_pair(b_dst, pb, fb, kbk, brow);
                    } else {
                        for (int b = 0; b < BNh / 64; ++b) tma_load_2d_pair(b_dst + 8192 * b, pb, fb, brow + 64 * b, kbk);
                    }
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
                // The pair's loads of every stage the leader expects land on its barrier:
                // wait (bounded, a flag of its own) for them before the pair retires.
                volatile int no_abort = 0;
                for (int s = 0; s < S; ++s)
                    if (issued_mask & (1u << s))
                        (void)mbar_wait(full0 + 8 * s, (issued_parity >> s) & 1u, &no_abort);
            }
        }
    } else if (warp == 1) {
        if (lane == 0 && leader) {
            // ---------------- MMA issuer (even CTA) ----------------
            const uint32_t idesc = idesc_bf16_f32((uint32_t)g.BN, A_MN, B_MN, 256);
            int stage = 0;
            uint32_t phase = 0;
            int it = 0;
            bool ok = true;
            for (int w = cid; w < nwork && ok; w += ncl, ++it) {
                const Work wi = work_item(g, w, tiles_m2);
                const int kb0 = wi.kb0, kb1 = wi.kb1;
                const int acc = it & 1;
                if (!mbar_wait(tempty0 + 8 * acc, (((uint32_t)it >> 1) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * g.BN);
                for (int kb = kb0; kb < kb1; ++kb) {
                    if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(sA + (size_t)stage * a_bytes);
                    const uint32_t b_addr = smem_u32(sB + (size_t)stage * b_bytes);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t ad = A_MN ? smem_desc_sw128(a_addr + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                        const uint64_t bd = B_MN ? smem_desc_sw128(b_addr + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(b_addr + kk * 32, 16, 1024);
                        umma_bf16_pair(d_tmem, ad, bd, idesc, (kb > kb0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit_pair(empty0 + 8 * stage, 3);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                umma_commit_pair(tfull0 + 8 * acc, 3);
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
            }
            umma_commit_pair(drain0, 1);
            volatile int no_abort = 0;
            if (!mbar_wait(drain0, 0u, &no_abort)) record_error(g.status, ATTT_ERR_TIMEOUT);
        }
    } else if (warp >= 2 && warp <= 5) {
        // ---------------- epilogue (warps 2..5, both CTAs) ----------------
        griddep_wait();  // what the epilogue reads or overwrites may come from the previous grid
        const int q = warp & 3;
        const int row = q * 32 + lane;
        F32Stage fst{smem_u32(sE) + (uint32_t)q * 8192u, smem_u32(sE) + 32768u + (uint32_t)q * 16u, 0u};
        uint32_t bec = 0;  // EPI_BF16 boxes stored by this warp
        uint32_t kl_ck = 0;  // EPI_KL chunks handed over by this warp pair
        int it = 0;
        for (int w = cid; w < nwork; w += ncl, ++it) {
            const Work wi = work_item(g, w, tiles_m2);
            const int acc = it & 1;
            const uint32_t par = ((uint32_t)it >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull0 + 8 * acc, par, abort_flag) ? 1 : 0;
            // one decision for all four epilogue warps
            ok = named_barrier_and(1, 128, __shfl_sync(0xffffffffu, ok, 0));
            if (!ok) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
            (void)mbar_try_wait(tfull0 + 8 * acc, par);
            tc_fence_after();
            const uint32_t taddr = tmem_base + ((uint32_t)(q * 32) << 16) + (uint32_t)(acc * g.BN);
            const int gm_base = wi.tm * 256 + 128 * (int)rank;
            if constexpr (EPI == EPI_KL) {
                epilogue_kl(g, wi.tm * 128 + 64 * (int)rank, wi.tn, q, lane, taddr, reinterpret_cast<float *>(sE),
                            kl_ck);
            } else if constexpr (EPI == EPI_F32_ACC) {
                if (wi.piece >= 0) {
                    epilogue_piece_f32_acc(g, wi, gm_base, (int)rank, 2, row, taddr, &tmC, fst, abort_flag);
                } else {
                    const int gm = gm_base + row;
                    const int n_base = wi.tn * g.BN;
                    f32_tile_store(g, &tmC, fst, lane, gm - lane, acc_row(g.ep, gm, gm < g.M), n_base,
                                   min(g.N, n_base + g.BN), abort_flag,
                                   [&](int c, float(&v)[32]) { tmem_ld_x32(taddr + (uint32_t)c, v); });
                }
            } else if constexpr (EPI == EPI_BF16) {
                bf16_tile_store(g, &tmC, smem_u32(sE) + (uint32_t)q * 4096u, bec, lane, gm_base + 32 * q,
                                wi.tn * g.BN, min(g.N, (wi.tn + 1) * g.BN), taddr);
            } else {
                epilogue_tile<EPI>(g, gm_base, wi.tn, row, taddr, &tmC, smem_u32(sE) + (uint32_t)q * 4096u);
            }
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive_cluster(lead_tempty0 + 8 * acc);
        }
        // every TMA store of the epilogue has landed before the CTA retires
        if constexpr (EPI == EPI_CE_EXP || EPI == EPI_F32_ACC || EPI == EPI_BF16) {
            if (lane == 0) bulk_wait<0>();
        }
    }

    tc_fence_before();
    cluster_sync();  // no CTA leaves while the pair's MMAs or signals are in flight
    tc_fence_after();
    if (warp == 1) tmem_dealloc_pair(tmem_base, g.tmem_cols);
}

}  // namespace attt
