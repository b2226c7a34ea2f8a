// lora_fused.cuh -- the LoRA adapter gradients of one group of projections
// that share an input x, in one persistent tcgen05 launch (Appendix C's
// adapter y = x W0 + s (x A) B; the gradient of Eq. 2):
//
//   pass 1   u = x [A_0 | A_1 | ...]   and   v_p = dy_p B_p^T        (bf16, u^T / v^T)
//   pass 2   dA_p = s x^T v_p          and   dB_p = s u_p^T dy_p      (fp32)
//
// Pass 2 reduces over the rows of x and dy that pass 1 reduced along, so a
// row block's x and dy are read by both.  The rows are cut into chunks small
// enough that two of them sit in L2 together (about 24 MiB each), and the
// work runs in the order
//
//   P1(0), P1(1), P2(0), P1(2), P2(1), ..., P1(C-1), P2(C-2), P2(C-1)
//
// so that pass 2 of a chunk re-reads its x and dy from L2 shortly after
// pass 1 brought them in from HBM, while pass 1 of the next chunk keeps HBM
// busy.  Work items are handed out in that order by one atomic counter, so a
// CTA only ever waits for items handed out before its own (never for a CTA
// that has not started), and the CTAs that finish early take the next items.
//
// Items:
//   P1 item  one 128-row tile of u or v_p over a piece of K (din or dout_p);
//            a tile cut into several pieces has each piece store an fp32
//            partial, and the piece that arrives last (ticket) sums them in
//            piece order and writes the tile as bf16.  The writer of a tile
//            bumps the chunk's done counter.
//   P2 item  one 128-row tile of dA (rows of din) or dB_p (rows of dout_p)
//            over one chunk's rows.  It starts once the chunk's pass-1 tiles
//            are all written (bounded wait on the done counter), adds the
//            running sum of the earlier chunks (an fp32 slot per tile,
//            folded in chunk order behind a per-tile flag) and, for the last
//            chunk, writes s times the sum.  The order of every sum is fixed,
//            so the gradients are the same bits whichever CTA runs an item.
//
// The pipeline is that of the other contraction kernels: warp 0 is the TMA
// producer (and takes the items), warp 1 issues the MMAs, warps 2-5 are the
// epilogue; the item of every step travels from the producer to the others
// through a ring in shared memory.  Every wait is bounded.
#pragma once

#include "tc_gemm.cuh"

namespace attt {

constexpr int kFusedRing = 4;  // item ids in flight between the producer and the other roles

struct FusedMaps {
    CUtensorMap x_k;   // x [L, din], box {64, 128}: pass-1 A (K-major, K = din)
    CUtensorMap x_mn;  // x,          box {64, 64}:  pass-2 A (MN-major, M = din, K = rows)
    CUtensorMap at;    // A^T padded [Nu, din], box {64, BNu}: the B operand of u
    CUtensorMap ut;    // u^T [Nu, L] (row pitch Lp), box {64, rpad}: the B operand of dB_p
    CUtensorMap vt;    // v^T [Nu, L], box {64, BNu}: the B operand of dA
    CUtensorMap dy_k[kMaxProj];   // dy_p [L, dout_p], box {64, 128}
    CUtensorMap dy_mn[kMaxProj];  // dy_p, box {64, 64}
    CUtensorMap bt[kMaxProj];     // B_p padded [rpad, dout_p], box {64, rpad}
};

struct FusedArgs {
    int P, r, rpad, Nu, BNu, tn_u;
    int L, Lp, din;
    int dout[kMaxProj];
    int Lc, C, mt_full, mt_last;  // chunk rows (multiple of 128), chunks, row tiles of a full / the last chunk
    int kpiece;                   // 64-deep K blocks per pass-1 piece
    int kb_u, np_u;               // K blocks and pieces of u
    int kb_v[kMaxProj], np_v[kMaxProj];
    int tm_dA;                    // 128-row tiles of din
    int tm_dB[kMaxProj];          // 128-row tiles of dout_p
    int t2_dB[kMaxProj];          // first pass-2 tile id of dB_p
    int n1_full, n1_last, n2;     // items of P1 (full chunk, last chunk) and of P2 (any chunk)
    int t1_full;                  // pass-1 tiles of a full chunk
    int total_items;
    int stages;
    uint32_t b_stage_bytes;       // BN max x 128 bytes
    uint32_t acc_cols;            // TMEM columns between the two accumulators
    float scale;
    __nv_bfloat16 *uT, *vT;       // [Nu, Lp] each
    float *dA[kMaxProj], *dB[kMaxProj];
    unsigned int *head;           // next item to hand out
    unsigned int *p1done;         // [C] pass-1 tiles written per chunk
    unsigned int *tickets;        // [C * t1_full] pieces arrived per pass-1 tile
    unsigned int *flags;          // [tiles of pass 2] chunks folded into each pass-2 sum
    float *slots;                 // pass-1 partials: chunk c at c * slot_chunk floats
    int64_t slot_chunk, slot_u;
    int64_t slot_v[kMaxProj];
    float *acc;                   // pass-2 running sums (C > 1)
    int64_t acc_dA;
    int64_t acc_dB[kMaxProj];
    int *status;
};

struct FusedItem {
    int phase;  // 1 or 2
    int c;      // chunk
    int q;      // 0: u / dA; 1 + p: v_p / dB_p
    int tn, mt, j, np;
    int kb0, kb1;  // K blocks [kb0, kb1) (pass 2: row blocks of 64)
    int BN;        // N of this item's MMAs
};

__device__ __forceinline__ int fused_mt(const FusedArgs &g, int c) { return c == g.C - 1 ? g.mt_last : g.mt_full; }

__device__ __forceinline__ void fused_decode_p1(const FusedArgs &g, int c, int loc, FusedItem &it) {
    const int mtc = fused_mt(g, c);
    it.phase = 1;
    it.c = c;
    const int nu = g.tn_u * mtc * g.np_u;
    if (loc < nu) {
        const int per = mtc * g.np_u;
        it.q = 0;
        it.np = g.np_u;
        it.tn = loc / per;
        const int rem = loc - it.tn * per;
        it.mt = rem / g.np_u;
        it.j = rem - it.mt * g.np_u;
        it.kb0 = it.j * g.kpiece;
        it.kb1 = min(g.kb_u, it.kb0 + g.kpiece);
        it.BN = min(g.BNu, g.Nu - it.tn * g.BNu);
        return;
    }
    loc -= nu;
    int p = 0;
    while (p + 1 < g.P && loc >= mtc * g.np_v[p]) {
        loc -= mtc * g.np_v[p];
        ++p;
    }
    it.q = 1 + p;
    it.np = g.np_v[p];
    it.tn = 0;
    it.mt = loc / it.np;
    it.j = loc - it.mt * it.np;
    it.kb0 = it.j * g.kpiece;
    it.kb1 = min(g.kb_v[p], it.kb0 + g.kpiece);
    it.BN = g.rpad;
}

__device__ __forceinline__ void fused_decode_p2(const FusedArgs &g, int c, int loc, FusedItem &it) {
    it.phase = 2;
    it.c = c;
    it.j = 0;
    it.np = 1;
    const int row0 = c * g.Lc;
    const int rows = min(g.Lc, g.L - row0);
    it.kb0 = row0 / 64;
    it.kb1 = (row0 + rows + 63) / 64;
    const int na = g.tn_u * g.tm_dA;
    if (loc < na) {
        it.q = 0;
        it.tn = loc / g.tm_dA;
        it.mt = loc - it.tn * g.tm_dA;
        it.BN = min(g.BNu, g.Nu - it.tn * g.BNu);
        return;
    }
    loc -= na;
    int p = 0;
    while (p + 1 < g.P && loc >= g.tm_dB[p]) {
        loc -= g.tm_dB[p];
        ++p;
    }
    it.q = 1 + p;
    it.tn = 0;
    it.mt = loc;
    it.BN = g.rpad;
}

// The item handed out as number `id`; false past the last one.
__device__ __forceinline__ bool fused_decode(const FusedArgs &g, unsigned int id, FusedItem &it) {
    if (id >= (unsigned int)g.total_items) return false;
    const int x0 = (int)id;
    if (g.C == 1) {
        if (x0 < g.n1_last) fused_decode_p1(g, 0, x0, it);
        else fused_decode_p2(g, 0, x0 - g.n1_last, it);
        return true;
    }
    if (x0 < g.n1_full) {
        fused_decode_p1(g, 0, x0, it);
        return true;
    }
    int x = x0 - g.n1_full;
    const int S = g.n1_full + g.n2;  // group k in [1, C - 2]: P1(k), then P2(k - 1)
    const int mid = (g.C - 2) * S;
    if (x < mid) {
        const int k = 1 + x / S;
        const int y = x - (k - 1) * S;
        if (y < g.n1_full) fused_decode_p1(g, k, y, it);
        else fused_decode_p2(g, k - 1, y - g.n1_full, it);
        return true;
    }
    x -= mid;
    if (x < g.n1_last + g.n2) {  // group C - 1
        if (x < g.n1_last) fused_decode_p1(g, g.C - 1, x, it);
        else fused_decode_p2(g, g.C - 2, x - g.n1_last, it);
        return true;
    }
    fused_decode_p2(g, g.C - 1, x - g.n1_last - g.n2, it);
    return true;
}

// Pass-1 tiles of chunk c.
__device__ __forceinline__ unsigned int fused_t1(const FusedArgs &g, int c) {
    return (unsigned int)((g.tn_u + g.P) * fused_mt(g, c));
}

// Final dA / dB columns [col0, col0 + 16) of tile row m: s * v.
__device__ __forceinline__ void fused_store_grad(const FusedArgs &g, const FusedItem &it, int m, int col0,
                                                 const float (&v)[16]) {
    if (it.q == 0) {
        // columns of [dA_0 | dA_1 | ...] (rpad each, a multiple of 16)
        const int n0 = it.tn * g.BNu + col0;
        const int pp = n0 / g.rpad, cc0 = n0 - pp * g.rpad;
        float *o = g.dA[pp] + (int64_t)m * g.r + cc0;
        if (cc0 + 16 <= g.r && (g.r & 3) == 0 && (reinterpret_cast<uintptr_t>(o) & 15) == 0) {
#pragma unroll
            for (int i = 0; i < 16; i += 4)
                *reinterpret_cast<float4 *>(o + i) =
                    make_float4(g.scale * v[i], g.scale * v[i + 1], g.scale * v[i + 2], g.scale * v[i + 3]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (cc0 + i < g.r) o[i] = g.scale * v[i];
        }
    } else {
        const int p = it.q - 1;
        float *o = g.dB[p] + m;
        const int64_t ld = g.dout[p];
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if (col0 + i < g.r) o[(int64_t)(col0 + i) * ld] = g.scale * v[i];
    }
}

// The epilogue of one item on the four epilogue warps (thread = tile row).
// Returns false if a bounded wait ran out.
__device__ __forceinline__ bool fused_epilogue(const FusedArgs &g, const FusedItem &it, int row, uint32_t taddr,
                                               volatile int *abort_flag) {
    const int BN = it.BN;
    if (it.phase == 1) {
        const int m = it.c * g.Lc + it.mt * 128 + row;
        const bool rv = m < g.L;
        __nv_bfloat16 *out = it.q == 0 ? g.uT + (int64_t)(it.tn * g.BNu) * g.Lp : g.vT + (int64_t)(it.q - 1) * g.rpad * g.Lp;
        if (it.np == 1) {
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld_x16(taddr + (uint32_t)c0, v);
                if (rv) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) out[(int64_t)(c0 + i) * g.Lp + m] = __float2bfloat16_rn(v[i]);
                }
            }
        } else {
            const int mtc = fused_mt(g, it.c);
            const int t1 = it.q == 0 ? it.tn * mtc + it.mt : (g.tn_u + it.q - 1) * mtc + it.mt;
            const int bna = it.q == 0 ? g.BNu : g.rpad;
            const int64_t slot = (int64_t)128 * bna;
            float *tile_slots = g.slots + (int64_t)it.c * g.slot_chunk + (it.q == 0 ? g.slot_u : g.slot_v[it.q - 1]) +
                                (int64_t)(it.tn * g.mt_full + it.mt) * it.np * slot;
            float4 *mine = reinterpret_cast<float4 *>(tile_slots + (int64_t)it.j * slot) + row;
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float v[16];
                tmem_ld_x16(taddr + (uint32_t)c0, v);
#pragma unroll
                for (int q = 0; q < 4; ++q)
                    __stcg(mine + (c0 / 4 + q) * 128, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
            }
            __threadfence();
            named_barrier_sync(1, 128);
            int last = 0;
            if (row == 0) {
                last = atomicAdd(g.tickets + (int64_t)it.c * g.t1_full + t1, 1u) == (unsigned int)(it.np - 1) ? 1 : 0;
                __threadfence();
            }
            if (!named_barrier_or(1, 128, last)) return true;  // another piece finishes the tile
            for (int c0 = 0; c0 < BN; c0 += 16) {
                float own[16];
                tmem_ld_x16(taddr + (uint32_t)c0, own);
                float s[16];
                // pieces in order, four partials in flight at a time
                for (int j0 = 0; j0 < it.np; j0 += 4) {
                    float4 f[4][4];
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const int j = j0 + b;
                        if (j < it.np && j != it.j) {
                            const float4 *src = reinterpret_cast<const float4 *>(tile_slots + (int64_t)j * slot) + row;
#pragma unroll
                            for (int q = 0; q < 4; ++q) f[b][q] = __ldcg(src + (c0 / 4 + q) * 128);
                        }
                    }
#pragma unroll
                    for (int b = 0; b < 4; ++b) {
                        const int j = j0 + b;
                        if (j >= it.np) break;
#pragma unroll
                        for (int q = 0; q < 4; ++q) {
                            const float4 x = j == it.j ? make_float4(own[4 * q], own[4 * q + 1], own[4 * q + 2], own[4 * q + 3])
                                                       : f[b][q];
                            if (j == 0) {
                                s[4 * q] = x.x; s[4 * q + 1] = x.y; s[4 * q + 2] = x.z; s[4 * q + 3] = x.w;
                            } else {
                                s[4 * q] += x.x; s[4 * q + 1] += x.y; s[4 * q + 2] += x.z; s[4 * q + 3] += x.w;
                            }
                        }
                    }
                }
                if (rv) {
#pragma unroll
                    for (int i = 0; i < 16; ++i) out[(int64_t)(c0 + i) * g.Lp + m] = __float2bfloat16_rn(s[i]);
                }
            }
        }
        // the tile is written: count it for pass 2 of this chunk, whose TMA
        // loads read it
        fence_proxy_async_global();
        __threadfence();
        named_barrier_sync(1, 128);
        if (row == 0) atomicAdd(g.p1done + it.c, 1u);
        return true;
    }

    // pass 2
    const int M = it.q == 0 ? g.din : g.dout[it.q - 1];
    const int m = it.mt * 128 + row;
    const bool rv = m < M;
    const bool first = it.c == 0, last = it.c == g.C - 1;
    const int t2 = it.q == 0 ? it.tn * g.tm_dA + it.mt : g.t2_dB[it.q - 1] + it.mt;
    float4 *accp = nullptr;
    if (g.C > 1) {
        const float *base = it.q == 0 ? g.acc + g.acc_dA + (int64_t)(it.tn * g.tm_dA + it.mt) * 128 * g.BNu
                                      : g.acc + g.acc_dB[it.q - 1] + (int64_t)it.mt * 128 * g.rpad;
        accp = reinterpret_cast<float4 *>(const_cast<float *>(base)) + row;
    }
    if (!first) {
        int ok = 1;
        if (row == 0) ok = wait_counter_geq(g.flags + t2, (unsigned int)it.c, abort_flag) ? 1 : 0;
        if (!named_barrier_and(1, 128, ok)) return false;
    }
    for (int c0 = 0; c0 < BN; c0 += 16) {
        float v[16];
        tmem_ld_x16(taddr + (uint32_t)c0, v);
        if (!first) {
            float4 f[4];
#pragma unroll
            for (int q = 0; q < 4; ++q) f[q] = __ldcg(accp + (c0 / 4 + q) * 128);
#pragma unroll
            for (int q = 0; q < 4; ++q) {
                v[4 * q] = f[q].x + v[4 * q];
                v[4 * q + 1] = f[q].y + v[4 * q + 1];
                v[4 * q + 2] = f[q].z + v[4 * q + 2];
                v[4 * q + 3] = f[q].w + v[4 * q + 3];
            }
        }
        if (!last) {
#pragma unroll
            for (int q = 0; q < 4; ++q)
                __stcg(accp + (c0 / 4 + q) * 128, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
        } else if (rv) {
            fused_store_grad(g, it, m, c0, v);
        }
    }
    if (!last) {
        __threadfence();
        named_barrier_sync(1, 128);
        if (row == 0) st_release_gpu(g.flags + t2, (unsigned int)(it.c + 1));
    }
    return true;
}

__global__ void __launch_bounds__(kGemmThreads, 1)
    lora_fused_kernel(const __grid_constant__ FusedMaps maps, const FusedArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = g.stages;
    uint8_t *sA = smem;
    uint8_t *sB = smem + (size_t)S * kABytes;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + (size_t)S * g.b_stage_bytes);
    const uint32_t full0 = smem_u32(bars);
    const uint32_t empty0 = smem_u32(bars + S);
    const uint32_t tfull0 = smem_u32(bars + 2 * S);
    const uint32_t tempty0 = smem_u32(bars + 2 * S + 2);
    const uint32_t rfull0 = smem_u32(bars + 2 * S + 4);
    const uint32_t rempty0 = smem_u32(bars + 2 * S + 4 + kFusedRing);
    const uint32_t drain0 = smem_u32(bars + 2 * S + 4 + 2 * kFusedRing);
    volatile unsigned int *ring = reinterpret_cast<volatile unsigned int *>(bars + 2 * S + 5 + 2 * kFusedRing);
    uint32_t *tmem_slot = const_cast<uint32_t *>(reinterpret_cast<volatile uint32_t *>(ring + kFusedRing));
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
        for (int i = 0; i < kFusedRing; ++i) {
            mbar_init(rfull0 + 8 * i, 1);
            mbar_init(rempty0 + 8 * i, 5);  // the MMA thread and the four epilogue warps
        }
        griddep_launch_dependents();
        mbar_init(drain0, 1);
        *abort_flag = 0;
        fence_mbar_init();
        tma_prefetch_desc(&maps.x_k);
        tma_prefetch_desc(&maps.x_mn);
        tma_prefetch_desc(&maps.at);
        tma_prefetch_desc(&maps.ut);
        tma_prefetch_desc(&maps.vt);
        for (int p = 0; p < g.P; ++p) {
            tma_prefetch_desc(&maps.dy_k[p]);
            tma_prefetch_desc(&maps.dy_mn[p]);
            tma_prefetch_desc(&maps.bt[p]);
        }
    }
    if (warp == 1) {
        tmem_alloc(smem_u32(tmem_slot), 2 * g.acc_cols);
        tmem_relinquish();
    }
    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    const uint32_t tmem_base = *tmem_slot;

    if (warp == 0) {
        if (lane == 0) {
            griddep_wait();  // the workspace (adapters, counters) comes from the prep grid
            int stage = 0, rs = 0;
            uint32_t phase = 0, rph = 0;
            uint32_t issued_mask = 0, issued_parity = 0;
            bool ok = true;
            unsigned int next = atomicAdd(g.head, 1u);
            while (true) {
                const unsigned int id = next;
                if (!mbar_wait(rempty0 + 8 * rs, rph ^ 1u, abort_flag)) { ok = false; break; }
                ring[rs] = id;
                mbar_arrive(rfull0 + 8 * rs);
                if (++rs == kFusedRing) { rs = 0; rph ^= 1u; }
                FusedItem it;
                if (!fused_decode(g, id, it)) break;
                next = atomicAdd(g.head, 1u);  // in flight while this item's loads issue
                if (it.phase == 2) {
                    // the chunk's u^T and v^T tiles, written by other CTAs
                    if (!wait_counter_geq(g.p1done + it.c, fused_t1(g, it.c), abort_flag)) { ok = false; break; }
                    fence_proxy_async_global();
                }
                const uint32_t tx = kABytes + (uint32_t)(it.phase == 1 ? (it.q == 0 ? g.BNu : g.rpad)
                                                                       : (it.q == 0 ? g.BNu : g.rpad)) * 128u;
                const int row0 = it.c * g.Lc + it.mt * 128;  // pass 1: first row of the tile
                for (int kb = it.kb0; kb < it.kb1; ++kb) {
                    if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) { ok = false; break; }
                    const uint32_t fb = full0 + 8 * stage;
                    mbar_arrive_expect_tx(fb, tx);  // rows and columns past the extents arrive as zeros
                    const uint32_t a_dst = smem_u32(sA + (size_t)stage * kABytes);
                    const uint32_t b_dst = smem_u32(sB + (size_t)stage * g.b_stage_bytes);
                    const int k = kb * 64;
                    if (it.phase == 1) {
                        if (it.q == 0) {
                            tma_load_2d(a_dst, &maps.x_k, fb, k, row0);
                            tma_load_2d(b_dst, &maps.at, fb, k, it.tn * g.BNu);
                        } else {
                            tma_load_2d(a_dst, &maps.dy_k[it.q - 1], fb, k, row0);
                            tma_load_2d(b_dst, &maps.bt[it.q - 1], fb, k, 0);
                        }
                    } else {
                        const CUtensorMap *am = it.q == 0 ? &maps.x_mn : &maps.dy_mn[it.q - 1];
                        tma_load_2d(a_dst, am, fb, it.mt * 128, k);
                        tma_load_2d(a_dst + 8192, am, fb, it.mt * 128 + 64, k);
                        if (it.q == 0) tma_load_2d(b_dst, &maps.vt, fb, k, it.tn * g.BNu);
                        else tma_load_2d(b_dst, &maps.ut, fb, k, (it.q - 1) * g.rpad);
                    }
                    issued_mask |= 1u << stage;
                    issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
                for (int s = 0; s < S; ++s)
                    if (issued_mask & (1u << s)) (void)mbar_wait(full0 + 8 * s, (issued_parity >> s) & 1u, abort_flag);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            int stage = 0, rs = 0, n = 0;
            uint32_t phase = 0, rph = 0;
            bool ok = true;
            while (true) {
                if (!mbar_wait(rfull0 + 8 * rs, rph, abort_flag)) { ok = false; break; }
                const unsigned int id = ring[rs];
                mbar_arrive(rempty0 + 8 * rs);
                if (++rs == kFusedRing) { rs = 0; rph ^= 1u; }
                FusedItem it;
                if (!fused_decode(g, id, it)) break;
                const int acc = n & 1;
                if (!mbar_wait(tempty0 + 8 * acc, (((uint32_t)n >> 1) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)acc * g.acc_cols;
                const bool a_mn = it.phase == 2;
                const uint32_t idesc = idesc_bf16_f32((uint32_t)it.BN, a_mn, false);
                for (int kb = it.kb0; kb < it.kb1; ++kb) {
                    if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    const uint32_t a_addr = smem_u32(sA + (size_t)stage * kABytes);
                    const uint32_t b_addr = smem_u32(sB + (size_t)stage * g.b_stage_bytes);
#pragma unroll
                    for (int kk = 0; kk < 4; ++kk) {
                        const uint64_t ad = a_mn ? smem_desc_sw128(a_addr + kk * 2048, 8192, 1024)
                                                 : smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                        const uint64_t bd = smem_desc_sw128(b_addr + kk * 32, 16, 1024);
                        umma_bf16(d_tmem, ad, bd, idesc, (kb > it.kb0 || kk > 0) ? 1u : 0u);
                    }
                    umma_commit(empty0 + 8 * stage);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
                if (!ok) break;
                umma_commit(tfull0 + 8 * acc);
                ++n;
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
            }
            umma_commit(drain0);
            volatile int no_abort = 0;
            if (!mbar_wait(drain0, 0u, &no_abort)) record_error(g.status, ATTT_ERR_TIMEOUT);
        }
    } else {
        griddep_wait();  // slots, tickets and counters follow the prep grid
        const int qw = warp & 3;
        const int row = qw * 32 + lane;
        int rs = 0, n = 0;
        uint32_t rph = 0;
        while (true) {
            int ok = 1;
            if (lane == 0) ok = mbar_wait(rfull0 + 8 * rs, rph, abort_flag) ? 1 : 0;
            ok = __shfl_sync(0xffffffffu, ok, 0);
            if (!ok) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
            (void)mbar_try_wait(rfull0 + 8 * rs, rph);  // this lane's own acquire of the ring slot
            const unsigned int id = ring[rs];
            __syncwarp();
            if (lane == 0) mbar_arrive(rempty0 + 8 * rs);
            if (++rs == kFusedRing) { rs = 0; rph ^= 1u; }
            FusedItem it;
            if (!fused_decode(g, id, it)) break;
            const int acc = n & 1;
            const uint32_t par = ((uint32_t)n >> 1) & 1u;
            int okt = 1;
            if (lane == 0) okt = mbar_wait(tfull0 + 8 * acc, par, abort_flag) ? 1 : 0;
            okt = named_barrier_and(1, 128, __shfl_sync(0xffffffffu, okt, 0));
            if (!okt) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
            (void)mbar_try_wait(tfull0 + 8 * acc, par);
            tc_fence_after();
            const uint32_t taddr = tmem_base + ((uint32_t)(qw * 32) << 16) + (uint32_t)acc * g.acc_cols;
            const bool done = fused_epilogue(g, it, row, taddr, abort_flag);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
            ++n;
            if (!done) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem_base, 2 * g.acc_cols);
}

}  // namespace attt
