// tc_group.cuh -- grouped tcgen05 contractions: several independent problems
// (own operands, sizes, K split and epilogue) in one persistent launch.
//
// The LoRA gradients are a handful of skinny, HBM-bound contractions (the
// rank on N); launched one by one, each pays a launch, a ramp and a tail
// that cost more than streaming its operands.  Grouping runs every
// contraction of a pass in one launch.  The pipeline is the single-CTA one
// of tc_gemm.cuh (TMA producer warp, MMA warp, four epilogue warps, two TMEM
// accumulators); only the tile -> problem decode and the per-problem tensor
// maps and epilogue differ.  All problems of a group share BN and the operand
// majors.
#pragma once

#include "tc_gemm.cuh"

namespace attt {

constexpr int kMaxGroup = kMaxProj + 1;

struct GroupProblem {
    int M, N;
    int tiles_m, tiles_n, splits, kb_per_split, kb_total;
    int a_m_off, a_k_off, b_n_off, b_k_off;
    int tile_begin;  // first group-wide tile index of this problem
    int epi;         // EPI_ATOMIC_T or EPI_ATOMIC_N
    EpiParams ep;
};

struct GroupMaps {
    CUtensorMap a[kMaxGroup];
    CUtensorMap b[kMaxGroup];
};

struct GroupArgs {
    int nprob, total_tiles;
    int BN, stages;
    int kbs;  // 64-deep K blocks per pipeline stage (each row is fetched in kbs x 128 B runs)
    uint32_t tmem_cols;
    int *status;
    GroupProblem prob[kMaxGroup];
};

__device__ __forceinline__ void decode_group(const GroupArgs &g, int t, int &q, int &tm, int &tn, int &split) {
    q = 0;
    while (q + 1 < g.nprob && t >= g.prob[q + 1].tile_begin) ++q;
    const GroupProblem &p = g.prob[q];
    const int local = t - p.tile_begin;
    const int per = p.tiles_m * p.tiles_n;
    split = local / per;
    const int rem = local - split * per;
    tn = rem / p.tiles_m;
    tm = rem - tn * p.tiles_m;
}

// A GemmArgs view of one problem, for the shared epilogues.
__device__ __forceinline__ GemmArgs group_view(const GroupArgs &g, const GroupProblem &p) {
    GemmArgs v{};
    v.M = p.M;
    v.N = p.N;
    v.BN = g.BN;
    v.tiles_m = p.tiles_m;
    v.tiles_n = p.tiles_n;
    v.splits = p.splits;
    v.status = g.status;
    v.ep = p.ep;
    return v;
}

// EPI_ATOMIC_T epilogue with an optional bf16 finalize: after this split's
// atomics, the split that takes the tile's last ticket converts the tile's
// fp32 sums (out[n, m]) to bf16 (out16[n, m]).  No CTA waits for another.
__device__ __forceinline__ void group_atomic_t_tile(const GemmArgs &v, int gm_base, int tm, int tn, int row,
                                                    uint32_t taddr) {
    epilogue_tile<EPI_ATOMIC_T>(v, gm_base, tn, row, taddr);
    const EpiParams &ep = v.ep;
    if (!ep.out16) return;
    __threadfence();
    named_barrier_sync(1, 128);
    __shared__ int s_last;
    if (threadIdx.x == 64) {
        unsigned int *tk = ep.tickets + (tm + tn * v.tiles_m);
        s_last = atomicAdd(tk, 1u) == (unsigned)(v.splits - 1);
        if (s_last) *tk = 0u;
    }
    named_barrier_sync(1, 128);
    if (!s_last) return;
    __threadfence();
    const int gm = gm_base + row;
    if (gm >= v.M) return;
    const int n_base = tn * v.BN;
    const int n_end = min(v.N, n_base + v.BN);
    for (int col = n_base; col < n_end; ++col) {
        const float x = __ldcg(ep.out + (int64_t)col * ep.out_ld + gm);
        ep.out16[(int64_t)col * ep.out_ld + gm] = __float2bfloat16_rn(x);
    }
}

template <bool A_MN, bool B_MN>
__global__ void __launch_bounds__(kGemmThreads, 1)
    tc_gemm_group_kernel(const __grid_constant__ GroupMaps maps, const GroupArgs g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = g.stages;
    const int KBS = g.kbs;
    const uint32_t a1 = kABytes, b1 = gemm_b_stage_bytes(g.BN);  // one K block
    const uint32_t kABytesS = a1 * KBS;
    const uint32_t b_bytes = b1 * KBS;
    uint8_t *sA = smem;
    uint8_t *sB = smem + (size_t)S * kABytesS;
    uint64_t *bars = reinterpret_cast<uint64_t *>(sB + (size_t)S * b_bytes);
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
        mbar_init(drain0, 1);
        *abort_flag = 0;
        fence_mbar_init();
        for (int q = 0; q < g.nprob; ++q) {
            tma_prefetch_desc(&maps.a[q]);
            tma_prefetch_desc(&maps.b[q]);
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

    if (warp == 0) {
        if (lane == 0) {
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < g.total_tiles && ok; t += gridDim.x) {
                int q, tm, tn, split;
                decode_group(g, t, q, tm, tn, split);
                const GroupProblem &p = g.prob[q];
                const CUtensorMap *ta = &maps.a[q];
                const CUtensorMap *tb = &maps.b[q];
                const int kb0 = split * p.kb_per_split;
                const int kb1 = min(p.kb_total, kb0 + p.kb_per_split);
                for (int kb = kb0; kb < kb1; kb += KBS) {
                    if (!mbar_wait(empty0 + 8 * stage, phase ^ 1u, abort_flag)) { ok = false; break; }
                    const uint32_t fb = full0 + 8 * stage;
                    mbar_arrive_expect_tx(fb, kABytesS + b_bytes);  // blocks past K arrive as zeros
                    for (int j = 0; j < KBS; ++j) {
                        const uint32_t a_dst = smem_u32(sA + (size_t)stage * kABytesS + (size_t)j * a1);
                        const uint32_t b_dst = smem_u32(sB + (size_t)stage * b_bytes + (size_t)j * b1);
                        const int k = (kb + j) * 64;
                        if (!A_MN) {
                            tma_load_2d(a_dst, ta, fb, p.a_k_off + k, p.a_m_off + tm * 128);
                        } else {
                            tma_load_2d(a_dst, ta, fb, p.a_m_off + tm * 128, p.a_k_off + k);
                            tma_load_2d(a_dst + 8192, ta, fb, p.a_m_off + tm * 128 + 64, p.a_k_off + k);
                        }
                        if (!B_MN) {
                            tma_load_2d(b_dst, tb, fb, p.b_k_off + k, p.b_n_off + tn * g.BN);
                        } else {
                            for (int b = 0; b < g.BN / 64; ++b)
                                tma_load_2d(b_dst + 8192 * b, tb, fb, p.b_n_off + tn * g.BN + 64 * b, p.b_k_off + k);
                        }
                    }
                    issued_mask |= 1u << stage;
                    issued_parity = (issued_parity & ~(1u << stage)) | (phase << stage);
                    if (++stage == S) { stage = 0; phase ^= 1u; }
                }
            }
            if (!ok) {
                *abort_flag = 1;
                record_error(g.status, ATTT_ERR_TIMEOUT);
                for (int s = 0; s < S; ++s)
                    if (issued_mask & (1u << s))
                        (void)mbar_wait(full0 + 8 * s, (issued_parity >> s) & 1u, abort_flag);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32((uint32_t)g.BN, A_MN, B_MN);
            int stage = 0;
            uint32_t phase = 0;
            int it = 0;
            bool ok = true;
            for (int t = blockIdx.x; t < g.total_tiles && ok; t += gridDim.x, ++it) {
                int q, tm, tn, split;
                decode_group(g, t, q, tm, tn, split);
                const GroupProblem &p = g.prob[q];
                const int kb0 = split * p.kb_per_split;
                const int kb1 = min(p.kb_total, kb0 + p.kb_per_split);
                const int acc = it & 1;
                if (!mbar_wait(tempty0 + 8 * acc, (((uint32_t)it >> 1) & 1u) ^ 1u, abort_flag)) { ok = false; break; }
                tc_fence_after();
                const uint32_t d_tmem = tmem_base + (uint32_t)(acc * g.BN);
                for (int kb = kb0; kb < kb1; kb += KBS) {
                    if (!mbar_wait(full0 + 8 * stage, phase, abort_flag)) { ok = false; break; }
                    tc_fence_after();
                    for (int j = 0; j < KBS; ++j) {
                        const uint32_t a_addr = smem_u32(sA + (size_t)stage * kABytesS + (size_t)j * a1);
                        const uint32_t b_addr = smem_u32(sB + (size_t)stage * b_bytes + (size_t)j * b1);
#pragma unroll
                        for (int kk = 0; kk < 4; ++kk) {
                            const uint64_t ad = A_MN ? smem_desc_sw128(a_addr + kk * 2048, 8192, 1024)
                                                     : smem_desc_sw128(a_addr + kk * 32, 16, 1024);
                            const uint64_t bd = B_MN ? smem_desc_sw128(b_addr + kk * 2048, 8192, 1024)
                                                     : smem_desc_sw128(b_addr + kk * 32, 16, 1024);
                            umma_bf16(d_tmem, ad, bd, idesc, (kb > kb0 || j > 0 || kk > 0) ? 1u : 0u);
                        }
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
            umma_commit(drain0);
            volatile int no_abort = 0;
            if (!mbar_wait(drain0, 0u, &no_abort)) record_error(g.status, ATTT_ERR_TIMEOUT);
        }
    } else {
        const int qw = warp & 3;
        const int row = qw * 32 + lane;
        int it = 0;
        for (int t = blockIdx.x; t < g.total_tiles; t += gridDim.x, ++it) {
            int q, tm, tn, split;
            decode_group(g, t, q, tm, tn, split);
            const int acc = it & 1;
            const uint32_t par = ((uint32_t)it >> 1) & 1u;
            int ok = 1;
            if (lane == 0) ok = mbar_wait(tfull0 + 8 * acc, par, abort_flag) ? 1 : 0;
            ok = named_barrier_and(1, 128, __shfl_sync(0xffffffffu, ok, 0));
            if (!ok) {
                if (lane == 0) { *abort_flag = 1; record_error(g.status, ATTT_ERR_TIMEOUT); }
                break;
            }
            (void)mbar_try_wait(tfull0 + 8 * acc, par);
            tc_fence_after();
            const uint32_t taddr = tmem_base + ((uint32_t)(qw * 32) << 16) + (uint32_t)(acc * g.BN);
            const GemmArgs v = group_view(g, g.prob[q]);
            if (g.prob[q].epi == EPI_ATOMIC_N)
                epilogue_tile<EPI_ATOMIC_N>(v, tm * 128, tn, row, taddr);
            else
                group_atomic_t_tile(v, tm * 128, tm, tn, row, taddr);
            tc_fence_before();
            __syncwarp();
            if (lane == 0) mbar_arrive(tempty0 + 8 * acc);
        }
    }

    tc_fence_before();
    __syncthreads();
    tc_fence_after();
    if (warp == 1) tmem_dealloc(tmem_base, g.tmem_cols);
}

}  // namespace attt
