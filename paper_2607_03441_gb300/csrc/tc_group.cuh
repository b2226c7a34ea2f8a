// tc_group.cuh -- grouped tcgen05 contractions: several independent problems
// (own operands, sizes and output) in one persistent launch.
//
// The LoRA gradients are a handful of skinny, HBM-bound contractions (the
// rank on N); launched one by one, each pays a launch, a ramp and a tail
// that cost more than streaming its operands.  Grouping runs every
// contraction of a pass in one launch.  The pipeline is the single-CTA one
// of tc_gemm.cuh (MMA warp, four epilogue warps, two TMEM accumulators) with
// two TMA producer warps instead of one; the work decode, the per-problem
// tensor maps and the epilogue differ.  All problems of a group share BN and the operand majors.
//
// Work is split stream-K style: the K stages of every tile of every problem
// are laid end to end (problem by problem, tile by tile), and CTA c takes the
// stages [c S / G, (c + 1) S / G) of the S stages for G CTAs, so every CTA
// streams the same number of stages.  A CTA's range is a few segments (the
// end of one tile, whole tiles, the start of another), each one accumulator
// pass.  A tile that one segment covers is written straight from TMEM; a tile
// split over several CTAs has each piece store its fp32 partial in a slot,
// and the piece that arrives last (ticket) sums the partials in CTA order and
// writes the tile.  No atomics on the outputs, and the result does not depend
// on which piece finishes last.
#pragma once

#include "tc_gemm.cuh"

namespace attt {

// Problems of one grouped launch at most.  The tensor maps and problems
// travel in the kernel's parameters, so the capacity is a template argument:
// kMaxGroup (u and every v of kMaxProj projections, ~3.7 KB) for one group
// of projections, kMaxGroupBatch (the u and v, or dA and dB, of kGroupEpisodes
// episodes of a batch, ~14 KB of the 32 KB parameter space) for a batch.
constexpr int kMaxGroup = kMaxProj + 1;
constexpr int kGroupEpisodes = 16;
constexpr int kMaxGroupBatch = 2 * kGroupEpisodes;
constexpr int kGroupMaxGrid = 256;  // CTAs of a grouped launch at most: partial slots are CTA + tile

// How a problem writes its result D (fp32 accumulator, rows m < M, columns
// n < N).
enum GroupOut : int {
    GOUT_T16 = 0,  // out16[n * ld + m] = bf16(alpha D[m, n])                          (transposed, bf16)
    GOUT_N32 = 1,  // outp[n / rpad][m * r + n % rpad] = alpha D[m, n], n % rpad < r   (a row-major block per rpad columns)
    GOUT_T32 = 2,  // out32[n * ld + m] = alpha D[m, n], n % rpad < r                  (transposed, fp32)
    GOUT_N16 = 3,  // out16[m * ld + n] = bf16(alpha D[m, n])                          (row-major, bf16)
};

struct GroupProblem {
    int M, N;
    int tiles_m, tiles_n, kb_total;
    int nst;  // K stages per tile (kbs K blocks each)
    int a_m_off, a_k_off, b_n_off, b_k_off;
    int64_t stage_begin;  // first group-wide stage of this problem
    int tile_begin;       // first group-wide tile of this problem
    int out;              // GroupOut
    float alpha;
    int r, rpad;
    int64_t ld;
    float *out32;
    __nv_bfloat16 *out16;
    float *outp[kMaxProj];
};

template <int NP>
struct GroupMaps {
    CUtensorMap a[NP];
    CUtensorMap b[NP];
};

template <int NP>
struct GroupArgs {
    int nprob;
    int64_t total_stages;  // S; the grid G is at most S, so no CTA's range is empty
    int BN, stages;
    int kbs;  // 64-deep K blocks per pipeline stage (each row is fetched in kbs x 128 B runs)
    uint32_t tmem_cols;
    int *status;
    float *part;            // partial slots of 128 x BN fp32, [BN / 4][128] float4 each; CTA + tile slots
    unsigned int *tickets;  // one arrival counter per group-wide tile, 0 between launches
    GroupProblem prob[NP];
};

// One segment of a CTA's stage range: problem q, tile (tm, tn), K blocks
// [kb0, kb1); ts / te bound the tile's own stages.
struct GroupSeg {
    int q, tm, tn, kb0, kb1;
    int64_t ts, te;
};

// The segment that starts at stage x of a range ending at xend; advances x.
template <int NP>
__device__ __forceinline__ bool group_next(const GroupArgs<NP> &g, int64_t &x, int64_t xend, GroupSeg &sg) {
    if (x >= xend) return false;
    int q = 0;
    while (q + 1 < g.nprob && x >= g.prob[q + 1].stage_begin) ++q;
    const GroupProblem &p = g.prob[q];
    const int64_t loc = x - p.stage_begin;
    const int tile = (int)(loc / p.nst);
    const int s0 = (int)(loc - (int64_t)tile * p.nst);
    sg.ts = p.stage_begin + (int64_t)tile * p.nst;
    sg.te = sg.ts + p.nst;
    const int64_t end = xend < sg.te ? xend : sg.te;
    sg.q = q;
    sg.tn = tile / p.tiles_m;
    sg.tm = tile - sg.tn * p.tiles_m;
    sg.kb0 = s0 * g.kbs;
    sg.kb1 = min(p.kb_total, (int)(s0 + (end - x)) * g.kbs);
    x = end;
    return true;
}

// The CTA whose range holds stage x: the largest c with floor(c S / G) <= x.
template <int NP>
__device__ __forceinline__ int64_t group_owner(const GroupArgs<NP> &g, int64_t x, int64_t G) {
    return ((x + 1) * G - 1) / g.total_stages;
}

// Writes the 16 columns [col0, col0 + 16) of row m (values already summed
// over the tile's pieces).
__device__ __forceinline__ void group_store16(const GroupProblem &p, int m, int col0, int n_end,
                                              const float (&v)[16]) {
    if (p.out == GOUT_T16) {
#pragma unroll
        for (int i = 0; i < 16; ++i)
            if (col0 + i < n_end) p.out16[(int64_t)(col0 + i) * p.ld + m] = __float2bfloat16_rn(p.alpha * v[i]);
    } else if (p.out == GOUT_N32) {
        // the 16 columns lie in one rpad block (rpad is a multiple of 16)
        const int blk = col0 / p.rpad, cc0 = col0 - blk * p.rpad;
        float *orow = p.outp[blk] + (int64_t)m * p.r;
        if (col0 + 16 <= n_end && (p.r & 3) == 0 && (reinterpret_cast<uintptr_t>(orow) & 15) == 0) {
#pragma unroll
            for (int i = 0; i < 16; i += 4)
                if (cc0 + i < p.r)
                    *reinterpret_cast<float4 *>(orow + cc0 + i) =
                        make_float4(p.alpha * v[i], p.alpha * v[i + 1], p.alpha * v[i + 2], p.alpha * v[i + 3]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (col0 + i < n_end && cc0 + i < p.r) orow[cc0 + i] = p.alpha * v[i];
        }
    } else if (p.out == GOUT_T32) {
#pragma unroll
        for (int i = 0; i < 16; ++i) {
            const int col = col0 + i;
            if (col < n_end && (col % p.rpad) < p.r) p.out32[(int64_t)col * p.ld + m] = p.alpha * v[i];
        }
    } else {
        __nv_bfloat16 *o = p.out16 + (int64_t)m * p.ld + col0;
        if (col0 + 16 <= n_end && (reinterpret_cast<uintptr_t>(o) & 15) == 0) {
            uint32_t pk[8];
#pragma unroll
            for (int i = 0; i < 16; i += 2) {
                __nv_bfloat162 b = __floats2bfloat162_rn(p.alpha * v[i], p.alpha * v[i + 1]);
                pk[i / 2] = *reinterpret_cast<uint32_t *>(&b);
            }
            reinterpret_cast<uint4 *>(o)[0] = make_uint4(pk[0], pk[1], pk[2], pk[3]);
            reinterpret_cast<uint4 *>(o)[1] = make_uint4(pk[4], pk[5], pk[6], pk[7]);
        } else {
#pragma unroll
            for (int i = 0; i < 16; ++i)
                if (col0 + i < n_end) o[i] = __float2bfloat16_rn(p.alpha * v[i]);
        }
    }
}

// Shared memory of the GOUT_T16 stores: two buffers of 16 columns x 128 rows
// of bf16.
constexpr uint32_t kGroupTBytes = 2 * 16 * 128 * 2;

// GOUT_T16 columns [col0, col0 + 16) of the tile's 128 rows (m0 + row), all
// four epilogue warps together: each thread puts its row's 16 values into a
// 16 x 128 buffer, then 16 rows of out16 go out as 16-byte vectors of 8
// consecutive m (out16 rows are ld elements long, ld a multiple of 8; rows m
// past M but below ld hold the accumulator's zero rows and are never read).
// Two buffers alternate, so one barrier per call orders the writes of a
// buffer after the reads of its previous use.
__device__ __forceinline__ void group_store_t16(const GroupProblem &p, int m0, int row, int col0, int n_end,
                                                const float (&v)[16], uint32_t sbase, uint32_t &chunk) {
    const uint32_t buf = sbase + (chunk & 1u) * (kGroupTBytes / 2);
    ++chunk;
#pragma unroll
    for (int i = 0; i < 16; ++i) {
        const __nv_bfloat16 b = __float2bfloat16_rn(p.alpha * v[i]);
        asm volatile("st.shared.b16 [%0], %1;" ::"r"(buf + (uint32_t)(i * 128 + row) * 2u),
                     "h"(*reinterpret_cast<const unsigned short *>(&b))
                     : "memory");
    }
    named_barrier_sync(1, 128);
#pragma unroll
    for (int k = 0; k < 2; ++k) {
        const int idx = row + 128 * k;  // 16 rows of out16 x 16 vectors of 8 m
        const int i = idx >> 4, j = idx & 15;
        const int col = col0 + i, m = m0 + j * 8;
        if (col < n_end && m < p.ld) {
            uint4 val;
            asm volatile("ld.shared.v4.b32 {%0, %1, %2, %3}, [%4];"
                         : "=r"(val.x), "=r"(val.y), "=r"(val.z), "=r"(val.w)
                         : "r"(buf + (uint32_t)(i * 256 + j * 16)));
            *reinterpret_cast<uint4 *>(p.out16 + (int64_t)col * p.ld + m) = val;
        }
    }
}

// Epilogue of one segment, on CTA `cta` of G (four warps, thread = row).
// sT / tchunk: the GOUT_T16 buffers (group_store_t16).
template <int NP>
__device__ __forceinline__ void group_segment_epilogue(const GroupArgs<NP> &g, const GroupSeg &sg, int64_t cta, int64_t G,
                                                       int row, uint32_t taddr, uint32_t sT, uint32_t &tchunk) {
    const GroupProblem &p = g.prob[sg.q];
    const int gm = sg.tm * 128 + row;
    const bool rv = gm < p.M;
    const int n_base = sg.tn * g.BN;
    const int n_end = min(p.N, n_base + g.BN);
    const int64_t c0 = group_owner(g, sg.ts, G), c1 = group_owner(g, sg.te - 1, G);
    if (c0 == c1) {  // the whole tile is this segment
        for (int c = 0; c < g.BN; c += 16) {
            if (n_base + c >= n_end) break;
            float v[16];
            tmem_ld_x16(taddr + (uint32_t)c, v);
            if (p.out == GOUT_T16) group_store_t16(p, sg.tm * 128, row, n_base + c, n_end, v, sT, tchunk);
            else if (rv) group_store16(p, gm, n_base + c, n_end, v);
        }
        return;
    }
    const int64_t gtile = p.tile_begin + sg.tm + (int64_t)sg.tn * p.tiles_m;
    const size_t slot = (size_t)128 * g.BN;
    float4 *mine = reinterpret_cast<float4 *>(g.part + (size_t)(cta + gtile) * slot) + row;
    for (int c = 0; c < g.BN; c += 16) {
        if (n_base + c >= n_end) break;
        float v[16];
        tmem_ld_x16(taddr + (uint32_t)c, v);
#pragma unroll
        for (int q = 0; q < 4; ++q)
            __stcg(mine + (size_t)(c / 4 + q) * 128, make_float4(v[4 * q], v[4 * q + 1], v[4 * q + 2], v[4 * q + 3]));
    }
    __threadfence();
    named_barrier_sync(1, 128);
    int last = 0;
    if (row == 0) {
        unsigned int *tk = g.tickets + gtile;
        last = atomicAdd(tk, 1u) == (unsigned int)(c1 - c0) ? 1 : 0;
        if (last) atomicExch(tk, 0u);  // every piece has arrived: ready for the next launch
        __threadfence();
    }
    if (!named_barrier_or(1, 128, last)) return;
    for (int c = 0; c < g.BN; c += 16) {
        if (n_base + c >= n_end) break;
        float own[16];
        tmem_ld_x16(taddr + (uint32_t)c, own);
        float s[16];
        // pieces in CTA order, four partials loaded together (their loads in
        // flight at once), summed in order after they land
        for (int64_t j0 = c0; j0 <= c1; j0 += 4) {
            float4 f[4][4];
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int64_t j = j0 + b;
                if (j <= c1 && j != cta) {
                    const float4 *src = reinterpret_cast<const float4 *>(g.part + (size_t)(j + gtile) * slot) + row;
#pragma unroll
                    for (int q = 0; q < 4; ++q) f[b][q] = __ldcg(src + (size_t)(c / 4 + q) * 128);
                }
            }
#pragma unroll
            for (int b = 0; b < 4; ++b) {
                const int64_t j = j0 + b;
                if (j > c1) break;
#pragma unroll
                for (int q = 0; q < 4; ++q) {
                    const float4 x = (j == cta) ? make_float4(own[4 * q], own[4 * q + 1], own[4 * q + 2], own[4 * q + 3])
                                                : f[b][q];
                    if (j == c0) {
                        s[4 * q] = x.x; s[4 * q + 1] = x.y; s[4 * q + 2] = x.z; s[4 * q + 3] = x.w;
                    } else {
                        s[4 * q] += x.x; s[4 * q + 1] += x.y; s[4 * q + 2] += x.z; s[4 * q + 3] += x.w;
                    }
                }
            }
        }
        if (p.out == GOUT_T16) group_store_t16(p, sg.tm * 128, row, n_base + c, n_end, s, sT, tchunk);
        else if (rv) group_store16(p, gm, n_base + c, n_end, s);
    }
}

// Warps 0 and 6 both feed the ring, taking alternate stages: one thread keeps
// about one stage of TMA loads in flight at a time (measured on GB300 for a CTA
// streaming alone), so two producers double what a lone CTA streams; with every
// SM streaming, the grid's read rate is HBM's either way.  Warp 1 issues the
// MMAs, warps 2-5 run the epilogue.
constexpr int kGroupThreads = 224;

template <bool A_MN, bool B_MN, int NP>
__global__ void __launch_bounds__(kGroupThreads, 1)
    tc_gemm_group_kernel(const __grid_constant__ GroupMaps<NP> maps, const GroupArgs<NP> g) {
    extern __shared__ uint8_t smem_raw[];
    uint8_t *smem = reinterpret_cast<uint8_t *>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
    const int S = g.stages;
    const int KBS = g.kbs;
    const uint32_t a1 = kABytes, b1 = gemm_b_stage_bytes(g.BN);  // one K block
    const uint32_t kABytesS = a1 * KBS;
    const uint32_t b_bytes = b1 * KBS;
    uint8_t *sA = smem;
    uint8_t *sB = smem + (size_t)S * kABytesS;
    uint8_t *sT = sB + (size_t)S * b_bytes;  // the GOUT_T16 store buffers
    uint64_t *bars = reinterpret_cast<uint64_t *>(sT + kGroupTBytes);
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
        griddep_launch_dependents();  // the next grid may launch; it waits for this one before reading its results
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
    const int64_t G = gridDim.x;
    const int64_t x0 = (int64_t)blockIdx.x * g.total_stages / G;
    const int64_t x1 = ((int64_t)blockIdx.x + 1) * g.total_stages / G;

    if (warp == 0 || warp == 6) {
        if (lane == 0) {
            griddep_wait();  // the B operands (adapters, u, v) come from the previous grid
            const uint32_t pid = warp == 0 ? 0u : 1u;  // this producer's stages: pos % 2 == pid
            uint32_t pos = 0;
            int stage = 0;
            uint32_t phase = 0;
            uint32_t issued_mask = 0, issued_parity = 0;
            bool ok = true;
            GroupSeg sg;
            for (int64_t x = x0; ok && group_next(g, x, x1, sg);) {
                const GroupProblem &p = g.prob[sg.q];
                const CUtensorMap *ta = &maps.a[sg.q];
                const CUtensorMap *tb = &maps.b[sg.q];
                const int tm = sg.tm, tn = sg.tn;
                for (int kb = sg.kb0; kb < sg.kb1; kb += KBS) {
                    if (((pos++) & 1u) != pid) {  // the other producer's stage
                        if (++stage == S) { stage = 0; phase ^= 1u; }
                        continue;
                    }
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
                // the loads already issued still land in shared memory: wait (bounded)
                // for them with a flag of its own, which the raised abort flag does not cut short
                volatile int no_abort = 0;
                for (int s = 0; s < S; ++s)
                    if (issued_mask & (1u << s))
                        (void)mbar_wait(full0 + 8 * s, (issued_parity >> s) & 1u, &no_abort);
            }
        }
    } else if (warp == 1) {
        if (lane == 0) {
            const uint32_t idesc = idesc_bf16_f32((uint32_t)g.BN, A_MN, B_MN);
            int stage = 0;
            uint32_t phase = 0;
            int it = 0;
            bool ok = true;
            GroupSeg sg;
            for (int64_t x = x0; ok && group_next(g, x, x1, sg); ++it) {
                const int kb0 = sg.kb0, kb1 = sg.kb1;
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
    } else if (warp >= 2 && warp <= 5) {
        griddep_wait();  // tickets, slots and outputs follow the previous grid
        const int qw = warp & 3;
        const int row = qw * 32 + lane;
        int it = 0;
        uint32_t tchunk = 0;
        GroupSeg sg;
        for (int64_t x = x0; group_next(g, x, x1, sg); ++it) {
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
            group_segment_epilogue(g, sg, (int64_t)blockIdx.x, G, row, taddr, smem_u32(sT), tchunk);
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
