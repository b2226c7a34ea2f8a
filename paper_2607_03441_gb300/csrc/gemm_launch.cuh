// gemm_launch.cuh -- host-side set-up and launch of tc_gemm_kernel.
#pragma once

#include "attt_host.h"
#include "tc_gemm.cuh"

namespace attt {

// Description of one contraction D = A * B^T (see tc_gemm.cuh).
struct GemmProblem {
    const void *a;        // A base pointer
    int64_t a_rows_ld;    // A: K-major -> row pitch in elements of the [rows, K] matrix;
                          //    MN-major -> row pitch of the [K, rows] matrix
    int64_t a_rows, a_k;  // extents of A's storage (rows = M extent, k = K extent)
    const void *b;
    int64_t b_rows_ld;
    int64_t b_rows, b_k;
    int M, N, K;
    // optional second operand pair over K2 more K (same majors, no offsets):
    // D = A B^T + A2 B2^T
    const void *a2 = nullptr;
    int64_t a2_rows_ld = 0, a2_rows = 0, a2_k = 0;
    const void *b2 = nullptr;
    int64_t b2_rows_ld = 0, b2_rows = 0, b2_k = 0;
    int K2 = 0;
    int BN;
    int a_m_off = 0, a_k_off = 0, b_n_off = 0, b_k_off = 0;
    bool pair = false;  // run on CTA pairs (256-row tiles, cta_group::2)
    // Launch as a programmatic dependent of the previous grid in the stream;
    // operands_ready: A and B do not come from that grid.
    bool pdl = false;
    bool operands_ready = false;
    // Tail split (EPI_F32_ACC): workspace for up to `split_regions` partials
    // of 128 x BN fp32 and as many arrival counters (zero on entry).
    float *split_ws = nullptr;
    unsigned int *split_tick = nullptr;
    int split_regions = 0;
};

// Pieces per tile for the tiles of a partial last wave: `tiles` tiles over
// `units` concurrent tile slots leave r = tiles mod units tiles for the last
// wave; cutting each into s K pieces (2 <= s <= 4, at least 8 K blocks each)
// runs that wave in ceil(r s / units) / s of a tile's time.  Returns 1 when the
// cut shortens the launch by less than a tenth (a long launch under the power
// cap gains nothing from filling idle SMs) or the partials would not fit
// `regions` (ranks per tile: `nranks`).
inline int tail_pieces(int tiles, int units, int kb_total, int nranks, int regions) {
    const int r = tiles % units;
    if (r == 0) return 1;
    int best_s = 1;
    double best = 1.0;
    for (int s = 2; s <= 4; ++s) {
        if (kb_total < 8 * s || r * s * nranks > regions) break;
        const double t = (double)cdiv(r * s, units) / s;
        if (t < best - 1e-9) { best = t; best_s = s; }
    }
    const double waves = (double)(tiles / units) + 1.0;
    return (1.0 - best) >= 0.1 * waves ? best_s : 1;
}

constexpr size_t kMaxSmem = 232448;  // 227 KB opt-in per CTA on sm_100-class parts

inline int gemm_stages(int BN, uint32_t extra = 0) {
    int s = 8;
    while (s > 2 && gemm_smem_bytes(BN, s, extra) > kMaxSmem) --s;
    return s;
}

inline uint32_t gemm_tmem_cols(int BN) {
    uint32_t need = 2u * (uint32_t)BN, c = 32;
    while (c < need) c <<= 1;
    return c;
}

// `status` is the device word that records a timed-out wait; nullptr selects
// the library's per-device status word.
template <int EPI, bool A_MN, bool B_MN>
attt_status launch_gemm(const GemmProblem &p, const EpiParams &ep, int dev, cudaStream_t stream,
                        int *status = nullptr) {
    if (p.BN < 16 || p.BN > 256 || p.BN % 16 != 0) return ATTT_ERR_INVALID_ARG;
    if (B_MN && (p.pair ? (p.BN / 2) % 64 : p.BN % 64) != 0) return ATTT_ERR_INVALID_ARG;
    if (p.pair && p.BN < 32) return ATTT_ERR_INVALID_ARG;  // BN/2 B rows per CTA (a multiple of 8)
    if (p.M <= 0 || p.N <= 0 || p.K <= 0) return ATTT_ERR_INVALID_ARG;
    CUtensorMap ta, tb;
    // K-major operand: storage [rows, K] (K contiguous), box 64 x rows_tile.
    // MN-major operand: storage [K, rows] (rows contiguous), box 64 x 64.
    bool ok;
    // EPI_KL loads 64 rows of A and 64 of A2 into one 128-row tile
    const uint32_t a_box_rows = EPI == EPI_KL ? 64u : 128u;
    if (!A_MN)
        ok = make_tmap_bf16(&ta, p.a, (uint64_t)p.a_k, (uint64_t)p.a_rows, (uint64_t)p.a_rows_ld * 2, 64, a_box_rows);
    else
        ok = make_tmap_bf16(&ta, p.a, (uint64_t)p.a_rows, (uint64_t)p.a_k, (uint64_t)p.a_rows_ld * 2, 64, 64);
    if (!ok) return ATTT_ERR_INVALID_ARG;
    if (!B_MN)
        ok = make_tmap_bf16(&tb, p.b, (uint64_t)p.b_k, (uint64_t)p.b_rows, (uint64_t)p.b_rows_ld * 2, 64,
                            (uint32_t)(p.pair ? p.BN / 2 : p.BN));
    else
        ok = make_tmap_bf16(&tb, p.b, (uint64_t)p.b_rows, (uint64_t)p.b_k, (uint64_t)p.b_rows_ld * 2, 64, 64);
    if (!ok) return ATTT_ERR_INVALID_ARG;
    CUtensorMap ta2 = ta, tb2 = tb;
    if (EPI == EPI_KL) {
        // the second A operand (same shape as A) shares every B tile
        if (!p.a2 || !p.pair || A_MN || B_MN) return ATTT_ERR_INVALID_ARG;
        if (!make_tmap_bf16(&ta2, p.a2, (uint64_t)p.a_k, (uint64_t)p.a_rows, (uint64_t)p.a2_rows_ld * 2, 64, 64))
            return ATTT_ERR_INVALID_ARG;
    } else if (p.K2 > 0) {
        if (!p.a2 || !p.b2) return ATTT_ERR_INVALID_ARG;
        if (!A_MN)
            ok = make_tmap_bf16(&ta2, p.a2, (uint64_t)p.a2_k, (uint64_t)p.a2_rows, (uint64_t)p.a2_rows_ld * 2, 64, 128);
        else
            ok = make_tmap_bf16(&ta2, p.a2, (uint64_t)p.a2_rows, (uint64_t)p.a2_k, (uint64_t)p.a2_rows_ld * 2, 64, 64);
        if (!ok) return ATTT_ERR_INVALID_ARG;
        if (!B_MN)
            ok = make_tmap_bf16(&tb2, p.b2, (uint64_t)p.b2_k, (uint64_t)p.b2_rows, (uint64_t)p.b2_rows_ld * 2, 64,
                                (uint32_t)(p.pair ? p.BN / 2 : p.BN));
        else
            ok = make_tmap_bf16(&tb2, p.b2, (uint64_t)p.b2_rows, (uint64_t)p.b2_k, (uint64_t)p.b2_rows_ld * 2, 64, 64);
        if (!ok) return ATTT_ERR_INVALID_ARG;
    }
    // EPI_CE_EXP writes E through TMA stores: [M, G_ld] bf16, 32 x 32 boxes
    // EPI_F32_ACC reads and writes `out` through TMA: [M, N] fp32 of pitch out_ld, 32 x 32 boxes
    CUtensorMap tc = tb;
    if (EPI == EPI_CE_EXP) {
        if (!make_tmap_bf16(&tc, ep.G, (uint64_t)ep.G_ld, (uint64_t)p.M, (uint64_t)ep.G_ld * 2, 32, 32, 64))
            return ATTT_ERR_INVALID_ARG;
    } else if (EPI == EPI_F32_ACC) {
        if (!make_tmap_f32(&tc, ep.out, (uint64_t)p.N, (uint64_t)p.M, (uint64_t)ep.out_ld * 4, 32, 32))
            return ATTT_ERR_INVALID_ARG;
    } else if (EPI == EPI_BF16) {
        if (!make_tmap_bf16(&tc, ep.out16, (uint64_t)p.N, (uint64_t)p.M, (uint64_t)ep.out_ld * 2, 32, 32, 64))
            return ATTT_ERR_INVALID_ARG;
    }

    GemmArgs g{};
    g.M = p.M;
    g.N = p.N;
    g.BN = p.BN;
    const int bn_cta = p.pair ? p.BN / 2 : p.BN;  // B rows one CTA stages
    g.e_stage_bytes = (EPI == EPI_CE_EXP || EPI == EPI_BF16) ? kEStageBytes
                      : EPI == EPI_F32_ACC                   ? kF32StageBytes
                      : EPI == EPI_KL                        ? kKlXBytes
                                                             : 0u;
    g.stages = gemm_stages(bn_cta, g.e_stage_bytes);
    // tiles_m counts tiles of 128 accumulator rows; an EPI_KL tile holds 64
    // rows of the problem (the other 64 are A2's)
    g.tiles_m = (int)cdiv(p.M, EPI == EPI_KL ? 64 : 128);
    g.tiles_n = (int)cdiv(p.N, p.BN);
    g.kb_split = (int)cdiv(p.K, 64);
    g.kb_total = g.kb_split + (p.K2 > 0 ? (int)cdiv(p.K2, 64) : 0);
    const int sms = num_sms(dev);
    const int units = p.pair ? sms / 2 : sms;  // concurrent tiles
    const int tiles = (p.pair ? (g.tiles_m + 1) / 2 : g.tiles_m) * g.tiles_n;
    g.splits = 1;
    g.kb_per_split = g.kb_total;
    g.whole_tiles = tiles;
    g.tail_s = 1;
    if (EPI == EPI_F32_ACC && p.split_ws && p.split_tick && p.BN % 32 == 0) {
        const int s = tail_pieces(tiles, units, g.kb_total, p.pair ? 2 : 1, p.split_regions);
        if (s > 1) {
            g.tail_s = s;
            g.whole_tiles = tiles - tiles % units;
            g.split_ws = p.split_ws;
            g.split_tick = p.split_tick;
        }
    }
    g.a_m_off = p.a_m_off;
    g.a_k_off = p.a_k_off;
    g.b_n_off = p.b_n_off;
    g.b_k_off = p.b_k_off;
    g.tmem_cols = gemm_tmem_cols(p.BN);
    g.operands_ready = p.operands_ready ? 1 : 0;
    g.status = status ? status : device_status_word(dev);
    g.ep = ep;

    const size_t smem = gemm_smem_bytes(bn_cta, g.stages, g.e_stage_bytes);
    const int ntiles = g.whole_tiles + (tiles - g.whole_tiles) * g.tail_s;  // work items
    cudaLaunchConfig_t cfg = {};
    cfg.blockDim = dim3(p.pair ? kGemmPairThreads : kGemmThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.stream = stream;
    cudaLaunchAttribute attr[2];
    unsigned na = 0;
    if (p.pdl) {
        attr[na].id = cudaLaunchAttributeProgrammaticStreamSerialization;
        attr[na].val.programmaticStreamSerializationAllowed = 1;
        ++na;
    }
    if (!p.pair) {
        if constexpr (EPI != EPI_KL) {  // EPI_KL runs on CTA pairs only
            auto kern = tc_gemm_kernel<EPI, A_MN, B_MN>;
            if (!set_smem_limit(reinterpret_cast<const void *>(kern), smem, dev)) return ATTT_ERR_CUDA;
            cfg.gridDim = dim3((unsigned)(ntiles < sms ? ntiles : sms));
            cfg.attrs = attr;
            cfg.numAttrs = na;
            if (cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, ta2, tb2, g) != cudaSuccess) return ATTT_ERR_CUDA;
        }
    } else {
        auto kern = tc_gemm_pair_kernel<EPI, A_MN, B_MN>;
        if (!set_smem_limit(reinterpret_cast<const void *>(kern), smem, dev)) return ATTT_ERR_CUDA;
        const int pairs = ntiles < units ? ntiles : units;
        cfg.gridDim = dim3((unsigned)(2 * pairs));
        attr[na].id = cudaLaunchAttributeClusterDimension;
        attr[na].val.clusterDim.x = 2;
        attr[na].val.clusterDim.y = 1;
        attr[na].val.clusterDim.z = 1;
        ++na;
        cfg.attrs = attr;
        cfg.numAttrs = na;
        if (cudaLaunchKernelEx(&cfg, kern, ta, tb, tc, ta2, tb2, g) != cudaSuccess) return ATTT_ERR_CUDA;
    }
    count_launch();
    return cudaGetLastError() == cudaSuccess ? ATTT_OK : ATTT_ERR_CUDA;
}

}  // namespace attt
