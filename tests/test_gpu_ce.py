"""GPU parity of Eq. 10 (weighted CE forward + backward through the frozen LM
head) against the CPU oracle.

Tolerances: loss within 1e-3 relative; lse within 1e-3 absolute (an lse is a
log, so its error is absolute); dh within 2e-2 relative L2 (bf16 products,
fp32 accumulation, the softmax-gradient block rounded to bf16 once).
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, f32_dev, i32_dev, rel_l2

pytestmark = pytest.mark.gpu

LOSS_RTOL = 1e-3
LSE_ATOL = 1e-3
DH_RL2 = 2e-2


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _run(attt, h, W, tgt, w):
    L = h.shape[0]
    lse = torch.empty(L, dtype=torch.float32, device=DEV)
    loss, dh, lse = attt.attt_weighted_ce_fwd_bwd(bf16_dev(h), bf16_dev(W), i32_dev(tgt), f32_dev(w), lse=lse)
    assert attt.attt_device_status() == 0
    return float(loss.item()), dh.cpu().numpy(), lse.cpu().numpy()


def _full_check(attt, h, W, tgt, w):
    loss, dh, lse = _run(attt, h, W, tgt, w)
    rloss, rlse, _, rdh = oracle.ce_loss(h, W, tgt, w)
    assert abs(loss - rloss) <= LOSS_RTOL * max(abs(rloss), 1e-30), (loss, rloss)
    np.testing.assert_allclose(lse, rlse, atol=LSE_ATOL, rtol=0)
    e = rel_l2(dh, rdh)
    assert e < DH_RL2, e
    return loss, dh


def test_tiny_workload(attt):
    """Tiny config: L 256, V 8192, d 512, weights from its own n-gram history."""
    wl = wk.WORKLOADS["tiny"]
    H = wk.history_tokens(wl)
    x = wk.update_tokens(wl, H)
    w = oracle.ngram_weights(H, x, wl.n)
    dense = wk.dense_inputs(wl)
    _full_check(attt, dense["h"], dense["W"], x, w)


@pytest.mark.parametrize("L,V,d", [(300, 1000, 200), (129, 257, 72), (1, 1, 8), (5, 3, 16), (130, 8448, 64),
                                   (64, 300, 1024)])
def test_ragged_shapes(attt, L, V, d):
    h = wk.normal_bf16(10 + L, "h", (L, d), 1.0)
    W = wk.normal_bf16(10 + V, "W", (V, d), 0.1)
    rng = wk.rng_for(L * 7 + V, "t")
    tgt = rng.integers(0, V, L).astype(np.int32)
    w = rng.choice(np.array([1.0, 0.5, 0.25, 0.05], np.float32), L).astype(np.float32)
    _full_check(attt, h, W, tgt, w)


def test_every_row_at_a_multi_tile_size(attt):
    """L 2,048, d 3,584 (the 7B-class rows and hidden size), V 4,000: eight
    256-row pair tiles of the logits contraction and 112 tiles of the dh
    contraction on 76 CTA pairs (a partial last wave, so the tail split);
    the loss, every row's lse and all of dh against the oracle."""
    L, V, d = 2048, 4000, 3584
    h = wk.normal_bf16(21, "h", (L, d), 1.0)
    W = wk.normal_bf16(21, "W", (V, d), 0.02)
    rng = wk.rng_for(21, "t")
    tgt = rng.integers(0, V, L).astype(np.int32)
    w = rng.choice(np.array([1.0, 0.5, 0.25, 0.05], np.float32), L).astype(np.float32)
    _full_check(attt, h, W, tgt, w)


def test_zero_weights_and_unit_weights(attt):
    L, V, d = 200, 700, 96
    h = wk.normal_bf16(3, "h", (L, d), 1.0)
    W = wk.normal_bf16(3, "W", (V, d), 0.1)
    tgt = wk.rng_for(3, "t").integers(0, V, L).astype(np.int32)
    loss, dh, _ = _run(attt, h, W, tgt, np.zeros(L, np.float32))
    assert loss == 0.0 and np.all(dh == 0.0)
    _full_check(attt, h, W, tgt, np.ones(L, np.float32))


def test_zero_hidden(attt):
    L, V, d = 70, 600, 64
    h = np.zeros((L, d), np.uint16)
    W = wk.normal_bf16(4, "W", (V, d), 0.1)
    tgt = wk.rng_for(4, "t").integers(0, V, L).astype(np.int32)
    w = np.full(L, 0.5, np.float32)
    loss, _ = _full_check(attt, h, W, tgt, w)
    assert loss == pytest.approx(np.log(V) * 0.5, rel=LOSS_RTOL)


def test_target_out_of_range(attt):
    from paper_2607_03441_gb300.attt import AtttError  # noqa: F401
    L, V, d = 16, 64, 32
    h = wk.normal_bf16(5, "h", (L, d), 1.0)
    W = wk.normal_bf16(5, "W", (V, d), 0.1)
    tgt = np.zeros(L, np.int32)
    tgt[3] = V
    loss, _, _ = attt.attt_weighted_ce_fwd_bwd(bf16_dev(h), bf16_dev(W), i32_dev(tgt), f32_dev(np.ones(L, np.float32)))
    assert np.isnan(loss.item())
    assert attt.attt_device_status() == 3  # ATTT_ERR_TOKEN_RANGE
    assert attt.attt_device_status() == 0  # read clears it
    # the row with the bad target is NaN; every other row is still exact
    w = np.ones(L, np.float32)
    lse_t = torch.empty(L, dtype=torch.float32, device=DEV)
    _, dh_t, _ = attt.attt_weighted_ce_fwd_bwd(bf16_dev(h), bf16_dev(W), i32_dev(tgt), f32_dev(w), lse=lse_t)
    assert attt.attt_device_status() == 3
    dh = dh_t.cpu().numpy()
    assert np.all(np.isnan(dh[3]))
    rows = np.array([j for j in range(L) if j != 3], np.int64)
    tgt_ok = tgt.copy()
    tgt_ok[3] = 0
    rlse, _, rdh = oracle.ce_rows(h, W, tgt_ok, w, rows)
    np.testing.assert_allclose(lse_t.cpu().numpy()[rows], rlse, atol=LSE_ATOL, rtol=0)
    assert rel_l2(dh[rows], rdh) < DH_RL2


def test_bad_arguments(attt):
    from paper_2607_03441_gb300.attt import AtttError
    L, V, d = 16, 64, 36  # d % 8 != 0
    h = torch.zeros(L, d, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(V, d, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(AtttError):
        attt.attt_weighted_ce_fwd_bwd(h, W, torch.zeros(L, dtype=torch.int32, device=DEV),
                                      torch.ones(L, device=DEV))
    h = torch.zeros(L, 32, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(V, 32, dtype=torch.bfloat16, device=DEV)
    with pytest.raises(AtttError):  # workspace too small
        attt.attt_weighted_ce_fwd_bwd(h, W, torch.zeros(L, dtype=torch.int32, device=DEV),
                                      torch.ones(L, device=DEV),
                                      workspace=torch.empty(256, dtype=torch.uint8, device=DEV))


def _sampled_check(attt, name, nrows=12):
    wl = wk.WORKLOADS[name]
    H = wk.history_tokens(wl) if wl.hist_len else np.zeros(0, np.int32)
    x = wk.update_tokens(wl, H)
    w = oracle.ngram_weights(H, x, wl.n)
    h = wk.normal_bf16(wl.seed, "hidden", (wl.L, wl.d), 1.0)
    W = wk.normal_bf16(wl.seed, "lm_head", (wl.V, wl.d), 0.02)
    loss, dh, lse = _run(attt, h, W, x, w)
    rng = wk.rng_for(wl.seed, "sample_rows")
    rows = np.unique(np.concatenate([[0, wl.L - 1], rng.choice(wl.L, nrows - 2, replace=False)])).astype(np.int64)
    rlse, rnll, rdh = oracle.ce_rows(h, W, x, w, rows)
    np.testing.assert_allclose(lse[rows], rlse, atol=LSE_ATOL, rtol=0)
    e = rel_l2(dh[rows], rdh)
    assert e < DH_RL2, e
    # every row: loss is the weighted mean of lse_j - z_{j, x_j} (z from the inputs)
    hf = wk.bf16_to_f32(h).astype(np.float64)
    Wt = wk.bf16_to_f32(W[x]).astype(np.float64)
    zt = np.einsum("ld,ld->l", hf, Wt)
    ref_loss = float(np.sum(w.astype(np.float64) * (lse.astype(np.float64) - zt)) / wl.L)
    assert abs(loss - ref_loss) <= LOSS_RTOL * abs(ref_loss)
    # sampled-row oracle nll agrees with the same decomposition
    np.testing.assert_allclose(rnll, rlse - zt[rows], rtol=1e-9, atol=1e-9)


def test_7b_sampled(attt):
    _sampled_check(attt, "7b")


def test_long_sampled(attt):
    _sampled_check(attt, "long", nrows=8)


@pytest.mark.slow
def test_32b_sampled(attt):
    _sampled_check(attt, "32b", nrows=6)


def test_multichunk_with_reference_jumps(attt):
    """Several vocab chunks, with rows whose max logit sits far above their
    reference (the target logit, then the running max): 2^92 in log2 units
    (E rewritten, in the first chunk for row 1500, the last for row 77) and
    2^61 (E written up to 2^61, no rewrite: row 300 in the first chunk, row
    900 in the last); row 5's target
    is its max, so the chunks before it sit far below the reference; sampled
    rows against the oracle."""
    L, V, d = 2048, 80000, 64
    rng = wk.rng_for(77, "jump")
    h = wk.normal_bf16(77, "h", (L, d), 0.5)
    W = wk.normal_bf16(77, "W", (V, d), 0.05)
    hot_rows = [5, 77, 1500, 300, 900]
    for j, v, x in zip(hot_rows, [60000, 79999, 30, 100, 79000], [8.0, 8.0, 8.0, 6.5, 6.5]):
        h[j] = 0
        h[j, 0] = wk.bf16_bits(np.array([x], np.float32))[0]
        W[v, 0] = wk.bf16_bits(np.array([x], np.float32))[0]  # z[j, v] = x^2 (64 or 42.25)
    tgt = rng.integers(0, V, L).astype(np.int32)
    tgt[5] = 60000
    w = rng.choice(np.array([1.0, 0.5, 0.05], np.float32), L).astype(np.float32)
    loss, dh, lse = _run(attt, h, W, tgt, w)
    rows = np.array(hot_rows + [0, 1, 1000, L - 1], np.int64)
    rlse, rnll, rdh = oracle.ce_rows(h, W, tgt, w, rows)
    np.testing.assert_allclose(lse[rows], rlse, atol=LSE_ATOL, rtol=0)
    for i in range(len(rows)):
        e = rel_l2(dh[rows[i]], rdh[i])
        assert e < DH_RL2, (rows[i], e)
    hf = wk.bf16_to_f32(h).astype(np.float64)
    zt = np.einsum("ld,ld->l", hf, wk.bf16_to_f32(W[tgt]).astype(np.float64))
    ref_loss = float(np.sum(w.astype(np.float64) * (lse.astype(np.float64) - zt)) / L)
    assert abs(loss - ref_loss) <= LOSS_RTOL * abs(ref_loss)


@pytest.mark.parametrize("L,V,d", [(1280, 6000, 1280), (2048, 3000, 3584), (100, 20000, 3584)])
def test_tail_pieces_deterministic(attt, L, V, d):
    """Shapes whose dh contraction leaves a partial last wave on a 152-SM
    part, so its tiles run as 2-4 K pieces (25 tiles: 3 pieces; 112 tiles:
    2; 14 single-CTA tiles: 4): sampled rows against the oracle, and two calls
    give the same bits whichever piece finishes last."""
    h = wk.normal_bf16(L + 1, "h", (L, d), 1.0)
    W = wk.normal_bf16(V + 1, "W", (V, d), 0.05)
    rng = wk.rng_for(L + V, "t")
    tgt = rng.integers(0, V, L).astype(np.int32)
    w = rng.choice(np.array([1.0, 0.5, 0.05], np.float32), L).astype(np.float32)
    loss, dh, lse = _run(attt, h, W, tgt, w)
    loss2, dh2, lse2 = _run(attt, h, W, tgt, w)
    assert loss == loss2
    np.testing.assert_array_equal(dh.view(np.uint32), dh2.view(np.uint32))
    np.testing.assert_array_equal(lse.view(np.uint32), lse2.view(np.uint32))
    rows = np.unique(np.concatenate([[0, 1, L - 1], rng.choice(L, 9, replace=False)])).astype(np.int64)
    rlse, _, rdh = oracle.ce_rows(h, W, tgt, w, rows)
    np.testing.assert_allclose(lse[rows], rlse, atol=LSE_ATOL, rtol=0)
    e = rel_l2(dh[rows], rdh)
    assert e < DH_RL2, e


def test_launch_counter_counts_every_kernel(attt):
    """One single-chunk call launches the reference kernel, GEMM1, the chunk
    kernel and GEMM2: four kernels, all counted."""
    L, V, d = 200, 1000, 64
    h = wk.normal_bf16(8, "h", (L, d), 1.0)
    W = wk.normal_bf16(8, "W", (V, d), 0.1)
    tgt = wk.rng_for(8, "t").integers(0, V, L).astype(np.int32)
    args = (bf16_dev(h), bf16_dev(W), i32_dev(tgt), f32_dev(np.ones(L, np.float32)))
    attt.attt_weighted_ce_fwd_bwd(*args)
    n0 = attt.attt_kernel_launches()
    attt.attt_weighted_ce_fwd_bwd(*args)
    assert attt.attt_kernel_launches() - n0 == 4
