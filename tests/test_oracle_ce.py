"""Pins for the oracle's Eq. 10 (token-weighted CE) and its gradient dh.

Checked against torch's CPU cross_entropy and autograd (library routines),
central finite differences of the oracle's own loss, and closed forms
(h = 0, constant weights).
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2607_03441_gb300 import workloads as wk


def _f64(bits):
    return wk.bf16_to_f32(bits).astype(np.float64)


def _case(seed, L, V, d, hstd=1.0, wstd=0.02):
    h = wk.normal_bf16(seed, "h", (L, d), hstd)
    W = wk.normal_bf16(seed, "W", (V, d), wstd)
    rng = wk.rng_for(seed, "t")
    tgt = rng.integers(0, V, L).astype(np.int32)
    w = rng.choice(np.array([1.0, 0.5, 1 / 3, 0.05], np.float32), L).astype(np.float32)
    return h, W, tgt, w


def _torch_loss(h, W, tgt, w):
    z = torch.from_numpy(_f64(h)) @ torch.from_numpy(_f64(W)).T
    ce = F.cross_entropy(z, torch.from_numpy(tgt).long(), reduction="none")
    return (torch.from_numpy(w.astype(np.float64)) * ce).sum().item() / h.shape[0], ce.numpy()


def test_unit_weights_equal_library_mean_ce(oracle_mod):
    h, W, tgt, _ = _case(1, 24, 300, 40, wstd=0.3)
    w = np.ones(24, np.float32)
    loss, lse, nll, _ = oracle_mod.ce_loss(h, W, tgt, w, with_dh=False)
    z = torch.from_numpy(_f64(h)) @ torch.from_numpy(_f64(W)).T
    ref = F.cross_entropy(z, torch.from_numpy(tgt).long(), reduction="mean").item()
    assert loss == pytest.approx(ref, rel=1e-12)
    np.testing.assert_allclose(lse, torch.logsumexp(z, dim=1).numpy(), rtol=1e-12)


def test_weighted_loss_matches_library(oracle_mod):
    h, W, tgt, w = _case(2, 33, 257, 24, wstd=0.5)
    loss, _, nll, _ = oracle_mod.ce_loss(h, W, tgt, w, with_dh=False)
    ref, ce = _torch_loss(h, W, tgt, w)
    assert loss == pytest.approx(ref, rel=1e-12)
    np.testing.assert_allclose(nll, ce, rtol=1e-12)


def test_constant_weight_scales_mean_nll(oracle_mod):
    h, W, tgt, _ = _case(3, 16, 100, 16, wstd=0.4)
    ones = np.ones(16, np.float32)
    base, *_ = oracle_mod.ce_loss(h, W, tgt, ones, with_dh=False)
    c = np.float32(0.25)
    scaled, *_ = oracle_mod.ce_loss(h, W, tgt, np.full(16, c, np.float32), with_dh=False)
    assert scaled == pytest.approx(float(c) * base, rel=1e-13)


def test_zero_hidden_closed_form(oracle_mod):
    """h = 0: every logit is 0, so lse = log V, loss = log V * sum(w) / L and
    dh_j = (w_j / L) (mean_v W_v - W_{x_j})."""
    L, V, d = 8, 64, 12
    _, W, tgt, w = _case(4, L, V, d)
    h = np.zeros((L, d), np.uint16)
    loss, lse, nll, dh = oracle_mod.ce_loss(h, W, tgt, w)
    assert loss == pytest.approx(np.log(V) * w.astype(np.float64).sum() / L, rel=1e-13)
    np.testing.assert_allclose(lse, np.log(V), rtol=1e-14)
    Wf = _f64(W)
    ref = (w.astype(np.float64)[:, None] / L) * (Wf.mean(0)[None, :] - Wf[tgt])
    np.testing.assert_allclose(dh, ref, rtol=1e-11, atol=1e-15)


def test_dh_matches_autograd(oracle_mod):
    h, W, tgt, w = _case(5, 12, 90, 20, wstd=0.3)
    _, _, _, dh = oracle_mod.ce_loss(h, W, tgt, w)
    ht = torch.from_numpy(_f64(h)).requires_grad_(True)
    z = ht @ torch.from_numpy(_f64(W)).T
    ce = F.cross_entropy(z, torch.from_numpy(tgt).long(), reduction="none")
    loss = (torch.from_numpy(w.astype(np.float64)) * ce).sum() / 12
    loss.backward()
    np.testing.assert_allclose(dh, ht.grad.numpy(), rtol=1e-10, atol=1e-14)


def test_dh_finite_differences(oracle_mod):
    """Central differences of the oracle's own loss, with h on a grid of
    multiples of 1/8 and a step of 2^-7 so that h +- eps are exact in bf16."""
    L, V, d = 4, 16, 8
    rng = np.random.default_rng(9)
    hv = rng.integers(-8, 9, (L, d)).astype(np.float32) / 8
    Wv = rng.integers(-8, 9, (V, d)).astype(np.float32) / 8
    tgt = rng.integers(0, V, L).astype(np.int32)
    w = np.array([1.0, 0.5, 0.25, 0.05], np.float32)
    W = wk.bf16_bits(Wv)
    _, _, _, dh = oracle_mod.ce_loss(wk.bf16_bits(hv), W, tgt, w)
    eps = np.float32(2.0 ** -7)
    fd = np.zeros((L, d))
    for j in range(L):
        for k in range(d):
            hp = hv.copy(); hp[j, k] += eps
            hm = hv.copy(); hm[j, k] -= eps
            assert wk.bf16_to_f32(wk.bf16_bits(hp))[j, k] == hp[j, k]
            lp, *_ = oracle_mod.ce_loss(wk.bf16_bits(hp), W, tgt, w, with_dh=False)
            lm, *_ = oracle_mod.ce_loss(wk.bf16_bits(hm), W, tgt, w, with_dh=False)
            fd[j, k] = (lp - lm) / (2 * float(eps))
    np.testing.assert_allclose(dh, fd, rtol=2e-3, atol=2e-5)


def test_rows_subset_matches_full(oracle_mod):
    h, W, tgt, w = _case(6, 20, 150, 16)
    _, lse, nll, dh = oracle_mod.ce_loss(h, W, tgt, w)
    rows = np.array([19, 0, 7], np.int64)
    lse_r, nll_r, dh_r = oracle_mod.ce_rows(h, W, tgt, w, rows)
    np.testing.assert_array_equal(lse_r, lse[rows])
    np.testing.assert_array_equal(nll_r, nll[rows])
    np.testing.assert_array_equal(dh_r, dh[rows])
