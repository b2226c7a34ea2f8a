"""Pins for the oracle's adapter-drift KL (Sec. 4, Fig. 6): the divergence
of the adapted model's next-token distribution from the base model's,
KL(softmax(h_p W^T) || softmax(h_q W^T)) per row.

Checked against torch CPU kl_div (a library routine), a two-token closed
form (the direction of the divergence), the zero cases (equal states, a
zero head), Gibbs' inequality, invariance to a constant logit shift, and a
planted mistake (the reversed direction).
"""
import math

import numpy as np
import torch
import torch.nn.functional as F

from paper_2607_03441_gb300 import workloads as wk


def _f64(bits):
    return wk.bf16_to_f32(bits).astype(np.float64)


def _case(seed, L=9, d=24, V=50, scale=0.3):
    hp = wk.normal_bf16(seed, "kl/hp", (L, d), 1.0)
    hq = wk.normal_bf16(seed, "kl/hq", (L, d), 1.0)
    W = wk.normal_bf16(seed, "kl/W", (V, d), scale)
    return hp, hq, W


def test_matches_torch_kl_div(oracle_mod):
    hp, hq, W = _case(1)
    zp = torch.from_numpy(_f64(hp)) @ torch.from_numpy(_f64(W)).T
    zq = torch.from_numpy(_f64(hq)) @ torch.from_numpy(_f64(W)).T
    ref = F.kl_div(F.log_softmax(zq, -1), F.log_softmax(zp, -1), reduction="none", log_target=True).sum(-1)
    np.testing.assert_allclose(oracle_mod.kl_rows(hp, hq, W), ref.numpy(), rtol=1e-10, atol=1e-13)


def test_two_token_closed_form_and_direction(oracle_mod):
    """z_p = [0, a], z_q = [0, 0]: p = (1, e^a) / (1 + e^a), q uniform;
    KL(p || q) = sum p log(2 p)."""
    d = 8
    a = wk.bf16_to_f32(wk.bf16_bits(np.array([math.log(3.0)], np.float32)))[0]
    hp = np.zeros((1, d), np.float32); hp[0, 0] = 1.0
    hq = np.zeros((1, d), np.float32)
    W = np.zeros((2, d), np.float32); W[1, 0] = a
    kl = oracle_mod.kl_rows(wk.bf16_bits(hp), wk.bf16_bits(hq), wk.bf16_bits(W))[0]
    p1 = math.exp(a) / (1 + math.exp(a))
    p = [1 - p1, p1]
    ref = sum(pi * math.log(2 * pi) for pi in p)
    assert abs(kl - ref) < 1e-12
    rev = sum(0.5 * math.log(0.5 / pi) for pi in p)   # KL(q || p), the other direction
    assert abs(kl - rev) > 1e-3


def test_zero_cases_and_gibbs(oracle_mod):
    hp, hq, W = _case(2)
    np.testing.assert_array_equal(oracle_mod.kl_rows(hp, hp, W), np.zeros(hp.shape[0]))
    assert np.all(oracle_mod.kl_rows(hp, hq, np.zeros_like(W)) == 0.0)
    kl = oracle_mod.kl_rows(hp, hq, W)
    assert np.all(kl > 0)
    # rows are independent: a subset equals the full result
    rows = np.array([4, 0, 7], np.int64)
    np.testing.assert_array_equal(oracle_mod.kl_rows(hp, hq, W, rows), kl[rows])


def test_shift_invariance(oracle_mod):
    """A logit shift common to every vocab entry of a row leaves p, q and KL
    unchanged: append a coordinate where every W row is 1 and move h_p there."""
    hp, hq, W = _case(3, d=16)
    L = hp.shape[0]
    W1 = np.concatenate([wk.bf16_to_f32(W), np.ones((W.shape[0], 8), np.float32)], axis=1)
    hp1 = np.concatenate([wk.bf16_to_f32(hp), np.zeros((L, 8), np.float32)], axis=1)
    hq1 = np.concatenate([wk.bf16_to_f32(hq), np.zeros((L, 8), np.float32)], axis=1)
    hp2 = hp1.copy(); hp2[:, 16] = 2.0
    base = oracle_mod.kl_rows(wk.bf16_bits(hp1), wk.bf16_bits(hq1), wk.bf16_bits(W1))
    shifted = oracle_mod.kl_rows(wk.bf16_bits(hp2), wk.bf16_bits(hq1), wk.bf16_bits(W1))
    np.testing.assert_allclose(shifted, base, rtol=1e-9, atol=1e-12)


def test_reversed_direction_is_caught(oracle_mod):
    hp, hq, W = _case(4, V=20, scale=0.5)
    fwd = oracle_mod.kl_rows(hp, hq, W)
    rev = oracle_mod.kl_rows(hq, hp, W)
    assert np.abs(fwd - rev).max() > 1e-3
