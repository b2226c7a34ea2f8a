"""Pins for the oracle's AdamW step (an optional optimizer of the update; the
paper's is the SGD step of Eq. 2): torch CPU torch.optim.AdamW over several
steps (bias corrections included), the beta = 0 sign-like case, pure
weight decay when the gradient is zero, and the episode's use of it."""
import numpy as np
import torch

from paper_2607_03441_gb300 import workloads as wk


def test_matches_torch_adamw(oracle_mod):
    rng = np.random.default_rng(3)
    p0 = rng.standard_normal(50).astype(np.float32)
    grads = [rng.standard_normal(50).astype(np.float32) for _ in range(5)]
    lr, b1, b2, eps, wd = 1e-2, 0.9, 0.999, 1e-8, 0.01
    tp = torch.nn.Parameter(torch.from_numpy(p0.astype(np.float64)))
    opt = torch.optim.AdamW([tp], lr=lr, betas=(b1, b2), eps=eps, weight_decay=wd)
    p, m, v = p0, np.zeros(50), np.zeros(50)
    for t, g in enumerate(grads, start=1):
        tp.grad = torch.from_numpy(g.astype(np.float64))
        opt.step()
        p, m, v = oracle_mod.adamw_step(p, g, m, v, t, lr, b1, b2, eps, wd)
        np.testing.assert_allclose(p, tp.detach().numpy(), rtol=2e-7, atol=1e-7)


def test_special_cases(oracle_mod):
    g = np.array([3.0, -0.5, 2e-3], np.float32)
    p = np.zeros(3, np.float32)
    # beta1 = beta2 = 0: the step is lr g / (|g| + eps), about lr sign(g)
    q, _, _ = oracle_mod.adamw_step(p, g, np.zeros(3), np.zeros(3), 1, 0.1, 0.0, 0.0, 1e-8, 0.0)
    np.testing.assert_allclose(q, -0.1 * np.sign(g), rtol=1e-5)
    # zero gradient: only the decoupled decay acts
    p = np.array([1.0, -2.0, 4.0], np.float32)
    q, m, v = oracle_mod.adamw_step(p, np.zeros(3, np.float32), np.zeros(3), np.zeros(3), 1, 0.5, weight_decay=0.1)
    np.testing.assert_allclose(q, p * (1 - 0.05), rtol=1e-7)
    assert not m.any() and not v.any()


def test_episode_with_adamw_moves_by_about_lr(oracle_mod):
    """Adam's first step moves every adapter entry with a nonzero gradient by
    about lr (|m_hat / sqrt(v_hat)| = 1), whatever the gradient's scale."""
    rng = np.random.default_rng(5)
    L, din, d, V, r = 24, 32, 32, 100, 8
    H = rng.integers(0, 9, 80).astype(np.int32)
    tok = rng.integers(0, 9, L).astype(np.int32)
    x = wk.normal_bf16(5, "adamw/x", (L, din), 1.0)
    W0 = wk.normal_bf16(5, "adamw/W0", (din, d), 0.2)
    Wlm = wk.normal_bf16(5, "adamw/W", (V, d), 0.3)
    A0 = wk.bf16_to_f32(wk.normal_bf16(5, "adamw/A", (din, r), 0.05))
    B0 = wk.bf16_to_f32(wk.normal_bf16(5, "adamw/B", (r, d), 0.05))
    st = {"t": 0, "mA": np.zeros((din, r)), "vA": np.zeros((din, r)), "mB": np.zeros((r, d)),
          "vB": np.zeros((r, d)), "beta1": 0.9, "beta2": 0.999, "eps": 1e-8, "weight_decay": 0.0}
    lr = 1e-3
    out = oracle_mod.episode_update(H, tok, x, W0, Wlm, A0, B0, n=3, w_min=0.05, scale=2.0, lr=lr, grad_steps=1,
                                    adamw=st)
    assert st["t"] == 1
    dBm = np.abs(out["B32"] - B0)
    np.testing.assert_allclose(dBm[dBm > 0], lr, rtol=1e-3)
