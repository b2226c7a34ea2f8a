"""Pins for the oracle's adapted projection of a chained update (the
Appendix C adapter y = x W0 + s (x A) B whose output feeds the LM head): the
forward h and the input gradient dx = dy W0^T + s (dy B^T) A^T.

Checked against torch CPU matmul and autograd (library routines), the zero
adapter cases, a rank-one closed form, linearity, and central finite
differences of the oracle's own forward.
"""
import numpy as np
import pytest
import torch

from paper_2607_03441_gb300 import workloads as wk


def _f64(bits):
    return wk.bf16_to_f32(bits).astype(np.float64)


def _inputs(seed, L, din, dout, r):
    x = wk.normal_bf16(seed, "x", (L, din), 1.0)
    dy = wk.normal_bf16(seed, "dy", (L, dout), 1.0)
    W0 = wk.normal_bf16(seed, "W0", (din, dout), 0.05)
    A = wk.normal_bf16(seed, "A", (din, r), 0.05)
    B = wk.normal_bf16(seed, "B", (r, dout), 0.05)
    return x, dy, W0, A, B


def test_forward_with_zero_adapter_is_the_base_projection(oracle_mod):
    x, _, W0, A, B = _inputs(1, 19, 24, 40, 8)
    ref = _f64(x) @ _f64(W0)
    np.testing.assert_allclose(oracle_mod.lora_forward(x, W0, A, np.zeros_like(B), 2.0), ref, rtol=1e-12, atol=1e-12)
    np.testing.assert_allclose(oracle_mod.lora_forward(x, W0, np.zeros_like(A), B, 2.0), ref, rtol=1e-12, atol=1e-12)


def test_forward_rank_one_closed_form(oracle_mod):
    """W0 = 0 and r = 1: h = s (x a) b^T, an outer product."""
    x, _, W0, A, B = _inputs(2, 11, 16, 24, 1)
    s = 0.75
    h = oracle_mod.lora_forward(x, np.zeros_like(W0), A, B, s)
    ref = s * np.outer(_f64(x) @ _f64(A)[:, 0], _f64(B)[0])
    np.testing.assert_allclose(h, ref, rtol=1e-12, atol=1e-14)


def test_forward_matches_library_and_is_linear(oracle_mod):
    x, _, W0, A, B = _inputs(3, 33, 48, 40, 8)
    s = 2.0
    ref = (torch.from_numpy(_f64(x)) @ torch.from_numpy(_f64(W0))
           + s * (torch.from_numpy(_f64(x)) @ torch.from_numpy(_f64(A))) @ torch.from_numpy(_f64(B))).numpy()
    h = oracle_mod.lora_forward(x, W0, A, B, s)
    np.testing.assert_allclose(h, ref, rtol=1e-10, atol=1e-12)
    # the scale enters only the adapter term
    h0 = oracle_mod.lora_forward(x, W0, A, B, 0.0)
    h1 = oracle_mod.lora_forward(x, W0, A, B, 1.0)
    np.testing.assert_allclose(h - h0, s * (h1 - h0), rtol=1e-10, atol=1e-12)


@pytest.mark.parametrize("shape", [(32, 48, 40, 8), (17, 16, 64, 1), (64, 24, 8, 5)])
def test_input_grad_matches_autograd(oracle_mod, shape):
    L, din, dout, r = shape
    x, dy, W0, A, B = _inputs(4 + r, L, din, dout, r)
    s = 2.0
    xt = torch.from_numpy(_f64(x)).requires_grad_(True)
    h = xt @ torch.from_numpy(_f64(W0)) + s * (xt @ torch.from_numpy(_f64(A))) @ torch.from_numpy(_f64(B))
    (h * torch.from_numpy(_f64(dy))).sum().backward()
    dx = oracle_mod.lora_input_grad(dy, W0, A, B, s)
    np.testing.assert_allclose(dx, xt.grad.numpy(), rtol=1e-10, atol=1e-12)


def test_input_grad_finite_differences(oracle_mod):
    """Central differences of <dy, h(x)> with the oracle's own forward, on
    bf16-exact perturbations (x on a grid of 1/8, step 2^-6)."""
    L, din, dout, r = 3, 6, 5, 2
    rng = np.random.default_rng(5)
    xv = rng.integers(-8, 9, (L, din)).astype(np.float32) / 8
    _, dy, W0, A, B = _inputs(5, L, din, dout, r)
    s = 0.5
    dx = oracle_mod.lora_input_grad(dy, W0, A, B, s)
    dyf = _f64(dy)
    eps = np.float32(2.0 ** -6)
    fd = np.zeros((L, din))
    for j in range(L):
        for k in range(din):
            xp = xv.copy(); xp[j, k] += eps
            xm = xv.copy(); xm[j, k] -= eps
            fp = (oracle_mod.lora_forward(wk.bf16_bits(xp), W0, A, B, s) * dyf).sum()
            fm = (oracle_mod.lora_forward(wk.bf16_bits(xm), W0, A, B, s) * dyf).sum()
            fd[j, k] = (fp - fm) / (2 * float(eps))
    np.testing.assert_allclose(dx, fd, rtol=1e-9, atol=1e-11)


def test_input_grad_uses_W0_transposed(oracle_mod):
    """A slip that used W0 without the transpose (possible only when din ==
    dout) changes the result on a non-symmetric W0."""
    x, dy, W0, A, B = _inputs(6, 7, 12, 12, 4)
    dx = oracle_mod.lora_input_grad(dy, W0, A, B, 1.0)
    wrong = _f64(dy) @ _f64(W0) + (_f64(dy) @ _f64(B).T) @ _f64(A).T
    assert np.abs(dx - wrong).max() > 1e-3
