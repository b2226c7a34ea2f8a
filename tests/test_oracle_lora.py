"""Pins for the oracle's LoRA adapter gradients and the SGD step (Eq. 2,
Algorithm 1's gradient step, the Appendix C adapter).

Checked against torch CPU autograd, finite differences of the adapter's
output functional, and the zero cases (B = 0 gives dA = 0; x = 0 gives
dA = dB = 0).  The SGD step is checked against numpy fp32 arithmetic and the
bf16 refresh against torch's round-to-nearest-even cast.
"""
import numpy as np
import pytest
import torch

from paper_2607_03441_gb300 import workloads as wk


def _f64(bits):
    return wk.bf16_to_f32(bits).astype(np.float64)


def _inputs(seed, L, din, dout, r, zero_B=False, zero_x=False):
    x = wk.normal_bf16(seed, "x", (L, din), 1.0)
    dy = wk.normal_bf16(seed, "dy", (L, dout), 1.0)
    A = wk.normal_bf16(seed, "A", (din, r), 0.02)
    B = wk.normal_bf16(seed, "B", (r, dout), 0.01)
    if zero_B:
        B = np.zeros_like(B)
    if zero_x:
        x = np.zeros_like(x)
    return x, dy, A, B


def _autograd(x, dy, A, B, s):
    At = torch.from_numpy(_f64(A)).requires_grad_(True)
    Bt = torch.from_numpy(_f64(B)).requires_grad_(True)
    y = s * (torch.from_numpy(_f64(x)) @ At) @ Bt
    (y * torch.from_numpy(_f64(dy))).sum().backward()
    return At.grad.numpy(), Bt.grad.numpy()


@pytest.mark.parametrize("shape", [(32, 48, 40, 8), (17, 16, 64, 1), (64, 24, 8, 5)])
def test_matches_autograd(oracle_mod, shape):
    L, din, dout, r = shape
    x, dy, A, B = _inputs(1, L, din, dout, r)
    s = 2.0
    dA, dB = oracle_mod.lora_grad(x, dy, A, B, s)
    gA, gB = _autograd(x, dy, A, B, s)
    np.testing.assert_allclose(dA, gA, rtol=1e-10, atol=1e-13)
    np.testing.assert_allclose(dB, gB, rtol=1e-10, atol=1e-13)


def test_zero_B_gives_zero_dA(oracle_mod):
    x, dy, A, B = _inputs(2, 40, 32, 24, 8, zero_B=True)
    dA, dB = oracle_mod.lora_grad(x, dy, A, B, 2.0)
    assert np.all(dA == 0.0)
    assert np.any(dB != 0.0)


def test_zero_x_gives_zero_grads(oracle_mod):
    x, dy, A, B = _inputs(3, 40, 32, 24, 8, zero_x=True)
    dA, dB = oracle_mod.lora_grad(x, dy, A, B, 2.0)
    assert np.all(dA == 0.0) and np.all(dB == 0.0)


def test_finite_differences(oracle_mod):
    """F(A, B) = sum(s (xA)B * dy) is bilinear, so its central differences are
    exact up to rounding; perturb single entries of A and B."""
    L, din, dout, r, s = 6, 5, 7, 3, 2.0
    x, dy, A, B = _inputs(4, L, din, dout, r)
    xf, dyf, Af, Bf = _f64(x), _f64(dy), _f64(A), _f64(B)
    dA, dB = oracle_mod.lora_grad(x, dy, A, B, s)

    def F(Am, Bm):
        return float(np.sum(s * (xf @ Am) @ Bm * dyf))

    eps = 1e-3
    for i in range(din):
        for c in range(r):
            Ap, Am = Af.copy(), Af.copy()
            Ap[i, c] += eps; Am[i, c] -= eps
            assert (F(Ap, Bf) - F(Am, Bf)) / (2 * eps) == pytest.approx(dA[i, c], rel=1e-8, abs=1e-10)
    for c in range(r):
        for o in range(dout):
            Bp, Bm = Bf.copy(), Bf.copy()
            Bp[c, o] += eps; Bm[c, o] -= eps
            assert (F(Af, Bp) - F(Af, Bm)) / (2 * eps) == pytest.approx(dB[c, o], rel=1e-8, abs=1e-10)


def test_rank_one_outer_products(oracle_mod):
    """r = 1: dB = s (x a)^T dy is the dy-weighted sum of rows, dA = s x^T (dy b)."""
    x, dy, A, B = _inputs(5, 30, 12, 9, 1)
    dA, dB = oracle_mod.lora_grad(x, dy, A, B, 1.5)
    u = _f64(x) @ _f64(A)[:, 0]
    v = _f64(dy) @ _f64(B)[0, :]
    np.testing.assert_allclose(dB[0], 1.5 * np.einsum("l,lo->o", u, _f64(dy)), rtol=1e-12)
    np.testing.assert_allclose(dA[:, 0], 1.5 * np.einsum("li,l->i", _f64(x), v), rtol=1e-12)


def test_sgd_step_closed_form(oracle_mod):
    rng = np.random.default_rng(1)
    p = rng.standard_normal(1000).astype(np.float32)
    g = rng.standard_normal(1000).astype(np.float32)
    lr = np.float32(5e-4)
    new, b = oracle_mod.sgd_step(p, g, float(lr))
    ref = p - (lr * g).astype(np.float32)
    np.testing.assert_array_equal(new, ref.astype(np.float32))
    ref16 = torch.from_numpy(new).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(b, ref16)


def test_bf16_round_to_nearest_even(oracle_mod):
    vals = np.array([1.0, 1.00390625, 1.005859375, -2.5, 3.0e38, 1e-40, 0.0, -0.0], np.float32)
    ref = torch.from_numpy(vals).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle_mod.to_bf16(vals), ref)
