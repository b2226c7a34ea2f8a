"""GPU parity of the adapted projection of a chained update against the CPU
oracle: the forward h = x W0 + s (x A) B (bf16 out) and the input gradient
dx = dy W0^T + s (dy B^T) A^T (fp32 out).

Tolerances: h within 1e-2 relative L2 (h is rounded to bf16, 2^-9 per
element, and s (x A) to bf16 once); dx within 2e-2 relative L2 (the adapter
gradients' bar; s (dy B^T) is rounded to bf16 once).  Rows are independent,
so large shapes are checked on sampled rows.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, rel_l2

pytestmark = pytest.mark.gpu

H_RL2 = 1e-2
DX_RL2 = 2e-2


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _inputs(seed, L, din, dout, r):
    x = wk.normal_bf16(seed, "x", (L, din), 1.0)
    dy = wk.normal_bf16(seed, "dy", (L, dout), 1.0)
    W0 = wk.normal_bf16(seed, "W0", (din, dout), 0.03)
    A = wk.normal_bf16(seed, "A", (din, r), 0.05)
    B = wk.normal_bf16(seed, "B", (r, dout), 0.05)
    return x, dy, W0, A, B


def _rows(L, k, seed):
    if L <= k:
        return np.arange(L)
    rng = np.random.default_rng(seed)
    return np.unique(np.concatenate([[0, L - 1], rng.choice(L, k - 2, replace=False)]))


@pytest.mark.parametrize("shape", [(256, 512, 512, 8), (100, 512, 384, 16), (300, 200, 136, 16), (129, 64, 264, 5),
                                   (2048, 3584, 3584, 16)])
def test_forward(attt, shape):
    L, din, dout, r = shape
    x, _, W0, A, B = _inputs(L + din, L, din, dout, r)
    s = 2.0
    h = attt.attt_lora_forward(bf16_dev(x), bf16_dev(W0), bf16_dev(A), bf16_dev(B), s)
    assert attt.attt_device_status() == 0
    h = h.float().cpu().numpy()
    rows = _rows(L, 24, L)
    ref = oracle.lora_forward(x[rows], W0, A, B, s)
    e = rel_l2(h[rows], ref)
    assert e < H_RL2, e


@pytest.mark.parametrize("shape", [(256, 512, 512, 8), (100, 512, 384, 16), (300, 200, 136, 16), (2048, 3584, 3584, 16),
                                   (1280, 1280, 1280, 64)])
def test_input_grad(attt, shape):
    L, din, dout, r = shape
    _, dy, W0, A, B = _inputs(L + dout, L, din, dout, r)
    s = 2.0
    args = (bf16_dev(dy), bf16_dev(W0), bf16_dev(A), bf16_dev(B), s)
    dx = attt.attt_lora_input_grad(*args)
    dx2 = attt.attt_lora_input_grad(*args)
    assert attt.attt_device_status() == 0
    dx, dx2 = dx.cpu().numpy(), dx2.cpu().numpy()
    np.testing.assert_array_equal(dx.view(np.uint32), dx2.view(np.uint32))  # deterministic
    rows = _rows(L, 24, L + 1)
    ref = oracle.lora_input_grad(dy[rows], W0, A, B, s)
    e = rel_l2(dx[rows], ref)
    assert e < DX_RL2, e


def test_zero_adapter_forward_is_the_base_projection(attt):
    L, din, dout, r = 200, 256, 512, 16
    x, _, W0, A, B = _inputs(7, L, din, dout, r)
    h = attt.attt_lora_forward(bf16_dev(x), bf16_dev(W0), bf16_dev(A), bf16_dev(np.zeros_like(B)), 2.0)
    ref = oracle.lora_forward(x, W0, A, np.zeros_like(B), 2.0)
    assert rel_l2(h.float().cpu().numpy(), ref) < H_RL2


def test_launch_counts_and_arguments(attt):
    from paper_2607_03441_gb300.attt import AtttError
    L, din, dout, r = 256, 256, 256, 16
    x, dy, W0, A, B = _inputs(8, L, din, dout, r)
    xd, dyd, W0d, Ad, Bd = (bf16_dev(t) for t in (x, dy, W0, A, B))
    attt.attt_lora_forward(xd, W0d, Ad, Bd, 1.0)
    n0 = attt.attt_kernel_launches()
    attt.attt_lora_forward(xd, W0d, Ad, Bd, 1.0)
    assert attt.attt_kernel_launches() - n0 == 3  # prep, s (x A), the contraction
    n0 = attt.attt_kernel_launches()
    attt.attt_lora_input_grad(dyd, W0d, Ad, Bd, 1.0)
    assert attt.attt_kernel_launches() - n0 == 2  # s (dy B^T), the contraction
    A12 = bf16_dev(wk.normal_bf16(9, "A", (din, 12), 0.05))
    B12 = bf16_dev(wk.normal_bf16(9, "B", (12, dout), 0.05))
    with pytest.raises(AtttError):  # r % 8 != 0: A cannot be read in place
        attt.attt_lora_input_grad(dyd, W0d, A12, B12, 1.0)
    with pytest.raises(AtttError):  # din not a multiple of 8
        attt.attt_lora_forward(torch.zeros(L, 36, dtype=torch.bfloat16, device=DEV),
                               torch.zeros(36, dout, dtype=torch.bfloat16, device=DEV),
                               torch.zeros(36, r, dtype=torch.bfloat16, device=DEV), Bd, 1.0)
