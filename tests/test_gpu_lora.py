"""GPU parity of the LoRA adapter gradients and the SGD step against the CPU
oracle.  Gradients within 2e-2 relative L2 per tensor (bf16 inputs, fp32
accumulation, u and v rounded to bf16 once); exact zeros where the
mathematics gives zeros; the SGD step bit-exact."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, f32_dev, rel_l2

pytestmark = pytest.mark.gpu

GRAD_RL2 = 2e-2


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _group(attt, x, dys, As, Bs, scale):
    dAs, dBs = attt.attt_lora_grad(bf16_dev(x), [bf16_dev(d) for d in dys], [bf16_dev(a) for a in As],
                                   [bf16_dev(b) for b in Bs], scale)
    assert attt.attt_device_status() == 0
    return [t.cpu().numpy() for t in dAs], [t.cpu().numpy() for t in dBs]


def _check_group(attt, x, dys, As, Bs, scale=2.0):
    gA, gB = _group(attt, x, dys, As, Bs, scale)
    for p in range(len(dys)):
        rA, rB = oracle.lora_grad(x, dys[p], As[p], Bs[p], scale)
        ea, eb = rel_l2(gA[p], rA), rel_l2(gB[p], rB)
        assert ea < GRAD_RL2 and eb < GRAD_RL2, (p, ea, eb)
    return gA, gB


def _inputs(seed, L, din, douts, r):
    x = wk.normal_bf16(seed, "x", (L, din), 1.0)
    dys = [wk.normal_bf16(seed, f"dy{p}", (L, do), 1.0) for p, do in enumerate(douts)]
    As = [wk.normal_bf16(seed, f"A{p}", (din, r), 0.02) for p in range(len(douts))]
    Bs = [wk.normal_bf16(seed, f"B{p}", (r, do), 0.01) for p, do in enumerate(douts)]
    return x, dys, As, Bs


@pytest.mark.parametrize("L,din,douts,r", [(256, 512, [512], 8), (300, 200, [72, 136], 5), (100, 64, [64], 1),
                                          (513, 384, [256, 128, 64], 64), (64, 8, [8], 16), (1000, 256, [1024], 32)])
def test_shapes(attt, L, din, douts, r):
    _check_group(attt, *_inputs(L + din, L, din, douts, r))


def test_largest_group(attt):
    """Eight projections on one x (the largest group), ragged douts."""
    douts = [64, 72, 128, 200, 8, 136, 256, 24]
    _check_group(attt, *_inputs(99, 330, 136, douts, 12))


def test_zero_B_and_zero_x(attt):
    x, dys, As, Bs = _inputs(7, 200, 128, [96], 8)
    gA, gB = _group(attt, x, dys, As, [np.zeros_like(Bs[0])], 2.0)
    assert np.all(gA[0] == 0.0)
    gA, gB = _group(attt, np.zeros_like(x), dys, As, Bs, 2.0)
    assert np.all(gA[0] == 0.0) and np.all(gB[0] == 0.0)


def test_tiny_chained_from_ce(attt):
    """Tiny config: dy of the projection is the Eq. 10 gradient dh cast to bf16,
    each side chaining its own dh (the oracle its fp64 dh)."""
    wl = wk.WORKLOADS["tiny"]
    H = wk.history_tokens(wl)
    xt = wk.update_tokens(wl, H)
    w = oracle.ngram_weights(H, xt, wl.n)
    dense = wk.dense_inputs(wl)
    _, dh, _ = attt.attt_weighted_ce_fwd_bwd(bf16_dev(dense["h"]), bf16_dev(dense["W"]),
                                             torch.from_numpy(xt).to(DEV), f32_dev(w))
    dy_gpu = dh.to(torch.bfloat16)
    _, _, _, rdh = oracle.ce_loss(dense["h"], dense["W"], xt, w)
    dy_ref = wk.bf16_bits(rdh.astype(np.float32))
    x, A, B = dense["x/proj"], dense["A/proj"], dense["B/proj"]
    dAs, dBs = attt.attt_lora_grad(bf16_dev(x), [dy_gpu], [bf16_dev(A)], [bf16_dev(B)], wl.scale)
    rA, rB = oracle.lora_grad(x, dy_ref, A, B, wl.scale)
    assert rel_l2(dAs[0].cpu().numpy(), rA) < GRAD_RL2
    assert rel_l2(dBs[0].cpu().numpy(), rB) < GRAD_RL2
    # and with the same dy on both sides
    _check_group(attt, x, [dy_ref], [A], [B], wl.scale)


def _workload_groups(name):
    wl = wk.WORKLOADS[name]
    dense = wk.dense_inputs(wl, with_lm_head=False)
    groups = {}
    for p in wl.projs:
        groups.setdefault(p.x_group, []).append(p)
    return wl, dense, groups


@pytest.mark.parametrize("name", ["7b", "long", "32b"])
def test_workload(attt, name):
    wl, dense, groups = _workload_groups(name)
    for g, projs in groups.items():
        x = dense[f"x/{projs[0].name}"]
        _check_group(attt, x, [dense[f"dy/{p.name}"] for p in projs], [dense[f"A/{p.name}"] for p in projs],
                     [dense[f"B/{p.name}"] for p in projs], wl.scale)


def _offset_view(arr, dtype, off):
    """A contiguous device copy of arr that starts `off` elements into its
    allocation (off = 1 leaves it without 16-byte alignment)."""
    n = int(np.prod(arr.shape))
    buf = torch.empty(n + off, dtype=dtype, device=DEV)
    v = buf[off:].view(*arr.shape)
    if arr.dtype != np.float32 or dtype != torch.float32:
        return v
    v.copy_(torch.from_numpy(arr))
    return v


@pytest.mark.parametrize("din,dout,r,off", [(384, 200, 16, 0), (37, 19, 3, 1), (130, 66, 5, 1), (64, 64, 4, 2)])
def test_sgd_step_bit_exact(attt, din, dout, r, off):
    """Both the four-wide path (aligned, sizes a multiple of four) and the
    one-wide path (offset buffers, ragged sizes) against the oracle."""
    rng = np.random.default_rng(din + dout + r + off)
    A = rng.standard_normal((din, r)).astype(np.float32) * 0.02
    B = rng.standard_normal((r, dout)).astype(np.float32) * 0.01
    dA = rng.standard_normal((din, r)).astype(np.float32)
    dB = rng.standard_normal((r, dout)).astype(np.float32)
    A32, B32 = _offset_view(A, torch.float32, off), _offset_view(B, torch.float32, off)
    A16 = _offset_view(A, torch.bfloat16, off)
    B16 = _offset_view(B, torch.bfloat16, off)
    attt.attt_lora_step(A32, B32, _offset_view(dA, torch.float32, off), _offset_view(dB, torch.float32, off), 5e-4,
                        A16, B16)
    pA, bA = oracle.sgd_step(A, dA, 5e-4)
    pB, bB = oracle.sgd_step(B, dB, 5e-4)
    np.testing.assert_array_equal(A32.cpu().numpy(), pA)
    np.testing.assert_array_equal(B32.cpu().numpy(), pB)
    np.testing.assert_array_equal(A16.view(torch.int16).cpu().numpy().view(np.uint16), bA)
    np.testing.assert_array_equal(B16.view(torch.int16).cpu().numpy().view(np.uint16), bB)


def test_launch_counter_counts_every_kernel(attt):
    """Two projections: prep, pass 1 (u and both v, grouped), pass 2 (dA and
    both dB, grouped) = 3 kernels; the SGD step is one more."""
    x, dys, As, Bs = _inputs(9, 200, 128, [64, 128], 8)
    n0 = attt.attt_kernel_launches()
    _group(attt, x, dys, As, Bs, 2.0)
    assert attt.attt_kernel_launches() - n0 == 3
    A32 = f32_dev(np.zeros((128, 8), np.float32))
    B32 = f32_dev(np.zeros((8, 64), np.float32))
    n1 = attt.attt_kernel_launches()
    attt.attt_lora_step(A32, B32, torch.zeros_like(A32), torch.zeros_like(B32), 5e-4)
    assert attt.attt_kernel_launches() - n1 == 1


@pytest.mark.parametrize("L,din,douts,r", [
    (2000, 3584, [3584, 512], 16),                               # ragged last row tile, tiles split over CTAs
    (1500, 256, [64, 72, 128, 200, 8, 136, 256, 24], 40),        # 8 x 48 = 384 rank columns: two N tiles
    (777, 1032, [520, 1032], 64),                                # ragged din / dout tiles
])
def test_ragged_shapes_and_repeatability(attt, L, din, douts, r):
    """Ragged row, din and dout tiles, a group whose rank columns take two N
    tiles of u and dA, and the stream-K split of long tiles; two calls give
    the same bits."""
    host = _inputs(L + r, L, din, douts, r)
    gA, gB = _check_group(attt, *host)
    hA, hB = _group(attt, *host, 2.0)
    for p in range(len(douts)):
        assert np.array_equal(gA[p].view(np.uint32), hA[p].view(np.uint32)), ("dA", p)
        assert np.array_equal(gB[p].view(np.uint32), hB[p].view(np.uint32)), ("dB", p)
