"""GPU parity of the adapter-drift KL (attt_kl_drift) against the oracle:
KL(softmax(h_p W^T) || softmax(h_q W^T)) per row and its mean.

Tolerance: |KL_gpu - KL_ref| <= 5e-5 + 1e-3 KL_ref.  Every term of the GPU's
KL comes from fp32 accumulators (logits of d bf16 products, sums of 128
exponentials per tile, online merges): the logits carry ~1e-6 relative
error and lse, E_p[z_p - z_q] a few 1e-6 absolute, so 5e-5 absolute covers
the cancellation of lse_p - lse_q for small divergences with a margin.
"""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev

pytestmark = pytest.mark.gpu

ATOL, RTOL = 5e-5, 1e-3


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _inputs(seed, L, d, V, drift):
    hq = wk.normal_bf16(seed, "klg/hq", (L, d), 1.0)
    noise = wk.bf16_to_f32(wk.normal_bf16(seed, "klg/noise", (L, d), drift))
    hp = wk.bf16_bits(wk.bf16_to_f32(hq) + noise)
    W = wk.normal_bf16(seed, "klg/W", (V, d), 0.02 if d >= 1024 else 0.1)
    return hp, hq, W


def _check(got, ref):
    err = np.abs(got.astype(np.float64) - ref)
    bad = err > ATOL + RTOL * np.abs(ref)
    assert not bad.any(), (np.flatnonzero(bad)[:5], got[bad][:5], ref[bad][:5])


@pytest.mark.parametrize("shape", [(300, 256, 5000, 0.3), (129, 72, 300, 1.0), (64, 512, 8192, 0.05),
                                   (1, 8, 1, 1.0), (257, 128, 129, 0.5)])
def test_kl_matches_oracle(attt, shape):
    L, d, V, drift = shape
    hp, hq, W = _inputs(L + V, L, d, V, drift)
    kl, mean = attt.attt_kl_drift(bf16_dev(hp), bf16_dev(hq), bf16_dev(W))
    got = kl.cpu().numpy()
    ref = oracle.kl_rows(hp, hq, W)
    _check(got, ref)
    assert abs(mean.item() - got.astype(np.float64).mean()) <= 1e-6 * max(1.0, abs(got.mean()))
    assert attt.attt_device_status() == 0


def test_equal_states_give_zero_and_calls_repeat(attt):
    L, d, V = 200, 256, 3000
    hp, hq, W = _inputs(5, L, d, V, 0.2)
    a, b = bf16_dev(hp), bf16_dev(W)
    kl0, m0 = attt.attt_kl_drift(a, a, b)
    assert torch.count_nonzero(kl0).item() == 0 and m0.item() == 0.0
    k1, m1 = attt.attt_kl_drift(a, bf16_dev(hq), b)
    k2, m2 = attt.attt_kl_drift(a, bf16_dev(hq), b)
    assert torch.equal(k1, k2) and torch.equal(m1, m2)


def test_adapter_drift_of_the_projection(attt):
    """The diagnostic as the episode uses it: h_q = x W0 (the base model),
    h_p = x W0 + s (x A) B (the adapted one), both from attt_lora_forward."""
    ew = wk.EPISODES["tiny-episode"]
    dense = wk.episode_dense(ew)
    x = wk.episode_x(ew, 1)
    W0, W = bf16_dev(dense["W0"]), bf16_dev(dense["W"])
    B = torch.from_numpy(wk.bf16_bits(20 * dense["B0"]).view(np.int16)).to(DEV).view(torch.bfloat16)
    A = bf16_dev(wk.bf16_bits(dense["A0"]))
    xd = bf16_dev(x)
    hp = attt.attt_lora_forward(xd, W0, A, B, ew.scale)
    hq = attt.attt_lora_forward(xd, W0, A, B, 0.0)
    kl, mean = attt.attt_kl_drift(hp, hq, W)
    hp_b = hp.view(torch.int16).cpu().numpy().view(np.uint16)
    hq_b = hq.view(torch.int16).cpu().numpy().view(np.uint16)
    ref = oracle.kl_rows(hp_b, hq_b, dense["W"])
    _check(kl.cpu().numpy(), ref)
    assert 1e-4 < ref.mean() < 10


@pytest.mark.slow
def test_7b_shapes_sampled_rows(attt):
    L, d, V = 2048, 3584, 152064
    hp, hq, W = _inputs(7, L, d, V, 0.1)
    kl, mean = attt.attt_kl_drift(bf16_dev(hp), bf16_dev(hq), bf16_dev(W))
    got = kl.cpu().numpy()
    rows = np.array([0, 1, 1000, 1777, L - 1], np.int64)
    _check(got[rows], oracle.kl_rows(hp, hq, W, rows))
    assert np.isfinite(got).all() and (got > -ATOL).all()
    assert abs(mean.item() - got.astype(np.float64).mean()) <= 1e-5 * abs(got.mean())


def test_bad_arguments(attt):
    a = torch.zeros(4, 16, dtype=torch.bfloat16, device=DEV)
    W = torch.zeros(10, 16, dtype=torch.bfloat16, device=DEV)
    ws = torch.empty(attt.attt_kl_workspace_bytes(4, 16, 10), dtype=torch.uint8, device=DEV)
    with pytest.raises(attt.AtttError) as e:
        attt.attt_kl_drift(a, a, W, workspace=ws[: ws.numel() // 2])
    assert e.value.code == attt.ATTT_ERR_WORKSPACE
    with pytest.raises(ValueError):
        attt.attt_kl_drift(a, a[:3], W)
