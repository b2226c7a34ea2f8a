"""Failure detection on the GPU without a fault: a device-side wait that
nothing completes runs out after the library's wall-clock limit, the device
status word reports ATTT_ERR_TIMEOUT to the host, and the context keeps
working (a call after it matches the oracle)."""
import time

import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, f32_dev, i32_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def test_wait_runs_out_and_the_context_survives(attt):
    assert attt.attt_device_status() == 0
    t0 = time.monotonic()
    attt.attt_selftest_wait_timeout()
    status = attt.attt_device_status()   # synchronises, reads and clears
    waited = time.monotonic() - t0
    assert status == attt.ATTT_ERR_TIMEOUT
    assert 1.5 < waited < 60.0
    assert attt.attt_device_status() == 0  # cleared by the read
    # the context is usable: an Eq. 10 call right after matches the oracle
    L, d, V = 96, 64, 700
    h = wk.normal_bf16(3, "fail/h", (L, d), 1.0)
    W = wk.normal_bf16(3, "fail/W", (V, d), 0.1)
    tgt = wk.zipf_ids(wk.rng_for(3, "fail/t"), L, V)
    w = np.ones(L, np.float32)
    loss, _, _ = attt.attt_weighted_ce_fwd_bwd(bf16_dev(h), bf16_dev(W), i32_dev(tgt), f32_dev(w))
    ref, _, _, _ = oracle.ce_loss(h, W, tgt, w)
    assert abs(loss.item() - ref) <= 1e-3 * abs(ref)
    assert attt.attt_device_status() == 0
