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


def test_injected_allocation_failure_cleans_up(attt):
    ew = wk.EPISODES["tiny-episode"]
    dense = wk.episode_dense(ew)
    args = (bf16_dev(dense["W0"]), bf16_dev(dense["W"]), f32_dev(dense["A0"]), f32_dev(dense["B0"]))
    kw = dict(n=ew.n, max_history=4 * ew.L, max_update=ew.L, scale=ew.scale, lr=1.0)
    free0 = torch.cuda.mem_get_info()[0]
    for make in (lambda: attt.History(4, 1000), lambda: attt.Episode(*args, **kw),
                 lambda: attt.Batch(*args, episodes=3, **kw)):
        attt.attt_fault_inject("alloc")
        with pytest.raises(attt.AtttError) as e:
            make()
        assert e.value.code == attt.ATTT_ERR_CUDA
        obj = make()                     # the fault was taken once: the next create works
        obj.close()
    torch.cuda.synchronize()
    assert torch.cuda.mem_get_info()[0] >= free0 - (64 << 20)  # nothing of the failed creates kept
    ep = attt.Episode(*args, **kw)       # and an update runs after it
    ep.update(i32_dev(wk.episode_texts(ew)[0]), bf16_dev(wk.episode_x(ew, 1)))
    assert attt.attt_device_status() == 0
    ep.close()


def test_injected_full_table_reaches_the_status_word(attt):
    h = attt.History(3, 1000)
    toks = i32_dev(np.arange(50, dtype=np.int32))
    attt.attt_fault_inject("table_full")
    attt.attt_history_insert(h, toks)
    assert attt.attt_history_status(h) == attt.ATTT_ERR_TABLE_FULL
    assert attt.attt_history_status(h) == 0          # read and cleared
    attt.attt_history_insert(h, toks)                 # the fault was taken: counts as usual
    q = i32_dev(np.array([[0, 1, 2], [10, 11, 12]], np.int32))
    assert attt.attt_history_count(h, q).cpu().tolist() == [1, 1]
    # a pending fault can be withdrawn; an unknown site is refused
    attt.attt_fault_inject("table_full")
    attt.attt_fault_inject("none")
    attt.attt_history_insert(h, toks)
    assert attt.attt_history_status(h) == 0
    with pytest.raises(attt.AtttError):
        attt.attt_fault_inject("disk")
    h.close()
