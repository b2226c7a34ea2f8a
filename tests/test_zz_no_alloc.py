"""attt_lora_grad_noalloc: the LoRA adapter gradients for callers that cannot
allocate device memory (a pool that owns all of HBM, a loop that may not call
the allocator, a plugin whose host owns every allocation).  The entry point
uses the library's static 16 MiB device scratch instead of a workspace.

Both entry points run the same deterministic kernels, so the no-allocation
call must reproduce attt_lora_grad bit for bit.  The calls come in a row and
in decreasing size (a problem whose scratch nearly fills the 16 MiB first,
then smaller ones with other inputs), so that anything left in the shared
scratch by an earlier, larger call would show.  The near-full case is also
checked against the oracle.  This file is collected last so that a run
stopping at its first failure has already run every other test."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, bits, rel_l2

pytestmark = pytest.mark.gpu

GRAD_RL2 = 2e-2  # the adapter-gradient tolerance of the LoRA parity tests


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _inputs(seed, L, din, douts, r):
    x = wk.normal_bf16(seed, "x", (L, din), 1.0)
    dys = [wk.normal_bf16(seed, f"dy{p}", (L, do), 1.0) for p, do in enumerate(douts)]
    As = [wk.normal_bf16(seed, f"A{p}", (din, r), 0.02) for p in range(len(douts))]
    Bs = [wk.normal_bf16(seed, f"B{p}", (r, do), 0.01) for p, do in enumerate(douts)]
    return x, dys, As, Bs


def _largest_L_within_scratch(attt, din, douts, r):
    """The largest row count whose scratch fits the static array (host-side
    size queries only)."""
    cap = attt.LORA_NOALLOC_SCRATCH_BYTES
    lo, hi = 1, 1 << 22
    assert attt.attt_lora_workspace_bytes(lo, din, douts, r) <= cap
    while hi - lo > 1:
        mid = (lo + hi) // 2
        if attt.attt_lora_workspace_bytes(mid, din, douts, r) <= cap:
            lo = mid
        else:
            hi = mid
    return lo


def _both(attt, host, scale=2.0):
    """(workspace entry point, no-allocation entry point) results, as numpy."""
    x, dys, As, Bs = host
    L, din = x.shape
    douts = [d.shape[1] for d in dys]
    r = As[0].shape[1]
    xd, dyd = bf16_dev(x), [bf16_dev(d) for d in dys]
    Ad, Bd = [bf16_dev(a) for a in As], [bf16_dev(b) for b in Bs]
    ref_dA, ref_dB = attt.attt_lora_grad(xd, dyd, Ad, Bd, scale)
    # outputs start as NaN, so that an element the call fails to write shows
    dA = [torch.full((din, r), float("nan"), dtype=torch.float32, device=DEV) for _ in douts]
    dB = [torch.full((r, do), float("nan"), dtype=torch.float32, device=DEV) for do in douts]
    attt.attt_lora_grad_noalloc(xd, dyd, Ad, Bd, scale, dA, dB)
    torch.cuda.synchronize()
    assert attt.attt_device_status() == 0
    np_ = lambda ts: [t.cpu().numpy() for t in ts]  # noqa: E731
    return (np_(ref_dA), np_(ref_dB)), (np_(dA), np_(dB))


def _assert_bit_equal(ref, got, what):
    for p in range(len(ref[0])):
        assert np.array_equal(bits(got[0][p]), bits(ref[0][p])), (what, "dA", p)
        assert np.array_equal(bits(got[1][p]), bits(ref[1][p])), (what, "dB", p)


def test_noalloc_matches_workspace_entry_point(attt):
    # 1. A problem whose scratch nearly fills the static array (ragged L).
    din, douts, r = 640, [640, 128], 16
    L_big = _largest_L_within_scratch(attt, din, douts, r)
    need = attt.attt_lora_workspace_bytes(L_big, din, douts, r)
    assert need > 0.9 * attt.LORA_NOALLOC_SCRATCH_BYTES, (L_big, need)
    host = _inputs(31, L_big, din, douts, r)
    ref, got = _both(attt, host)
    _assert_bit_equal(ref, got, f"near-full scratch, L={L_big}")
    x, dys, As, Bs = host
    for p in range(len(douts)):
        rA, rB = oracle.lora_grad(x, dys[p], As[p], Bs[p], 2.0)
        ea, eb = rel_l2(got[0][p], rA), rel_l2(got[1][p], rB)
        assert ea < GRAD_RL2 and eb < GRAD_RL2, (p, ea, eb)
    # 2, 3. Smaller problems with other inputs right after it (the 7B-class q
    #       and v projections, then a ragged three-projection group).
    for what, seed, L, din, douts, r in (("7b q+v", 21, 2048, 3584, [3584, 512], 16),
                                         ("ragged", 22, 300, 200, [72, 136, 8], 5)):
        assert attt.attt_lora_workspace_bytes(L, din, douts, r) < need
        ref, got = _both(attt, _inputs(seed, L, din, douts, r))
        _assert_bit_equal(ref, got, what)


def test_noalloc_rejects_problems_beyond_its_scratch(attt):
    from paper_2607_03441_gb300.attt import AtttError
    L, din, douts, r = 8192, 5120, [5120, 1024, 1024], 64  # needs more scratch than the static 16 MiB
    assert attt.attt_lora_workspace_bytes(L, din, douts, r) > attt.LORA_NOALLOC_SCRATCH_BYTES
    x = torch.zeros(L, din, dtype=torch.bfloat16, device=DEV)
    dys = [torch.zeros(L, do, dtype=torch.bfloat16, device=DEV) for do in douts]
    As = [torch.zeros(din, r, dtype=torch.bfloat16, device=DEV) for _ in douts]
    Bs = [torch.zeros(r, do, dtype=torch.bfloat16, device=DEV) for do in douts]
    dAs = [torch.empty(din, r, dtype=torch.float32, device=DEV) for _ in douts]
    dBs = [torch.empty(r, do, dtype=torch.float32, device=DEV) for do in douts]
    with pytest.raises(AtttError) as e:
        attt.attt_lora_grad_noalloc(x, dys, As, Bs, 2.0, dAs, dBs)
    assert e.value.code == 5  # ATTT_ERR_WORKSPACE
    assert attt.attt_device_status() == 0
