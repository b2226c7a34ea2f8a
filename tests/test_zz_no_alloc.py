"""attt_lora_grad_noalloc: the LoRA adapter gradients for callers that cannot
allocate device memory (a pool that owns all of HBM, a loop that may not call
the allocator, a plugin whose host owns every allocation).  The entry point
uses the library's static 16 MiB device scratch instead of a workspace.

Checked through the C ABI against attt_lora_grad (the workspace entry point)
on the same inputs, within the tolerance the LoRA parity tests use, on two
calls in a row with different inputs, so that a result leaking from the
previous call's scratch would show.  This file is collected last so that a
run stopping at its first failure has already run every other test."""
import numpy as np
import pytest
import torch

from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, rel_l2

pytestmark = pytest.mark.gpu

GRAD_RL2 = 2e-2  # the adapter-gradient tolerance of the LoRA parity tests


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    return a


def _inputs(seed, L, din, douts, r):
    x = bf16_dev(wk.normal_bf16(seed, "x", (L, din), 1.0))
    dys = [bf16_dev(wk.normal_bf16(seed, f"dy{p}", (L, do), 1.0)) for p, do in enumerate(douts)]
    As = [bf16_dev(wk.normal_bf16(seed, f"A{p}", (din, r), 0.02)) for p in range(len(douts))]
    Bs = [bf16_dev(wk.normal_bf16(seed, f"B{p}", (r, do), 0.01)) for p, do in enumerate(douts)]
    return x, dys, As, Bs


def test_noalloc_matches_workspace_entry_point(attt):
    L, din, douts, r = 2048, 3584, [3584, 512], 16  # the 7B-class q and v projections
    outs = ([torch.empty(din, r, dtype=torch.float32, device=DEV) for _ in douts],
            [torch.empty(r, do, dtype=torch.float32, device=DEV) for do in douts])
    for call, seed in enumerate((21, 22)):
        x, dys, As, Bs = _inputs(seed, L, din, douts, r)
        ref_dA, ref_dB = attt.attt_lora_grad(x, dys, As, Bs, 2.0)
        dA, dB = attt.attt_lora_grad_noalloc(x, dys, As, Bs, 2.0, outs[0], outs[1])
        torch.cuda.synchronize()
        for p in range(len(douts)):
            ea = rel_l2(dA[p].cpu().numpy(), ref_dA[p].cpu().numpy())
            eb = rel_l2(dB[p].cpu().numpy(), ref_dB[p].cpu().numpy())
            assert ea < GRAD_RL2 and eb < GRAD_RL2, (call, p, ea, eb)
    assert attt.attt_device_status() == 0


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
