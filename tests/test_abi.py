"""The C-ABI library builds, loads without a GPU and exports every entry point
that include/attt.h declares; host-only calls answer without a device."""
import ctypes
import os
import re
import subprocess

import pytest

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "attt.h")


def declared_symbols():
    text = open(HEADER).read()
    return sorted(set(re.findall(r"ATTT_API[^;(]*?\b(attt_\w+)\s*\(", text)))


@pytest.fixture(scope="module")
def lib_path():
    from paper_2607_03441_gb300 import build
    return build.build()


def test_header_declares_the_update_calls():
    names = declared_symbols()
    for must in ("attt_history_insert", "attt_ngram_weights", "attt_weighted_ce_fwd_bwd", "attt_lora_grad",
                 "attt_lora_step"):
        assert must in names


def test_library_exports_every_declared_symbol(lib_path):
    out = subprocess.run(["nm", "-D", "--defined-only", lib_path], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (attt_\w+)", out))
    missing = [s for s in declared_symbols() if s not in exported]
    assert not missing, f"not exported: {missing}"
    lib = ctypes.CDLL(lib_path)
    for s in declared_symbols():
        assert getattr(lib, s) is not None


def test_host_only_calls(lib_path):
    from paper_2607_03441_gb300 import attt
    assert attt.attt_abi_version() == 100
    assert attt.attt_status_string(0) == "ATTT_OK"
    assert attt.attt_status_string(8) == "ATTT_ERR_CAPACITY"
    assert attt.attt_status_string(99) == "ATTT_ERR_UNKNOWN"
    assert attt.attt_ce_workspace_bytes(256, 512, 8192) > 0
    assert attt.attt_ce_workspace_bytes(0, 512, 8192) == 0
    assert attt.attt_lora_workspace_bytes(256, 512, [512], 8) > 0
    assert attt.attt_lora_workspace_bytes(256, 512, [512], 65) == 0


def test_product_has_no_oracle_or_cpu_path():
    """Nothing on the product path imports the oracle or falls back to torch
    compute: the binding only marshals arguments to libattt."""
    pkg = os.path.join(ROOT, "paper_2607_03441_gb300")
    for dirpath, _, files in os.walk(pkg):
        for f in files:
            if f.endswith((".py", ".cu", ".cuh", ".h")):
                src = open(os.path.join(dirpath, f)).read()
                assert "import oracle" not in src and "from oracle" not in src, f
                assert "liboracle" not in src, f
    binding = open(os.path.join(pkg, "attt.py")).read()
    for forbidden in ("torch.matmul", "F.cross_entropy", "torch.nn.functional", "@ ", ".mm("):
        assert forbidden not in binding


def test_missing_library_fails_loudly(tmp_path):
    from paper_2607_03441_gb300 import attt
    saved = attt._lib
    try:
        attt._lib = None
        with pytest.raises(RuntimeError):
            attt.load_library(str(tmp_path / "nope.so"))
    finally:
        attt._lib = saved


def test_fault_injection_switch_is_host_only():
    """attt_fault_inject only arms a host-side fault (no device needed)."""
    from paper_2607_03441_gb300 import attt
    attt.attt_fault_inject("table_full")
    attt.attt_fault_inject("alloc")
    attt.attt_fault_inject("none")
    with pytest.raises(attt.AtttError):
        attt.attt_fault_inject("network")


def test_checked_build_exports_the_same_calls():
    """The checked build (-DATTT_CHECKED=1: device-side bounds checks) builds
    and exports every declared entry point, as the normal build does."""
    from paper_2607_03441_gb300 import build
    path = build.build(checked=True)
    out = subprocess.run(["nm", "-D", "--defined-only", path], capture_output=True, text=True, check=True).stdout
    exported = set(re.findall(r"\bT (attt_\w+)", out))
    assert not [s for s in declared_symbols() if s not in exported]
    assert ctypes.CDLL(path).attt_status_string(9) is not None


def test_ce_workspace_max_is_the_maximum_over_lengths(lib_path):
    """attt_ce_workspace_max_bytes(Lmax) equals the largest
    attt_ce_workspace_bytes(L) over every L <= Lmax (host-only; the size is
    not monotone in L because the vocabulary chunk depends on L)."""
    from paper_2607_03441_gb300 import attt
    lib = attt.load_library()
    assert attt.attt_ce_workspace_max_bytes(0, 512, 8192) == 0
    for Lmax, d, V in ((256, 512, 8192), (2048, 3584, 152064), (4096, 4096, 128256), (9000, 5120, 152064),
                       (40000, 3584, 152064), (3000, 64, 300), (5000, 128, 100000)):
        exhaustive = max(lib.attt_ce_workspace_bytes(L, d, V) for L in range(1, Lmax + 1))
        assert attt.attt_ce_workspace_max_bytes(Lmax, d, V) == exhaustive, (Lmax, d, V)


def test_binding_rejects_mismatched_shapes():
    """The C ABI takes sizes on trust, so the binding checks every tensor's
    shape and dtype against the sizes it passes (host-only: the checks run
    before any pointer is taken)."""
    import torch
    from paper_2607_03441_gb300 import attt
    bf, f32 = torch.bfloat16, torch.float32
    x = torch.zeros(8, 16, dtype=bf)
    with pytest.raises(ValueError, match="dys"):
        attt.attt_lora_grad(x, [torch.zeros(7, 32, dtype=bf)], [torch.zeros(16, 4, dtype=bf)],
                            [torch.zeros(4, 32, dtype=bf)], 2.0)
    with pytest.raises(ValueError, match="Bs"):
        attt.attt_lora_grad(x, [torch.zeros(8, 32, dtype=bf)], [torch.zeros(16, 4, dtype=bf)],
                            [torch.zeros(4, 24, dtype=bf)], 2.0)
    with pytest.raises(ValueError, match="one entry per projection"):
        attt.attt_lora_grad(x, [torch.zeros(8, 32, dtype=bf)] * 2, [torch.zeros(16, 4, dtype=bf)],
                            [torch.zeros(4, 32, dtype=bf)], 2.0)
    with pytest.raises(ValueError, match="tgt"):
        attt.attt_weighted_ce_fwd_bwd(x, torch.zeros(10, 16, dtype=bf), torch.zeros(7, dtype=torch.int32),
                                      torch.zeros(8, dtype=f32))
    with pytest.raises(ValueError, match="W"):
        attt.attt_weighted_ce_fwd_bwd(x, torch.zeros(10, 12, dtype=bf), torch.zeros(8, dtype=torch.int32),
                                      torch.zeros(8, dtype=f32))
    with pytest.raises(ValueError, match="dB"):
        attt.attt_lora_step(torch.zeros(16, 4), torch.zeros(4, 32), torch.zeros(16, 4), torch.zeros(4, 31), 1e-3)
    with pytest.raises(ValueError, match="B"):
        attt.attt_lora_forward(x, torch.zeros(16, 32, dtype=bf), torch.zeros(16, 4, dtype=bf),
                               torch.zeros(4, 33, dtype=bf), 2.0)
    with pytest.raises(ValueError, match="dx"):
        attt.attt_lora_input_grad(torch.zeros(8, 32, dtype=bf), torch.zeros(16, 32, dtype=bf),
                                  torch.zeros(16, 4, dtype=bf), torch.zeros(4, 32, dtype=bf), 2.0,
                                  dx=torch.zeros(8, 15))


def test_noalloc_scratch_size_matches_the_header():
    """The binding's size constant is the header's ATTT_LORA_NOALLOC_SCRATCH_BYTES."""
    from paper_2607_03441_gb300 import attt
    m = re.search(r"#define\s+ATTT_LORA_NOALLOC_SCRATCH_BYTES\s+\(\(size_t\)(\d+)\s*<<\s*(\d+)\)", open(HEADER).read())
    assert m, "ATTT_LORA_NOALLOC_SCRATCH_BYTES not found in include/attt.h"
    assert int(m.group(1)) << int(m.group(2)) == attt.LORA_NOALLOC_SCRATCH_BYTES
    src = open(os.path.join(ROOT, "paper_2607_03441_gb300", "csrc", "lora_noalloc.cu")).read()
    assert re.search(r"static __device__ __align__\(256\) unsigned char g_scratch\[kScratchBytes\]", src)
    assert "kScratchBytes = ATTT_LORA_NOALLOC_SCRATCH_BYTES" in src


@pytest.mark.parametrize("entry", ["attt_lora_grad", "attt_lora_grad_noalloc"])
def test_lora_entry_points_check_arguments_before_any_call(entry):
    """A wrong dtype, shape or list length raises ValueError on the host,
    before a pointer reaches the C ABI (CPU tensors: nothing could launch)."""
    import torch
    from paper_2607_03441_gb300 import attt
    L, din, douts, r = 32, 16, [24, 8], 4
    bf = torch.bfloat16

    def args(**over):
        a = dict(x=torch.zeros(L, din, dtype=bf), dys=[torch.zeros(L, d, dtype=bf) for d in douts],
                 As=[torch.zeros(din, r, dtype=bf) for _ in douts], Bs=[torch.zeros(r, d, dtype=bf) for d in douts],
                 dAs=[torch.zeros(din, r) for _ in douts], dBs=[torch.zeros(r, d) for d in douts])
        a.update(over)
        return a

    bad = {
        "dys[1]": args(dys=[torch.zeros(L, 24, dtype=bf), torch.zeros(L, 8)]),             # fp32 dy
        "As[0]": args(As=[torch.zeros(din + 1, r, dtype=bf), torch.zeros(din, r, dtype=bf)]),
        "Bs[1]": args(Bs=[torch.zeros(r, 24, dtype=bf), torch.zeros(r, 16, dtype=bf)]),    # narrower than dout
        "dAs[0]": args(dAs=[torch.zeros(din, r, dtype=bf), torch.zeros(din, r)]),           # bf16 gradient
        "dBs[1]": args(dBs=[torch.zeros(r, 24), torch.zeros(r, 4)]),                       # smaller than r x dout
        "x": args(x=torch.zeros(L, din)),                                                    # fp32 x
        "one entry per projection": args(Bs=[torch.zeros(r, 24, dtype=bf)]),
    }
    fn = getattr(attt, entry)
    for name, a in bad.items():
        with pytest.raises(ValueError, match=re.escape(name)):
            fn(a["x"], a["dys"], a["As"], a["Bs"], 2.0, a["dAs"], a["dBs"])
