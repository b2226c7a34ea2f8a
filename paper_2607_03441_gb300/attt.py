"""ctypes binding of libattt (include/attt.h), argument marshalling only.

Each function has the name of the C entry point it calls and takes torch
tensors (device memory) plus an optional torch.cuda.Stream; every step of the
computation runs in the library's CUDA kernels.  There is no fallback: if
libattt.so is missing or the device is not a GB300-class part, the call
raises.
"""
from __future__ import annotations

import ctypes
import os
import threading
from typing import Optional, Sequence

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libattt.so")

ATTT_OK = 0
STATUS_NAMES = {
    0: "ATTT_OK", 1: "ATTT_ERR_INVALID_ARG", 2: "ATTT_ERR_TABLE_FULL", 3: "ATTT_ERR_TOKEN_RANGE",
    4: "ATTT_ERR_TIMEOUT", 5: "ATTT_ERR_WORKSPACE", 6: "ATTT_ERR_CUDA", 7: "ATTT_ERR_UNSUPPORTED",
    8: "ATTT_ERR_CAPACITY",
}

_lock = threading.Lock()
_lib = None


class AtttError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = int(code)
        super().__init__(f"{where}: {STATUS_NAMES.get(int(code), code)}")


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Loads libattt.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or LIB_PATH
        if not os.path.exists(p):
            raise RuntimeError(f"libattt.so not found at {p}; run paper_2607_03441_gb300.build.build()")
        lib = ctypes.CDLL(p)
        P, i64, i32, f32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        sig = {
            "attt_status_string": (ctypes.c_char_p, [i32]),
            "attt_abi_version": (i32, []),
            "attt_kernel_launches": (ctypes.c_uint64, []),
            "attt_device_status": (i32, [P]),
            "attt_history_create": (i32, [i32, i64, ctypes.POINTER(P)]),
            "attt_history_destroy": (i32, [P]),
            "attt_history_reset": (i32, [P, P]),
            "attt_history_insert": (i32, [P, P, i64, P]),
            "attt_history_length": (i64, [P]),
            "attt_history_ngram": (i32, [P]),
            "attt_history_status": (i32, [P, P]),
            "attt_history_count": (i32, [P, P, i64, P, P]),
            "attt_ngram_weights": (i32, [P, P, i64, f32, P, P]),
            "attt_ce_workspace_bytes": (sz, [i64, i64, i64]),
            "attt_weighted_ce_fwd_bwd": (i32, [P, P, P, P, i64, i64, i64, P, P, P, P, sz, P]),
            "attt_lora_workspace_bytes": (sz, [i64, i64, i32, P, i32]),
            "attt_lora_grad": (i32, [P, i64, i64, i32, P, P, P, P, i32, f32, P, P, P, sz, P]),
            "attt_lora_step": (i32, [P, P, P, P, i64, i64, i32, f32, P, P, P]),
            "attt_lora_grad_noalloc": (i32, [P, i64, i64, i32, P, P, P, P, i32, f32, P, P, P]),
            "attt_lora_forward_workspace_bytes": (sz, [i64, i64, i64, i32]),
            "attt_lora_input_grad_workspace_bytes": (sz, [i64, i64, i64, i32]),
            "attt_lora_forward": (i32, [P, P, P, P, i64, i64, i64, i32, f32, P, P, sz, P]),
            "attt_lora_input_grad": (i32, [P, P, P, P, i64, i64, i64, i32, f32, P, P, sz, P]),
        }
        for name, (res, args) in sig.items():
            fn = getattr(lib, name)
            fn.restype = res
            fn.argtypes = args
        _lib = lib
        return lib


def _check(code: int, where: str) -> None:
    if code != ATTT_OK:
        raise AtttError(code, where)


def _stream(stream: Optional[torch.cuda.Stream]) -> ctypes.c_void_p:
    s = stream if stream is not None else torch.cuda.current_stream()
    return ctypes.c_void_p(s.cuda_stream)


def _ptr(t: Optional[torch.Tensor]) -> Optional[int]:
    if t is None:
        return None
    if not t.is_cuda:
        raise ValueError("expected a CUDA tensor")
    if not t.is_contiguous():
        raise ValueError("expected a contiguous tensor")
    return t.data_ptr()


def _bf16(t: torch.Tensor) -> int:
    if t.dtype != torch.bfloat16:
        raise ValueError(f"expected bfloat16, got {t.dtype}")
    return _ptr(t)


# --------------------------------------------------------------------------
# status
# --------------------------------------------------------------------------

def attt_status_string(code: int) -> str:
    return load_library().attt_status_string(int(code)).decode()


def attt_abi_version() -> int:
    return int(load_library().attt_abi_version())


def attt_kernel_launches() -> int:
    """Kernels launched by libattt in this process so far."""
    return int(load_library().attt_kernel_launches())


def attt_device_status(stream=None) -> int:
    """Synchronises and returns (and clears) the device-side status word."""
    return int(load_library().attt_device_status(_stream(stream)))


# --------------------------------------------------------------------------
# history
# --------------------------------------------------------------------------

class History:
    """Owning handle of an attt_history (destroyed with the object)."""

    def __init__(self, n: int, max_tokens: int):
        self._lib = load_library()
        h = ctypes.c_void_p()
        _check(self._lib.attt_history_create(int(n), int(max_tokens), ctypes.byref(h)), "attt_history_create")
        self.handle = h
        self.n = int(n)
        self.max_tokens = int(max_tokens)

    def close(self) -> None:
        if getattr(self, "handle", None):
            self._lib.attt_history_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __len__(self) -> int:
        return int(self._lib.attt_history_length(self.handle))


def attt_history_create(n: int, max_tokens: int) -> History:
    return History(n, max_tokens)


def attt_history_destroy(h: History) -> None:
    h.close()


def attt_history_reset(h: History, stream=None) -> None:
    _check(load_library().attt_history_reset(h.handle, _stream(stream)), "attt_history_reset")


def attt_history_insert(h: History, tokens: torch.Tensor, stream=None) -> None:
    if tokens.dtype != torch.int32:
        raise ValueError("tokens must be int32")
    _check(load_library().attt_history_insert(h.handle, _ptr(tokens), tokens.numel(), _stream(stream)),
           "attt_history_insert")


def attt_history_length(h: History) -> int:
    return int(load_library().attt_history_length(h.handle))


def attt_history_status(h: History, stream=None) -> int:
    return int(load_library().attt_history_status(h.handle, _stream(stream)))


def attt_history_count(h: History, ngrams: torch.Tensor, out: Optional[torch.Tensor] = None,
                       stream=None) -> torch.Tensor:
    """count(g, H) for each row g of an int32 [m, n] tensor -> int32 [m]."""
    if ngrams.dtype != torch.int32 or ngrams.dim() != 2 or ngrams.shape[1] != h.n:
        raise ValueError("ngrams must be int32 [m, n]")
    m = ngrams.shape[0]
    if out is None:
        out = torch.empty(m, dtype=torch.int32, device=ngrams.device)
    _check(load_library().attt_history_count(h.handle, _ptr(ngrams), m, _ptr(out), _stream(stream)),
           "attt_history_count")
    return out


def attt_ngram_weights(h: History, tokens: torch.Tensor, w_min: float = 0.05,
                       out: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """Eq. 8 / Eq. 9 weights (fp32 [L]) of the update `tokens` (int32 [L])."""
    if tokens.dtype != torch.int32:
        raise ValueError("tokens must be int32")
    L = tokens.numel()
    if out is None:
        out = torch.empty(L, dtype=torch.float32, device=tokens.device)
    _check(load_library().attt_ngram_weights(h.handle, _ptr(tokens), L, float(w_min), _ptr(out), _stream(stream)),
           "attt_ngram_weights")
    return out


# --------------------------------------------------------------------------
# Eq. 10
# --------------------------------------------------------------------------

def attt_ce_workspace_bytes(L: int, d: int, V: int) -> int:
    return int(load_library().attt_ce_workspace_bytes(int(L), int(d), int(V)))


def attt_weighted_ce_fwd_bwd(h: torch.Tensor, W: torch.Tensor, tgt: torch.Tensor, w: torch.Tensor,
                             loss: Optional[torch.Tensor] = None, dh: Optional[torch.Tensor] = None,
                             lse: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                             stream=None):
    """Eq. 10 loss (fp32 [1]), dh (fp32 [L, d]) and optionally lse (fp32 [L])."""
    L, d = h.shape
    V = W.shape[0]
    dev = h.device
    if loss is None:
        loss = torch.empty(1, dtype=torch.float32, device=dev)
    if dh is None:
        dh = torch.empty(L, d, dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = torch.empty(attt_ce_workspace_bytes(L, d, V), dtype=torch.uint8, device=dev)
    if tgt.dtype != torch.int32 or w.dtype != torch.float32:
        raise ValueError("tgt must be int32 and w float32")
    _check(load_library().attt_weighted_ce_fwd_bwd(
        _bf16(h), _bf16(W), _ptr(tgt), _ptr(w), L, d, V, _ptr(loss), _ptr(dh), _ptr(lse),
        _ptr(workspace), workspace.numel(), _stream(stream)), "attt_weighted_ce_fwd_bwd")
    return loss, dh, lse


# --------------------------------------------------------------------------
# LoRA
# --------------------------------------------------------------------------

def attt_lora_workspace_bytes(L: int, din: int, douts: Sequence[int], r: int) -> int:
    arr = (ctypes.c_int64 * len(douts))(*[int(x) for x in douts])
    return int(load_library().attt_lora_workspace_bytes(int(L), int(din), len(douts), arr, int(r)))


def attt_lora_grad(x: torch.Tensor, dys: Sequence[torch.Tensor], As: Sequence[torch.Tensor],
                   Bs: Sequence[torch.Tensor], scale: float, dAs: Optional[Sequence[torch.Tensor]] = None,
                   dBs: Optional[Sequence[torch.Tensor]] = None, workspace: Optional[torch.Tensor] = None,
                   stream=None):
    """Adapter gradients for projections sharing the input x.  Returns (dAs, dBs)."""
    L, din = x.shape
    k = len(dys)
    r = As[0].shape[1]
    douts = [int(t.shape[1]) for t in dys]
    dev = x.device
    if dAs is None:
        dAs = [torch.empty(din, r, dtype=torch.float32, device=dev) for _ in range(k)]
    if dBs is None:
        dBs = [torch.empty(r, do, dtype=torch.float32, device=dev) for do in douts]
    if workspace is None:
        workspace = torch.empty(attt_lora_workspace_bytes(L, din, douts, r), dtype=torch.uint8, device=dev)
    P = ctypes.c_void_p
    arr = lambda ts, f: (P * k)(*[f(t) for t in ts])  # noqa: E731
    douts_arr = (ctypes.c_int64 * k)(*douts)
    _check(load_library().attt_lora_grad(
        _bf16(x), L, din, k, arr(dys, _bf16), douts_arr, arr(As, _bf16), arr(Bs, _bf16), int(r), float(scale),
        arr(dAs, _ptr), arr(dBs, _ptr), _ptr(workspace), workspace.numel(), _stream(stream)), "attt_lora_grad")
    return dAs, dBs


LORA_NOALLOC_SCRATCH_BYTES = 16 << 20


def attt_lora_grad_noalloc(x: torch.Tensor, dys: Sequence[torch.Tensor], As: Sequence[torch.Tensor],
                           Bs: Sequence[torch.Tensor], scale: float, dAs: Sequence[torch.Tensor],
                           dBs: Sequence[torch.Tensor], stream=None):
    """attt_lora_grad without a workspace: the library uses its own static
    16 MiB device scratch and allocates nothing.  The caller passes the output
    tensors.  Returns (dAs, dBs)."""
    L, din = x.shape
    k = len(dys)
    r = As[0].shape[1]
    P = ctypes.c_void_p
    arr = lambda ts, f: (P * k)(*[f(t) for t in ts])  # noqa: E731
    douts_arr = (ctypes.c_int64 * k)(*[int(t.shape[1]) for t in dys])
    _check(load_library().attt_lora_grad_noalloc(
        _bf16(x), L, din, k, arr(dys, _bf16), douts_arr, arr(As, _bf16), arr(Bs, _bf16), int(r), float(scale),
        arr(dAs, _ptr), arr(dBs, _ptr), _stream(stream)), "attt_lora_grad_noalloc")
    return dAs, dBs


def attt_lora_step(A32: torch.Tensor, B32: torch.Tensor, dA: torch.Tensor, dB: torch.Tensor, lr: float,
                   A16: Optional[torch.Tensor] = None, B16: Optional[torch.Tensor] = None, stream=None) -> None:
    """In-place SGD step on the fp32 masters and bf16 refresh (Eq. 2)."""
    din, r = A32.shape
    dout = B32.shape[1]
    _check(load_library().attt_lora_step(
        _ptr(A32), _ptr(B32), _ptr(dA), _ptr(dB), din, dout, r, float(lr),
        _bf16(A16) if A16 is not None else None, _bf16(B16) if B16 is not None else None, _stream(stream)),
        "attt_lora_step")


# --------------------------------------------------------------------------
# the adapted projection of a chained update
# --------------------------------------------------------------------------

def attt_lora_forward_workspace_bytes(L: int, din: int, dout: int, r: int) -> int:
    return int(load_library().attt_lora_forward_workspace_bytes(int(L), int(din), int(dout), int(r)))


def attt_lora_input_grad_workspace_bytes(L: int, din: int, dout: int, r: int) -> int:
    return int(load_library().attt_lora_input_grad_workspace_bytes(int(L), int(din), int(dout), int(r)))


def attt_lora_forward(x: torch.Tensor, W0: torch.Tensor, A: torch.Tensor, B: torch.Tensor, scale: float,
                      h: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                      stream=None) -> torch.Tensor:
    """h = x W0 + s (x A) B (bf16).  Returns h."""
    L, din = x.shape
    dout = W0.shape[1]
    r = A.shape[1]
    if h is None:
        h = torch.empty(L, dout, dtype=torch.bfloat16, device=x.device)
    if workspace is None:
        workspace = torch.empty(attt_lora_forward_workspace_bytes(L, din, dout, r), dtype=torch.uint8,
                                device=x.device)
    _check(load_library().attt_lora_forward(
        _bf16(x), _bf16(W0), _bf16(A), _bf16(B), L, din, dout, int(r), float(scale), _bf16(h), _ptr(workspace),
        workspace.numel(), _stream(stream)), "attt_lora_forward")
    return h


def attt_lora_input_grad(dy: torch.Tensor, W0: torch.Tensor, A: torch.Tensor, B: torch.Tensor, scale: float,
                         dx: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                         stream=None) -> torch.Tensor:
    """dx = dy W0^T + s (dy B^T) A^T (fp32).  Returns dx."""
    L, dout = dy.shape
    din = W0.shape[0]
    r = A.shape[1]
    if dx is None:
        dx = torch.empty(L, din, dtype=torch.float32, device=dy.device)
    if workspace is None:
        workspace = torch.empty(attt_lora_input_grad_workspace_bytes(L, din, dout, r), dtype=torch.uint8,
                                device=dy.device)
    _check(load_library().attt_lora_input_grad(
        _bf16(dy), _bf16(W0), _bf16(A), _bf16(B), L, din, dout, int(r), float(scale), _ptr(dx), _ptr(workspace),
        workspace.numel(), _stream(stream)), "attt_lora_input_grad")
    return dx
