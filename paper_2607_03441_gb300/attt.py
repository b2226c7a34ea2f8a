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
from typing import Optional, Sequence, Tuple

import torch

_HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_HERE, "libattt.so")
# ATTT_CHECKED=1 selects the checked build (device-side bounds checks)
LIB_CHECKED_PATH = os.path.join(_HERE, "libattt_checked.so")

ATTT_OK = 0
ATTT_ERR_INVALID_ARG = 1
ATTT_ERR_TABLE_FULL = 2
ATTT_ERR_TOKEN_RANGE = 3
ATTT_ERR_TIMEOUT = 4
ATTT_ERR_WORKSPACE = 5
ATTT_ERR_CUDA = 6
ATTT_ERR_UNSUPPORTED = 7
ATTT_ERR_CAPACITY = 8
ATTT_ERR_CHECK = 9
STATUS_NAMES = {
    0: "ATTT_OK", 1: "ATTT_ERR_INVALID_ARG", 2: "ATTT_ERR_TABLE_FULL", 3: "ATTT_ERR_TOKEN_RANGE",
    4: "ATTT_ERR_TIMEOUT", 5: "ATTT_ERR_WORKSPACE", 6: "ATTT_ERR_CUDA", 7: "ATTT_ERR_UNSUPPORTED",
    8: "ATTT_ERR_CAPACITY", 9: "ATTT_ERR_CHECK",
}

_lock = threading.Lock()
_lib = None


class AtttError(RuntimeError):
    def __init__(self, code: int, where: str):
        self.code = int(code)
        super().__init__(f"{where}: {STATUS_NAMES.get(int(code), code)}")


class EpisodeConfig(ctypes.Structure):
    """attt_episode_config (field order and types as in attt.h)."""
    _fields_ = [("n", ctypes.c_int), ("w_min", ctypes.c_float), ("max_history", ctypes.c_int64),
                ("max_update", ctypes.c_int64), ("din", ctypes.c_int64), ("d", ctypes.c_int64),
                ("V", ctypes.c_int64), ("r", ctypes.c_int), ("scale", ctypes.c_float), ("lr", ctypes.c_float),
                ("grad_steps", ctypes.c_int), ("cadence", ctypes.c_int), ("optimizer", ctypes.c_int),
                ("beta1", ctypes.c_double), ("beta2", ctypes.c_double), ("eps", ctypes.c_double),
                ("weight_decay", ctypes.c_double)]


class BatchConfig(ctypes.Structure):
    """attt_batch_config (field order and types as in attt.h)."""
    _fields_ = [("episodes", ctypes.c_int), ("n", ctypes.c_int), ("w_min", ctypes.c_float),
                ("max_history", ctypes.c_int64), ("max_update", ctypes.c_int64), ("din", ctypes.c_int64),
                ("d", ctypes.c_int64), ("V", ctypes.c_int64), ("r", ctypes.c_int), ("scale", ctypes.c_float),
                ("lr", ctypes.c_float), ("grad_steps", ctypes.c_int)]


def load_library(path: Optional[str] = None) -> ctypes.CDLL:
    """Loads libattt.so (raises if it has not been built)."""
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        p = path or (LIB_CHECKED_PATH if os.environ.get("ATTT_CHECKED") == "1" else LIB_PATH)
        if not os.path.exists(p):
            raise RuntimeError(f"libattt.so not found at {p}; run paper_2607_03441_gb300.build.build()")
        lib = ctypes.CDLL(p)
        P, i64, i32, f32, sz = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int, ctypes.c_float, ctypes.c_size_t
        f64 = ctypes.c_double
        sig = {
            "attt_status_string": (ctypes.c_char_p, [i32]),
            "attt_abi_version": (i32, []),
            "attt_kernel_launches": (ctypes.c_uint64, []),
            "attt_device_status": (i32, [P]),
            "attt_selftest_wait_timeout": (i32, [P]),
            "attt_fault_inject": (i32, [ctypes.c_char_p]),
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
            "attt_ce_workspace_max_bytes": (sz, [i64, i64, i64]),
            "attt_weighted_ce_fwd_bwd": (i32, [P, P, P, P, i64, i64, i64, P, P, P, P, sz, P]),
            "attt_lora_workspace_bytes": (sz, [i64, i64, i32, P, i32]),
            "attt_lora_grad": (i32, [P, i64, i64, i32, P, P, P, P, i32, f32, P, P, P, sz, P]),
            "attt_lora_step": (i32, [P, P, P, P, i64, i64, i32, f32, P, P, P]),
            "attt_lora_grad_noalloc": (i32, [P, i64, i64, i32, P, P, P, P, i32, f32, P, P, P]),
            "attt_lora_forward_workspace_bytes": (sz, [i64, i64, i64, i32]),
            "attt_lora_input_grad_workspace_bytes": (sz, [i64, i64, i64, i32]),
            "attt_lora_forward": (i32, [P, P, P, P, i64, i64, i64, i32, f32, P, P, sz, P]),
            "attt_lora_input_grad": (i32, [P, P, P, P, i64, i64, i64, i32, f32, P, P, sz, P]),
            "attt_cast_bf16": (i32, [P, P, i64, P]),
            "attt_lora_adamw_step": (i32, [P, P, P, P, P, P, P, P, i64, i64, i32, f32, f64, f64, f64, f64, i32, P,
                                           P, P]),
            "attt_episode_create": (i32, [ctypes.POINTER(EpisodeConfig), P, P, P, P, ctypes.POINTER(P)]),
            "attt_episode_destroy": (i32, [P]),
            "attt_episode_reset": (i32, [P, P]),
            "attt_episode_update": (i32, [P, P, P, i64, P, P, P]),
            "attt_episode_agent_step": (i32, [P, P, P, i64, P, P, ctypes.POINTER(i32), P]),
            "attt_episode_read_adapter": (i32, [P, P, P, P]),
            "attt_episode_drift": (i32, [P, P, i64, P, P, P]),
            "attt_episode_checkpoint_bytes": (sz, [P]),
            "attt_episode_save": (i32, [P, P, sz, P]),
            "attt_episode_load": (i32, [P, P, sz, P]),
            "attt_history_save": (i32, [P, P, P]),
            "attt_history_restore": (i32, [P, P, i64, P]),
            "attt_episode_history": (P, [P]),
            "attt_episode_pending_tokens": (i64, [P]),
            "attt_kl_workspace_bytes": (sz, [i64, i64, i64]),
            "attt_kl_drift": (i32, [P, P, P, i64, i64, i64, P, P, P, sz, P]),
            "attt_batch_create": (i32, [ctypes.POINTER(BatchConfig), P, P, P, P, ctypes.POINTER(P)]),
            "attt_batch_destroy": (i32, [P]),
            "attt_batch_reset": (i32, [P, i32, P]),
            "attt_batch_update": (i32, [P, P, P, P, P, P, P]),
            "attt_batch_read_adapter": (i32, [P, i32, P, P, P]),
            "attt_batch_history": (P, [P, i32]),
            "attt_wordsets_create": (i32, [i32, i64, ctypes.POINTER(P)]),
            "attt_wordsets_destroy": (i32, [P]),
            "attt_wordsets_reset": (i32, [P, P]),
            "attt_repetition": (i32, [P, P, i64, f32, P, P, P, P]),
            "attt_wordsets_updates": (i32, [P]),
            "attt_wordsets_status": (i32, [P, P]),
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


def _expect(t: Optional[torch.Tensor], shape, dtype, name: str) -> None:
    """Raises ValueError unless t (when given) has this shape and dtype: the
    C ABI takes sizes on trust, so a smaller tensor would be read or written
    past its end."""
    if t is None:
        return
    if tuple(t.shape) != tuple(int(x) for x in shape):
        raise ValueError(f"{name}: expected shape {tuple(shape)}, got {tuple(t.shape)}")
    if t.dtype != dtype:
        raise ValueError(f"{name}: expected {dtype}, got {t.dtype}")


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


def attt_selftest_wait_timeout(stream=None) -> None:
    """Launches the bounded-wait self-test (a wait that runs out after 2 s)."""
    _check(load_library().attt_selftest_wait_timeout(_stream(stream)), "attt_selftest_wait_timeout")


def attt_fault_inject(site: str) -> None:
    """One pending host-side fault: "alloc", "table_full" or "none"."""
    _check(load_library().attt_fault_inject(site.encode()), "attt_fault_inject")


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
        self._owned = True

    @classmethod
    def _view(cls, handle: int, n: int, max_tokens: int, owner) -> "History":
        """Non-owning handle of a history that another object owns."""
        self = cls.__new__(cls)
        self._lib = load_library()
        self.handle = ctypes.c_void_p(handle)
        self.n = int(n)
        self.max_tokens = int(max_tokens)
        self._owned = False
        self._owner = owner
        return self

    def close(self) -> None:
        if getattr(self, "handle", None):
            if self._owned:
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


def attt_history_save(h: History, stream=None):
    """The history's token stream (int32 numpy array), for a checkpoint."""
    import numpy as np
    n = len(h)
    out = np.empty(n, dtype=np.int32)
    _check(load_library().attt_history_save(h.handle, out.ctypes.data_as(ctypes.c_void_p) if n else None,
                                            _stream(stream)), "attt_history_save")
    return out


def attt_history_restore(h: History, tokens, stream=None) -> None:
    """Makes h the history of `tokens` (int32 numpy array), counts rebuilt exactly."""
    import numpy as np
    t = np.ascontiguousarray(tokens, dtype=np.int32)
    _check(load_library().attt_history_restore(h.handle, t.ctypes.data_as(ctypes.c_void_p) if t.size else None,
                                               t.size, _stream(stream)), "attt_history_restore")


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
    _expect(out, (m,), torch.int32, "out")
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
    _expect(out, (L,), torch.float32, "out")
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


def attt_ce_workspace_max_bytes(Lmax: int, d: int, V: int) -> int:
    """One workspace for every update length 1..Lmax (host-only)."""
    return int(load_library().attt_ce_workspace_max_bytes(int(Lmax), int(d), int(V)))


def attt_weighted_ce_fwd_bwd(h: torch.Tensor, W: torch.Tensor, tgt: torch.Tensor, w: torch.Tensor,
                             loss: Optional[torch.Tensor] = None, dh: Optional[torch.Tensor] = None,
                             lse: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None,
                             stream=None):
    """Eq. 10 loss (fp32 [1]), dh (fp32 [L, d]) and optionally lse (fp32 [L])."""
    L, d = h.shape
    V = W.shape[0]
    dev = h.device
    _expect(W, (V, d), torch.bfloat16, "W")
    _expect(tgt, (L,), torch.int32, "tgt")
    _expect(w, (L,), torch.float32, "w")
    _expect(dh, (L, d), torch.float32, "dh")
    _expect(lse, (L,), torch.float32, "lse")
    if loss is not None and (loss.numel() < 1 or loss.dtype != torch.float32):
        raise ValueError("loss: expected a float32 tensor of at least one element")
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


def _lora_check(x: torch.Tensor, dys, As, Bs, dAs, dBs):
    """Shapes of one attt_lora_grad group: (L, din, r, douts).  Raises
    ValueError before any launch unless every list has one entry per
    projection and every tensor has its shape and dtype (the C ABI takes the
    sizes on trust, so a smaller or wider-typed tensor would be read or written
    past its end)."""
    if x.dim() != 2:
        raise ValueError(f"x: expected a 2-D [L, din] tensor, got shape {tuple(x.shape)}")
    L, din = x.shape
    k = len(dys)
    if k < 1:
        raise ValueError("at least one projection (dys) is required")
    if not (len(As) == len(Bs) == k) or (dAs is not None and len(dAs) != k) or (dBs is not None and len(dBs) != k):
        raise ValueError("dys, As, Bs (and dAs, dBs) must have one entry per projection")
    _expect(x, (L, din), torch.bfloat16, "x")
    if As[0].dim() != 2:
        raise ValueError(f"As[0]: expected a 2-D [din, r] tensor, got shape {tuple(As[0].shape)}")
    r = int(As[0].shape[1])
    douts = []
    for p in range(k):
        if dys[p].dim() != 2:
            raise ValueError(f"dys[{p}]: expected a 2-D [L, dout] tensor, got shape {tuple(dys[p].shape)}")
        douts.append(int(dys[p].shape[1]))
        _expect(dys[p], (L, douts[p]), torch.bfloat16, f"dys[{p}]")
        _expect(As[p], (din, r), torch.bfloat16, f"As[{p}]")
        _expect(Bs[p], (r, douts[p]), torch.bfloat16, f"Bs[{p}]")
        _expect(dAs[p] if dAs is not None else None, (din, r), torch.float32, f"dAs[{p}]")
        _expect(dBs[p] if dBs is not None else None, (r, douts[p]), torch.float32, f"dBs[{p}]")
    return int(L), int(din), r, douts


def attt_lora_grad(x: torch.Tensor, dys: Sequence[torch.Tensor], As: Sequence[torch.Tensor],
                   Bs: Sequence[torch.Tensor], scale: float, dAs: Optional[Sequence[torch.Tensor]] = None,
                   dBs: Optional[Sequence[torch.Tensor]] = None, workspace: Optional[torch.Tensor] = None,
                   stream=None):
    """Adapter gradients for projections sharing the input x.  Returns (dAs, dBs)."""
    L, din, r, douts = _lora_check(x, dys, As, Bs, dAs, dBs)
    k = len(dys)
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
    tensors, which are checked like every other argument before the call.
    Returns (dAs, dBs)."""
    if dAs is None or dBs is None:
        raise ValueError("attt_lora_grad_noalloc: the caller passes the output tensors dAs and dBs")
    L, din, r, douts = _lora_check(x, dys, As, Bs, dAs, dBs)
    k = len(dys)
    P = ctypes.c_void_p
    arr = lambda ts, f: (P * k)(*[f(t) for t in ts])  # noqa: E731
    douts_arr = (ctypes.c_int64 * k)(*douts)
    _check(load_library().attt_lora_grad_noalloc(
        _bf16(x), L, din, k, arr(dys, _bf16), douts_arr, arr(As, _bf16), arr(Bs, _bf16), int(r), float(scale),
        arr(dAs, _ptr), arr(dBs, _ptr), _stream(stream)), "attt_lora_grad_noalloc")
    return dAs, dBs


def attt_lora_step(A32: torch.Tensor, B32: torch.Tensor, dA: torch.Tensor, dB: torch.Tensor, lr: float,
                   A16: Optional[torch.Tensor] = None, B16: Optional[torch.Tensor] = None, stream=None) -> None:
    """In-place SGD step on the fp32 masters and bf16 refresh (Eq. 2)."""
    din, r = A32.shape
    dout = B32.shape[1]
    _expect(A32, (din, r), torch.float32, "A32")
    _expect(B32, (r, dout), torch.float32, "B32")
    _expect(dA, (din, r), torch.float32, "dA")
    _expect(dB, (r, dout), torch.float32, "dB")
    _expect(A16, (din, r), torch.bfloat16, "A16")
    _expect(B16, (r, dout), torch.bfloat16, "B16")
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
    _expect(W0, (din, dout), torch.bfloat16, "W0")
    _expect(A, (din, r), torch.bfloat16, "A")
    _expect(B, (r, dout), torch.bfloat16, "B")
    _expect(h, (L, dout), torch.bfloat16, "h")
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
    _expect(W0, (din, dout), torch.bfloat16, "W0")
    _expect(A, (din, r), torch.bfloat16, "A")
    _expect(B, (r, dout), torch.bfloat16, "B")
    _expect(dx, (L, din), torch.float32, "dx")
    if dx is None:
        dx = torch.empty(L, din, dtype=torch.float32, device=dy.device)
    if workspace is None:
        workspace = torch.empty(attt_lora_input_grad_workspace_bytes(L, din, dout, r), dtype=torch.uint8,
                                device=dy.device)
    _check(load_library().attt_lora_input_grad(
        _bf16(dy), _bf16(W0), _bf16(A), _bf16(B), L, din, dout, int(r), float(scale), _ptr(dx), _ptr(workspace),
        workspace.numel(), _stream(stream)), "attt_lora_input_grad")
    return dx


def attt_cast_bf16(src: torch.Tensor, dst: Optional[torch.Tensor] = None, stream=None) -> torch.Tensor:
    """dst = bf16(src) (round to nearest even).  Returns dst."""
    if src.dtype != torch.float32:
        raise ValueError(f"expected float32, got {src.dtype}")
    if dst is None:
        dst = torch.empty(src.shape, dtype=torch.bfloat16, device=src.device)
    if dst.numel() != src.numel():
        raise ValueError(f"dst: expected {src.numel()} elements, got {dst.numel()}")
    _check(load_library().attt_cast_bf16(_ptr(src), _bf16(dst), src.numel(), _stream(stream)), "attt_cast_bf16")
    return dst


# --------------------------------------------------------------------------
# the episode (Algorithm 1 with the Sec. 4 / Appendix C schedule)
# --------------------------------------------------------------------------

class Episode:
    """Owning handle of an attt_episode.

    W0 (bf16 [din, d]) and Wlm (bf16 [V, d]) are borrowed by the library: this
    object keeps references to them so they outlive the episode.  A0 / B0
    (fp32) are the adapter's initial value, restored by reset().
    """

    def __init__(self, W0: torch.Tensor, Wlm: torch.Tensor, A0: torch.Tensor, B0: torch.Tensor, *, n: int,
                 max_history: int, max_update: int, scale: float, lr: float, w_min: float = 0.05,
                 grad_steps: int = 2, cadence: int = 5, optimizer: str = "sgd", betas=(0.9, 0.999),
                 eps: float = 1e-8, weight_decay: float = 0.01):
        self._lib = load_library()
        din, d = W0.shape
        V = Wlm.shape[0]
        r = A0.shape[1]
        if Wlm.shape[1] != d or A0.shape[0] != din or tuple(B0.shape) != (r, d):
            raise ValueError("shape mismatch between W0, Wlm, A0, B0")
        if A0.dtype != torch.float32 or B0.dtype != torch.float32:
            raise ValueError("A0 and B0 must be float32")
        self.cfg = EpisodeConfig(n=int(n), w_min=float(w_min), max_history=int(max_history),
                                 max_update=int(max_update), din=int(din), d=int(d), V=int(V), r=int(r),
                                 scale=float(scale), lr=float(lr), grad_steps=int(grad_steps),
                                 cadence=int(cadence), optimizer={"sgd": 0, "adamw": 1}[optimizer],
                                 beta1=float(betas[0]), beta2=float(betas[1]), eps=float(eps),
                                 weight_decay=float(weight_decay))
        e = ctypes.c_void_p()
        _check(self._lib.attt_episode_create(ctypes.byref(self.cfg), _bf16(W0), _bf16(Wlm), _ptr(A0), _ptr(B0),
                                             ctypes.byref(e)), "attt_episode_create")
        self.handle = e
        self._keep = (W0, Wlm)
        self.device = W0.device

    def close(self) -> None:
        if getattr(self, "handle", None):
            self._lib.attt_episode_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def _out(self, losses, dx, L):
        c = self.cfg
        if losses is not None and (losses.dtype != torch.float32 or losses.numel() < c.grad_steps):
            raise ValueError("losses must be float32 with grad_steps entries")
        if dx is not None and (dx.dtype != torch.float32 or dx.numel() < c.grad_steps * L * c.din):
            raise ValueError("dx must be float32 [grad_steps, L, din]")
        return _ptr(losses), _ptr(dx)

    def update(self, tokens: torch.Tensor, x: torch.Tensor, losses: Optional[torch.Tensor] = None,
               dx: Optional[torch.Tensor] = None, stream=None) -> None:
        """One update on `tokens` (int32 [L]) with projection inputs `x` (bf16 [L, din])."""
        if tokens.dtype != torch.int32:
            raise ValueError("tokens must be int32")
        L = tokens.numel()
        if tuple(x.shape) != (L, self.cfg.din):
            raise ValueError("x must be [L, din]")
        pl, pd = self._out(losses, dx, L)
        _check(self._lib.attt_episode_update(self.handle, _ptr(tokens), _bf16(x), L, pl, pd, _stream(stream)),
               "attt_episode_update")

    def agent_step(self, tokens: torch.Tensor, x: torch.Tensor, losses: Optional[torch.Tensor] = None,
                   dx: Optional[torch.Tensor] = None, stream=None) -> bool:
        """Appends one agent step's text; returns True if it triggered an update."""
        if tokens.dtype != torch.int32:
            raise ValueError("tokens must be int32")
        n = tokens.numel()
        if tuple(x.shape) != (n, self.cfg.din):
            raise ValueError("x must be [len, din]")
        pending = self.pending_tokens()
        pl, pd = self._out(losses, dx, pending + n)
        up = ctypes.c_int(0)
        _check(self._lib.attt_episode_agent_step(self.handle, _ptr(tokens) if n else None,
                                                 _bf16(x) if n else None, n, pl, pd, ctypes.byref(up),
                                                 _stream(stream)), "attt_episode_agent_step")
        return bool(up.value)

    def reset(self, stream=None) -> None:
        _check(self._lib.attt_episode_reset(self.handle, _stream(stream)), "attt_episode_reset")

    def drift(self, x: torch.Tensor, kl: Optional[torch.Tensor] = None, kl_mean: Optional[torch.Tensor] = None,
              stream=None):
        """KL of the adapted from the base next-token distribution on the rows
        of x (bf16 [L, din]).  Returns (kl [L], kl_mean [1])."""
        L = x.shape[0]
        if tuple(x.shape) != (L, self.cfg.din):
            raise ValueError("x must be [L, din]")
        if kl is None:
            kl = torch.empty(L, dtype=torch.float32, device=x.device)
        if kl_mean is None:
            kl_mean = torch.empty(1, dtype=torch.float32, device=x.device)
        _check(self._lib.attt_episode_drift(self.handle, _bf16(x), L, _ptr(kl), _ptr(kl_mean), _stream(stream)),
               "attt_episode_drift")
        return kl, kl_mean

    def read_adapter(self, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
        """(A [din, r], B [r, d]) fp32 copies of the current adapter."""
        c = self.cfg
        A = torch.empty((c.din, c.r), dtype=torch.float32, device=self.device)
        B = torch.empty((c.r, c.d), dtype=torch.float32, device=self.device)
        _check(self._lib.attt_episode_read_adapter(self.handle, _ptr(A), _ptr(B), _stream(stream)),
               "attt_episode_read_adapter")
        return A, B

    def history(self) -> History:
        h = self._lib.attt_episode_history(self.handle)
        return History._view(h, self.cfg.n, self.cfg.max_history, self)

    def pending_tokens(self) -> int:
        return int(self._lib.attt_episode_pending_tokens(self.handle))

    def save(self, stream=None) -> bytes:
        """A checkpoint of the episode (adapter, optimizer state, history, pending text)."""
        n = int(self._lib.attt_episode_checkpoint_bytes(self.handle))
        buf = ctypes.create_string_buffer(n)
        _check(self._lib.attt_episode_save(self.handle, buf, n, _stream(stream)), "attt_episode_save")
        return buf.raw

    def load(self, blob: bytes, stream=None) -> None:
        """Restores a checkpoint made by save() of an episode with the same configuration."""
        buf = ctypes.create_string_buffer(bytes(blob), len(blob))
        _check(self._lib.attt_episode_load(self.handle, buf, len(blob), _stream(stream)), "attt_episode_load")


# --------------------------------------------------------------------------
# adapter drift (Sec. 4, Fig. 6)
# --------------------------------------------------------------------------

def attt_kl_workspace_bytes(L: int, d: int, V: int) -> int:
    return int(load_library().attt_kl_workspace_bytes(L, d, V))


def attt_kl_drift(hp: torch.Tensor, hq: torch.Tensor, W: torch.Tensor, kl: Optional[torch.Tensor] = None,
                  kl_mean: Optional[torch.Tensor] = None, workspace: Optional[torch.Tensor] = None, stream=None):
    """KL(softmax(h_p W^T) || softmax(h_q W^T)) per row (fp32 [L]) and its
    mean (fp32 [1]).  Returns (kl, kl_mean)."""
    L, d = hp.shape
    V = W.shape[0]
    if tuple(hq.shape) != (L, d) or W.shape[1] != d:
        raise ValueError("shape mismatch")
    _expect(kl, (L,), torch.float32, "kl")
    _expect(kl_mean, (1,), torch.float32, "kl_mean")
    dev = hp.device
    if kl is None:
        kl = torch.empty(L, dtype=torch.float32, device=dev)
    if kl_mean is None:
        kl_mean = torch.empty(1, dtype=torch.float32, device=dev)
    if workspace is None:
        workspace = torch.empty(attt_kl_workspace_bytes(L, d, V), dtype=torch.uint8, device=dev)
    _check(load_library().attt_kl_drift(_bf16(hp), _bf16(hq), _bf16(W), L, d, V, _ptr(kl), _ptr(kl_mean),
                                        _ptr(workspace), workspace.numel(), _stream(stream)), "attt_kl_drift")
    return kl, kl_mean


# --------------------------------------------------------------------------
# update-text repetition (Eq. 6), novelty (Eq. 7), the sequence filter
# --------------------------------------------------------------------------

class WordSets:
    """Owning handle of an attt_wordsets (the episode's update texts)."""

    def __init__(self, max_updates: int, max_bytes: int):
        self._lib = load_library()
        s = ctypes.c_void_p()
        _check(self._lib.attt_wordsets_create(int(max_updates), int(max_bytes), ctypes.byref(s)),
               "attt_wordsets_create")
        self.handle = s

    def close(self) -> None:
        if getattr(self, "handle", None):
            self._lib.attt_wordsets_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def __len__(self) -> int:
        return int(self._lib.attt_wordsets_updates(self.handle))


def attt_wordsets_create(max_updates: int, max_bytes: int) -> WordSets:
    return WordSets(max_updates, max_bytes)


def attt_wordsets_destroy(s: WordSets) -> None:
    s.close()


def attt_wordsets_reset(s: WordSets, stream=None) -> None:
    _check(load_library().attt_wordsets_reset(s.handle, _stream(stream)), "attt_wordsets_reset")


def attt_wordsets_updates(s: WordSets) -> int:
    return int(load_library().attt_wordsets_updates(s.handle))


def attt_wordsets_status(s: WordSets, stream=None) -> int:
    return int(load_library().attt_wordsets_status(s.handle, _stream(stream)))


def attt_repetition(s: WordSets, text: torch.Tensor, tau: float = 0.5, out: Optional[torch.Tensor] = None,
                    keep: Optional[torch.Tensor] = None, stream=None):
    """Eq. 6 / Eq. 7 for the update text `text` (uint8 bytes on the device):
    returns (out, keep) with out = float32 [2] (rho, nu) and keep = int32 [1]."""
    if text.dtype != torch.uint8:
        raise ValueError("text must be uint8 bytes")
    _expect(out, (2,), torch.float32, "out")
    _expect(keep, (1,), torch.int32, "keep")
    dev = text.device
    if out is None:
        out = torch.empty(2, dtype=torch.float32, device=dev)
    if keep is None:
        keep = torch.empty(1, dtype=torch.int32, device=dev)
    n = text.numel()
    base = _ptr(out)
    _check(load_library().attt_repetition(s.handle, _ptr(text) if n else None, n, float(tau), base, base + 4,
                                          _ptr(keep), _stream(stream)), "attt_repetition")
    return out, keep


# --------------------------------------------------------------------------
# a batch of concurrent episodes
# --------------------------------------------------------------------------

class Batch:
    """Owning handle of an attt_batch: E episodes sharing W0 and the LM head
    (borrowed: kept referenced here), each adapter starting at (A0, B0)."""

    def __init__(self, W0: torch.Tensor, Wlm: torch.Tensor, A0: torch.Tensor, B0: torch.Tensor, *, episodes: int,
                 n: int, max_history: int, max_update: int, scale: float, lr: float, w_min: float = 0.05,
                 grad_steps: int = 2):
        self._lib = load_library()
        din, d = W0.shape
        r = A0.shape[1]
        if Wlm.shape[1] != d or A0.shape[0] != din or tuple(B0.shape) != (r, d):
            raise ValueError("shape mismatch between W0, Wlm, A0, B0")
        self.cfg = BatchConfig(episodes=int(episodes), n=int(n), w_min=float(w_min), max_history=int(max_history),
                               max_update=int(max_update), din=int(din), d=int(d), V=int(Wlm.shape[0]), r=int(r),
                               scale=float(scale), lr=float(lr), grad_steps=int(grad_steps))
        b = ctypes.c_void_p()
        _check(self._lib.attt_batch_create(ctypes.byref(self.cfg), _bf16(W0), _bf16(Wlm), _ptr(A0), _ptr(B0),
                                           ctypes.byref(b)), "attt_batch_create")
        self.handle = b
        self._keep = (W0, Wlm)
        self.device = W0.device

    def close(self) -> None:
        if getattr(self, "handle", None):
            self._lib.attt_batch_destroy(self.handle)
            self.handle = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def update(self, tokens: torch.Tensor, x: torch.Tensor, lens: Sequence[int],
               losses: Optional[torch.Tensor] = None, dx: Optional[torch.Tensor] = None, stream=None) -> None:
        """One update of every episode with lens[e] > 0; tokens (int32) and x
        (bf16 [sum lens, din]) hold the episodes' rows one after another."""
        c = self.cfg
        if len(lens) != c.episodes:
            raise ValueError("one length per episode")
        R = int(sum(lens))
        if tokens.dtype != torch.int32 or tokens.numel() != R or tuple(x.shape) != (R, c.din):
            raise ValueError("tokens must be int32 [sum lens] and x [sum lens, din]")
        if losses is not None and (losses.dtype != torch.float32 or losses.numel() < c.episodes * c.grad_steps):
            raise ValueError("losses must be float32 [E, grad_steps]")
        if dx is not None and (dx.dtype != torch.float32 or dx.numel() < c.grad_steps * R * c.din):
            raise ValueError("dx must be float32 [grad_steps, sum lens, din]")
        arr = (ctypes.c_int64 * c.episodes)(*[int(v) for v in lens])
        _check(self._lib.attt_batch_update(self.handle, _ptr(tokens), _bf16(x), arr, _ptr(losses), _ptr(dx),
                                           _stream(stream)), "attt_batch_update")

    def reset(self, e: int = -1, stream=None) -> None:
        _check(self._lib.attt_batch_reset(self.handle, int(e), _stream(stream)), "attt_batch_reset")

    def read_adapter(self, e: int, stream=None) -> Tuple[torch.Tensor, torch.Tensor]:
        c = self.cfg
        A = torch.empty((c.din, c.r), dtype=torch.float32, device=self.device)
        B = torch.empty((c.r, c.d), dtype=torch.float32, device=self.device)
        _check(self._lib.attt_batch_read_adapter(self.handle, int(e), _ptr(A), _ptr(B), _stream(stream)),
               "attt_batch_read_adapter")
        return A, B

    def history(self, e: int) -> History:
        h = self._lib.attt_batch_history(self.handle, int(e))
        return History._view(h, self.cfg.n, self.cfg.max_history, self)


def attt_lora_adamw_step(A32: torch.Tensor, B32: torch.Tensor, dA: torch.Tensor, dB: torch.Tensor,
                         mA: torch.Tensor, vA: torch.Tensor, mB: torch.Tensor, vB: torch.Tensor, lr: float, step: int,
                         betas=(0.9, 0.999), eps: float = 1e-8, weight_decay: float = 0.01,
                         A16: Optional[torch.Tensor] = None, B16: Optional[torch.Tensor] = None, stream=None) -> None:
    """In-place AdamW step on the fp32 masters (moments mA, vA, mB, vB), bf16 refresh."""
    din, r = A32.shape
    dout = B32.shape[1]
    _check(load_library().attt_lora_adamw_step(
        _ptr(A32), _ptr(B32), _ptr(dA), _ptr(dB), _ptr(mA), _ptr(vA), _ptr(mB), _ptr(vB), din, dout, r, float(lr),
        float(betas[0]), float(betas[1]), float(eps), float(weight_decay), int(step),
        _bf16(A16) if A16 is not None else None, _bf16(B16) if B16 is not None else None, _stream(stream)),
        "attt_lora_adamw_step")
