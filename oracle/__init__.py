"""Plain CPU oracle for the aTTT update step -- TEST INFRASTRUCTURE ONLY.

Only ``tests/``, ``__graft_entry__.smoke()`` and the CPU-baseline leg and
reference arm (``--impl reference``) of ``bench.py`` may import this package.  The CUDA library never imports, links
or calls it, and it shares no code with that library.

The arithmetic lives in ``attt_oracle.c`` (fp64 sums over the bf16 inputs,
Eqs. 8-10, Eq. 2 and Algorithm 1 of the aTTT paper); this module only builds
it with gcc and marshals numpy arrays through ctypes.

Every function here has a pin in ``tests/test_oracle_*.py`` (hand-worked
example, brute force, two independent counters, finite differences, torch CPU
library routines, closed forms); none is "parity unpinned".
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "attt_oracle.c")
_LIB_PATH = os.path.join(_HERE, "liboracle.so")
_lock = threading.Lock()
_lib = None


def build(force: bool = False) -> str:
    """Compile attt_oracle.c into liboracle.so next to it (gcc, OpenMP)."""
    if (not force and os.path.exists(_LIB_PATH)
            and os.path.getmtime(_LIB_PATH) >= os.path.getmtime(_SRC)):
        return _LIB_PATH
    tmp = _LIB_PATH + f".tmp{os.getpid()}"
    cmd = ["gcc", "-O2", "-fPIC", "-shared", "-fopenmp", "-ffp-contract=off",
           "-fno-fast-math", "-std=c11", _SRC, "-o", tmp, "-lm"]
    subprocess.run(cmd, check=True)
    os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def _load():
    global _lib
    with _lock:
        if _lib is not None:
            return _lib
        lib = ctypes.CDLL(build())
        P = ctypes.c_void_p
        i64 = ctypes.c_int64
        lib.oracle_count_naive.restype = i64
        lib.oracle_count_naive.argtypes = [P, i64, P, ctypes.c_int]
        lib.oracle_exposure_naive.restype = None
        lib.oracle_exposure_naive.argtypes = [P, i64, P, i64, ctypes.c_int, P]
        lib.oracle_exposure_sorted.restype = None
        lib.oracle_exposure_sorted.argtypes = [P, i64, P, i64, ctypes.c_int, P]
        lib.oracle_weights_from_exposure.restype = None
        lib.oracle_weights_from_exposure.argtypes = [P, i64, ctypes.c_float, P]
        lib.oracle_kl_rows.restype = None
        lib.oracle_kl_rows.argtypes = [P, P, P, i64, i64, P, i64, P]
        lib.oracle_ce_rows.restype = None
        lib.oracle_ce_rows.argtypes = [P, P, P, P, i64, i64, i64, P, i64, P, P, P]
        lib.oracle_ce_loss.restype = ctypes.c_double
        lib.oracle_ce_loss.argtypes = [P, P, P, P, i64, i64, i64, P, P, P]
        lib.oracle_lora_grad.restype = None
        lib.oracle_lora_grad.argtypes = [P, P, P, P, i64, i64, i64, ctypes.c_int,
                                         ctypes.c_double, P, P]
        lib.oracle_sgd_step.restype = None
        lib.oracle_lora_forward.argtypes = [P, P, P, P, i64, i64, i64, ctypes.c_int, ctypes.c_double, P]
        lib.oracle_lora_forward.restype = None
        lib.oracle_lora_input_grad.argtypes = [P, P, P, P, i64, i64, i64, ctypes.c_int, ctypes.c_double, P]
        lib.oracle_lora_input_grad.restype = None
        lib.oracle_sgd_step.argtypes = [P, P, i64, ctypes.c_float]
        lib.oracle_to_bf16.restype = None
        lib.oracle_to_bf16.argtypes = [P, P, i64]
        lib.oracle_num_threads.restype = ctypes.c_int
        lib.oracle_num_threads.argtypes = []
        lib.oracle_set_num_threads.restype = None
        lib.oracle_set_num_threads.argtypes = [ctypes.c_int]
        _lib = lib
        return lib


def _c(a, dtype):
    a = np.ascontiguousarray(a, dtype=dtype)
    return a, a.ctypes.data_as(ctypes.c_void_p)


def num_threads() -> int:
    return int(_load().oracle_num_threads())


def set_num_threads(t: int) -> None:
    _load().oracle_set_num_threads(int(t))


# --------------------------------------------------------------------------
# Eq. 8 / Eq. 9
# --------------------------------------------------------------------------

def count_naive(H, g) -> int:
    """count(g, H) of Eq. 8: every start position, overlaps included."""
    H, pH = _c(H, np.int32)
    g, pg = _c(g, np.int32)
    return int(_load().oracle_count_naive(pH, H.size, pg, g.size))


def exposure(H, x, n: int, method: str = "sorted") -> np.ndarray:
    """f_k(j) of Eq. 8 for every position j of x (int64)."""
    H, pH = _c(H, np.int32)
    x, px = _c(x, np.int32)
    f = np.zeros(x.size, dtype=np.int64)
    fn = {"naive": _load().oracle_exposure_naive,
          "sorted": _load().oracle_exposure_sorted}[method]
    fn(pH, H.size, px, x.size, int(n), f.ctypes.data_as(ctypes.c_void_p))
    return f


def weights_from_exposure(f, w_min: float) -> np.ndarray:
    """w_{k,j} of Eq. 9 in fp32 (IEEE divide, then the floor)."""
    f, pf = _c(f, np.int64)
    w = np.zeros(f.size, dtype=np.float32)
    _load().oracle_weights_from_exposure(pf, f.size, ctypes.c_float(w_min),
                                         w.ctypes.data_as(ctypes.c_void_p))
    return w


def ngram_weights(H, x, n: int, w_min: float = 0.05, method: str = "sorted") -> np.ndarray:
    """Algorithm 1's per-token weight loop: Eq. 8 then Eq. 9."""
    return weights_from_exposure(exposure(H, x, n, method), w_min)


# --------------------------------------------------------------------------
# Eq. 10 and dh
# --------------------------------------------------------------------------

def ce_rows(h_bf16, W_bf16, tgt, w, rows, with_dh: bool = True):
    """Per-row lse, nll and (optionally) dh of Eq. 10 for the given rows.

    h_bf16 [L, d] and W_bf16 [V, d] are uint16 arrays holding bf16 bits."""
    h, ph = _c(h_bf16, np.uint16)
    W, pW = _c(W_bf16, np.uint16)
    t, pt = _c(tgt, np.int32)
    wv, pw = _c(w, np.float32)
    rows, pr = _c(rows, np.int64)
    L, d = h.shape
    V = W.shape[0]
    lse = np.zeros(rows.size, dtype=np.float64)
    nll = np.zeros(rows.size, dtype=np.float64)
    dh = np.zeros((rows.size, d), dtype=np.float64) if with_dh else None
    _load().oracle_ce_rows(ph, pW, pt, pw, L, d, V, pr, rows.size,
                           lse.ctypes.data_as(ctypes.c_void_p),
                           nll.ctypes.data_as(ctypes.c_void_p),
                           dh.ctypes.data_as(ctypes.c_void_p) if with_dh else None)
    return lse, nll, dh


def ce_loss(h_bf16, W_bf16, tgt, w, with_dh: bool = True):
    """Eq. 10 over all rows: (loss, lse[L], nll[L], dh[L, d] or None)."""
    h, ph = _c(h_bf16, np.uint16)
    W, pW = _c(W_bf16, np.uint16)
    t, pt = _c(tgt, np.int32)
    wv, pw = _c(w, np.float32)
    L, d = h.shape
    V = W.shape[0]
    lse = np.zeros(L, dtype=np.float64)
    nll = np.zeros(L, dtype=np.float64)
    dh = np.zeros((L, d), dtype=np.float64) if with_dh else None
    loss = _load().oracle_ce_loss(ph, pW, pt, pw, L, d, V,
                                  lse.ctypes.data_as(ctypes.c_void_p),
                                  nll.ctypes.data_as(ctypes.c_void_p),
                                  dh.ctypes.data_as(ctypes.c_void_p) if with_dh else None)
    return float(loss), lse, nll, dh


# --------------------------------------------------------------------------
# LoRA gradients and the SGD step
# --------------------------------------------------------------------------

def lora_grad(x_bf16, dy_bf16, A_bf16, B_bf16, scale: float):
    """(dA [din, r], dB [r, dout]) in fp64 for y = x W0 + s (x A) B."""
    x, px = _c(x_bf16, np.uint16)
    dy, pdy = _c(dy_bf16, np.uint16)
    A, pA = _c(A_bf16, np.uint16)
    B, pB = _c(B_bf16, np.uint16)
    L, din = x.shape
    dout = dy.shape[1]
    r = A.shape[1]
    assert dy.shape[0] == L and A.shape[0] == din and B.shape == (r, dout)
    dA = np.zeros((din, r), dtype=np.float64)
    dB = np.zeros((r, dout), dtype=np.float64)
    _load().oracle_lora_grad(px, pdy, pA, pB, L, din, dout, r, float(scale),
                             dA.ctypes.data_as(ctypes.c_void_p),
                             dB.ctypes.data_as(ctypes.c_void_p))
    return dA, dB


def lora_forward(x_bf16, W0_bf16, A_bf16, B_bf16, scale: float):
    """h = x W0 + s (x A) B in fp64 [L, dout] (the adapted projection)."""
    x, px = _c(x_bf16, np.uint16)
    W0, pW = _c(W0_bf16, np.uint16)
    A, pA = _c(A_bf16, np.uint16)
    B, pB = _c(B_bf16, np.uint16)
    L, din = x.shape
    dout = W0.shape[1]
    r = A.shape[1]
    assert W0.shape[0] == din and A.shape[0] == din and B.shape == (r, dout)
    h = np.zeros((L, dout), dtype=np.float64)
    _load().oracle_lora_forward(px, pW, pA, pB, L, din, dout, r, float(scale), h.ctypes.data_as(ctypes.c_void_p))
    return h


def lora_input_grad(dy_bf16, W0_bf16, A_bf16, B_bf16, scale: float):
    """dx = dy W0^T + s (dy B^T) A^T in fp64 [L, din]."""
    dy, pdy = _c(dy_bf16, np.uint16)
    W0, pW = _c(W0_bf16, np.uint16)
    A, pA = _c(A_bf16, np.uint16)
    B, pB = _c(B_bf16, np.uint16)
    L, dout = dy.shape
    din = W0.shape[0]
    r = A.shape[1]
    assert W0.shape[1] == dout and A.shape[0] == din and B.shape == (r, dout)
    dx = np.zeros((L, din), dtype=np.float64)
    _load().oracle_lora_input_grad(pdy, pW, pA, pB, L, din, dout, r, float(scale),
                                   dx.ctypes.data_as(ctypes.c_void_p))
    return dx


def sgd_step(p32, g32, lr: float):
    """Eq. 2: returns (p - lr*g in fp32, its bf16 refresh as uint16)."""
    p = np.array(p32, dtype=np.float32, copy=True)
    g, pg = _c(g32, np.float32)
    _load().oracle_sgd_step(p.ctypes.data_as(ctypes.c_void_p), pg, p.size,
                            ctypes.c_float(lr))
    b = np.zeros(p.shape, dtype=np.uint16)
    _load().oracle_to_bf16(p.ctypes.data_as(ctypes.c_void_p),
                           b.ctypes.data_as(ctypes.c_void_p), p.size)
    return p, b


def to_bf16(p32) -> np.ndarray:
    """fp32 -> bf16 bits, round to nearest even."""
    p, pp = _c(p32, np.float32)
    b = np.zeros(p.shape, dtype=np.uint16)
    _load().oracle_to_bf16(pp, b.ctypes.data_as(ctypes.c_void_p), p.size)
    return b


# --------------------------------------------------------------------------
# One update of Algorithm 1, chained through the adapted projection
# --------------------------------------------------------------------------

def episode_update(H, tokens, x_bf16, W0_bf16, Wlm_bf16, A32, B32, *, n: int, w_min: float, scale: float,
                   lr: float, grad_steps: int = 2, want_dx: bool = True, adamw=None):
    """Algorithm 1 for update x_k (= `tokens`, also the Eq. 10 targets) with
    the adapter on the projection whose output is the LM head's input:

      w = Eq. 9(Eq. 8(x_k, H))                       (once per update)
      grad_steps times (Appendix C: two):
        h = x W0 + s (x A) B, stored as bf16          (A, B: bf16 copies)
        loss, dh = Eq. 10(h, W_lm, x_k, w)
        dy = bf16(fp32(dh))
        dA, dB = the adapter gradients; dx = dy W0^T + s (dy B^T) A^T
        A, B <- A - lr dA, B - lr dB (Eq. 2, fp32) and refresh the bf16 copies
      H <- H || x_k

    Returns a dict with w, losses [grad_steps], dx (list, or None), A32, B32
    (fp32 after the update) and H (the new history).

    adamw: None for the paper's SGD, else a dict {"t", "mA", "vA", "mB", "vB",
    "beta1", "beta2", "eps", "weight_decay"} of AdamW's state and settings,
    advanced in place (t counts the steps taken so far)."""
    w = ngram_weights(H, tokens, n, w_min)
    A = np.array(A32, dtype=np.float32, copy=True)
    B = np.array(B32, dtype=np.float32, copy=True)
    A16, B16 = to_bf16(A), to_bf16(B)
    losses, dxs = [], []
    for _ in range(int(grad_steps)):
        h16 = to_bf16(lora_forward(x_bf16, W0_bf16, A16, B16, scale).astype(np.float32))
        loss, _, _, dh = ce_loss(h16, Wlm_bf16, tokens, w)
        dy = to_bf16(dh.astype(np.float32))
        dA, dB = lora_grad(x_bf16, dy, A16, B16, scale)
        if want_dx:
            dxs.append(lora_input_grad(dy, W0_bf16, A16, B16, scale))
        if adamw is None:
            A, A16 = sgd_step(A, dA.astype(np.float32), lr)
            B, B16 = sgd_step(B, dB.astype(np.float32), lr)
        else:
            o = adamw
            o["t"] += 1
            kw = dict(beta1=o["beta1"], beta2=o["beta2"], eps=o["eps"], weight_decay=o["weight_decay"])
            A, o["mA"], o["vA"] = adamw_step(A, dA.astype(np.float32), o["mA"], o["vA"], o["t"], lr, **kw)
            B, o["mB"], o["vB"] = adamw_step(B, dB.astype(np.float32), o["mB"], o["vB"], o["t"], lr, **kw)
            A16, B16 = to_bf16(A), to_bf16(B)
        losses.append(loss)
    H = np.concatenate([np.asarray(H, dtype=np.int32), np.asarray(tokens, dtype=np.int32)])
    return {"w": w, "losses": np.array(losses), "dx": dxs if want_dx else None, "A32": A, "B32": B, "H": H}


# --------------------------------------------------------------------------
# Eq. 6 / Eq. 7: update-text repetition and the sequence-level filter
# --------------------------------------------------------------------------

def words(text: bytes) -> set:
    """W(x): the set of whitespace-separated words of the update text, split
    on runs of the ASCII whitespace bytes (space, tab, LF, VT, FF, CR), the
    words compared byte for byte."""
    return set(bytes(text).split())


def jaccard(a: set, b: set) -> np.float32:
    """J(a, b) = |a & b| / |a | b| as one fp32 division of the two integer
    sizes; 0 when both sets are empty."""
    union = len(a | b)
    if union == 0:
        return np.float32(0.0)
    return np.float32(len(a & b)) / np.float32(union)


def repetition(previous, text: bytes):
    """Eq. 6 and Eq. 7: (rho, nu) of update text `text` given the episode's
    previous update texts; rho = 0 for the first update, nu = 1 - rho (fp32)."""
    cur = words(text)
    rho = np.float32(0.0)
    for prev in previous:
        rho = max(rho, jaccard(cur, words(prev)))
    return rho, np.float32(1.0) - rho


def sequence_filter(texts, tau: float):
    """The sequence-level filter over an episode's candidate update texts in
    order: [(rho, nu, keep)] with keep = not (nu < tau).  Every candidate text
    joins the previous texts of the later ones, kept or not."""
    out = []
    for k, text in enumerate(texts):
        rho, nu = repetition(texts[:k], text)
        out.append((rho, nu, not bool(nu < np.float32(tau))))
    return out


# --------------------------------------------------------------------------
# Adapter drift: KL of the adapted from the base next-token distribution
# --------------------------------------------------------------------------

def kl_rows(hp_bf16, hq_bf16, W_bf16, rows=None):
    """KL(softmax(h_p W^T) || softmax(h_q W^T)) per row (fp64), for `rows`
    (all rows when None)."""
    hp, php = _c(hp_bf16, np.uint16)
    hq, phq = _c(hq_bf16, np.uint16)
    W, pW = _c(W_bf16, np.uint16)
    L, d = hp.shape
    assert hq.shape == (L, d) and W.shape[1] == d
    rows = np.arange(L, dtype=np.int64) if rows is None else rows
    rows, pr = _c(rows, np.int64)
    out = np.zeros(rows.size, dtype=np.float64)
    _load().oracle_kl_rows(php, phq, pW, d, W.shape[0], pr, rows.size, out.ctypes.data_as(ctypes.c_void_p))
    return out


# --------------------------------------------------------------------------
# AdamW (an optional optimizer for the update; the paper's is SGD, Eq. 2)
# --------------------------------------------------------------------------

def adamw_step(p32, g32, m, v, t: int, lr: float, beta1: float = 0.9, beta2: float = 0.999, eps: float = 1e-8,
               weight_decay: float = 0.01):
    """One AdamW step (Adam with decoupled weight decay, Loshchilov and
    Hutter), in fp64 on fp32 inputs: step t (1-based),
      p <- p (1 - lr wd);  m <- b1 m + (1 - b1) g;  v <- b2 v + (1 - b2) g^2
      p <- p - (lr / (1 - b1^t)) m / (sqrt(v) / sqrt(1 - b2^t) + eps)
    Returns (p as fp32, m, v) with m, v in fp64."""
    p = np.asarray(p32, dtype=np.float32).astype(np.float64)
    g = np.asarray(g32, dtype=np.float32).astype(np.float64)
    m = np.asarray(m, dtype=np.float64)
    v = np.asarray(v, dtype=np.float64)
    p = p * (1.0 - lr * weight_decay)
    m = beta1 * m + (1.0 - beta1) * g
    v = beta2 * v + (1.0 - beta2) * g * g
    step_size = lr / (1.0 - beta1 ** t)
    denom = np.sqrt(v) / np.sqrt(1.0 - beta2 ** t) + eps
    p = p - step_size * m / denom
    return p.astype(np.float32), m, v
