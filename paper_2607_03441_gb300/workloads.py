"""Seeded synthetic inputs for the aTTT update step.

This module only draws random inputs; it holds none of the method's
arithmetic (no counting, no weighting, no loss, no gradients), so both the
CUDA path and the CPU oracle may take their inputs from it.

Recipe (stands in for the paper's ALFWorld / SWE-bench update texts and the
Qwen / Gemma weights, none of which are available here):

* Token ids: truncated Zipf(1.1) over the vocabulary, P(k) proportional to
  k^-1.1 for k = 1..V, drawn by inverse CDF over an fp64 cumulative table,
  id = k - 1 (no permutation, so low ids are the hot ones).
* History: iid Zipf ids of the stated length.
* Repeated spans: a fraction ``frac`` of the update's positions is overwritten
  by spans copied from the history.  Span lengths are uniform in [8, 32]
  (the last one truncated so exactly round(frac * L) positions are covered),
  source starts are uniform in the history, and the spans are laid out in a
  random order with uniformly random gaps between them (no overlaps).
* Dense tensors: fp32 normal samples rounded once to bf16 (round to nearest
  even); hidden ~ N(0, 1), LM head ~ N(0, 0.02), LoRA A ~ N(0, 0.02),
  B = 0.01 * N(0, 1), activations x and upstream grads dy ~ N(0, 1).
* Update texts as bytes (Eq. 6 works on whitespace-separated words): a
  synthetic vocabulary of words (1-12 characters over lowercase letters,
  digits and ``._/()-:``), Zipf(1.1) word ids, joined by a space (80%), a
  newline (10%), a tab (4%), two spaces (4%) or CR LF (2%); spans of words
  copied from the previous update's text at a fraction rising linearly from
  5% to 95% (an episode drifting into the repetitive, stuck regime).
* Chained episodes (the adapted projection's output is the LM head's input):
  the frozen projection W0 [din, d] ~ N(0, 1/din), so that h = x W0 has unit
  variance like the hidden states above; one x ~ N(0, 1) per update; update
  texts copy spans from the episode's history so far, with the repeat
  fraction rising like the long episode's.

Every array comes from its own numpy PCG64 stream keyed by (seed, name).
"""
from __future__ import annotations

import dataclasses
import functools
import zlib
from typing import Dict, List, Optional, Tuple

import numpy as np

W_MIN = 0.05          # the paper's weight floor (Appendix C)
LORA_LR = 5e-4        # the paper's learning rate (Appendix C)


def rng_for(seed: int, name: str) -> np.random.Generator:
    """Independent, reproducible stream for one named array of one config."""
    return np.random.default_rng([int(seed), zlib.crc32(name.encode())])


@functools.lru_cache(maxsize=8)
def _zipf_cdf(V: int, a: float) -> np.ndarray:
    k = np.arange(1, V + 1, dtype=np.float64)
    c = np.cumsum(k ** (-a))
    return c / c[-1]


def zipf_ids(rng: np.random.Generator, n: int, V: int, a: float = 1.1) -> np.ndarray:
    """n iid token ids in [0, V) from a truncated Zipf(a) (inverse CDF)."""
    u = rng.random(n)
    ids = np.searchsorted(_zipf_cdf(int(V), float(a)), u, side="right")
    return np.minimum(ids, V - 1).astype(np.int32)


def copy_spans(rng: np.random.Generator, x: np.ndarray, H: np.ndarray, frac: float) -> np.ndarray:
    """Overwrite round(frac*len(x)) positions of x with spans copied from H."""
    x = np.array(x, dtype=np.int32, copy=True)
    L = x.size
    target = int(round(frac * L))
    if target <= 0 or H.size == 0:
        return x
    target = min(target, L)
    max_len = int(min(32, H.size))
    min_len = int(min(8, max_len))
    lens: List[int] = []
    while sum(lens) < target:
        lens.append(int(rng.integers(min_len, max_len + 1)))
    lens[-1] -= sum(lens) - target
    if lens[-1] <= 0:
        lens.pop()
    k = len(lens)
    gap_total = L - target
    # random composition of gap_total into k+1 non-negative gaps
    cuts = np.sort(rng.integers(0, gap_total + 1, size=k))
    gaps = np.diff(np.concatenate([[0], cuts, [gap_total]]))
    pos = 0
    for i, ln in enumerate(lens):
        pos += int(gaps[i])
        src = int(rng.integers(0, H.size - ln + 1))
        x[pos:pos + ln] = H[src:src + ln]
        pos += ln
    return x


def bf16_bits(a: np.ndarray) -> np.ndarray:
    """fp32 array -> bf16 bit patterns (uint16), round to nearest even."""
    a = np.ascontiguousarray(a, dtype=np.float32)
    out = np.empty(a.shape, dtype=np.uint16)
    flat_in = a.reshape(-1).view(np.uint32)
    flat_out = out.reshape(-1)
    step = 1 << 24
    for s in range(0, flat_in.size, step):
        u = flat_in[s:s + step].astype(np.uint64)
        lsb = (u >> 16) & 1
        flat_out[s:s + step] = ((u + 0x7FFF + lsb) >> 16).astype(np.uint16)
    return out


def bf16_to_f32(b: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> fp32 values (exact)."""
    return (np.asarray(b, dtype=np.uint16).astype(np.uint32) << 16).view(np.float32)


def normal_bf16(seed: int, name: str, shape: Tuple[int, ...], std: float = 1.0) -> np.ndarray:
    """bf16 bits of fp32 N(0, std^2) samples, generated in chunks."""
    rng = rng_for(seed, name)
    n = int(np.prod(shape))
    out = np.empty(n, dtype=np.uint16)
    step = 1 << 24
    for s in range(0, n, step):
        m = min(step, n - s)
        v = rng.standard_normal(m, dtype=np.float32)
        if std != 1.0:
            v *= np.float32(std)
        out[s:s + m] = bf16_bits(v)
    return out.reshape(shape)


# --------------------------------------------------------------------------
# The five workloads
# --------------------------------------------------------------------------

@dataclasses.dataclass
class LoraProj:
    name: str
    din: int
    dout: int
    x_group: str          # projections with the same x_group share one x


@dataclasses.dataclass
class Workload:
    name: str
    seed: int
    L: int                # update tokens
    V: int                # vocabulary
    n: int                # n-gram size
    hist_len: int         # prior-update history length
    frac: float           # repeated-span fraction
    d: int = 0            # hidden size (0: integer path only)
    r: int = 0            # LoRA rank
    projs: Tuple[LoraProj, ...] = ()
    updates: int = 1      # sequential updates (long episode)
    w_min: float = W_MIN

    @property
    def scale(self) -> float:
        """LoRA scale s = alpha / r with alpha = 2r (the paper's 16 / 8)."""
        return 2.0


def _qkvo(d: int, kv: int) -> Tuple[LoraProj, ...]:
    return (LoraProj("q", d, d, "attn"), LoraProj("k", d, kv, "attn"),
            LoraProj("v", d, kv, "attn"), LoraProj("o", d, d, "o"))


WORKLOADS: Dict[str, Workload] = {
    "tiny": Workload("tiny", 0, L=256, V=8192, n=4, hist_len=2048, frac=0.30, d=512, r=8,
                     projs=(LoraProj("proj", 512, 512, "x"),)),
    "7b": Workload("7b", 1, L=2048, V=152064, n=4, hist_len=65536, frac=0.40, d=3584, r=16,
                   projs=(LoraProj("q", 3584, 3584, "attn"), LoraProj("v", 3584, 512, "attn"))),
    "stress": Workload("stress", 2, L=8192, V=128256, n=4, hist_len=1 << 20, frac=0.30),
    "long": Workload("long", 3, L=4096, V=128256, n=4, hist_len=0, frac=0.05, d=4096, r=32,
                     projs=_qkvo(4096, 1024) + (LoraProj("gate", 4096, 14336, "mlp"),
                                                 LoraProj("up", 4096, 14336, "mlp"),
                                                 LoraProj("down", 14336, 4096, "down")),
                     updates=32),
    "32b": Workload("32b", 4, L=8192, V=152064, n=4, hist_len=262144, frac=0.50, d=5120, r=64,
                    projs=_qkvo(5120, 1024)),
}


def long_episode_frac(k: int, updates: int = 32) -> float:
    """Repeat fraction of update k (1-based): 5% rising linearly to 80%."""
    if updates <= 1:
        return 0.05
    return 0.05 + 0.75 * (k - 1) / (updates - 1)


def history_tokens(wl: Workload, seed: Optional[int] = None) -> np.ndarray:
    s = wl.seed if seed is None else seed
    return zipf_ids(rng_for(s, "history"), wl.hist_len, wl.V)


def update_tokens(wl: Workload, H: np.ndarray, frac: Optional[float] = None,
                  tag: str = "update", seed: Optional[int] = None) -> np.ndarray:
    s = wl.seed if seed is None else seed
    x = zipf_ids(rng_for(s, tag + "/ids"), wl.L, wl.V)
    return copy_spans(rng_for(s, tag + "/spans"), x, H, wl.frac if frac is None else frac)


def stress_case(n: int, frac: float, seed: int = 2, L: int = 8192, hist_len: int = 1 << 20,
                V: int = 128256) -> Tuple[np.ndarray, np.ndarray]:
    """(history, update) for one point of the n-gram stress sweep."""
    H = zipf_ids(rng_for(seed, "stress/history"), hist_len, V)
    x = zipf_ids(rng_for(seed, f"stress/ids/n{n}/f{frac:.2f}"), L, V)
    x = copy_spans(rng_for(seed, f"stress/spans/n{n}/f{frac:.2f}"), x, H, frac)
    return H, x


def long_episode_updates(wl: Workload) -> List[np.ndarray]:
    """The 32 update texts of the long episode; each copies spans from the
    concatenation of the updates before it."""
    out: List[np.ndarray] = []
    H = np.zeros(0, dtype=np.int32)
    for k in range(1, wl.updates + 1):
        x = update_tokens(wl, H, frac=long_episode_frac(k, wl.updates), tag=f"update{k}")
        out.append(x)
        H = np.concatenate([H, x])
    return out


def dense_inputs(wl: Workload, with_lm_head: bool = True) -> Dict[str, np.ndarray]:
    """bf16 bit arrays for the CE and LoRA parts of one update."""
    s = wl.seed
    out: Dict[str, np.ndarray] = {}
    out["h"] = normal_bf16(s, "hidden", (wl.L, wl.d), 1.0)
    if with_lm_head:
        out["W"] = normal_bf16(s, "lm_head", (wl.V, wl.d), 0.02)
    groups = {}
    for p in wl.projs:
        if p.x_group not in groups:
            groups[p.x_group] = normal_bf16(s, f"x/{p.x_group}", (wl.L, p.din), 1.0)
        out[f"x/{p.name}"] = groups[p.x_group]
        out[f"A/{p.name}"] = normal_bf16(s, f"A/{p.name}", (p.din, wl.r), 0.02)
        out[f"B/{p.name}"] = normal_bf16(s, f"B/{p.name}", (wl.r, p.dout), 0.01)
        out[f"dy/{p.name}"] = normal_bf16(s, f"dy/{p.name}", (wl.L, p.dout), 1.0)
    return out


# --------------------------------------------------------------------------
# chained episodes: the adapted projection feeds the LM head
# --------------------------------------------------------------------------

@dataclasses.dataclass
class EpisodeWorkload:
    name: str
    seed: int
    L: int                # update tokens
    V: int
    n: int
    din: int              # adapted projection input width
    d: int                # its output width = LM head input
    r: int
    updates: int          # updates per episode
    hist_len: int = 0     # prior history before the first update
    grad_steps: int = 2   # Appendix C
    cadence: int = 5      # Sec. 4 default K
    frac_first: float = 0.05
    frac_last: float = 0.80
    w_min: float = W_MIN
    lr: float = LORA_LR

    @property
    def scale(self) -> float:
        return 2.0


EPISODES: Dict[str, EpisodeWorkload] = {
    # Tiny shapes (512 x 512 projection, vocab 8192), three updates after the
    # 2,048-token prior history.
    "tiny-episode": EpisodeWorkload("tiny-episode", 0, L=256, V=8192, n=4, din=512, d=512, r=8, updates=3,
                                    hist_len=2048),
    # 7B-class shapes (hidden 3584, vocab 152064, rank 16): 16 updates of
    # 2,048 tokens from an empty history.
    "7b-episode": EpisodeWorkload("7b-episode", 1, L=2048, V=152064, n=4, din=3584, d=3584, r=16, updates=16),
}


def episode_frac(ew: EpisodeWorkload, k: int) -> float:
    """Repeat fraction of update k (1-based), linear from first to last."""
    if ew.updates <= 1:
        return ew.frac_first
    return ew.frac_first + (ew.frac_last - ew.frac_first) * (k - 1) / (ew.updates - 1)


def episode_history(ew: EpisodeWorkload) -> np.ndarray:
    return zipf_ids(rng_for(ew.seed, "episode/history"), ew.hist_len, ew.V)


def episode_texts(ew: EpisodeWorkload) -> List[np.ndarray]:
    """Update texts of one episode; update k copies spans from the prior
    history and the updates before it."""
    out: List[np.ndarray] = []
    H = episode_history(ew)
    for k in range(1, ew.updates + 1):
        x = zipf_ids(rng_for(ew.seed, f"episode/ids{k}"), ew.L, ew.V)
        x = copy_spans(rng_for(ew.seed, f"episode/spans{k}"), x, H, episode_frac(ew, k))
        out.append(x)
        H = np.concatenate([H, x])
    return out


def episode_dense(ew: EpisodeWorkload) -> Dict[str, np.ndarray]:
    """bf16 bits of W0 [din, d] and the LM head [V, d]; fp32 A0 [din, r] and
    B0 [r, d] (the bf16-rounded draws, so both copies start equal)."""
    s = ew.seed
    return {
        "W0": normal_bf16(s, "episode/W0", (ew.din, ew.d), float(1.0 / np.sqrt(ew.din))),
        "W": normal_bf16(s, "episode/lm_head", (ew.V, ew.d), 0.02),
        "A0": bf16_to_f32(normal_bf16(s, "episode/A0", (ew.din, ew.r), 0.02)),
        "B0": bf16_to_f32(normal_bf16(s, "episode/B0", (ew.r, ew.d), 0.01)),
    }


def episode_x(ew: EpisodeWorkload, k: int) -> np.ndarray:
    """bf16 bits of the projection inputs [L, din] of update k (1-based)."""
    return normal_bf16(ew.seed, f"episode/x{k}", (ew.L, ew.din), 1.0)


# --------------------------------------------------------------------------
# update texts as bytes (Eq. 6 / Eq. 7)
# --------------------------------------------------------------------------

_WORD_ALPHABET = np.frombuffer(b"abcdefghijklmnopqrstuvwxyzabcdefghijklmnopqrstuvwxyz0123456789._/()-:", dtype=np.uint8)
_SEPS = (b" ", b"\n", b"\t", b"  ", b"\r\n")
_SEP_P = np.array([0.80, 0.10, 0.04, 0.04, 0.02])


@functools.lru_cache(maxsize=4)
def word_vocab(seed: int, size: int) -> Tuple[bytes, ...]:
    """`size` distinct synthetic words (1-12 characters)."""
    rng = rng_for(seed, "words/vocab")
    out, seen = [], set()
    while len(out) < size:
        n = int(rng.integers(1, 13))
        w = bytes(_WORD_ALPHABET[rng.integers(0, _WORD_ALPHABET.size, n)])
        if w not in seen:
            seen.add(w)
            out.append(w)
    return tuple(out)


def text_bytes(rng: np.random.Generator, ids: np.ndarray, vocab: Tuple[bytes, ...]) -> bytes:
    """Words `ids` of `vocab` joined by random whitespace separators."""
    seps = rng.choice(len(_SEPS), size=len(ids), p=_SEP_P)
    return b"".join(vocab[int(i)] + _SEPS[int(j)] for i, j in zip(ids, seps))


@dataclasses.dataclass
class TextWorkload:
    name: str
    seed: int
    updates: int
    words: int            # words per update text
    vocab: int            # synthetic word vocabulary
    frac_first: float = 0.05
    frac_last: float = 0.95
    tau: float = 0.5      # Appendix C


TEXT_WORKLOADS: Dict[str, TextWorkload] = {
    # a long-episode-shaped run of update texts: 32 updates of ~1,536 words
    # (a 2,048-token update at ~1.33 tokens per word)
    "texts": TextWorkload("texts", 5, updates=32, words=1536, vocab=50000),
    # larger texts for throughput: 64 updates of 131,072 words (~0.8 MB each)
    "texts-stress": TextWorkload("texts-stress", 6, updates=64, words=131072, vocab=200000),
}


def episode_update_texts(tw: TextWorkload) -> List[bytes]:
    """The update texts of one episode: Zipf words, with spans of words
    copied from the previous update's text at a fraction rising linearly."""
    vocab = word_vocab(tw.seed, tw.vocab)
    texts: List[bytes] = []
    prev = np.zeros(0, dtype=np.int32)
    for k in range(1, tw.updates + 1):
        frac = tw.frac_first if tw.updates <= 1 else \
            tw.frac_first + (tw.frac_last - tw.frac_first) * (k - 1) / (tw.updates - 1)
        ids = zipf_ids(rng_for(tw.seed, f"texts/ids{k}"), tw.words, tw.vocab)
        ids = copy_spans(rng_for(tw.seed, f"texts/spans{k}"), ids, prev, frac)
        texts.append(text_bytes(rng_for(tw.seed, f"texts/seps{k}"), ids, vocab))
        prev = ids
    return texts
