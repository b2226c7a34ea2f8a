"""Pins for the oracle's update-text repetition (Eq. 6), novelty (Eq. 7) and
the sequence-level filter (Sec. 4; tau = 0.5 in Appendix C).

Checked against hand-worked examples (tests/golden/jaccard_worked_examples.json),
an independent sort-and-merge count of the word sets, closed forms
(identical texts, disjoint texts, a subset, word order and repeats do not
matter) and the filter's order of update texts.
"""
import json
import os

import numpy as np
import pytest

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "jaccard_worked_examples.json")


def _cases():
    with open(GOLDEN) as f:
        return json.load(f)["cases"]


def _f32(bits: str) -> np.float32:
    return np.array([int(bits, 16)], dtype=np.uint32).view(np.float32)[0]


@pytest.mark.parametrize("case", _cases(), ids=lambda c: c["name"])
def test_golden(oracle_mod, case):
    prev = [bytes.fromhex(h) for h in case["prev_hex"]]
    cur = bytes.fromhex(case["cur_hex"])
    rho, nu = oracle_mod.repetition(prev, cur)
    assert np.float32(rho).view(np.uint32) == _f32(case["rho_bits"]).view(np.uint32)
    assert np.float32(nu).view(np.uint32) == _f32(case["nu_bits"]).view(np.uint32)
    out = oracle_mod.sequence_filter(prev + [cur], case["tau"])
    assert out[-1][2] == case["keep"]


def _merge_counts(a: bytes, b: bytes):
    """|W(a) & W(b)| and |W(a) | W(b)| by sorting each word list, dropping
    repeats and merging (no hashing, no set type)."""
    def uniq(text):
        ws, cur = [], bytearray()
        for ch in text + b" ":
            if ch in b" \t\n\x0b\x0c\r":
                if cur:
                    ws.append(bytes(cur))
                    cur = bytearray()
            else:
                cur.append(ch)
        ws.sort()
        return [w for i, w in enumerate(ws) if i == 0 or w != ws[i - 1]]
    x, y = uniq(a), uniq(b)
    i = j = inter = 0
    while i < len(x) and j < len(y):
        if x[i] == y[j]:
            inter += 1
            i += 1
            j += 1
        elif x[i] < y[j]:
            i += 1
        else:
            j += 1
    return inter, len(x) + len(y) - inter


def _random_text(rng, nwords, vocab):
    seps = [b" ", b" ", b" ", b"\n", b"\t", b"  ", b"\r\n"]
    parts = []
    for _ in range(nwords):
        parts.append(vocab[int(rng.integers(0, len(vocab)))])
        parts.append(seps[int(rng.integers(0, len(seps)))])
    return b"".join(parts)


def test_against_sort_merge(oracle_mod):
    rng = np.random.default_rng(7)
    vocab = [bytes(rng.integers(97, 123, int(rng.integers(1, 6))).astype(np.uint8)) for _ in range(40)]
    for _ in range(200):
        texts = [_random_text(rng, int(rng.integers(0, 30)), vocab) for _ in range(int(rng.integers(1, 6)))]
        cur = texts[-1]
        ref = np.float32(0.0)
        for prev in texts[:-1]:
            inter, union = _merge_counts(cur, prev)
            if union:
                ref = max(ref, np.float32(inter) / np.float32(union))
        rho, nu = oracle_mod.repetition(texts[:-1], cur)
        assert rho == ref
        assert nu == np.float32(1) - ref


def test_closed_forms(oracle_mod):
    a = b"go to shelf 3 then take the mug"
    assert oracle_mod.repetition([a], a) == (np.float32(1), np.float32(0))
    assert oracle_mod.repetition([b"alpha beta"], b"gamma delta")[0] == 0
    # a subset: |small| / |big|
    assert oracle_mod.repetition([b"a b c d"], b"b d")[0] == np.float32(2) / np.float32(4)
    # word order and repeats do not matter; the argument order of J does not either
    assert oracle_mod.repetition([b"c b a"], b"a b b c a")[0] == 1
    x, y = b"one two three four", b"three four five"
    assert oracle_mod.repetition([x], y)[0] == oracle_mod.repetition([y], x)[0]


def test_filter_sees_every_earlier_candidate(oracle_mod):
    """A skipped update's text still counts for the later ones."""
    texts = [b"a b c d", b"a b c d", b"a b c d e f"]
    out = oracle_mod.sequence_filter(texts, 0.5)
    assert [o[2] for o in out] == [True, False, False]
    assert out[0][0] == 0
    assert out[2][0] == np.float32(4) / np.float32(6)
    # tau = 0 keeps every update, tau above 1 skips every update
    assert all(o[2] for o in oracle_mod.sequence_filter(texts, 0.0))
    assert not any(o[2] for o in oracle_mod.sequence_filter(texts, 1.5))


def test_mutations_fail_a_pin(oracle_mod, monkeypatch):
    """A plausible slip (splitting on the space byte only) changes a golden
    case."""
    prev = [bytes.fromhex(h) for h in _cases()[3]["prev_hex"]]
    cur = bytes.fromhex(_cases()[3]["cur_hex"])
    good = oracle_mod.repetition(prev, cur)[0]
    monkeypatch.setattr(oracle_mod, "words", lambda t: set(bytes(t).split(b" ")) - {b""})
    assert oracle_mod.repetition(prev, cur)[0] != good
