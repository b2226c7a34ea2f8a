"""Pins for the oracle's Eq. 8 / Eq. 9 (n-gram exposure and token weights).

The oracle is checked against things other than itself: hand-worked cases
(tests/golden), a brute-force Counter over every n-gram of tiny inputs, the
agreement of its two independent counters, a histogram for n = 1, and the
invariants the definitions imply.
"""
import collections
import itertools
import json
import os

import numpy as np
import pytest

from paper_2607_03441_gb300 import workloads as wk

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "ngram_worked_examples.json")


def _bits(w):
    return [f"0x{int(b):08x}" for b in np.asarray(w, dtype=np.float32).view(np.uint32)]


def brute_force_exposure(H, x, n):
    """Count every n-gram of H with a Counter, then take the max over the
    n-grams of x that cover each position (Eq. 8, written as a hash count)."""
    cnt = collections.Counter(tuple(H[p:p + n]) for p in range(len(H) - n + 1))
    f = [0] * len(x)
    for s in range(len(x) - n + 1):
        c = cnt.get(tuple(x[s:s + n]), 0)
        for j in range(s, s + n):
            f[j] = max(f[j], c)
    return f


@pytest.mark.parametrize("case", json.load(open(GOLDEN))["cases"], ids=lambda c: c["name"])
@pytest.mark.parametrize("method", ["naive", "sorted"])
def test_worked_examples(oracle_mod, case, method):
    H = np.array(case["history"], dtype=np.int32)
    x = np.array(case["update"], dtype=np.int32)
    f = oracle_mod.exposure(H, x, case["n"], method)
    assert f.tolist() == case["f"]
    w = oracle_mod.weights_from_exposure(f, case["w_min"])
    assert _bits(w) == case["w_bits"]


def test_exhaustive_tiny(oracle_mod):
    """Every history of length <= 5 and update of length <= 4 over a 2-letter
    alphabet, n in 1..3: both counters equal the brute force."""
    for n in (1, 2, 3):
        for lh in range(0, 6):
            for H in itertools.product((0, 1), repeat=lh):
                for lx in range(0, 5):
                    for x in itertools.product((0, 1), repeat=lx):
                        ref = brute_force_exposure(list(H), list(x), n)
                        Ha = np.array(H, dtype=np.int32)
                        xa = np.array(x, dtype=np.int32)
                        assert oracle_mod.exposure(Ha, xa, n, "naive").tolist() == ref
                        assert oracle_mod.exposure(Ha, xa, n, "sorted").tolist() == ref


def test_random_brute_force(oracle_mod):
    rng = np.random.default_rng(7)
    for trial in range(300):
        V = int(rng.integers(1, 9))
        L = int(rng.integers(0, 13))
        nH = int(rng.integers(0, 41))
        n = int(rng.integers(1, 6))
        H = rng.integers(0, V, nH).astype(np.int32)
        x = rng.integers(0, V, L).astype(np.int32)
        ref = brute_force_exposure(H.tolist(), x.tolist(), n)
        assert oracle_mod.exposure(H, x, n, "naive").tolist() == ref
        assert oracle_mod.exposure(H, x, n, "sorted").tolist() == ref


def test_counters_agree_medium(oracle_mod):
    """The naive scan and the sort-based counter on a Zipf workload."""
    rng = wk.rng_for(11, "agree")
    H = wk.zipf_ids(rng, 6000, 512)
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 400, 512), H, 0.5)
    for n in (2, 3, 4, 5):
        a = oracle_mod.exposure(H, x, n, "naive")
        b = oracle_mod.exposure(H, x, n, "sorted")
        np.testing.assert_array_equal(a, b)


def test_unigram_is_histogram(oracle_mod):
    rng = np.random.default_rng(3)
    H = rng.integers(0, 50, 3000).astype(np.int32)
    x = rng.integers(0, 60, 500).astype(np.int32)
    hist = np.bincount(H, minlength=60)
    f = oracle_mod.exposure(H, x, 1)
    np.testing.assert_array_equal(f, hist[x])


def test_invariants(oracle_mod):
    rng = wk.rng_for(5, "inv")
    H = wk.zipf_ids(rng, 20000, 300)
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 1000, 300), H, 0.4)
    for n in (3, 4):
        # empty history: every weight is 1
        w0 = oracle_mod.ngram_weights(np.zeros(0, np.int32), x, n)
        assert np.all(w0 == np.float32(1.0))
        # weights in [w_min, 1]
        w = oracle_mod.ngram_weights(H, x, n)
        assert np.all(w >= np.float32(0.05)) and np.all(w <= np.float32(1.0))
        # more history never raises a weight
        w_more = oracle_mod.ngram_weights(np.concatenate([H, wk.zipf_ids(rng, 5000, 300)]), x, n)
        assert np.all(w_more <= w)
        # a contiguous copy of the history (L >= n): every weight <= 1/2
        src = H[1234:1234 + 64]
        wc = oracle_mod.ngram_weights(H, src, n)
        assert np.all(wc <= np.float32(0.5))


def test_floor_saturation(oracle_mod):
    """Every exposure at or above 19 gives exactly the floor 0.05f, because
    RN(1/20) == 0.05f; below 19 the weight is strictly above the floor."""
    f = np.arange(0, 200, dtype=np.int64)
    w = oracle_mod.weights_from_exposure(f, 0.05)
    assert np.all(w[19:] == np.float32(0.05))
    assert np.all(w[:19] > np.float32(0.05))
    # and the weights are exactly the fp32 quotients
    q = (np.float32(1.0) / (np.float32(1.0) + f[:19].astype(np.float32))).astype(np.float32)
    np.testing.assert_array_equal(w[:19], q)


def test_mutations_are_caught(oracle_mod):
    """A plausible slip in Eq. 8 (max over only the window starting at j, or an
    off-by-one end of the history scan) changes a golden case."""
    case = [c for c in json.load(open(GOLDEN))["cases"] if c["name"] == "window_max_over_covering_ngrams"][0]
    H, x, n = case["history"], case["update"], case["n"]
    cnt = collections.Counter(tuple(H[p:p + n]) for p in range(len(H) - n + 1))
    only_start = [cnt.get(tuple(x[j:j + n]), 0) if j + n <= len(x) else 0 for j in range(len(x))]
    assert only_start != case["f"]
    cnt_short = collections.Counter(tuple(H[p:p + n]) for p in range(len(H) - n))
    f_short = [0] * len(x)
    for s in range(len(x) - n + 1):
        for j in range(s, s + n):
            f_short[j] = max(f_short[j], cnt_short.get(tuple(x[s:s + n]), 0))
    assert f_short != case["f"]
