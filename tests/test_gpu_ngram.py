"""GPU parity of Eq. 8 / Eq. 9 (history insert + n-gram weights) against the
CPU oracle: bit-exact weights on every workload, plus edge cases."""
import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bits, i32_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _weights(attt, H, x, n, w_min=0.05, chunks=None, max_tokens=None):
    h = attt.attt_history_create(n, max_tokens or max(len(H), 1))
    if chunks is None:
        chunks = [H]
    for c in chunks:
        if len(c):
            attt.attt_history_insert(h, i32_dev(c))
    w = attt.attt_ngram_weights(h, i32_dev(x), w_min).cpu().numpy()
    assert attt.attt_history_status(h) == 0
    h.close()
    return w


def _assert_bit_exact(w, ref):
    diff = np.nonzero(bits(w) != bits(ref))[0]
    assert diff.size == 0, f"{diff.size} weights differ, first at {diff[:5]}: {w[diff[:5]]} vs {ref[diff[:5]]}"


def test_worked_examples(attt):
    import json, os
    cases = json.load(open(os.path.join(os.path.dirname(__file__), "golden", "ngram_worked_examples.json")))["cases"]
    for c in cases:
        H = np.array(c["history"], np.int32)
        x = np.array(c["update"], np.int32)
        chunks = [np.array(ch, np.int32) for ch in c.get("history_chunks", [c["history"]])]
        w = _weights(attt, H, x, c["n"], c["w_min"], chunks=chunks, max_tokens=max(len(H), 1))
        assert [f"0x{b:08x}" for b in bits(w)] == c["w_bits"], c["name"]


@pytest.mark.parametrize("name", ["tiny", "7b", "32b"])
def test_workload_weights(attt, name):
    wl = wk.WORKLOADS[name]
    H = wk.history_tokens(wl)
    x = wk.update_tokens(wl, H)
    w = _weights(attt, H, x, wl.n)
    _assert_bit_exact(w, oracle.ngram_weights(H, x, wl.n))


@pytest.mark.parametrize("n", [3, 4, 5])
@pytest.mark.parametrize("frac", [0.0, 0.3, 0.6, 0.9])
def test_stress_sweep(attt, n, frac):
    """8,192 update tokens against a 1,048,576-token history."""
    H, x = wk.stress_case(n, frac)
    w = _weights(attt, H, x, n)
    _assert_bit_exact(w, oracle.ngram_weights(H, x, n))


def test_long_episode(attt):
    """32 sequential updates, each inserted before the next (Algorithm 1)."""
    wl = wk.WORKLOADS["long"]
    ups = wk.long_episode_updates(wl)
    h = attt.attt_history_create(wl.n, wl.L * wl.updates)
    H = np.zeros(0, np.int32)
    for k, x in enumerate(ups):
        w = attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy()
        _assert_bit_exact(w, oracle.ngram_weights(H, x, wl.n))
        if k == 0:
            assert np.all(w == np.float32(1.0))
        attt.attt_history_insert(h, i32_dev(x))
        H = np.concatenate([H, x])
    assert attt.attt_history_status(h) == 0
    h.close()


def test_chunked_insert_equals_single(attt):
    rng = wk.rng_for(1, "chunks")
    H = wk.zipf_ids(rng, 5000, 64)
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 700, 64), H, 0.5)
    cuts = [0, 1, 2, 3, 50, 1234, 1235, 4999, 5000]
    chunks = [H[a:b] for a, b in zip(cuts[:-1], cuts[1:])]
    for n in (1, 2, 3, 5, 8):
        w1 = _weights(attt, H, x, n)
        w2 = _weights(attt, H, x, n, chunks=chunks, max_tokens=len(H))
        _assert_bit_exact(w1, w2)
        _assert_bit_exact(w1, oracle.ngram_weights(H, x, n))


def test_counts_exact(attt):
    """Table counts equal the brute-force count for present and absent n-grams."""
    rng = wk.rng_for(2, "counts")
    H = wk.zipf_ids(rng, 20000, 40)
    n = 3
    h = attt.attt_history_create(n, len(H))
    attt.attt_history_insert(h, i32_dev(H))
    q = np.concatenate([np.stack([H[p:p + n] for p in range(0, 2000, 7)]),
                        rng.integers(0, 60, (300, n)).astype(np.int32)])
    got = attt.attt_history_count(h, i32_dev(q)).cpu().numpy()
    ref = [oracle.count_naive(H, g) for g in q]
    np.testing.assert_array_equal(got, ref)
    h.close()


def test_edge_cases(attt):
    rng = wk.rng_for(3, "edge")
    H = wk.zipf_ids(rng, 3000, 16)
    # L < n, L == n, L == 1, L == 0, and ragged tile tails
    for L in (0, 1, 2, 3, 4, 5, 47, 48, 49, 95, 96, 97, 255, 256, 257, 511, 513):
        x = wk.zipf_ids(rng, L, 16)
        for n in (1, 4, 16):
            if L == 0:
                h = attt.attt_history_create(n, len(H))
                attt.attt_history_insert(h, i32_dev(H))
                out = torch.empty(0, dtype=torch.float32, device=DEV)
                attt.attt_ngram_weights(h, torch.empty(0, dtype=torch.int32, device=DEV), 0.05, out=out)
                h.close()
                continue
            _assert_bit_exact(_weights(attt, H, x, n), oracle.ngram_weights(H, x, n))
    # empty history
    x = wk.zipf_ids(rng, 100, 16)
    w = _weights(attt, np.zeros(0, np.int32), x, 3, max_tokens=10)
    assert np.all(w == np.float32(1.0))
    # history shorter than n
    w = _weights(attt, np.array([1, 2], np.int32), x, 3, max_tokens=10)
    assert np.all(w == np.float32(1.0))
    # a different floor
    _assert_bit_exact(_weights(attt, H, x, 2, w_min=0.2), oracle.ngram_weights(H, x, 2, 0.2))


def test_reset_and_capacity(attt):
    from paper_2607_03441_gb300.attt import AtttError
    rng = wk.rng_for(4, "reset")
    H = wk.zipf_ids(rng, 1000, 8)
    x = wk.zipf_ids(rng, 64, 8)
    h = attt.attt_history_create(2, 1000)
    attt.attt_history_insert(h, i32_dev(H))
    with pytest.raises(AtttError):
        attt.attt_history_insert(h, i32_dev(H[:1]))  # would exceed max_tokens
    attt.attt_history_reset(h)
    assert attt.attt_history_length(h) == 0
    w = attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy()
    assert np.all(w == np.float32(1.0))
    attt.attt_history_insert(h, i32_dev(H[:500]))
    _assert_bit_exact(attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy(),
                      oracle.ngram_weights(H[:500], x, 2))
    h.close()


def test_invalid_args(attt):
    from paper_2607_03441_gb300.attt import AtttError
    with pytest.raises(AtttError):
        attt.attt_history_create(0, 10)
    with pytest.raises(AtttError):
        attt.attt_history_create(17, 10)
    h = attt.attt_history_create(3, 10)
    with pytest.raises(AtttError):
        attt.attt_ngram_weights(h, i32_dev(np.zeros(4, np.int32)), 0.0)
    h.close()


def test_extreme_ids_and_every_n(attt):
    """Any int32 token value (the sign bit set, 0, INT32_MAX) and n from 1 up
    to the largest, 16: five symbols with copied spans, so that long n-grams
    repeat; weights bit-exact and table counts equal to brute force."""
    rng = wk.rng_for(11, "extreme")
    i32 = np.iinfo(np.int32)
    alphabet = np.array([i32.min, -1, 0, 1, i32.max], np.int32)
    H0 = alphabet[rng.integers(0, 5, 3000)]
    H = wk.copy_spans(rng, H0, H0[:800], 0.5)
    x = wk.copy_spans(rng, alphabet[rng.integers(0, 5, 600)], H, 0.6)
    for n in (1, 2, 3, 8, 15, 16):
        ref = oracle.ngram_weights(H, x, n)
        if n >= 8:
            assert (ref < 1.0).any()  # some n-grams of x do repeat from H
        _assert_bit_exact(_weights(attt, H, x, n), ref)
    n = 16
    h = attt.attt_history_create(n, len(H))
    attt.attt_history_insert(h, i32_dev(H))
    q = np.stack([H[p:p + n] for p in range(0, len(H) - n, 37)] + [x[p:p + n] for p in range(0, 580, 29)])
    got = attt.attt_history_count(h, i32_dev(q)).cpu().numpy()
    np.testing.assert_array_equal(got, [oracle.count_naive(H, g) for g in q])
    assert attt.attt_history_status(h) == 0
    h.close()


def _count_check(attt, h, H, n, rng, picks=300, absent=100, vocab=60):
    q = np.concatenate([np.stack([H[p:p + n] for p in rng.integers(0, len(H) - n + 1, picks)]),
                        rng.integers(0, vocab, (absent, n)).astype(np.int32)])
    got = attt.attt_history_count(h, i32_dev(q)).cpu().numpy()
    np.testing.assert_array_equal(got, [oracle.count_naive(H, g) for g in q])


def test_large_append_between_small_ones_heavy_repeats(attt):
    """A 180,000-token append between small appends, into one table, over a
    50-symbol vocabulary (most n-grams repeat, so most inserts compare tokens
    and add to a count): weights bit-exact, counts exact."""
    rng = wk.rng_for(13, "bulk")
    n = 3
    H = wk.zipf_ids(rng, 200_000, 50)
    h = attt.attt_history_create(n, len(H))
    for a, b in ((0, 5000), (5000, 185_000), (185_000, len(H))):
        attt.attt_history_insert(h, i32_dev(H[a:b]))
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 3000, 50), H, 0.5)
    w = attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy()
    _assert_bit_exact(w, oracle.ngram_weights(H, x, n))
    _count_check(attt, h, H, n, rng, vocab=50)
    assert attt.attt_history_status(h) == 0
    h.close()


def test_append_of_two_and_a_half_million_tokens(attt):
    """One append of 2.5 M Zipf tokens over 128,256 ids (a 16 M-slot table):
    weights bit-exact on an update of copied spans, counts exact."""
    rng = wk.rng_for(14, "bulk_rounds")
    n = 4
    H = wk.zipf_ids(rng, 2_500_000, 128256)
    h = attt.attt_history_create(n, len(H))
    attt.attt_history_insert(h, i32_dev(H))
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 4096, 128256), H, 0.5)
    w = attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy()
    _assert_bit_exact(w, oracle.ngram_weights(H, x, n))
    _count_check(attt, h, H, n, rng, vocab=128256)
    assert attt.attt_history_status(h) == 0
    h.close()


@pytest.mark.slow
def test_history_at_maximum_length(attt):
    """A history filled to its limit, 2^24 - 2 tokens (the 24-bit position and
    count fields at their largest), inserted in three chunks: weights
    bit-exact, counts exact (an n-gram whose only occurrence ends the history
    included), and one token more is refused."""
    from paper_2607_03441_gb300.attt import AtttError
    MAXH = (1 << 24) - 2
    n = 4
    rng = wk.rng_for(12, "maxhist")
    H = wk.zipf_ids(rng, MAXH, 128256)
    tail = np.arange(40, dtype=np.int32) + 200000  # ids that occur nowhere else
    H[-40:] = tail
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 1024, 128256), H[-2_000_000:], 0.4)
    x[500:540] = tail
    h = attt.attt_history_create(n, MAXH)
    for a, b in ((0, 5_000_001), (5_000_001, MAXH - 20), (MAXH - 20, MAXH)):
        attt.attt_history_insert(h, i32_dev(H[a:b]))
    assert attt.attt_history_length(h) == MAXH
    with pytest.raises(AtttError):
        attt.attt_history_insert(h, i32_dev(H[:1]))
    w = attt.attt_ngram_weights(h, i32_dev(x), 0.05).cpu().numpy()
    _assert_bit_exact(w, oracle.ngram_weights(H, x, n))
    assert np.all(w[500:540] == np.float32(0.5))
    q = np.stack([H[p:p + n] for p in (0, 1, 12345, MAXH // 2, MAXH - 41, MAXH - n)] + [tail[:n], tail[-n:]])
    got = attt.attt_history_count(h, i32_dev(q)).cpu().numpy()
    np.testing.assert_array_equal(got, [oracle.count_naive(H, g) for g in q])
    assert got[-1] == 1 and attt.attt_history_status(h) == 0
    h.close()


_M64 = (1 << 64) - 1


def _table_home(tokens, mask):
    """Home slot of an n-gram in the device table: the table's 64-bit hash
    (an odd multiply per token, then a finalizer) masked to the capacity.
    White-box: used only to build inputs with long probe runs."""
    h = (0x9e3779b97f4a7c15 * (len(tokens) + 1)) & _M64
    for t in tokens:
        h = ((h ^ (int(t) & 0xFFFFFFFF)) * 0xbf58476d1ce4e5b9) & _M64
    for mul in (0xff51afd7ed558ccd, 0xc4ceb9fe1a85ec53):
        h ^= h >> 33
        h = (h * mul) & _M64
    h ^= h >> 33
    return h & mask


@pytest.mark.parametrize("n", [1, 2])
def test_long_probe_runs(attt, n):
    """N-grams whose home slots crowd into a few slots of a 1,024-slot table
    form one probe run of ~40 slots, so inserts probe past their home and a
    lookup (present or absent) reads several eight-slot windows.  Weights and
    counts against the oracle."""
    mask = 1023  # the table of a history of <= 256 tokens
    rng = np.random.default_rng(40 + n)
    crowd = []
    while len(crowd) < 60:
        g = rng.integers(0, 1 << 20, n).astype(np.int32)
        if 500 <= _table_home(g, mask) < 504:
            crowd.append(g)
    present, absent = crowd[:40], crowd[40:]
    H = np.concatenate(present).astype(np.int32)  # every window of H starting at a multiple of n is crowded
    # the run: linear probing of H's n-grams, in order, from their home slots
    used = set()
    for p in range(len(H) - n + 1):
        s = _table_home(H[p:p + n], mask)
        while s in used:
            s = (s + 1) & mask
        used.add(s)
    run = 0
    while (500 + run) & mask in used:
        run += 1
    assert run > 3 * 8, run
    x = np.concatenate(present[::3] + absent + present[1::5]).astype(np.int32)
    w = _weights(attt, H, x, n, max_tokens=len(H))
    _assert_bit_exact(w, oracle.ngram_weights(H, x, n))
    h = attt.attt_history_create(n, len(H))
    attt.attt_history_insert(h, i32_dev(H))
    q = np.stack(crowd).astype(np.int32)
    got = attt.attt_history_count(h, i32_dev(q)).cpu().numpy()
    assert attt.attt_history_status(h) == 0
    h.close()
    np.testing.assert_array_equal(got, [oracle.count_naive(H, g) for g in q])
