"""GPU parity of the update-text repetition (Eq. 6), novelty (Eq. 7) and the
sequence-level filter (attt_wordsets_*, attt_repetition) against the oracle:
rho and nu bit-exact, keep exact, on the hand-worked cases, a synthetic
episode drifting into repetition, more than 64 updates (several mask
words), words longer than the 16-bit length field, and the edge cases.
"""
import json
import os

import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV

pytestmark = pytest.mark.gpu

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "jaccard_worked_examples.json")


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    return a


def _dev(text: bytes) -> torch.Tensor:
    return torch.frombuffer(bytearray(text), dtype=torch.uint8).to(DEV) if text else \
        torch.empty(0, dtype=torch.uint8, device=DEV)


def _run(attt, ws, texts, tau):
    outs, keeps = [], []
    for t in texts:
        o, k = attt.attt_repetition(ws, _dev(t), tau)
        outs.append(o)
        keeps.append(k)
    torch.cuda.synchronize()
    return [(o.cpu().numpy(), int(k.item())) for o, k in zip(outs, keeps)]


def _check(got, ref):
    assert len(got) == len(ref)
    for i, ((o, keep), (rho, nu, kref)) in enumerate(zip(got, ref)):
        assert o[0].view(np.uint32) == np.float32(rho).view(np.uint32), (i, o[0], rho)
        assert o[1].view(np.uint32) == np.float32(nu).view(np.uint32), (i, o[1], nu)
        assert keep == int(kref), i


def test_golden_cases(attt):
    with open(GOLDEN) as f:
        cases = json.load(f)["cases"]
    for c in cases:
        texts = [bytes.fromhex(h) for h in c["prev_hex"]] + [bytes.fromhex(c["cur_hex"])]
        ws = attt.WordSets(8, 4096)
        got = _run(attt, ws, texts, c["tau"])
        (o, keep) = got[-1]
        assert o[0].view(np.uint32) == int(c["rho_bits"], 16), c["name"]
        assert o[1].view(np.uint32) == int(c["nu_bits"], 16), c["name"]
        assert keep == int(c["keep"]), c["name"]
        assert attt.attt_wordsets_status(ws) == 0
        ws.close()


def test_synthetic_episode_matches_oracle(attt):
    tw = wk.TEXT_WORKLOADS["texts"]
    texts = wk.episode_update_texts(tw)
    ws = attt.WordSets(tw.updates, sum(len(t) for t in texts))
    got = _run(attt, ws, texts, tw.tau)
    ref = oracle.sequence_filter(texts, tw.tau)
    _check(got, ref)
    assert any(not k for _, _, k in ref) and any(k for _, _, k in ref)  # the filter both keeps and skips
    assert attt.attt_wordsets_status(ws) == 0 and len(ws) == tw.updates
    # reset: the episode starts over with the same results
    attt.attt_wordsets_reset(ws)
    _check(_run(attt, ws, texts[:5], tw.tau), ref[:5])
    ws.close()


def test_many_updates_cross_mask_words(attt):
    """150 updates: the update bits span three 64-bit mask words."""
    rng = np.random.default_rng(11)
    vocab = wk.word_vocab(3, 300)
    texts = []
    for k in range(150):
        ids = wk.zipf_ids(rng, int(rng.integers(0, 40)), len(vocab))
        if k % 7 == 3 and texts:
            texts.append(texts[int(rng.integers(0, len(texts)))])  # an exact repeat of an earlier text
        else:
            texts.append(wk.text_bytes(rng, ids, vocab))
    ws = attt.WordSets(200, sum(len(t) for t in texts))
    _check(_run(attt, ws, texts, 0.5), oracle.sequence_filter(texts, 0.5))
    ws.close()


def test_edge_texts(attt):
    long_a = b"x" * 70000 + b"a"
    long_b = b"x" * 70000 + b"b"
    texts = [b"", b"   \n\t", b"word", b"word", long_a, long_b + b" " + long_a, b"\x00\xff \x80",
             b"\x00\xff", b"no-trailing-space", b"a\x0bb\x0cc\rd", b"a b c d"]
    ws = attt.WordSets(len(texts), sum(len(t) for t in texts))
    _check(_run(attt, ws, texts, 0.5), oracle.sequence_filter(texts, 0.5))
    ws.close()


def test_capacity_errors_launch_nothing(attt):
    ws = attt.WordSets(2, 10)
    attt.attt_repetition(ws, _dev(b"abc"), 0.5)
    n0 = attt.attt_kernel_launches()
    with pytest.raises(attt.AtttError) as e:       # text bytes beyond max_bytes
        attt.attt_repetition(ws, _dev(b"0123456789"), 0.5)
    assert e.value.code == attt.ATTT_ERR_CAPACITY
    attt.attt_repetition(ws, _dev(b"de"), 0.5)
    n1 = attt.attt_kernel_launches()
    with pytest.raises(attt.AtttError) as e:       # a third update
        attt.attt_repetition(ws, _dev(b"f"), 0.5)
    assert e.value.code == attt.ATTT_ERR_CAPACITY
    assert attt.attt_kernel_launches() == n1 and n1 - n0 == 1  # one launch per update
    assert len(ws) == 2 and attt.attt_wordsets_status(ws) == 0
    ws.close()
    with pytest.raises(attt.AtttError):
        attt.WordSets(0, 10)


@pytest.mark.slow
def test_stress_texts_first_updates(attt):
    """The stress texts (~1 MB, 131,072 words each): the first eight updates
    of the episode, bit-exact with the oracle, through the launch the bench
    times (chunks of 2,048 bytes, every SM)."""
    tw = wk.TEXT_WORKLOADS["texts-stress"]
    texts = wk.episode_update_texts(tw)[:8]
    ws = attt.WordSets(tw.updates, sum(len(t) for t in texts))
    _check(_run(attt, ws, texts, tw.tau), oracle.sequence_filter(texts, tw.tau))
    assert attt.attt_wordsets_status(ws) == 0
    ws.close()
