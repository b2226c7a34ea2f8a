"""Checkpoint and resume: a history saved and restored gives bit-identical
weights and counts, and an episode saved mid-way (with pending agent-step
text, with SGD or AdamW) and loaded into a fresh episode continues bit for
bit as the original does."""
import numpy as np
import pytest
import torch

from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, f32_dev, i32_dev

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    return a


def test_history_save_restore(attt):
    rng = wk.rng_for(4, "ckpt/h")
    H = wk.zipf_ids(rng, 5003, 300)
    x = wk.copy_spans(rng, wk.zipf_ids(rng, 777, 300), H, 0.5)
    a = attt.History(4, 20000)
    attt.attt_history_insert(a, i32_dev(H[:1000]))
    attt.attt_history_insert(a, i32_dev(H[1000:]))
    saved = attt.attt_history_save(a)
    np.testing.assert_array_equal(saved, H)
    b = attt.History(4, 20000)
    attt.attt_history_insert(b, i32_dev(x))         # whatever it held is replaced
    attt.attt_history_restore(b, saved)
    assert len(b) == len(a) == H.size
    wa = attt.attt_ngram_weights(a, i32_dev(x), 0.05)
    wb = attt.attt_ngram_weights(b, i32_dev(x), 0.05)
    assert torch.equal(wa, wb)
    q = torch.from_numpy(np.lib.stride_tricks.sliding_window_view(x, 4).copy()).to(DEV)
    assert torch.equal(attt.attt_history_count(a, q), attt.attt_history_count(b, q))
    # both go on the same way
    attt.attt_history_insert(a, i32_dev(x))
    attt.attt_history_insert(b, i32_dev(x))
    assert torch.equal(attt.attt_ngram_weights(a, i32_dev(x), 0.05), attt.attt_ngram_weights(b, i32_dev(x), 0.05))
    with pytest.raises(attt.AtttError) as e:
        attt.attt_history_restore(attt.History(4, 100), saved)
    assert e.value.code == attt.ATTT_ERR_CAPACITY
    assert attt.attt_history_status(a) == 0 and attt.attt_history_status(b) == 0


@pytest.mark.parametrize("optimizer", ["sgd", "adamw"])
def test_episode_save_load_continues_bit_for_bit(attt, optimizer):
    ew = wk.EPISODES["tiny-episode"]
    texts, dense = wk.episode_texts(ew), wk.episode_dense(ew)
    xs = [wk.episode_x(ew, k) for k in range(1, ew.updates + 1)]
    kw = dict(n=ew.n, max_history=ew.hist_len + ew.L * ew.updates, max_update=ew.L, scale=ew.scale,
              lr=2.0 if optimizer == "sgd" else 1e-3, w_min=ew.w_min, grad_steps=ew.grad_steps, cadence=3,
              optimizer=optimizer)
    args = (bf16_dev(dense["W0"]), bf16_dev(dense["W"]), f32_dev(dense["A0"]), f32_dev(dense["B0"]))
    ep = attt.Episode(*args, **kw)
    attt.attt_history_insert(ep.history(), i32_dev(wk.episode_history(ew)))
    ep.update(i32_dev(texts[0]), bf16_dev(xs[0]))
    # two agent steps of the next update: text pending when the checkpoint is taken
    for s, e in ((0, 100), (100, 180)):
        ep.agent_step(i32_dev(texts[1][s:e]), bf16_dev(xs[1][s:e]))
    blob = ep.save()

    def finish(episode):
        losses = torch.empty(ew.grad_steps, dtype=torch.float32, device=DEV)
        fired = episode.agent_step(i32_dev(texts[1][180:]), bf16_dev(xs[1][180:]), losses=losses)
        assert fired
        episode.update(i32_dev(texts[2]), bf16_dev(xs[2]), losses=losses)
        return (losses, *episode.read_adapter()), len(episode.history())

    ref, ref_len = finish(ep)
    fresh = attt.Episode(*args, **kw)
    fresh.load(blob)
    assert fresh.pending_tokens() == 180
    got, got_len = finish(fresh)
    assert got_len == ref_len
    for p, q in zip(ref, got):
        assert torch.equal(p, q)
    # a checkpoint of another configuration, or a cut one, is refused
    other = attt.Episode(*args, **dict(kw, lr=kw["lr"] * 2))
    with pytest.raises(attt.AtttError):
        other.load(blob)
    with pytest.raises(attt.AtttError):
        fresh.load(blob[: len(blob) // 2])
    assert attt.attt_device_status() == 0
    for x in (ep, fresh, other):
        x.close()
