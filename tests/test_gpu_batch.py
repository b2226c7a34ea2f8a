"""GPU parity of the batched multi-episode update (attt_batch_*) against the
oracle's chained update of each episode on its own: E episodes with private
adapters and histories, updated together (Eq. 8/9, the cast, the SGD step
and the history append as one launch each, Eq. 10 as one call over every
episode's rows), some episodes sitting a round out.

Tolerances as for one episode: Eq. 10 loss 1e-3 relative, dx and the
adapter's change 2e-2 relative L2, the next update's weights bit-exact; an
episode without rows keeps its adapter bit for bit.
"""
import dataclasses

import numpy as np
import pytest
import torch

import oracle
from paper_2607_03441_gb300 import workloads as wk
from tests.gpu_util import DEV, bf16_dev, f32_dev, i32_dev, rel_l2

pytestmark = pytest.mark.gpu

LR = 2.0


@pytest.fixture(scope="module")
def attt():
    from paper_2607_03441_gb300 import attt as a
    from paper_2607_03441_gb300 import build
    build.build()
    oracle.build()
    return a


def _episodes(E):
    base = wk.EPISODES["tiny-episode"]
    eps = []
    for e in range(E):
        ew = dataclasses.replace(base, seed=20 + e, L=base.L - 37 * e)  # ragged update lengths
        eps.append({"ew": ew, "H": wk.episode_history(ew), "texts": wk.episode_texts(ew),
                    "xs": [wk.episode_x(ew, k) for k in range(1, ew.updates + 1)]})
    return base, eps, wk.episode_dense(base)


def _batch(attt, base, eps, dense, E):
    b = attt.Batch(bf16_dev(dense["W0"]), bf16_dev(dense["W"]), f32_dev(dense["A0"]), f32_dev(dense["B0"]),
                   episodes=E, n=base.n, max_history=base.hist_len + base.L * base.updates, max_update=base.L,
                   scale=base.scale, lr=LR, w_min=base.w_min, grad_steps=base.grad_steps)
    for e, ep in enumerate(eps):
        attt.attt_history_insert(b.history(e), i32_dev(ep["H"]))
    return b


def test_batch_matches_each_episode(attt):
    E = 4
    base, eps, dense = _episodes(E)
    b = _batch(attt, base, eps, dense, E)
    state = [{"H": ep["H"], "A": dense["A0"], "B": dense["B0"]} for ep in eps]
    rounds = [[0, 0, 0, 0], [1, None, 1, 1], [2, 1, None, 2]]  # text index per episode; None: no update
    for rnd in rounds:
        lens = [0 if k is None else eps[e]["texts"][k].size for e, k in enumerate(rnd)]
        toks = np.concatenate([eps[e]["texts"][k] for e, k in enumerate(rnd) if k is not None])
        xs = np.concatenate([eps[e]["xs"][k] for e, k in enumerate(rnd) if k is not None])
        R = int(sum(lens))
        losses = torch.full((E, base.grad_steps), -1.0, dtype=torch.float32, device=DEV)
        dx = torch.empty(base.grad_steps, R, base.din, dtype=torch.float32, device=DEV)
        before = [b.read_adapter(e) for e in range(E)]
        b.update(i32_dev(toks), bf16_dev(xs), lens, losses=losses, dx=dx)
        off = np.concatenate([[0], np.cumsum(lens)])
        for e, k in enumerate(rnd):
            A, B = (t.cpu().numpy() for t in b.read_adapter(e))
            if k is None:
                assert torch.equal(b.read_adapter(e)[0], before[e][0]) and torch.equal(b.read_adapter(e)[1], before[e][1])
                assert (losses[e].cpu().numpy() == 0).all()
                continue
            s = state[e]
            ref = oracle.episode_update(s["H"], eps[e]["texts"][k], eps[e]["xs"][k], dense["W0"], dense["W"],
                                        s["A"], s["B"], n=base.n, w_min=base.w_min, scale=base.scale, lr=LR,
                                        grad_steps=base.grad_steps)
            np.testing.assert_allclose(losses[e].cpu().numpy(), ref["losses"], rtol=1e-3)
            for g in range(base.grad_steps):
                assert rel_l2(dx[g, off[e]:off[e + 1]].cpu().numpy(), ref["dx"][g]) < 2e-2, (e, g)
            assert rel_l2(A - s["A"], ref["A32"] - s["A"]) < 2e-2, e
            assert rel_l2(B - s["B"], ref["B32"] - s["B"]) < 2e-2, e
            s["H"], s["A"], s["B"] = ref["H"], ref["A32"], ref["B32"]
        for e in range(E):
            assert attt.attt_history_length(b.history(e)) == state[e]["H"].size
            nxt = eps[e]["texts"][-1]
            w = attt.attt_ngram_weights(b.history(e), i32_dev(nxt), base.w_min).cpu().numpy()
            np.testing.assert_array_equal(w, oracle.ngram_weights(state[e]["H"], nxt, base.n, base.w_min))
    assert attt.attt_device_status() == 0
    # the episode boundary of one episode
    b.reset(1)
    A, B = b.read_adapter(1)
    np.testing.assert_array_equal(A.cpu().numpy(), dense["A0"])
    assert attt.attt_history_length(b.history(1)) == 0
    assert attt.attt_history_length(b.history(0)) == state[0]["H"].size
    b.close()


def test_batch_of_one_equals_the_episode(attt):
    """E = 1: the batch's update is the episode driver's update (same calls
    but Eq. 10 with per-row normalisers: equal to rounding)."""
    base, eps, dense = _episodes(1)
    b = _batch(attt, base, eps, dense, 1)
    ep = attt.Episode(bf16_dev(dense["W0"]), bf16_dev(dense["W"]), f32_dev(dense["A0"]), f32_dev(dense["B0"]),
                      n=base.n, max_history=base.hist_len + base.L * base.updates, max_update=base.L,
                      scale=base.scale, lr=LR, w_min=base.w_min, grad_steps=base.grad_steps)
    attt.attt_history_insert(ep.history(), i32_dev(eps[0]["H"]))
    t, x = i32_dev(eps[0]["texts"][0]), bf16_dev(eps[0]["xs"][0])
    lb = torch.empty(1, base.grad_steps, dtype=torch.float32, device=DEV)
    le = torch.empty(base.grad_steps, dtype=torch.float32, device=DEV)
    b.update(t, x, [t.numel()], losses=lb)
    ep.update(t, x, losses=le)
    np.testing.assert_allclose(lb[0].cpu().numpy(), le.cpu().numpy(), rtol=1e-6)
    (Ab, Bb), (Ae, Be) = b.read_adapter(0), ep.read_adapter()
    assert rel_l2(Ab.cpu().numpy() - dense["A0"], Ae.cpu().numpy() - dense["A0"]) < 1e-3
    assert rel_l2(Bb.cpu().numpy() - dense["B0"], Be.cpu().numpy() - dense["B0"]) < 1e-3
    b.close()
    ep.close()


def test_batch_errors_launch_nothing(attt):
    base, eps, dense = _episodes(2)
    b = attt.Batch(bf16_dev(dense["W0"]), bf16_dev(dense["W"]), f32_dev(dense["A0"]), f32_dev(dense["B0"]),
                   episodes=2, n=base.n, max_history=300, max_update=base.L, scale=2.0, lr=1.0)
    t = i32_dev(np.concatenate([eps[0]["texts"][0], eps[1]["texts"][0]]))
    x = bf16_dev(np.concatenate([eps[0]["xs"][0], eps[1]["xs"][0]]))
    lens = [eps[0]["texts"][0].size, eps[1]["texts"][0].size]
    b.update(t, x, lens)
    n0 = attt.attt_kernel_launches()
    with pytest.raises(attt.AtttError) as e:     # episode 0's history would exceed 300 tokens
        b.update(t, x, lens)
    assert e.value.code == attt.ATTT_ERR_CAPACITY
    with pytest.raises(attt.AtttError) as e:     # an update longer than max_update
        b.update(t, x, [base.L + 1, sum(lens) - base.L - 1])
    assert e.value.code == attt.ATTT_ERR_INVALID_ARG
    assert attt.attt_kernel_launches() == n0
    b.update(t[:0], x[:0], [0, 0])               # nobody has text: nothing happens
    assert attt.attt_kernel_launches() == n0
    b.close()


@pytest.mark.slow
def test_7b_shapes_batch_equals_episodes(attt):
    """Two 7B-class episodes (2,048-token updates, 152,064-entry head,
    3,584 x 3,584 projection, rank 16) updated as a batch equal the same
    episodes updated one by one: losses to 1e-5, adapter changes to 1e-3
    relative L2 (Eq. 10 over 4,096 rows takes other vocabulary chunks than
    over 2,048, so only rounding differs)."""
    ew = wk.EPISODES["7b-episode"]
    dense = wk.episode_dense(ew)
    texts = wk.episode_texts(ew)[:2]
    xs = [wk.episode_x(ew, k) for k in (1, 2)]
    W0, W = bf16_dev(dense["W0"]), bf16_dev(dense["W"])
    A0, B0 = f32_dev(dense["A0"]), f32_dev(dense["B0"])
    kw = dict(n=ew.n, max_history=4 * ew.L, max_update=ew.L, scale=ew.scale, lr=0.5, w_min=ew.w_min,
              grad_steps=ew.grad_steps)
    b = attt.Batch(W0, W, A0, B0, episodes=2, **kw)
    lb = torch.empty(2, ew.grad_steps, dtype=torch.float32, device=DEV)
    b.update(i32_dev(np.concatenate(texts)), bf16_dev(np.concatenate(xs)), [ew.L, ew.L], losses=lb)
    for e in range(2):
        ep = attt.Episode(W0, W, A0, B0, cadence=1, **kw)
        le = torch.empty(ew.grad_steps, dtype=torch.float32, device=DEV)
        ep.update(i32_dev(texts[e]), bf16_dev(xs[e]), losses=le)
        np.testing.assert_allclose(lb[e].cpu().numpy(), le.cpu().numpy(), rtol=1e-5)
        (Ab, Bb), (Ae, Be) = b.read_adapter(e), ep.read_adapter()
        assert rel_l2(Ab.cpu().numpy() - dense["A0"], Ae.cpu().numpy() - dense["A0"]) < 1e-3
        assert rel_l2(Bb.cpu().numpy() - dense["B0"], Be.cpu().numpy() - dense["B0"]) < 1e-3
        ep.close()
    assert attt.attt_device_status() == 0
    b.close()


def test_batch_of_twenty_episodes(attt):
    """20 episodes: the adapter gradients run as two grouped launches per pass
    (16 episodes each at most); every episode against the oracle."""
    E = 20
    base, eps, dense = _episodes(E if E <= 6 else 6)
    # 20 episodes from 6 generated ones, with their lengths cut apart
    eps = [dict(eps[e % 6], cut=min(eps[e % 6]["texts"][0].size, base.L - 9 * e)) for e in range(E)]
    b = _batch(attt, base, [{"H": ep["H"]} for ep in eps], dense, E)
    lens = [ep["cut"] for ep in eps]
    toks = np.concatenate([ep["texts"][0][:n] for ep, n in zip(eps, lens)])
    xs = np.concatenate([ep["xs"][0][:n] for ep, n in zip(eps, lens)])
    losses = torch.empty(E, base.grad_steps, dtype=torch.float32, device=DEV)
    R = int(sum(lens))
    dx = torch.empty(base.grad_steps, R, base.din, dtype=torch.float32, device=DEV)
    b.update(i32_dev(toks), bf16_dev(xs), lens, losses=losses, dx=dx)
    off = np.concatenate([[0], np.cumsum(lens)])
    for e in (0, 7, 15, 16, 19):     # both launches of each pass, and their edges
        ep = eps[e]
        ref = oracle.episode_update(ep["H"], ep["texts"][0][:lens[e]], ep["xs"][0][:lens[e]], dense["W0"],
                                    dense["W"], dense["A0"], dense["B0"], n=base.n, w_min=base.w_min,
                                    scale=base.scale, lr=LR, grad_steps=base.grad_steps)
        np.testing.assert_allclose(losses[e].cpu().numpy(), ref["losses"], rtol=1e-3)
        A, B = (t.cpu().numpy() for t in b.read_adapter(e))
        assert rel_l2(A - dense["A0"], ref["A32"] - dense["A0"]) < 2e-2, e
        assert rel_l2(B - dense["B0"], ref["B32"] - dense["B0"]) < 2e-2, e
        assert rel_l2(dx[1, off[e]:off[e + 1]].cpu().numpy(), ref["dx"][1]) < 2e-2, e
    assert attt.attt_device_status() == 0
    b.close()
