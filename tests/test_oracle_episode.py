"""Pins for the oracle's chained update (Algorithm 1 with the adapted
projection feeding the LM head; two gradient steps per update, Appendix C).

Checked against torch CPU autograd of the whole one-layer model (fp64, two
SGD steps, the adapter's bf16 copies rounded by torch's own cast), and the
special cases the algorithm fixes: lr = 0 (nothing moves, both steps agree),
B = 0 (the first step leaves A unchanged), one step equals the first of two,
and the history after the update is H || x_k.
"""
import numpy as np
import pytest
import torch
import torch.nn.functional as F

from paper_2607_03441_gb300 import workloads as wk


def _f64(bits):
    return wk.bf16_to_f32(bits).astype(np.float64)


def _case(seed, L=40, din=48, d=32, V=300, r=8, hist=200, n=3):
    rng = wk.rng_for(seed, "episode-pin/tokens")
    H = rng.integers(0, 12, hist).astype(np.int32)       # small alphabet: repeats
    x_tok = rng.integers(0, 12, L).astype(np.int32)
    x = wk.normal_bf16(seed, "episode-pin/x", (L, din), 1.0)
    W0 = wk.normal_bf16(seed, "episode-pin/W0", (din, d), float(1 / np.sqrt(din)))
    Wlm = wk.normal_bf16(seed, "episode-pin/Wlm", (V, d), 0.3)
    A0 = wk.bf16_to_f32(wk.normal_bf16(seed, "episode-pin/A0", (din, r), 0.05))
    B0 = wk.bf16_to_f32(wk.normal_bf16(seed, "episode-pin/B0", (r, d), 0.05))
    return dict(H=H, tokens=x_tok, x=x, W0=W0, Wlm=Wlm, A0=A0, B0=B0, n=n)


def _rel(a, b):
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    return np.linalg.norm(a - b) / max(np.linalg.norm(b), 1e-300)


def _torch_update(c, w, scale, lr, steps):
    """The same update by torch autograd: fp64 sums, no rounding of h or dy;
    the forward uses bf16 copies of the adapter (torch's cast)."""
    x = torch.from_numpy(_f64(c["x"]))
    W0 = torch.from_numpy(_f64(c["W0"]))
    Wlm = torch.from_numpy(_f64(c["Wlm"]))
    tgt = torch.from_numpy(c["tokens"].astype(np.int64))
    wt = torch.from_numpy(np.asarray(w, np.float64))
    A = torch.from_numpy(c["A0"].astype(np.float64))
    B = torch.from_numpy(c["B0"].astype(np.float64))
    L = x.shape[0]
    losses, dxs = [], []
    for _ in range(steps):
        Ap = A.float().bfloat16().double().requires_grad_(True)
        Bp = B.float().bfloat16().double().requires_grad_(True)
        xp = x.clone().requires_grad_(True)
        h = xp @ W0 + scale * (xp @ Ap) @ Bp
        loss = (wt * F.cross_entropy(h @ Wlm.T, tgt, reduction="none")).sum() / L
        loss.backward()
        losses.append(loss.item())
        dxs.append(xp.grad.numpy())
        A = A - lr * Ap.grad
        B = B - lr * Bp.grad
    return np.array(losses), dxs, A.numpy(), B.numpy()


@pytest.mark.parametrize("lr", [5e-4, 0.5])
def test_two_steps_match_autograd(oracle_mod, lr):
    c = _case(1)
    scale = 2.0
    r = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"], n=c["n"],
                                  w_min=0.05, scale=scale, lr=lr, grad_steps=2)
    losses, dxs, A, B = _torch_update(c, r["w"], scale, lr, 2)
    # h and dy are rounded to bf16 once each on the oracle's side only
    np.testing.assert_allclose(r["losses"], losses, rtol=1e-3)
    for g in range(2):
        assert _rel(r["dx"][g], dxs[g]) < 2e-2
    assert _rel(r["A32"] - c["A0"], A - c["A0"]) < 2e-2
    assert _rel(r["B32"] - c["B0"], B - c["B0"]) < 2e-2
    if lr >= 0.5:
        # the second step sees the adapter the first one moved
        assert abs(losses[1] - losses[0]) > 1e-3 * abs(losses[0])
        assert abs(r["losses"][1] - r["losses"][0]) > 1e-3 * abs(r["losses"][0])


def test_second_step_uses_the_moved_adapter(oracle_mod):
    """A slip that took both steps at the initial adapter gives twice the
    first step's delta; the true second gradient differs from the first."""
    c = _case(2)
    r = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"], n=c["n"],
                                  w_min=0.05, scale=2.0, lr=0.5, grad_steps=2)
    r1 = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"], n=c["n"],
                                   w_min=0.05, scale=2.0, lr=0.5, grad_steps=1)
    wrong = c["B0"] + 2 * (r1["B32"] - c["B0"])
    assert _rel(r["B32"] - c["B0"], wrong - c["B0"]) > 5e-2


def test_lr_zero_moves_nothing(oracle_mod):
    c = _case(3)
    r = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"], n=c["n"],
                                  w_min=0.05, scale=2.0, lr=0.0, grad_steps=2)
    np.testing.assert_array_equal(r["A32"], c["A0"])
    np.testing.assert_array_equal(r["B32"], c["B0"])
    assert r["losses"][0] == r["losses"][1]
    np.testing.assert_array_equal(r["dx"][0], r["dx"][1])


def test_zero_B_leaves_A_after_one_step(oracle_mod):
    """B = 0: v = dy B^T = 0, so dA = 0 and A is unchanged by the first step,
    while B moves (dB = s (x A)^T dy is not zero)."""
    c = _case(4)
    B0 = np.zeros_like(c["B0"])
    r = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], B0, n=c["n"],
                                  w_min=0.05, scale=2.0, lr=0.5, grad_steps=1)
    np.testing.assert_array_equal(r["A32"], c["A0"])
    assert np.abs(r["B32"]).max() > 0
    # and the loss is the base projection's alone
    _, dxs, _, _ = _torch_update(dict(c, B0=B0), r["w"], 2.0, 0.5, 1)
    assert _rel(r["dx"][0], dxs[0]) < 2e-2


def test_one_step_is_the_first_of_two_and_history_grows(oracle_mod):
    c = _case(5)
    kw = dict(n=c["n"], w_min=0.05, scale=2.0, lr=0.5)
    r2 = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"],
                                   grad_steps=2, **kw)
    r1 = oracle_mod.episode_update(c["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], c["A0"], c["B0"],
                                   grad_steps=1, **kw)
    assert r1["losses"][0] == r2["losses"][0]
    np.testing.assert_array_equal(r1["dx"][0], r2["dx"][0])
    np.testing.assert_array_equal(r2["H"], np.concatenate([c["H"], c["tokens"]]))
    # Eq. 8 counts the earlier history only: the weights of this update
    np.testing.assert_array_equal(r2["w"], oracle_mod.ngram_weights(c["H"], c["tokens"], c["n"], 0.05))
    # a second update sees the first one's tokens
    r_next = oracle_mod.episode_update(r2["H"], c["tokens"], c["x"], c["W0"], c["Wlm"], r2["A32"], r2["B32"],
                                       grad_steps=1, **kw)
    assert r_next["w"].max() < 1.0 or len(c["tokens"]) < c["n"]
