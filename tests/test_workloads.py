"""The seeded input generators (no method arithmetic): the recipe the
synthetic workloads follow -- truncated Zipf(1.1) ids, spans copied from the
history covering round(frac L) positions, the long episode's rising repeat
fraction, shared projection inputs, bf16 round-to-nearest-even."""
import numpy as np
import torch

from paper_2607_03441_gb300 import workloads as wk


def test_streams_are_reproducible_and_independent():
    a = wk.zipf_ids(wk.rng_for(3, "x"), 1000, 5000)
    b = wk.zipf_ids(wk.rng_for(3, "x"), 1000, 5000)
    c = wk.zipf_ids(wk.rng_for(3, "y"), 1000, 5000)
    d = wk.zipf_ids(wk.rng_for(4, "x"), 1000, 5000)
    assert np.array_equal(a, b) and not np.array_equal(a, c) and not np.array_equal(a, d)


def test_zipf_ids_follow_the_truncated_law():
    V, n, a = 1000, 400_000, 1.1
    ids = wk.zipf_ids(wk.rng_for(0, "zipf"), n, V, a)
    assert ids.dtype == np.int32 and ids.min() >= 0 and ids.max() < V
    p = np.arange(1, V + 1, dtype=np.float64) ** -a
    p /= p.sum()
    counts = np.bincount(ids, minlength=V)
    # the ten most frequent ranks, each within 4 standard deviations of n p_k
    for k in range(10):
        sd = np.sqrt(n * p[k] * (1 - p[k]))
        assert abs(counts[k] - n * p[k]) < 4 * sd, (k, counts[k], n * p[k])
    # hot ids are low: frequencies fall with the id
    assert counts[0] > counts[1] > counts[2] > counts[9] > counts[99]


def test_copy_spans_covers_the_stated_fraction_from_the_history():
    rng = wk.rng_for(1, "spans")
    H = wk.zipf_ids(rng, 5000, 800)
    for L, frac in ((2048, 0.4), (256, 0.3), (1000, 0.0), (100, 1.0), (4096, 0.8)):
        x = np.full(L, -1, np.int32)
        y = wk.copy_spans(wk.rng_for(2, f"s{L}"), x, H, frac)
        covered = y != -1
        assert covered.sum() == round(frac * L)
        assert np.isin(y[covered], H).all()
    # the input is not modified
    x = np.full(50, -1, np.int32)
    wk.copy_spans(rng, x, H, 0.5)
    assert (x == -1).all()


def test_long_episode_fraction_rises_linearly():
    assert wk.long_episode_frac(1) == 0.05
    assert abs(wk.long_episode_frac(32) - 0.80) < 1e-12
    f = [wk.long_episode_frac(k) for k in range(1, 33)]
    assert np.allclose(np.diff(f), 0.75 / 31)


def test_projections_sharing_an_input_share_x():
    wl = wk.WORKLOADS["tiny"]
    dense = wk.dense_inputs(wl, with_lm_head=False)
    assert dense["x/proj"].shape == (wl.L, 512) and dense["dy/proj"].shape == (wl.L, 512)
    wl = wk.WORKLOADS["7b"]
    groups = {p.x_group for p in wl.projs}
    assert groups == {"attn"}  # q and v read the same attention input
    h = wk.bf16_to_f32(wk.normal_bf16(1, "hidden", (256, 512), 1.0))
    W = wk.bf16_to_f32(wk.normal_bf16(1, "lm_head", (512, 512), 0.02))
    assert abs(h.std() - 1.0) < 0.02 and abs(W.std() - 0.02) < 0.0005


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(5)
    v = np.concatenate([rng.standard_normal(10000).astype(np.float32) * 10.0 ** rng.integers(-8, 8, 10000),
                        np.array([0.0, -0.0, np.inf, -np.inf, 1.0 + 2.0 ** -8, 1.0 + 3 * 2.0 ** -8,
                                  3.3895314e38, 1e-40], np.float32)]).astype(np.float32)
    ours = wk.bf16_bits(v)
    ref = torch.from_numpy(v).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    assert np.array_equal(wk.bf16_to_f32(ours), torch.from_numpy(v).to(torch.bfloat16).float().numpy())
