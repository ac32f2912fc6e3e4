"""The seeded synthetic inputs follow their stated recipes (shapes, dtypes, value
distributions, masks) and are reproducible window by window.  CPU only, small draws."""

import math

import pytest
import torch

import synth


@pytest.mark.parametrize("name", sorted(synth.WORKLOADS))
def test_shapes_dtypes_and_masks(name):
    w = synth.workload(name)
    t, d, m = synth.make_logits(name, seed=1, n_windows=2, V=min(w.V, 512))
    assert t.shape == d.shape == (2, w.K, min(w.V, 512))
    assert t.dtype == d.dtype == w.dtype
    if w.recipe == "peak":
        assert m.shape == (2, w.K) and m.dtype == torch.uint8
    else:
        assert m is None


def test_first_windows_are_the_same_bytes_and_seeds_differ():
    a, b, ma = synth.make_logits("v32k", seed=3, n_windows=256, V=64)
    c, d, mc = synth.make_logits("v32k", seed=3, n_windows=300, V=64)
    assert torch.equal(a, c[:256]) and torch.equal(b, d[:256]) and torch.equal(ma, mc[:256])
    e, _, _ = synth.make_logits("v32k", seed=4, n_windows=256, V=64)
    assert not torch.equal(a, e)


def test_gauss_recipe_moments():
    t, d, _ = synth.make_logits("tiny", seed=0)
    assert abs(t.mean().item()) < 0.05 and abs(t.std().item() - 3.0) < 0.03
    noise = d - t
    assert abs(noise.mean().item()) < 0.02 and abs(noise.std().item() - 1.0) < 0.02


def test_peak_recipe_plants_eight_and_masks_a_tenth():
    # with V = 2 the planted +8 is half of each row's expected sum
    t, d, m = synth.make_logits("v32k", seed=0, V=2)
    rows = t.float().reshape(-1, 2)
    assert abs(rows.sum(1).mean().item() - 8.0) < 0.25            # se 0.06
    noise = (d.float() - 0.8 * t.float())
    assert abs(noise.std().item() - 1.5) < 0.05
    assert abs((m == 0).float().mean().item() - 0.1) < 0.015      # 10240 positions


def test_zipf_recipe_mean_rank_and_random_permutation():
    V = 4096
    t, d, _ = synth.make_logits("v128k", seed=0, n_windows=10, V=V, dtype=torch.float32)
    rows = t.reshape(-1, V)
    # mean of -1.1 ln(rank) over ranks 1..V (the N(0, 0.5^2) term has mean 0)
    expect = -1.1 * math.lgamma(V + 1) / V
    assert abs(rows.mean().item() - expect) < 0.03
    # the rank order is a fresh permutation per row: the argmaxes are spread over the row
    assert len(set(rows.argmax(1).tolist())) > 60
    assert abs((d - t).std().item() - 1.0) < 0.02


def test_gumbel_recipe_moments_and_replaced_rows():
    t, d, _ = synth.make_logits("v152k", seed=0, n_windows=100, V=512, dtype=torch.float32)
    euler = 0.5772156649
    assert abs(t.mean().item() - 3 * euler) < 0.03
    assert abs(t.std().item() - 3 * math.pi / math.sqrt(6)) < 0.05
    same = (t == d).reshape(-1, 512).all(1).float().mean().item()  # 600 rows
    assert abs(same - 0.8) < 0.06


def test_sequence_mask_is_prompt_then_trained_then_padding():
    w = synth.SEQUENCES["seq_v128k"]
    t, d, m = synth.make_seq_logits("seq_v128k", seed=5, V=8)
    assert t.shape == d.shape == (w.B, w.seq_len, 8) and m.shape == (w.B, w.seq_len)
    for b in range(w.B):
        row = m[b].tolist()
        first = row.index(1)
        last = len(row) - 1 - row[::-1].index(1)
        assert all(row[first:last + 1])                       # one contiguous trained span
        assert w.prompt[0] <= first < w.prompt[1]
        assert w.end_lo <= last + 1 <= w.seq_len


def test_reward_groups_are_reproducible_and_distinct():
    kw = dict(windows_per_rollout=2, rollouts_per_group=3, K=4, V=64, with_ref=True)
    t0, d0, r0 = synth.make_reward_logits(0, seed=2, **kw)
    t0b, d0b, r0b = synth.make_reward_logits(0, seed=2, **kw)
    t1, _, _ = synth.make_reward_logits(1, seed=2, **kw)
    assert t0.shape == d0.shape == r0.shape == (6, 4, 64)
    assert torch.equal(t0, t0b) and torch.equal(d0, d0b) and torch.equal(r0, r0b)
    assert not torch.equal(t0, t1)
    # the reference draft is the target plus its own noise, independent of the draft's
    nd, nr = (d0.float() - t0.float()).flatten(), (r0.float() - t0.float()).flatten()
    assert abs(torch.corrcoef(torch.stack([nd, nr]))[0, 1].item()) < 0.1
