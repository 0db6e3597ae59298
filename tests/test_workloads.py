"""Checks of the seeded input generator (CPU only): its FP8-E4M3 emulation of
the rollout engine and the structure of each workload."""

import numpy as np
import pytest
import torch

import workloads as W


def test_e4m3_grid_is_the_format():
    v = W.e4m3_values()
    assert v.numel() == 127 and float(v[-1]) == 448.0 and float(v[1]) == 2.0 ** -9
    assert torch.all(v[1:] > v[:-1])
    # every representable value survives both roundings unchanged
    for mode in ("nearest", "trunc"):
        assert torch.equal(W.e4m3_roundtrip(v, mode), v)
        assert torch.equal(W.e4m3_roundtrip(-v, mode), -v)


def test_e4m3_rounding_rules():
    # spacing 0.125 in [1, 2): ties go to the even mantissa
    x = torch.tensor([1.0625, 1.1875, 1.3125, -1.0625, 1.06, 1.07, 500.0])
    assert W.e4m3_roundtrip(x, "nearest").tolist() == [1.0, 1.25, 1.25, -1.0, 1.0, 1.125, 448.0]
    # truncation goes toward zero (Sec. 5.3 stress quantiser)
    y = torch.tensor([1.124, 1.126, -1.126, 0.0019, 447.0])
    assert W.e4m3_roundtrip(y, "trunc").tolist() == [1.0, 1.125, -1.125, 0.0, 416.0]


def test_nearest_matches_bruteforce_grid():
    g = torch.Generator().manual_seed(0)
    x = (torch.rand(4000, generator=g) - 0.5) * 900
    grid = torch.cat([-W.e4m3_values().flip(0), W.e4m3_values()])
    q = W.e4m3_roundtrip(x, "nearest")
    dist = (x.view(-1, 1) - grid.view(1, -1)).abs()
    best = dist.min(dim=1).values
    assert torch.all((q - x).abs() <= best + 1e-6)


@pytest.mark.parametrize("name", ["tiny", "grpo", "qwen", "long"])
def test_structure(name):
    spec = W.SPECS[name]
    st = W.make_structure(spec, W.seed_for(name))
    S = spec.n_seqs
    assert st.seq_offsets.numel() == S + 1 and int(st.seq_offsets[0]) == 0
    assert torch.all(st.lengths >= spec.len_lo) and torch.all(st.lengths <= spec.len_hi)
    assert int(st.mask.sum()) == int(st.lengths.sum())
    assert st.group_offsets.tolist() == [k * spec.group_size for k in range(spec.n_prompts + 1)]
    if spec.pad_multiple:
        assert torch.all((st.seq_offsets[1:] - st.seq_offsets[:-1]) % spec.pad_multiple == 0)
    # same seed, same structure
    st2 = W.make_structure(spec, W.seed_for(name))
    assert torch.equal(st.seq_offsets, st2.seq_offsets) and torch.equal(st.rewards, st2.rewards)


def test_generate_small_is_deterministic_and_valid():
    spec = W.small_variant(W.GRPO, n_prompts=2, group_size=3, len_lo=5, len_hi=70, V=1003, ld_pad=8)
    a = W.generate(spec, seed=5)
    b = W.generate(spec, seed=5)
    assert torch.equal(a.logits.view(torch.int16), b.logits.view(torch.int16))
    assert a.ld % 8 == 0 and a.ld >= a.V
    assert torch.all(a.logits[:, a.V:] == 0)
    assert torch.all((a.ids >= 0) & (a.ids < a.V))
    assert torch.all(a.logp_mu <= 0) and torch.all(torch.isfinite(a.logp_mu))
    assert np.isclose(float(a.logits[:, :a.V].float().std()), 3.0 * np.sqrt(1 + 0.01 * 64 / 9 - 0.0), rtol=0.2)
