"""The seeded synthetic workloads have the structure their recipes state (the
shapes, masks, group layouts and reward draws that stand in for the paper's
rollouts), and the same seed gives the same bits.  CPU only; the dense H and W
are left out except on the tiny case."""

import numpy as np
import torch

from paper_2607_20908_gb300 import inputs


def _seq_lengths(c):
    cu = c["cu_seqlens"].numpy().astype(np.int64)
    assert cu[0] == 0 and cu[-1] == c["T"] and np.all(np.diff(cu) >= 0)
    return np.diff(cu)


def test_tiny_case():
    c = inputs.tiny_case()
    assert (c["T"], c["d"], c["V"]) == (256, 256, 4096)
    assert c["H"].dtype == torch.bfloat16 and c["W"].dtype == torch.bfloat16
    assert c["H"].shape == (256, 256) and c["W"].shape == (4096, 256)
    assert abs(c["H"].float().std().item() - 1.0) < 0.02
    assert abs(c["W"].float().std().item() - 0.02) < 0.001
    assert np.all(_seq_lengths(c) == 16)
    np.testing.assert_array_equal(c["group_id"].numpy(), np.repeat(np.arange(4), 4))
    r = c["rewards"].numpy()
    assert r.shape == (16,) and r.min() >= 0 and r.max() <= 3
    assert int(c["mask"].sum()) == 256
    t = c["tgt"].numpy()
    assert t.min() >= 0 and t.max() < 4096


def test_full_case_layout():
    c = inputs.full_case(with_HW=False)
    assert (c["T"], c["d"], c["V"]) == (16384, 5120, 151936)
    assert np.all(_seq_lengths(c) == 128) and c["cu_seqlens"].numel() == 129
    np.testing.assert_array_equal(c["group_id"].numpy(), np.repeat(np.arange(16), 8))
    assert int(c["mask"].sum()) == c["T"]
    assert (c["clip_eps"], c["kl_beta"], c["window"]) == (0.2, 0.04, 1024)
    assert abs(c["old_noise"].std().item() - 0.05) < 0.002


def test_composite_reward_distribution():
    r = inputs.composite_rewards(200000, torch.Generator().manual_seed(3)).double()
    # Bernoulli(0.5) + N(0.3, 0.5^2) + U[0, 1]: mean 1.3, variance 0.25 + 0.25 + 1/12
    assert abs(r.mean().item() - 1.3) < 0.01
    assert abs(r.var().item() - (0.25 + 0.25 + 1.0 / 12.0)) < 0.01


def test_ragged_case_layout():
    c = inputs.ragged_case(with_HW=False)
    lens = _seq_lengths(c)
    assert c["T"] == 65536 and lens.sum() == 65536 and lens.min() >= 16
    gid = c["group_id"].numpy()
    assert c["n_groups"] == 32 and np.all(np.diff(gid) >= 0)
    per_group = np.bincount(gid, minlength=32)
    assert per_group.min() >= 8 and per_group.max() <= 32       # 8 rollouts x 1-4 turns
    # a masked prefix of 30-50 % of each sequence: about 40 % of all tokens
    m = c["mask"].numpy()
    cu = c["cu_seqlens"].numpy()
    fracs = np.array([1.0 - m[cu[i]:cu[i + 1]].mean() for i in range(lens.size)])
    long_ = lens >= 64
    assert np.all(fracs[long_] >= 0.28) and np.all(fracs[long_] <= 0.51)
    assert 0.37 < 1.0 - m.mean() < 0.43
    for i in range(lens.size):                                   # a prefix, then all ones
        seg = m[cu[i]:cu[i + 1]]
        k = int((seg == 0).sum())
        assert np.all(seg[:k] == 0) and np.all(seg[k:] == 1)
    # turn lengths were drawn in [64, 1024] before the scaling to 65536 tokens
    assert c["raw_token_total"] >= 64 * lens.size and c["raw_token_total"] <= 1024 * lens.size


def test_large_case_layout():
    c = inputs.large_case(with_HW=False)
    lens = _seq_lengths(c)
    assert c["T"] == 131072 and lens.sum() == 131072
    assert lens.max() <= 1024 and np.all(lens[:-1] >= 64)      # the last one may be truncated
    gid = c["group_id"].numpy()
    sizes = np.bincount(gid, minlength=c["n_groups"])
    assert set(sizes[:-1].tolist()) <= {4, 8, 16} and sizes[-1] <= 16
    r = c["rewards"].numpy()
    zero = c["zero_var_groups"]
    members = np.isin(gid, zero)
    assert members.sum() >= round(0.05 * lens.size) and members.mean() < 0.10
    for g in zero:
        assert np.unique(r[gid == g]).size == 1                  # advantage = 0 path
    others = [g for g in range(c["n_groups"]) if g not in zero and sizes[g] > 1]
    assert all(np.unique(r[gid == g]).size > 1 for g in others)


def test_same_seed_same_bits():
    a, b = inputs.tiny_case(seed=77), inputs.tiny_case(seed=77)
    for k in ("H", "W", "tgt", "rewards", "old_noise", "ref_noise"):
        x, y = a[k], b[k]
        if x.dtype == torch.bfloat16:
            x, y = x.view(torch.int16), y.view(torch.int16)
        assert torch.equal(x, y), k
    c = inputs.tiny_case(seed=78)
    assert not torch.equal(a["H"].view(torch.int16), c["H"].view(torch.int16))
    r1, r2 = inputs.ragged_case(with_HW=False), inputs.ragged_case(with_HW=False)
    assert torch.equal(r1["cu_seqlens"], r2["cu_seqlens"]) and torch.equal(r1["mask"], r2["mask"])
