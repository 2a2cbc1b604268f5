"""Seeded synthetic workloads for the GRPO log-prob / policy-loss path.

This module only draws random inputs; it contains none of the method's
arithmetic (no softmax, no advantage, no loss).  Both the CUDA path and the
fp64 oracle consume exactly the tensors produced here, so a parity test is a
comparison on identical inputs.

The shapes follow the workloads of the paper's online RL phase (§3 "Multi-turn
RL Training"): groups of g rollouts per task (g = 16 in the paper), up to five
refinement turns, generations of at most 1536 tokens and a 1024-token
log-prob window.  The policy's hidden states H and LM-head weight W are
synthetic stand-ins for Qwen-3-32B activations (no weights are available):
H ~ N(0, 1), W ~ N(0, 0.02^2), both rounded to bf16 (round-to-nearest-even).

Old- and reference-policy log-probs are "current log-probs + noise" in the
workload recipe; the generator returns only the noise (``old_noise``,
``ref_noise``) and the caller adds it to whichever log-probs it holds.

Every case is a plain dict of CPU (or ``device``) torch tensors plus scalars.
"""

from __future__ import annotations

import math
from dataclasses import dataclass

import torch


@dataclass(frozen=True)
class CaseSpec:
    name: str
    T: int
    d: int
    V: int


def _gen(seed: int, device: str = "cpu") -> torch.Generator:
    g = torch.Generator(device=device)
    g.manual_seed(int(seed))
    return g


def _bf16_normal(shape, std: float, gen: torch.Generator, device: str) -> torch.Tensor:
    x = torch.randn(shape, generator=gen, device=device, dtype=torch.float32)
    if std != 1.0:
        x.mul_(std)
    return x.to(torch.bfloat16)


def _dense_H_W(T: int, d: int, V: int, seed: int, device: str):
    gh = _gen(seed, device)
    H = _bf16_normal((T, d), 1.0, gh, device)
    gw = _gen(seed + 7919, device)
    W = _bf16_normal((V, d), 0.02, gw, device)
    return H, W


def _targets(T: int, V: int, gen: torch.Generator) -> torch.Tensor:
    return torch.randint(0, V, (T,), generator=gen, dtype=torch.int64).to(torch.int32)


def _cu_seqlens(lengths) -> torch.Tensor:
    cu = [0]
    for n in lengths:
        cu.append(cu[-1] + int(n))
    return torch.tensor(cu, dtype=torch.int32)


def tiny_case(seed: int = 1001, old_noise_std: float = 0.05, T_per_seq: int = 16,
              n_groups: int = 4, rollouts: int = 4, d: int = 256, V: int = 4096,
              device: str = "cpu") -> dict:
    """Small case the oracle finishes in well under a second.

    Default: T = 256 tokens as 4 groups x 4 rollouts x 16 tokens, d = 256,
    V = 4096, every token a loss token, rewards U[0, 3] per rollout,
    clip eps = 0.2, KL beta = 0.04.  ``old_noise_std = 0.3`` gives the
    variant in which the clip actually binds on many tokens.
    """
    n_seq = n_groups * rollouts
    T = n_seq * T_per_seq
    H, W = _dense_H_W(T, d, V, seed, device)
    g = _gen(seed + 1)
    tgt = _targets(T, V, g)
    old_noise = torch.randn(T, generator=g) * old_noise_std
    ref_noise = torch.randn(T, generator=g) * 0.05
    rewards = torch.rand(n_seq, generator=g) * 3.0
    return dict(
        name="tiny", T=T, d=d, V=V, H=H, W=W, tgt=tgt,
        mask=torch.ones(T, dtype=torch.uint8),
        cu_seqlens=_cu_seqlens([T_per_seq] * n_seq),
        group_id=torch.arange(n_groups, dtype=torch.int32).repeat_interleave(rollouts),
        n_groups=n_groups, rewards=rewards.float(),
        old_noise=old_noise.float(), ref_noise=ref_noise.float(),
        clip_eps=0.2, kl_beta=0.04, inv_temp=1.0, window=1024,
    )


def forward_case(seed: int = 1002, T: int = 8192, d: int = 4096, V: int = 151936,
                 device: str = "cpu") -> dict:
    """Forward-only workload: 8 rollouts x 1024 tokens, d = 4096, full vocab."""
    H, W = _dense_H_W(T, d, V, seed, device)
    g = _gen(seed + 1)
    tgt = _targets(T, V, g)
    return dict(name="forward", T=T, d=d, V=V, H=H, W=W, tgt=tgt,
                mask=torch.ones(T, dtype=torch.uint8), inv_temp=1.0)


def composite_rewards(n: int, gen: torch.Generator) -> torch.Tensor:
    """Synthetic composite reward r = correctness + log-speedup + structural.

    correctness ~ Bernoulli(0.5), log-speedup ~ N(0.3, 0.5^2), structural ~ U[0, 1];
    drawn per rollout (the paper's r_i = R_ver(i) + R_str(i), §3).
    """
    corr = (torch.rand(n, generator=gen) < 0.5).float()
    spd = 0.3 + 0.5 * torch.randn(n, generator=gen)
    struct = torch.rand(n, generator=gen)
    return (corr + spd + struct).float()


def full_case(seed: int = 1003, n_groups: int = 16, rollouts: int = 8, T_per_seq: int = 128,
              d: int = 5120, V: int = 151936, device: str = "cpu", with_HW: bool = True) -> dict:
    """Full loss fwd+bwd workload: 16 groups x 8 rollouts x 128 tokens = 16384 tokens,
    d = 5120, V = 151936, clip eps = 0.2, KL beta = 0.04."""
    n_seq = n_groups * rollouts
    T = n_seq * T_per_seq
    H = W = None
    if with_HW:
        H, W = _dense_H_W(T, d, V, seed, device)
    g = _gen(seed + 1)
    tgt = _targets(T, V, g)
    return dict(
        name="full", T=T, d=d, V=V, H=H, W=W, tgt=tgt,
        mask=torch.ones(T, dtype=torch.uint8),
        cu_seqlens=_cu_seqlens([T_per_seq] * n_seq),
        group_id=torch.arange(n_groups, dtype=torch.int32).repeat_interleave(rollouts),
        n_groups=n_groups, rewards=composite_rewards(n_seq, g),
        old_noise=(torch.randn(T, generator=g) * 0.05).float(),
        ref_noise=(torch.randn(T, generator=g) * 0.05).float(),
        clip_eps=0.2, kl_beta=0.04, inv_temp=1.0, window=1024,
    )


def ragged_case(seed: int = 1004, n_groups: int = 32, rollouts: int = 8, T_total: int = 65536,
                d: int = 5120, V: int = 151936, device: str = "cpu", with_HW: bool = True) -> dict:
    """Multi-turn ragged workload.

    32 groups x 8 rollouts, each rollout 1-4 turns (uniform); every
    (rollout, turn) is one sequence with its own reward.  Turn lengths are
    drawn U[64, 1024] and then all scaled by T_total / sum (floor 16, the last
    sequence absorbing the remainder) so that exactly T_total tokens are packed.
    In each sequence a prompt/feedback prefix of U[0.3, 0.5] of its length is
    masked out.  The group of a sequence is its task (all turns of the
    task's rollouts).
    """
    g = _gen(seed + 1)
    lengths, gid = [], []
    for grp in range(n_groups):
        for _ in range(rollouts):
            turns = int(torch.randint(1, 5, (1,), generator=g))
            for _ in range(turns):
                lengths.append(int(torch.randint(64, 1025, (1,), generator=g)))
                gid.append(grp)
    raw_total = sum(lengths)
    scale = T_total / raw_total
    lengths = [max(16, int(math.floor(n * scale))) for n in lengths]
    lengths[-1] += T_total - sum(lengths)
    assert lengths[-1] >= 16 and sum(lengths) == T_total
    n_seq = len(lengths)
    mask = torch.ones(T_total, dtype=torch.uint8)
    pos = 0
    for n in lengths:
        frac = 0.3 + 0.2 * float(torch.rand(1, generator=g))
        mask[pos:pos + int(frac * n)] = 0
        pos += n
    T = T_total
    H = W = None
    if with_HW:
        H, W = _dense_H_W(T, d, V, seed, device)
    tgt = _targets(T, V, g)
    return dict(
        name="ragged", T=T, d=d, V=V, H=H, W=W, tgt=tgt, mask=mask,
        cu_seqlens=_cu_seqlens(lengths),
        group_id=torch.tensor(gid, dtype=torch.int32), n_groups=n_groups,
        rewards=composite_rewards(n_seq, g),
        old_noise=(torch.randn(T, generator=g) * 0.05).float(),
        ref_noise=(torch.randn(T, generator=g) * 0.05).float(),
        clip_eps=0.2, kl_beta=0.04, inv_temp=1.0, window=1024,
        raw_token_total=raw_total,
    )


def large_case(seed: int = 1005, T_total: int = 131072, d: int = 5120, V: int = 151936,
               device: str = "cpu", with_HW: bool = True, zero_var_frac: float = 0.05) -> dict:
    """Large packed batch with variable group size G in {4, 8, 16}.

    Rollout lengths U[64, 1024]; the last rollout is truncated so that exactly
    T_total tokens are packed.  About ``zero_var_frac`` of the rollouts sit in
    groups whose members all carry the same reward (advantage = 0 path).
    """
    g = _gen(seed + 1)
    lengths, gid, sizes = [], [], []
    total, grp = 0, 0
    while total < T_total:
        G = [4, 8, 16][int(torch.randint(0, 3, (1,), generator=g))]
        sizes.append(G)
        for _ in range(G):
            if total >= T_total:
                break
            n = int(torch.randint(64, 1025, (1,), generator=g))
            n = min(n, T_total - total)
            lengths.append(n)
            gid.append(grp)
            total += n
        grp += 1
    n_groups = grp
    n_seq = len(lengths)
    rewards = composite_rewards(n_seq, g)
    # Pick whole groups for the zero-variance path until ~zero_var_frac of rollouts.
    gid_t = torch.tensor(gid, dtype=torch.int32)
    target = int(round(zero_var_frac * n_seq))
    order = torch.randperm(n_groups, generator=g).tolist()
    chosen, count = [], 0
    for grp_i in order:
        if count >= target:
            break
        members = (gid_t == grp_i).nonzero().flatten()
        rewards[members] = rewards[members[0]].clone()
        chosen.append(grp_i)
        count += len(members)
    T = T_total
    H = W = None
    if with_HW:
        H, W = _dense_H_W(T, d, V, seed, device)
    tgt = _targets(T, V, g)
    return dict(
        name="large", T=T, d=d, V=V, H=H, W=W, tgt=tgt,
        mask=torch.ones(T, dtype=torch.uint8),
        cu_seqlens=_cu_seqlens(lengths), group_id=gid_t, n_groups=n_groups,
        rewards=rewards.float(),
        old_noise=(torch.randn(T, generator=g) * 0.05).float(),
        ref_noise=(torch.randn(T, generator=g) * 0.05).float(),
        clip_eps=0.2, kl_beta=0.04, inv_temp=1.0, window=1024,
        zero_var_groups=chosen,
    )


def bf16_bits(x: torch.Tensor):
    """uint16 numpy view of a bf16 tensor (the exact bit patterns both sides consume)."""
    return x.contiguous().view(torch.int16).cpu().numpy().view("uint16")


def ranker_case(n_programs: int = 4096, n_pairs: int = 1000, seed: int = 1006,
                init_scale: float = 1.0) -> dict:
    """Synthetic structural-feature vectors and ranking pairs.

    The 11 features follow the appendix's definitions in range and type:
    coalescing score (mean over two kernels of {1, 0.4, 0.1, -0.5, 0.2, 0}),
    arithmetic-intensity proxy in [0, 1), occupancy proxy
    {1, 0.4, -0.3}, divergence (minus a count), transfer-overhead score,
    atomics count, syncthreads count, kernel count, threads per block,
    global-memory access count and operation count.  Pairs (y+, y-) are random
    row indices.  MLP parameters: uniform(+-1/sqrt(fan_in)) * init_scale,
    packed W1, b1, W2, b2, w3, b3.
    """
    g = _gen(seed)
    n = n_programs

    def pick(vals, k):
        v = torch.tensor(vals, dtype=torch.float32)
        return v[torch.randint(0, len(vals), (k,), generator=g)]

    kernels = torch.randint(1, 6, (n,), generator=g).float()
    coal = (pick([1.0, 0.4, 0.1, -0.5, 0.2, 0.0], n) + pick([1.0, 0.4, 0.1, -0.5, 0.2, 0.0], n)) / 2
    ai = torch.rand(n, generator=g) * 0.999             # the proxy's range [0, 1)
    occ = pick([1.0, 0.4, -0.3], n)
    div = -torch.randint(0, 8, (n,), generator=g).float() * 0.5
    xfer = -torch.randint(0, 4, (n,), generator=g).float() + (torch.rand(n, generator=g) < 0.5).float()
    atomics = torch.randint(0, 10, (n,), generator=g).float()
    sync = torch.randint(0, 20, (n,), generator=g).float()
    tpb = pick([32.0, 64.0, 128.0, 256.0, 512.0, 1024.0], n)
    gmem = torch.randint(0, 200, (n,), generator=g).float()
    ops = torch.randint(0, 2000, (n,), generator=g).float()
    phi = torch.stack([coal, ai, occ, div, xfer, atomics, sync, kernels, tpb, gmem, ops], dim=1)
    pos = torch.randint(0, n, (n_pairs,), generator=g, dtype=torch.int64).to(torch.int32)
    neg = torch.randint(0, n, (n_pairs,), generator=g, dtype=torch.int64).to(torch.int32)
    parts = []
    for fan_in, count in ((11, 64 * 11), (11, 64), (64, 32 * 64), (64, 32), (32, 32), (32, 1)):
        bound = init_scale / math.sqrt(fan_in)
        parts.append((torch.rand(count, generator=g) * 2 - 1) * bound)
    params = torch.cat(parts).float()
    return dict(phi=phi.contiguous(), pos=pos, neg=neg, params=params, n=n, n_pairs=n_pairs)
