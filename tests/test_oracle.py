"""Pins for the fp64 oracle: closed forms, hand cases, brute force, library
routines and finite differences -- none of them re-types the oracle's own
formula.  CPU only."""

import json
import math
import os

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O


def _golden(golden_dir, name):
    with open(os.path.join(golden_dir, name)) as f:
        return json.load(f)


def _rand_hw(T, d, V, seed, scale_w=0.5):
    rng = np.random.default_rng(seed)
    return rng.standard_normal((T, d)), scale_w * rng.standard_normal((V, d))


# ---------------------------------------------------------------- bf16 widening
def test_bf16_widening_exact():
    x = torch.tensor([1.0, -2.5, 3.140625, 1e-3, -65504.0, 0.0], dtype=torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(O.bf16_bits_to_f64(bits), x.double().numpy())


# ---------------------------------------------------------------- log-probs
def test_uniform_logits_closed_form(golden_dir):
    for case in _golden(golden_dir, "uniform_logits.json")["cases"]:
        V = case["V"]
        d = 8
        H = np.zeros((3, d))
        W = np.random.default_rng(0).standard_normal((V, d))
        lp, ent, lse = O.logprobs(H, W, np.array([0, V // 2, V - 1]))
        np.testing.assert_allclose(lp, case["logp"], rtol=0, atol=1e-12)
        np.testing.assert_allclose(ent, case["entropy"], rtol=0, atol=1e-12)
        np.testing.assert_allclose(lse, -np.asarray(case["logp"]), atol=1e-12)


def test_logprobs_normalise_over_vocab():
    # exp(logp) summed over every possible target is 1 for each token
    T, d, V = 4, 6, 37
    H, W = _rand_hw(T, d, V, 1)
    Hrep = np.repeat(H, V, axis=0)
    tgt = np.tile(np.arange(V), T)
    lp, _, _ = O.logprobs(Hrep, W, tgt)
    sums = np.exp(lp).reshape(T, V).sum(axis=1)
    np.testing.assert_allclose(sums, 1.0, atol=1e-13)
    assert (lp <= 0).all()


def test_logprobs_brute_force_tiny():
    T, d, V = 3, 4, 5
    H, W = _rand_hw(T, d, V, 2)
    tgt = np.array([4, 0, 2])
    tau_inv = 0.7
    lp, ent, lse = O.logprobs(H, W, tgt, inv_temp=tau_inv)
    for t in range(T):
        z = []
        for v in range(V):
            acc = 0.0
            for k in range(d):
                acc += H[t][k] * W[v][k]
            z.append(tau_inv * acc)
        norm = sum(math.exp(x) for x in z)
        probs = [math.exp(x) / norm for x in z]
        assert abs(lp[t] - math.log(probs[tgt[t]])) < 1e-12
        assert abs(ent[t] - (-sum(p * math.log(p) for p in probs))) < 1e-12
        assert abs(lse[t] - math.log(norm)) < 1e-12


def test_logprobs_vs_torch_fp64():
    T, d, V = 17, 32, 301
    H, W = _rand_hw(T, d, V, 3)
    tgt = np.random.default_rng(4).integers(0, V, T)
    lp, ent, lse = O.logprobs(H, W, tgt, inv_temp=1.3)
    z = 1.3 * (torch.from_numpy(H) @ torch.from_numpy(W).T)
    ref_lp = torch.log_softmax(z, dim=-1)[torch.arange(T), torch.from_numpy(tgt)]
    ref_ent = torch.distributions.Categorical(logits=z).entropy()
    np.testing.assert_allclose(lp, ref_lp.numpy(), atol=1e-12)
    np.testing.assert_allclose(ent, ref_ent.numpy(), atol=1e-12)
    np.testing.assert_allclose(lse, torch.logsumexp(z, -1).numpy(), atol=1e-12)


def test_logprobs_dominant_logit_and_shift():
    d, V = 4, 50
    W = np.zeros((V, d))
    W[7, 0] = 1.0
    H = np.array([[60.0, 0, 0, 0]])
    lp, ent, _ = O.logprobs(H, W, np.array([7]))
    assert abs(lp[0]) < 1e-20
    assert ent[0] < 1e-20
    # a bias shared by every vocab entry leaves log-probs unchanged
    H2, W2 = _rand_hw(5, 3, 11, 5)
    tgt = np.arange(5)
    a, ea, _ = O.logprobs(H2, W2, tgt)
    Hb = np.concatenate([H2, np.full((5, 1), 3.7)], axis=1)
    Wb = np.concatenate([W2, np.ones((11, 1))], axis=1)
    b, eb, lb = O.logprobs(Hb, Wb, tgt)
    np.testing.assert_allclose(a, b, atol=1e-12)
    np.testing.assert_allclose(ea, eb, atol=1e-12)


def test_logprobs_mask_and_ignore_index():
    H, W = _rand_hw(6, 4, 9, 6)
    tgt = np.array([1, -100, 3, 4, 5, 6])
    mask = np.array([1, 1, 0, 1, 1, 1], dtype=np.uint8)
    lp, ent, lse = O.logprobs(H, W, tgt, mask=mask)
    assert lp[1] == 0 and lp[2] == 0 and ent[2] == 0 and lse[1] == 0
    full, _, _ = O.logprobs(H, W, np.array([1, 2, 3, 4, 5, 6]))
    np.testing.assert_allclose(lp[[0, 3, 4, 5]], full[[0, 3, 4, 5]], atol=1e-14)


# ---------------------------------------------------------------- token select
def test_token_select_hand_case():
    cu = [0, 6, 10]
    mask = np.array([0, 1, 1, 1, 1, 1, 1, 0, 1, 1], dtype=np.uint8)
    tgt = np.array([5, 5, -100, 5, 5, 5, 5, 5, 5, 5])
    lm, n = O.token_select(cu, mask, tgt, window=3)
    assert lm.tolist() == [0, 1, 0, 1, 1, 0, 1, 0, 1, 1]
    assert n.tolist() == [3, 3]
    lm2, n2 = O.token_select(cu, mask, tgt, window=0)
    assert lm2.tolist() == [0, 1, 0, 1, 1, 1, 1, 0, 1, 1]
    assert n2.tolist() == [4, 3]


# ---------------------------------------------------------------- advantages
def test_advantage_worked_example(golden_dir):
    gold = _golden(golden_dir, "advantage_worked_example.json")
    r = gold["rewards"]
    a = O.group_advantages(r, [0, 0, 0, 0], 1, O.STD_UNBIASED, eps=0.0)
    np.testing.assert_allclose(a, gold["unbiased"], atol=1e-15)
    a = O.group_advantages(r, [0, 0, 0, 0], 1, O.STD_POPULATION, eps=0.0)
    np.testing.assert_allclose(a, gold["population"], atol=1e-15)
    a32 = O.group_advantages_f32(r, [0, 0, 0, 0], 1, O.STD_UNBIASED, eps=0.0)
    np.testing.assert_allclose(a32, gold["unbiased"], atol=1e-6)


def test_advantage_invariants():
    rng = np.random.default_rng(7)
    n_groups, per = 6, 16
    r = rng.uniform(0, 3, n_groups * per)
    gid = np.repeat(np.arange(n_groups), per)
    perm = rng.permutation(r.size)          # members need not be contiguous
    r, gid = r[perm], gid[perm]
    a = O.group_advantages(r, gid, n_groups, O.STD_UNBIASED, eps=0.0)
    for g in range(n_groups):
        ag = a[gid == g]
        assert abs(ag.sum()) < 1e-12
        assert abs((ag ** 2).sum() - (per - 1)) < 1e-10
    # affine invariance for a positive scale
    b = O.group_advantages(2.5 * r - 7.0, gid, n_groups, O.STD_UNBIASED, eps=0.0)
    np.testing.assert_allclose(a, b, atol=1e-12)


def test_advantage_degenerate_groups():
    r = np.array([1.5, 1.5, 1.5, 0.3, 7.0, 2.0])
    gid = np.array([0, 0, 0, 1, 2, 2])
    for fn in (O.group_advantages, O.group_advantages_f32):
        a = fn(r, gid, 4, O.STD_UNBIASED, 1e-6)
        assert a[0] == 0 and a[1] == 0 and a[2] == 0      # zero variance
        assert a[3] == 0                                   # singleton group
        assert a[4] > 0 > a[5]
    # identical rewards whose mean is not exact in binary (3 x 0.1 sums to 0.30000000000000004):
    # the zero-variance rule, not the arithmetic, gives exactly 0, even with eps = 0
    r = np.array([0.1, 0.1, 0.1, 0.7, 0.7, 0.7])
    gid = np.array([0, 0, 0, 1, 1, 1])
    for fn in (O.group_advantages, O.group_advantages_f32):
        assert not fn(r, gid, 2, O.STD_UNBIASED, 0.0).any()


def test_advantage_f32_matches_f64():
    rng = np.random.default_rng(8)
    r = rng.normal(0.3, 1.0, 4096).astype(np.float32)
    gid = rng.integers(0, 256, r.size)
    a64 = O.group_advantages(r.astype(np.float64), gid, 256)
    a32 = O.group_advantages_f32(r, gid, 256)
    np.testing.assert_allclose(a32, a64, atol=2e-6, rtol=0)


# Exact IEEE binary32 rounding (to nearest, ties to even) of a rational, in
# integer arithmetic: checks the fixture's steps without any float32 unit.
def _b32(bits_hex):
    from fractions import Fraction
    b = int(bits_hex, 16)
    sign = -1 if b >> 31 else 1
    e, m = (b >> 23) & 0xFF, b & 0x7FFFFF
    assert 0 < e < 255, "fixture holds normal numbers only"
    return sign * Fraction((1 << 23) | m, 1 << 23) * Fraction(2) ** (e - 127)


def _round_b32(x):
    from fractions import Fraction
    x = Fraction(x)
    if x == 0:
        return "00000000"
    a = abs(x)
    e = a.numerator.bit_length() - a.denominator.bit_length()
    while Fraction(2) ** e > a:
        e -= 1
    while Fraction(2) ** (e + 1) <= a:
        e += 1
    sc = a / Fraction(2) ** (e - 23)                      # in [2^23, 2^24)
    q, rem = divmod(sc.numerator, sc.denominator)
    rem = Fraction(rem, sc.denominator)
    if rem > Fraction(1, 2) or (rem == Fraction(1, 2) and q % 2 == 1):
        q += 1
    if q == 1 << 24:
        q, e = 1 << 23, e + 1
    assert -126 <= e <= 127
    return f"{((1 if x < 0 else 0) << 31) | ((e + 127) << 23) | (q - (1 << 23)):08x}"


def _sqrt_b32(bits_hex):
    """Correctly rounded binary32 square root of a binary32, by integer isqrt."""
    from fractions import Fraction
    x = _b32(bits_hex)
    e = x.numerator.bit_length() - x.denominator.bit_length()
    while Fraction(2) ** e > x:
        e -= 1
    es = e // 2                                            # floor(log2(sqrt(x)))
    N = x * Fraction(2) ** (46 - 2 * es + 16)             # 8 guard bits beyond the 24
    assert N.denominator == 1
    r = math.isqrt(N.numerator)
    exact = r * r == N.numerator
    q, low = r >> 8, r & 0xFF
    if low > 0x80 or (low == 0x80 and (not exact or q % 2 == 1)):
        q += 1
    return _round_b32(q * Fraction(2) ** (es - 23))


def test_advantage_f32_bit_patterns(golden_dir):
    """group_advantages_f32 reproduces, bit for bit, advantages derived step by
    step in the fixed binary32 order (tests/golden/advantage_f32_bits.json).
    The fixture's own steps are first re-derived here in exact integer
    arithmetic, each one rounding of the previous listed values."""
    gold = _golden(golden_dir, "advantage_f32_bits.json")
    eps = _b32(gold["eps_bits"])
    assert _round_b32(__import__("fractions").Fraction(gold["eps"])) == gold["eps_bits"]
    for case in gold["cases"]:
        r = np.asarray(case["rewards"], dtype=np.float32)
        n = r.size
        for mode_name, mode in case["modes"].items():
            # the fixture's derivation, one rounded operation at a time
            assert [f"{int(b):08x}" for b in r.view(np.uint32)] == mode["rewards_bits"]
            rv = [_b32(b) for b in mode["rewards_bits"]]
            acc = 0
            for k in range(n):
                acc_hex = _round_b32(acc + rv[k])
                assert acc_hex == mode["running_sum"][k]
                acc = _b32(acc_hex)
            assert mode["sum"] == mode["running_sum"][-1]
            assert _round_b32(acc / n) == mode["mean"]
            mu = _b32(mode["mean"])
            ss = 0
            for k in range(n):
                assert _round_b32(rv[k] - mu) == mode["deviations"][k]
                dv = _b32(mode["deviations"][k])
                assert _round_b32(dv * dv) == mode["rounded_squares"][k]
                ss = _b32(_round_b32(ss + _b32(mode["rounded_squares"][k])))
            assert _round_b32(ss) == mode["sum_sq"]
            dof = n - 1 if mode_name == "unbiased" else n
            assert _round_b32(_b32(mode["sum_sq"]) / dof) == mode["var"]
            assert _sqrt_b32(mode["var"]) == mode["std"]
            assert _round_b32(_b32(mode["std"]) + eps) == mode["den"]
            den = _b32(mode["den"])
            assert [_round_b32(_b32(d) / den) for d in mode["deviations"]] == mode["adv"]
            # the pin: the oracle's fp32-order advantages carry exactly these bits
            std_mode = O.STD_UNBIASED if mode_name == "unbiased" else O.STD_POPULATION
            a = O.group_advantages_f32(r, np.zeros(n, np.int64), 1, std_mode, gold["eps"])
            assert a.dtype == np.float32
            assert [f"{int(b):08x}" for b in a.view(np.uint32)] == mode["adv"], (case["name"],
                                                                                mode_name)
            # group order does not matter: the same members scattered among another group
            gid = np.array([0, 1] * n)[: 2 * n]
            rr = np.empty(2 * n, np.float32)
            rr[0::2] = r
            rr[1::2] = np.float32(7.0)
            a2 = O.group_advantages_f32(rr, gid, 2, std_mode, gold["eps"])
            assert [f"{int(b):08x}" for b in a2[0::2].view(np.uint32)] == mode["adv"]


# ---------------------------------------------------------------- loss
def _single_token(rho, adv, beta, logp=None, ref=None, eps=0.2):
    lp = np.log(rho) if logp is None else logp
    old = lp - np.log(rho)
    loss, g, st = O.policy_loss(np.array([lp]), np.array([old]),
                                None if ref is None else np.array([ref]), np.array([adv]),
                                [0, 1], [0], 1, np.array([1], np.uint8), eps, beta)
    return loss, g[0], st


def test_surrogate_hand_cases(golden_dir):
    gold = _golden(golden_dir, "surrogate_hand_cases.json")
    for c in gold["cases"]:
        loss, g, _ = _single_token(c["rho"], c["adv"], c["beta"], c.get("logp"), c.get("ref"),
                                   gold["clip_eps"])
        assert abs(loss - c["loss"]) < 1e-12, c
        assert abs(g - c["g"]) < 1e-12, c


def test_ratio_one_no_kl_is_minus_mean_advantage():
    # with pi_theta == pi_old and beta = 0 the objective is the weighted mean advantage
    rng = np.random.default_rng(9)
    lens = [5, 9, 3, 7, 4, 6]
    cu = np.concatenate([[0], np.cumsum(lens)])
    gid = np.array([0, 0, 1, 1, 1, 2])
    adv = rng.standard_normal(len(lens))          # arbitrary, not group-normalised
    T = cu[-1]
    lp = -rng.uniform(0.1, 5, T)
    lm = np.ones(T, np.uint8)
    loss, g, st = O.policy_loss(lp, lp, None, adv, cu, gid, 3, lm, 0.2, 0.0, O.AGG_SEQ_GROUP)
    # SEQ_GROUP: mean over groups of mean over outputs of A_i
    want = -np.mean([adv[gid == k].mean() for k in range(3)])
    assert abs(loss - want) < 1e-12
    loss_t, _, _ = O.policy_loss(lp, lp, None, adv, cu, gid, 3, lm, 0.2, 0.0, O.AGG_TOKEN)
    want_t = -(np.repeat(adv, lens)).mean()
    assert abs(loss_t - want_t) < 1e-12
    assert st["clip_frac"] == 0 and abs(st["mean_ratio"] - 1) < 1e-15
    # with masked tokens the means run over loss tokens only
    lm = (rng.random(T) > 0.4).astype(np.uint8)
    lm[cu[:-1]] = 1                               # every output keeps at least one token
    per_tok = np.repeat(adv, lens)
    loss_t, _, st = O.policy_loss(lp, lp, None, adv, cu, gid, 3, lm, 0.2, 0.0, O.AGG_TOKEN)
    assert abs(loss_t + per_tok[lm == 1].mean()) < 1e-12
    loss_s, _, _ = O.policy_loss(lp, lp, None, adv, cu, gid, 3, lm, 0.2, 0.0, O.AGG_SEQ_GROUP)
    assert abs(loss_s - want) < 1e-12              # per-output token means: masks cancel
    assert st["n_loss_tokens"] == int(lm.sum())


def test_kl_properties():
    rng = np.random.default_rng(10)
    T = 50
    lp = -rng.uniform(0.1, 5, T)
    cu = [0, 20, 50]
    lm = np.ones(T, np.uint8)
    _, g0, st0 = O.policy_loss(lp, lp, lp, np.zeros(2), cu, [0, 0], 1, lm, 0.2, 0.3)
    assert st0["mean_kl"] == 0 and np.all(g0 == 0)
    ref = lp + rng.normal(0, 0.5, T)
    _, _, st = O.policy_loss(lp, lp, ref, np.zeros(2), cu, [0, 0], 1, lm, 0.2, 0.3)
    assert st["mean_kl"] > 0


def test_aggregations_agree_on_uniform_layout():
    rng = np.random.default_rng(11)
    lens = [8] * 8
    cu = np.concatenate([[0], np.cumsum(lens)])
    gid = np.repeat(np.arange(2), 4)
    T = cu[-1]
    lp = -rng.uniform(0.1, 3, T)
    old = lp + rng.normal(0, 0.3, T)
    ref = lp + rng.normal(0, 0.1, T)
    adv = rng.standard_normal(8)
    lm = np.ones(T, np.uint8)
    a = O.policy_loss(lp, old, ref, adv, cu, gid, 2, lm, 0.2, 0.04, O.AGG_SEQ_GROUP)
    b = O.policy_loss(lp, old, ref, adv, cu, gid, 2, lm, 0.2, 0.04, O.AGG_TOKEN)
    assert abs(a[0] - b[0]) < 1e-13
    np.testing.assert_allclose(a[1], b[1], atol=1e-15)


def test_dloss_dlogp_finite_difference():
    rng = np.random.default_rng(12)
    lens = [6, 4, 9, 5]
    cu = np.concatenate([[0], np.cumsum(lens)])
    gid = np.array([0, 0, 1, 1])
    T = cu[-1]
    lp = -rng.uniform(0.1, 3, T)
    old = lp + rng.normal(0, 0.4, T)
    ref = lp + rng.normal(0, 0.2, T)
    adv = rng.standard_normal(4)
    lm = np.ones(T, np.uint8)
    lm[3] = 0
    eps = 0.2
    rho = np.exp(lp - old)
    for agg in (O.AGG_SEQ_GROUP, O.AGG_TOKEN):
        _, g, _ = O.policy_loss(lp, old, ref, adv, cu, gid, 2, lm, eps, 0.07, agg)
        h = 1e-6
        for t in range(T):
            if min(abs(rho[t] - 1 - eps), abs(rho[t] - 1 + eps)) < 1e-4:
                continue
            lp_p, lp_m = lp.copy(), lp.copy()
            lp_p[t] += h
            lp_m[t] -= h
            fp = O.policy_loss(lp_p, old, ref, adv, cu, gid, 2, lm, eps, 0.07, agg)[0]
            fm = O.policy_loss(lp_m, old, ref, adv, cu, gid, 2, lm, eps, 0.07, agg)[0]
            assert abs((fp - fm) / (2 * h) - g[t]) < 1e-8, (agg, t)
        assert g[3] == 0


# ---------------------------------------------------------------- backward
def _loss_of_hw(H, W, tgt, cu, gid, n_groups, lm, old, ref, adv, eps, beta, tau):
    lp, _, _ = O.logprobs(H, W, tgt, tau, lm)
    return O.policy_loss(lp, old, ref, adv, cu, gid, n_groups, lm, eps, beta)


def test_backward_finite_difference():
    rng = np.random.default_rng(13)
    T, d, V = 7, 5, 11
    H, W = _rand_hw(T, d, V, 14)
    tgt = rng.integers(0, V, T)
    cu = [0, 3, 7]
    gid = [0, 0]
    lm = np.array([1, 1, 0, 1, 1, 1, 1], np.uint8)
    tau = 0.8
    lp0, _, _ = O.logprobs(H, W, tgt, tau, lm)
    old = lp0 + rng.normal(0, 0.05, T)
    ref = lp0 + rng.normal(0, 0.05, T)
    adv = np.array([0.7, -1.3])
    args = (tgt, cu, gid, 1, lm, old, ref, adv, 0.2, 0.05, tau)
    _, g, _ = _loss_of_hw(H, W, *args)
    dH, dW = O.policy_loss_bwd(H, W, tgt, g, tau)
    h = 1e-6
    for (t, k) in [(0, 0), (1, 4), (2, 2), (4, 1), (6, 3)]:
        Hp, Hm = H.copy(), H.copy()
        Hp[t, k] += h
        Hm[t, k] -= h
        fd = (_loss_of_hw(Hp, W, *args)[0] - _loss_of_hw(Hm, W, *args)[0]) / (2 * h)
        assert abs(fd - dH[t, k]) < 1e-8, (t, k, fd, dH[t, k])
    for (v, k) in [(0, 0), (int(tgt[0]), 2), (5, 4), (10, 1), (int(tgt[6]), 3)]:
        Wp, Wm = W.copy(), W.copy()
        Wp[v, k] += h
        Wm[v, k] -= h
        fd = (_loss_of_hw(H, Wp, *args)[0] - _loss_of_hw(H, Wm, *args)[0]) / (2 * h)
        assert abs(fd - dW[v, k]) < 1e-8, (v, k, fd, dW[v, k])
    assert np.all(dH[2] == 0)


def test_backward_vs_torch_cross_entropy_autograd():
    # rho = 1, beta = 0: L = sum_t c_t A_i * CE(z_t, y_t) + const, so torch's
    # fp64 cross_entropy autograd gives the same dH and dW.
    rng = np.random.default_rng(15)
    T, d, V = 12, 9, 23
    H, W = _rand_hw(T, d, V, 16)
    tgt = rng.integers(0, V, T)
    cu = np.array([0, 5, 12])
    gid = [0, 1]
    lm = np.ones(T, np.uint8)
    adv = np.array([0.9, -0.4])
    lp, _, _ = O.logprobs(H, W, tgt, 1.0, lm)
    _, g, _ = O.policy_loss(lp, lp, None, adv, cu, gid, 2, lm, 0.2, 0.0)
    dH, dW = O.policy_loss_bwd(H, W, tgt, g, 1.0)
    Ht = torch.tensor(H, requires_grad=True)
    Wt = torch.tensor(W, requires_grad=True)
    ce = torch.nn.functional.cross_entropy(Ht @ Wt.T, torch.tensor(tgt), reduction="none")
    c = torch.tensor(np.concatenate([np.full(5, adv[0] / (2 * 5)), np.full(7, adv[1] / (2 * 7))]))
    (c * ce).sum().backward()
    np.testing.assert_allclose(dH, Ht.grad.numpy(), atol=1e-13)
    np.testing.assert_allclose(dW, Wt.grad.numpy(), atol=1e-13)


def test_backward_invariants():
    rng = np.random.default_rng(17)
    T, d, V = 9, 6, 14
    H, W = _rand_hw(T, d, V, 18)
    tgt = rng.integers(0, V, T)
    g = rng.standard_normal(T)
    g[4] = 0.0
    _, dW = O.policy_loss_bwd(H, W, tgt, g)
    # each row of G sums to zero over the vocabulary
    np.testing.assert_allclose(dW.sum(axis=0), 0.0, atol=1e-12)
    Wsame = np.tile(W[:1], (V, 1))
    dH, _ = O.policy_loss_bwd(H, Wsame, tgt, g)
    np.testing.assert_allclose(dH, 0.0, atol=1e-12)
    dH, _ = O.policy_loss_bwd(H, W, tgt, g)
    assert np.all(dH[4] == 0)


def test_grpo_step_runs_on_tiny_workload():
    from paper_2607_20908_gb300 import inputs
    case = inputs.tiny_case()
    H = O.bf16_bits_to_f64(inputs.bf16_bits(case["H"]))
    W = O.bf16_bits_to_f64(inputs.bf16_bits(case["W"]))
    tgt = case["tgt"].numpy()
    lp, _, _ = O.logprobs(H, W, tgt)
    old = lp + case["old_noise"].double().numpy()
    ref = lp + case["ref_noise"].double().numpy()
    out = O.grpo_step(H, W, tgt, case["mask"].numpy(), case["cu_seqlens"].numpy(),
                      case["group_id"].numpy(), case["n_groups"], case["rewards"].numpy(),
                      old, ref, case["clip_eps"], case["kl_beta"])
    assert np.isfinite(out["loss"]) and out["stats"]["n_loss_tokens"] == case["T"]
    assert np.all(out["logp"] <= 0)


# ---------------------------------------------------------------- vocabulary split
def _slices(V, cuts):
    edges = [0] + list(cuts) + [V]
    return list(zip(edges[:-1], edges[1:]))


@pytest.mark.parametrize("cuts", [[], [40], [8, 56], [32, 64, 88]])
def test_slice_records_merge_to_the_full_softmax(cuts):
    """The logsumexp of a union of slices, assembled from per-slice (max, sumexp,
    sumexp*z, target) records, against the full-vocabulary definition and
    torch.log_softmax; uneven slices, a skipped token, an ignored target."""
    T, d, V = 24, 12, 96
    H, W = _rand_hw(T, d, V, seed=11, scale_w=1.5)
    rng = np.random.default_rng(12)
    tgt = rng.integers(0, V, T)
    tgt[5] = -1
    mask = (rng.random(T) > 0.2).astype(np.uint8)
    recs = [O.logprobs_slice_record(H, W[a:b], a, tgt, 0.8, mask) for a, b in _slices(V, cuts)]
    lp, ent, lse = O.merge_slice_records(recs)
    keep = (tgt >= 0) & (mask == 1)
    z = torch.from_numpy(0.8 * H @ W.T)
    ls = torch.log_softmax(z, dim=1).numpy()
    ref_lp = np.where(keep, ls[np.arange(T), np.where(keep, tgt, 0)], 0.0)
    ref_ent = np.where(keep, -(np.exp(ls) * ls).sum(axis=1), 0.0)
    ref_lse = np.where(keep, torch.logsumexp(z, dim=1).numpy(), 0.0)
    np.testing.assert_allclose(lp, ref_lp, atol=1e-12)
    np.testing.assert_allclose(ent, ref_ent, atol=1e-12)
    np.testing.assert_allclose(lse, ref_lse, atol=1e-12)
    # the merge does not depend on the order of the slices
    lp2, ent2, lse2 = O.merge_slice_records(recs[::-1])
    np.testing.assert_allclose(lp2, lp, atol=1e-13)
    np.testing.assert_allclose(ent2, ent, atol=1e-13)


def test_slice_record_fields_brute_force():
    """One token, one slice, written out element by element."""
    H = np.array([[0.5, -1.0, 2.0]])
    W = np.array([[1.0, 0.0, 0.0], [0.0, 1.0, 0.0], [0.0, 0.0, 1.0], [1.0, 1.0, 1.0]])
    rec = O.logprobs_slice_record(H, W[1:3], 1, np.array([2]))[0]
    z = [-1.0, 2.0]                         # logits of vocabulary ids 1 and 2
    assert rec[0] == 2.0
    assert math.isclose(rec[1], math.exp(-3.0) + 1.0, rel_tol=1e-15)
    assert math.isclose(rec[2], math.exp(-3.0) * z[0] + z[1], rel_tol=1e-15)
    assert rec[3] == 2.0
    other = O.logprobs_slice_record(H, W[3:4], 3, np.array([2]))[0]
    assert other[3] == -np.inf and other[1] == 1.0


@pytest.mark.parametrize("cuts", [[48], [16, 24, 72]])
def test_backward_slices_sum_to_the_full_backward(cuts):
    """Sum over slices of the dH parts is dH; the slices' dW rows stacked are dW
    (both against autograd of the fp64 log_softmax, not the oracle)."""
    T, d, V = 16, 10, 96
    H, W = _rand_hw(T, d, V, seed=21, scale_w=1.0)
    rng = np.random.default_rng(22)
    tgt = rng.integers(0, V, T)
    g = rng.standard_normal(T)
    g[[2, 9]] = 0.0
    tau = 0.7
    Ht = torch.from_numpy(H).requires_grad_(True)
    Wt = torch.from_numpy(W).requires_grad_(True)
    ls = torch.log_softmax(tau * Ht @ Wt.T, dim=1)
    (ls[torch.arange(T), torch.from_numpy(tgt)] * torch.from_numpy(g)).sum().backward()
    lse = torch.logsumexp(torch.from_numpy(tau * H @ W.T), dim=1).numpy()
    parts = [O.policy_loss_bwd_slice(H, W[a:b], a, tgt, lse, g, tau) for a, b in _slices(V, cuts)]
    dH = sum(p[0] for p in parts)
    dW = np.concatenate([p[1] for p in parts])
    np.testing.assert_allclose(dH, Ht.grad.numpy(), atol=1e-12)
    np.testing.assert_allclose(dW, Wt.grad.numpy(), atol=1e-12)
    assert not dH[[2, 9]].any()


# ---------------------------------------------------------------- reward composition
def test_verifiable_reward_hand_cases(golden_dir):
    gold = _golden(golden_dir, "verifiable_reward_hand_cases.json")
    cs = gold["cases"]
    r = O.reward_compose([c["compiled"] for c in cs], [c["pass_rate"] for c in cs],
                         [c["speedup"] for c in cs], [c["cv"] for c in cs],
                         [c["r_struct"] for c in cs])
    np.testing.assert_allclose(r, [c["reward"] for c in cs], atol=1e-12)


def test_verifiable_reward_properties():
    rng = np.random.default_rng(20)
    n = 200
    S = np.exp2(rng.uniform(-3, 7, n))
    cv = rng.uniform(0, 1, n)
    full = O.reward_compose(np.ones(n), np.ones(n), S, cv)
    # bounded by the clip: alpha_speed*[s_min, s_max] minus the stability term
    assert np.all(full <= 4.0 + 1e-12) and np.all(full >= -0.5 - 0.5 * 1.0 - 1e-12)
    # monotone in speedup for fixed cv
    order = np.argsort(S)
    fixed = O.reward_compose(np.ones(n), np.ones(n), S[order], np.full(n, 0.2))
    assert np.all(np.diff(fixed) >= -1e-12)
    # partial pass rates ignore speed and cv; a non-positive speedup is the lower bound
    part = O.reward_compose(np.ones(3), [0.5, 0.5, 0.999], [1e6, 1e-6, 5.0], [0.0, 9.0, 0.0])
    np.testing.assert_allclose(part, [-1.0, -1.0, -0.002], atol=1e-12)
    z = O.reward_compose([1, 1], [1.0, 1.0], [0.0, -3.0], [0.0, 0.0])
    np.testing.assert_allclose(z, [-0.5, -0.5], atol=1e-12)


# ---------------------------------------------------------------- offline ranker
def _ranker_case(seed, n=40, P=25):
    rng = np.random.default_rng(seed)
    phi = rng.standard_normal((n, 11)) * 3 + 1
    mu, sigma = phi.mean(axis=0), phi.std(axis=0) + 0.1
    flat = rng.standard_normal(O.RANKER_NPARAMS) * 0.3
    pos, neg = rng.integers(0, n, P), rng.integers(0, n, P)
    return phi, mu, sigma, flat, pos, neg


def test_ranker_shapes_and_equal_scores():
    assert O.RANKER_NPARAMS == 64 * 11 + 64 + 32 * 64 + 32 + 32 + 1
    phi, mu, sigma, flat, _, _ = _ranker_case(30)
    # identical members of a pair: loss = softplus(0) = ln 2 and the gradient vanishes
    loss, grad = O.ranker_pair_loss(phi, mu, sigma, flat, [3, 7], [3, 7])
    assert abs(loss - math.log(2.0)) < 1e-15 and np.abs(grad).max() < 1e-15
    # swapping every pair turns softplus(-d) into softplus(d): the sum is mean(|d|) + 2 mean(softplus(-|d|))
    _, _, _, _, pos, neg = _ranker_case(31)
    l1, _ = O.ranker_pair_loss(phi, mu, sigma, flat, pos, neg)
    l2, _ = O.ranker_pair_loss(phi, mu, sigma, flat, neg, pos)
    s, _ = O.ranker_scores(phi, mu, sigma, flat)
    d = s[pos] - s[neg]
    assert abs(l1 + l2 - (np.abs(d).mean() + 2 * np.logaddexp(0, -np.abs(d)).mean())) < 1e-12


def test_ranker_vs_torch_autograd():
    phi, mu, sigma, flat, pos, neg = _ranker_case(32)
    rng = np.random.default_rng(33)
    keep1 = (rng.random((pos.size, 2, 64)) > 0.1).astype(np.uint8)
    keep2 = (rng.random((pos.size, 2, 32)) > 0.1).astype(np.uint8)
    loss, grad = O.ranker_pair_loss(phi, mu, sigma, flat, pos, neg, keep1, keep2, 0.1)
    t = torch.tensor(flat, requires_grad=True)
    off, Pt = 0, {}
    for name, sh in O.RANKER_SHAPES:
        n = int(np.prod(sh))
        Pt[name] = t[off:off + n].reshape(sh)
        off += n
    x = (torch.tensor(phi) - torch.tensor(mu)) / torch.tensor(sigma)

    def score(rows, k1, k2):
        h1 = torch.relu(x[rows] @ Pt["W1"].T + Pt["b1"]) * torch.tensor(k1, dtype=torch.float64) / 0.9
        h2 = torch.relu(h1 @ Pt["W2"].T + Pt["b2"]) * torch.tensor(k2, dtype=torch.float64) / 0.9
        return h2 @ Pt["w3"] + Pt["b3"][0]

    d = score(torch.tensor(pos), keep1[:, 0], keep2[:, 0]) - score(torch.tensor(neg), keep1[:, 1], keep2[:, 1])
    lt = torch.nn.functional.softplus(-d).mean()
    lt.backward()
    assert abs(lt.item() - loss) < 1e-12
    np.testing.assert_allclose(grad, t.grad.numpy(), atol=1e-12)


def test_ranker_finite_difference():
    phi, mu, sigma, flat, pos, neg = _ranker_case(34, n=12, P=9)
    _, grad = O.ranker_pair_loss(phi, mu, sigma, flat, pos, neg)
    h = 1e-6
    for j in np.random.default_rng(35).choice(O.RANKER_NPARAMS, 40, replace=False):
        fp, fm = flat.copy(), flat.copy()
        fp[j] += h
        fm[j] -= h
        fd = (O.ranker_pair_loss(phi, mu, sigma, fp, pos, neg)[0] -
              O.ranker_pair_loss(phi, mu, sigma, fm, pos, neg)[0]) / (2 * h)
        assert abs(fd - grad[j]) < 1e-7, (j, fd, grad[j])
