"""Seeded shape fuzzing of the whole path against the fp64 oracle: 64 random
small configurations, each with its own T (ragged sequence lengths, some
empty), d (a multiple of 64), V (any multiple of 8 from 256), group layout,
mask density, ignored targets, window, temperature, clip, KL weight,
aggregation and std mode; the first 24 of them also through the
kept-exponential form and through the vocabulary split (2-4 slices at random
multiples of 8); and 32 random group layouts for both advantage calls,
bit-exact.  The bars are the path's (|d logp| <= 2e-2, loss relative
error <= 1e-3, g / dH / dW relative L2 <= 2e-2); the configurations are fixed
by the seed, so a failure reproduces."""

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O
from paper_2607_20908_gb300 import inputs
from tests import pipeline as P

pytestmark = pytest.mark.gpu

N_CASES = 64


def _config(k):
    rng = np.random.default_rng(9000 + k)
    n_groups = int(rng.integers(1, 7))
    sizes = rng.integers(1, 6, n_groups)
    lens = rng.integers(0, 160, int(sizes.sum()))
    lens[0] = max(lens[0], 1)
    d = 64 * int(rng.integers(1, 9))
    V = 8 * int(rng.integers(32, 1200))
    return dict(rng=rng, sizes=sizes, lens=lens, d=d, V=V,
                mask_p=float(rng.choice([1.0, 0.9, 0.6])),
                ignore_p=float(rng.choice([0.0, 0.03])),
                window=int(rng.choice([0, 5, 40, 1024])),
                inv_temp=float(rng.choice([1.0, 1.0 / 0.7, 1.0 / 0.2])),
                clip_eps=float(rng.choice([0.1, 0.2, 0.3])),
                kl_beta=float(rng.choice([0.0, 0.04, 0.2])),
                agg=int(rng.integers(0, 2)), std_mode=int(rng.integers(0, 2)),
                old_std=float(rng.choice([0.05, 0.3])))


def _case(k):
    c = _config(k)
    rng = c["rng"]
    lens = c["lens"]
    T = int(lens.sum())
    H, W = inputs._dense_H_W(T, c["d"], c["V"], 9100 + k, "cpu")
    tgt = torch.from_numpy(rng.integers(0, c["V"], T).astype(np.int32))
    tgt[torch.from_numpy(rng.random(T) < c["ignore_p"])] = -100
    mask = torch.from_numpy((rng.random(T) < c["mask_p"]).astype(np.uint8))
    cu = torch.from_numpy(np.concatenate([[0], np.cumsum(lens)]).astype(np.int32))
    gid = torch.from_numpy(np.repeat(np.arange(c["sizes"].size), c["sizes"]).astype(np.int32))
    return dict(name=f"fuzz{k}", T=T, d=c["d"], V=c["V"], H=H, W=W, tgt=tgt, mask=mask,
                cu_seqlens=cu, group_id=gid, n_groups=int(c["sizes"].size),
                rewards=torch.from_numpy(rng.uniform(0, 3, c["sizes"].sum()).astype(np.float32)),
                old_noise=torch.from_numpy((rng.normal(0, c["old_std"], T)).astype(np.float32)),
                ref_noise=torch.from_numpy((rng.normal(0, 0.05, T)).astype(np.float32)),
                clip_eps=c["clip_eps"], kl_beta=c["kl_beta"], inv_temp=c["inv_temp"],
                window=c["window"]), c


@pytest.mark.parametrize("k", range(N_CASES))
def test_random_configuration(k):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    case, c = _case(k)
    if case["T"] == 0:
        pytest.skip("no tokens drawn")
    o = P.run_oracle(case, agg=c["agg"], std_mode=c["std_mode"])
    g = P.run_gpu(case, o["old"], o["ref"], agg=c["agg"], std_mode=c["std_mode"])
    desc = {x: c[x] for x in ("d", "V", "window", "inv_temp", "clip_eps", "kl_beta", "agg",
                              "std_mode", "mask_p", "ignore_p")}
    np.testing.assert_array_equal(g["loss_mask"], o["loss_mask"], err_msg=str(desc))
    for key in ("logp", "entropy", "lse"):
        assert np.abs(g[key] - o[key]).max() <= P.TOL_LOGP, (key, desc)
    # the loss's advantage-weighted terms cancel within groups, so beside the
    # relative bar its error may reach the first-order propagation of the
    # log-prob error through g = dL/dlogp
    err_lp = np.abs(g["logp"] - o["logp"]).max()
    bound = P.TOL_LOSS_REL * abs(o["loss"]) + 2.0 * np.abs(o["g"]).sum() * err_lp + 1e-9
    assert abs(g["loss"] - o["loss"]) <= bound, desc
    for key in ("g", "dH", "dW"):
        assert P.rel_l2(g[key], o[key]) <= P.TOL_GRAD_REL, (key, desc)


def _oracle_and_inputs(k):
    case, c = _case(k)
    if case["T"] == 0:
        pytest.skip("no tokens drawn")
    o = P.run_oracle(case, agg=c["agg"], std_mode=c["std_mode"])
    dev = torch.device("cuda")
    t = {n: case[n].to(dev) for n in ("H", "W", "tgt", "mask", "cu_seqlens", "group_id", "rewards")}
    return case, c, o, t


def _loss_and_g(spo, case, c, o, t, logp, lm):
    dev = torch.device("cuda")
    adv = spo.spo_group_advantages(t["rewards"], t["group_id"], case["n_groups"], c["std_mode"])
    loss, g, _ = spo.spo_policy_loss_fwd(logp, torch.from_numpy(o["old"]).to(dev),
                                         torch.from_numpy(o["ref"]).to(dev), adv,
                                         t["cu_seqlens"], t["group_id"], case["n_groups"], lm,
                                         case["clip_eps"], case["kl_beta"], c["agg"])
    return loss, g


@pytest.mark.parametrize("k", range(24))
def test_random_configuration_kept_form(k):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import spo
    case, c, o, t = _oracle_and_inputs(k)
    lm, _ = spo.spo_token_select(t["cu_seqlens"], t["mask"], t["tgt"], case["window"])
    logp, ent, lse, keep, fws = spo.spo_logprobs_fwd_keep(t["H"], t["W"], t["tgt"], lm,
                                                         case["inv_temp"])
    assert np.abs(logp.cpu().numpy() - o["logp"]).max() <= P.TOL_LOGP
    loss, g = _loss_and_g(spo, case, c, o, t, logp, lm)
    dH, dW = spo.spo_policy_loss_bwd_kept(t["W"], lse, g, keep, fws, case["T"], case["d"],
                                         case["inv_temp"])
    torch.cuda.synchronize()
    assert P.rel_l2(g.cpu().numpy(), o["g"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(dH.float().cpu().numpy(), o["dH"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), o["dW"]) <= P.TOL_GRAD_REL
    assert spo.spo_device_error() == 0


@pytest.mark.parametrize("k", range(24))
def test_random_configuration_vocab_split(k):
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import spo
    case, c, o, t = _oracle_and_inputs(k)
    V = case["V"]
    rng = np.random.default_rng(9500 + k)
    n_sl = min(int(rng.integers(2, 5)), V // 256)    # each slice >= 256 rows (the call's minimum)
    if n_sl < 2:
        pytest.skip("vocabulary too small to split")
    units = V // 8                                    # slice sizes are multiples of 8 rows
    sizes = 32 + rng.multinomial(units - 32 * n_sl, np.ones(n_sl) / n_sl)
    bounds = (8 * np.concatenate([[0], np.cumsum(sizes)])).tolist()
    lm, _ = spo.spo_token_select(t["cu_seqlens"], t["mask"], t["tgt"], case["window"])
    recs = [spo.spo_logprobs_fwd_slice(t["H"], t["W"][a:z], a, t["tgt"], lm, case["inv_temp"])
            for a, z in zip(bounds[:-1], bounds[1:])]
    logp, ent, lse = spo.spo_logprobs_merge_slices(torch.stack(recs))
    assert np.abs(logp.cpu().numpy() - o["logp"]).max() <= P.TOL_LOGP
    assert np.abs(ent.cpu().numpy() - o["entropy"]).max() <= P.TOL_LOGP
    loss, g = _loss_and_g(spo, case, c, o, t, logp, lm)
    dH = torch.zeros(case["T"], case["d"], device="cuda")
    dWs = []
    for a, z in zip(bounds[:-1], bounds[1:]):
        part, dw = spo.spo_policy_loss_bwd_slice(t["H"], t["W"][a:z], a, t["tgt"], lse, g,
                                                 case["inv_temp"])
        dH += part
        dWs.append(dw)
    torch.cuda.synchronize()
    assert P.rel_l2(dH.cpu().numpy(), o["dH"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(torch.cat(dWs).cpu().numpy(), o["dW"]) <= P.TOL_GRAD_REL
    assert spo.spo_device_error() == 0



@pytest.mark.parametrize("k", range(32))
def test_random_advantage_layouts(k):
    """Both advantage calls, bit-exact against the fp32-order oracle, on random
    group layouts: sorted runs, runs in shuffled order, scattered members,
    and (some cases) ids outside [0, n_groups), whose advantages stay as the
    caller left them."""
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(9700 + k)
    ng = int(rng.integers(1, 400))
    sizes = rng.integers(1, int(rng.choice([3, 17, 40])), ng)
    gid = np.repeat(np.arange(ng), sizes).astype(np.int32)
    layout = ("sorted", "shuffled_runs", "scattered")[k % 3]
    if layout == "shuffled_runs":
        order = rng.permutation(ng)
        gid = np.repeat(order, sizes[order]).astype(np.int32)
    elif layout == "scattered":
        gid = gid[rng.permutation(gid.size)]
    n = gid.size
    r = rng.normal(0.5, 1.0, n).astype(np.float32)
    r[gid == 0] = 2.0                                   # one zero-variance group
    invalid = k % 4 == 3
    if invalid:
        gid[rng.choice(n, max(1, n // 50), replace=False)] = rng.choice([-1, ng, ng + 7])
    ok = (gid >= 0) & (gid < ng)
    std_mode = int(rng.integers(0, 2))
    # ids outside the range go to one extra oracle group whose values are not compared
    want = O.group_advantages_f32(r, np.where(ok, gid, ng), ng + 1, std_mode)
    rd, gd = torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda()
    scan = spo.spo_group_advantages(rd, gd, ng, std_mode).cpu().numpy()
    runs = spo.spo_group_advantages_ws(rd, gd, ng, std_mode,
                                       adv=torch.full((n,), 7.0, device="cuda")).cpu().numpy()
    for name, got in (("scan", scan), ("runs", runs)):
        np.testing.assert_array_equal(got[ok].view(np.uint32), want[ok].view(np.uint32),
                                      err_msg=f"{name} {layout}")
    assert np.all(runs[~ok] == 7.0)
