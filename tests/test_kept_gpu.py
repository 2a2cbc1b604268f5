"""GPU parity of the kept-exponential form: the forward keeps
E = exp(z - tile max) in bf16 and the backward forms G from it instead of
recomputing the logits.  Checked against the fp64 oracle (log-probs, the kept
values themselves, dH, dW) and against the recompute path."""

import math

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O
from paper_2607_20908_gb300 import inputs
from tests import pipeline as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spo():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import build
    build.build()
    from paper_2607_20908_gb300 import spo as mod
    return mod


def _case(seed=1501):
    """600 tokens (ragged last tile row), d = 256, V = 5000 (ragged last vocab tile),
    ~20 % of tokens masked, one ignored target."""
    case = inputs.tiny_case(seed=seed, T_per_seq=30, n_groups=5, rollouts=4, V=5000)
    gen = torch.Generator().manual_seed(seed + 3)
    case["mask"] = (torch.rand(case["T"], generator=gen) > 0.2).to(torch.uint8)
    case["tgt"][11] = -1
    case["inv_temp"] = 0.9
    return case


def test_kept_path_matches_oracle(spo):
    c = _case()
    dev = torch.device("cuda")
    H, W, tgt, mask = (c[k].to(dev) for k in ("H", "W", "tgt", "mask"))
    T, d, V, tau = c["T"], c["d"], c["V"], c["inv_temp"]
    logp, ent, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt, mask, tau)
    Ho, Wo = P.oracle_hw(c)
    lp_o, ent_o, lse_o = O.logprobs(Ho, Wo, c["tgt"].numpy(), tau, c["mask"].numpy())
    for gpu, ora in ((logp, lp_o), (ent, ent_o), (lse, lse_o)):
        assert np.abs(gpu.cpu().numpy() - ora).max() <= P.TOL_LOGP
    # the kept values: E[r][v] = exp(z - max over v's 256-entry tile), rows in the order of the
    # kept tokens
    kept = np.nonzero((c["mask"].numpy() == 1) & (c["tgt"].numpy() >= 0))[0]
    E = keep.view(torch.bfloat16).view(-1, V)[: kept.size].float().cpu().numpy()
    z = O.logits(Ho[kept], Wo, tau)
    tiles = np.repeat(np.arange((V + 255) // 256), 256)[:V]
    m = np.stack([z[:, tiles == k].max(axis=1) for k in range((V + 255) // 256)], axis=1)
    want = np.exp(z - m[:, tiles])
    assert np.abs(E - want).max() <= 2.0 ** -7          # bf16 of values in (0, 1]
    # backward from the kept forward against the oracle's backward with the same g (seeded)
    gen = torch.Generator().manual_seed(9)
    g = torch.where(torch.from_numpy((c["mask"].numpy() == 1) & (c["tgt"].numpy() >= 0)),
                    torch.randn(T, generator=gen) * 1e-2, torch.zeros(T)).float()
    dH, dW = spo.spo_policy_loss_bwd_kept(W, lse, g.to(dev), keep, fws, T, d, tau)
    torch.cuda.synchronize()
    dH_o, dW_o = O.policy_loss_bwd(Ho, Wo, c["tgt"].numpy(), g.double().numpy(), tau)
    assert P.rel_l2(dH.float().cpu().numpy(), dH_o) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), dW_o) <= P.TOL_GRAD_REL
    assert not dH.float().cpu().numpy()[np.setdiff1d(np.arange(T), kept)].any()
    # the recompute path on the same inputs
    dH1, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse, g.to(dev), tau)
    assert P.rel_l2(dH.float().cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-2
    assert P.rel_l2(dW.cpu().numpy(), dW1.cpu().numpy()) <= 1e-2
    assert spo.spo_device_error() == 0


def test_kept_whole_step_matches_oracle(spo):
    """Token select, kept forward, advantages, loss, kept backward: the whole
    step in the kept form against the oracle's step."""
    c = inputs.tiny_case(seed=1502, T_per_seq=40, n_groups=4, rollouts=4)
    o = P.run_oracle(c)
    dev = torch.device("cuda")
    H, W, tgt = c["H"].to(dev), c["W"].to(dev), c["tgt"].to(dev)
    cu, gid = c["cu_seqlens"].to(dev), c["group_id"].to(dev)
    lm, _ = spo.spo_token_select(cu, c["mask"].to(dev), tgt, c["window"])
    logp, ent, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt, lm, c["inv_temp"])
    adv = spo.spo_group_advantages(c["rewards"].to(dev), gid, c["n_groups"])
    loss, g, _ = spo.spo_policy_loss_fwd(logp, torch.from_numpy(o["old"]).to(dev),
                                         torch.from_numpy(o["ref"]).to(dev), adv, cu, gid,
                                         c["n_groups"], lm, c["clip_eps"], c["kl_beta"])
    dH, dW = spo.spo_policy_loss_bwd_kept(W, lse, g, keep, fws, c["T"], c["d"], c["inv_temp"])
    torch.cuda.synchronize()
    assert np.abs(logp.cpu().numpy() - o["logp"]).max() <= P.TOL_LOGP
    assert abs(loss.item() - o["loss"]) / abs(o["loss"]) <= P.TOL_LOSS_REL
    assert P.rel_l2(dH.float().cpu().numpy(), o["dH"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), o["dW"]) <= P.TOL_GRAD_REL


def test_full_workload_kept_backward_sampled(spo):
    """The benchmark's head (d = 5120, V = 151936, 16384 tokens) in the kept form:
    g N(0, 1e-2) on 48 sampled tokens, +-1e-20 elsewhere, against the oracle on
    the sampled tokens and against the recompute path on everything."""
    case = inputs.full_case(device="cuda")
    H, W, tgt = case["H"], case["W"], case["tgt"].cuda()
    T, d = case["T"], case["d"]
    logp, _, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt)
    lp1, _, lse1 = spo.spo_logprobs_fwd(H, W, tgt)
    assert float((logp - lp1).abs().max()) <= 1e-4 and float((lse - lse1).abs().max()) <= 1e-4
    gen = torch.Generator().manual_seed(3)
    g = torch.where(torch.rand(T, generator=gen) < 0.5, -1e-20, 1e-20).float()
    sel = np.sort(np.random.default_rng(2).choice(T, size=48, replace=False))
    g[torch.from_numpy(sel)] = (torch.randn(48, generator=gen) * 1e-2).float()
    g = g.cuda()
    dH, dW = spo.spo_policy_loss_bwd_kept(W, lse, g, keep, fws, T, d)
    dH1, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse1, g)
    torch.cuda.synchronize()
    assert P.rel_l2(dW.cpu().numpy(), dW1.cpu().numpy()) <= 1e-2
    assert P.rel_l2(dH.float().cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-2
    Wd = W.double().cpu().numpy()
    Hs = H[torch.from_numpy(sel).cuda()].double().cpu().numpy()
    dH_o, dW_o = O.policy_loss_bwd(Hs, Wd, tgt.cpu().numpy()[sel], g.double().cpu().numpy()[sel])
    assert P.rel_l2(dH[torch.from_numpy(sel).cuda()].float().cpu().numpy(), dH_o) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), dW_o) <= P.TOL_GRAD_REL
    del keep, fws, dW, dW1
    torch.cuda.empty_cache()


def test_kept_backward_optional_outputs(spo):
    """dW added into an existing buffer, dH or dW skipped, against the recompute
    path's own accumulate and skip behaviour on the same inputs."""
    c = _case(seed=1503)
    dev = torch.device("cuda")
    H, W, tgt, mask = (c[k].to(dev) for k in ("H", "W", "tgt", "mask"))
    T, d, V, tau = c["T"], c["d"], c["V"], c["inv_temp"]
    gen = torch.Generator().manual_seed(4)
    g = (torch.randn(T, generator=gen) * 1e-2).float().to(dev)
    base = torch.randn(V, d, generator=gen).float().to(dev)
    # each kept backward overwrites E with G, so every call gets its own kept forward
    _, _, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt, mask, tau)
    dH, dW = spo.spo_policy_loss_bwd_kept(W, lse, g, keep, fws, T, d, tau, dW=base.clone(),
                                          accumulate_dW=True)
    _, _, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt, mask, tau)
    dH2, none_w = spo.spo_policy_loss_bwd_kept(W, lse, g, keep, fws, T, d, tau, want_dW=False)
    _, _, lse, keep, fws = spo.spo_logprobs_fwd_keep(H, W, tgt, mask, tau)
    none_h, dW3 = spo.spo_policy_loss_bwd_kept(W, lse, g, keep, fws, T, d, tau, want_dH=False)
    torch.cuda.synchronize()
    assert none_w is None and none_h is None
    assert torch.equal(dH.view(torch.int16), dH2.view(torch.int16))
    torch.testing.assert_close(dW, base + dW3, rtol=1e-5, atol=1e-6)
    lm = (mask == 1) & (tgt >= 0)
    dH1, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse, torch.where(lm, g, torch.zeros_like(g)), tau)
    assert P.rel_l2(dW3.cpu().numpy(), dW1.cpu().numpy()) <= 1e-2
    assert P.rel_l2(dH2.float().cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-2
