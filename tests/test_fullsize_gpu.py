"""GPU parity at the workloads' full sizes, in the launch configuration the
benchmark times (every row active, the same grids and tiles), checked on
outputs the fp64 oracle can compute one by one: sampled rows of log-probs
and dH, dW restricted to a sampled token set, and the whole loss (O(T))."""

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


@pytest.fixture(autouse=True)
def _free():
    yield
    torch.cuda.empty_cache()


def _sample(T, n, seed):
    return np.sort(np.random.default_rng(seed).choice(T, size=n, replace=False))


def _fwd_check(spo, H, W, tgt, mask, rows, inv_temp=1.0):
    """GPU forward over the whole batch; oracle on the sampled rows only."""
    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt, mask, inv_temp)
    torch.cuda.synchronize()
    Hs = H[torch.from_numpy(rows).cuda()].double().cpu().numpy()
    Wd = W.double().cpu().numpy()
    ts = tgt.cpu().numpy()[rows]
    lp_o, ent_o, lse_o = O.logprobs(Hs, Wd, ts, inv_temp)
    got = [t.cpu().numpy()[rows] for t in (logp, ent, lse)]
    errs = [np.abs(g - o).max() for g, o in zip(got, (lp_o, ent_o, lse_o))]
    assert max(errs) <= P.TOL_LOGP, errs
    assert np.all(got[0] <= 0)
    return logp, ent, lse, Wd, errs


def test_full_workload_forward_sampled_rows(spo):
    """16384 tokens, d=5120, V=151936: 64 sampled rows against fp64."""
    case = inputs.full_case(device="cuda")
    H, W, tgt = case["H"], case["W"], case["tgt"].cuda()
    rows = _sample(case["T"], 64, 1)
    *_, errs = _fwd_check(spo, H, W, tgt, None, rows)
    print(f"\nfull fwd: max |dlogp|={errs[0]:.2e} |dent|={errs[1]:.2e} |dlse|={errs[2]:.2e}")


def test_full_workload_backward_sampled(spo):
    """Backward in the benchmark's launch shape (all 16384 rows have g != 0).
    dH: 32 sampled rows (each row depends on its own token only).  dW: g is
    N(0, 1e-2) on 48 sampled tokens and +-1e-20 elsewhere, so dW is the sampled
    tokens' sum to within |g_rest| * sum_t |G_t| |H_t| < 1e-14 relative."""
    case = inputs.full_case(device="cuda")
    H, W, tgt = case["H"], case["W"], case["tgt"].cuda()
    T = case["T"]
    _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
    gen = torch.Generator().manual_seed(3)
    g = torch.where(torch.rand(T, generator=gen) < 0.5, -1e-20, 1e-20).float()
    sel = _sample(T, 48, 2)
    g[torch.from_numpy(sel)] = (torch.randn(48, generator=gen) * 1e-2).float()
    dH, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, g.cuda())
    torch.cuda.synchronize()
    Wd = W.double().cpu().numpy()
    Hs = H[torch.from_numpy(sel).cuda()].double().cpu().numpy()
    dH_o, dW_o = O.policy_loss_bwd(Hs, Wd, tgt.cpu().numpy()[sel], g.double().numpy()[sel])
    e_dH = P.rel_l2(dH[torch.from_numpy(sel).cuda()].float().cpu().numpy(), dH_o)
    e_dW = P.rel_l2(dW.cpu().numpy(), dW_o)
    print(f"\nfull bwd: dH rel={e_dH:.2e} dW rel={e_dW:.2e}")
    assert e_dH <= P.TOL_GRAD_REL and e_dW <= P.TOL_GRAD_REL
    # rows with g = +-1e-20 carry a gradient of that order
    rest = np.setdiff1d(np.arange(T), sel)[:64]
    assert dH[torch.from_numpy(rest).cuda()].float().abs().max().item() < 1e-15


def _loss_inputs(case, seed):
    """Synthetic log-probs (not from either side) for the O(T) loss check."""
    T = case["T"]
    gen = torch.Generator().manual_seed(seed)
    logp = -torch.rand(T, generator=gen) * 8
    noise = torch.from_numpy(P.away_from_clip(case["old_noise"].double().numpy(),
                                              case["clip_eps"])).float()
    return logp.float(), (logp + noise).float(), (logp + case["ref_noise"]).float()


def _loss_check(spo, case, loss_mask_gpu, loss_mask_np, seed, agg=0):
    logp, old, ref = _loss_inputs(case, seed)
    adv_o = O.group_advantages(case["rewards"].numpy(), case["group_id"].numpy(), case["n_groups"])
    adv = spo.spo_group_advantages(case["rewards"].cuda(), case["group_id"].cuda(), case["n_groups"])
    np.testing.assert_allclose(adv.cpu().numpy(), adv_o, atol=1e-6, rtol=0)
    adv32 = O.group_advantages_f32(case["rewards"].numpy(), case["group_id"].numpy(), case["n_groups"])
    np.testing.assert_array_equal(adv.cpu().numpy().view(np.uint32), adv32.view(np.uint32))
    loss, g, stats = spo.spo_policy_loss_fwd(
        logp.cuda(), old.cuda(), ref.cuda(), adv, case["cu_seqlens"].cuda(), case["group_id"].cuda(),
        case["n_groups"], loss_mask_gpu, case["clip_eps"], case["kl_beta"], agg)
    # the oracle's own fp32-order advantages (the same bits as the kernel's, checked above)
    loss_o, g_o, st_o = O.policy_loss(logp.double().numpy(), old.double().numpy(),
                                      ref.double().numpy(), adv32.astype(np.float64),
                                      case["cu_seqlens"].numpy(), case["group_id"].numpy(),
                                      case["n_groups"], loss_mask_np, case["clip_eps"],
                                      case["kl_beta"], agg)
    rel = abs(loss.item() - loss_o) / max(abs(loss_o), 1e-12)
    assert rel <= P.TOL_LOSS_REL, (loss.item(), loss_o)
    assert P.rel_l2(g.cpu().numpy(), g_o) <= 1e-5
    assert stats[3].item() == st_o["n_loss_tokens"]
    return rel


def test_full_workload_loss(spo):
    case = inputs.full_case(with_HW=False)
    lm, n_tok = spo.spo_token_select(case["cu_seqlens"].cuda(), case["mask"].cuda(), case["tgt"].cuda(),
                                     case["window"])
    lm_o, n_o = O.token_select(case["cu_seqlens"].numpy(), case["mask"].numpy(), case["tgt"].numpy(),
                               case["window"])
    np.testing.assert_array_equal(lm.cpu().numpy(), lm_o)
    np.testing.assert_array_equal(n_tok.cpu().numpy(), n_o)
    for agg in (0, 1):
        _loss_check(spo, case, lm, lm_o, 11 + agg, agg)


def test_forward_only_workload_sampled_rows(spo):
    """8 rollouts x 1024 tokens, d=4096, V=151936, and a sampling temperature."""
    case = inputs.forward_case(device="cuda")
    rows = _sample(case["T"], 48, 4)
    _fwd_check(spo, case["H"], case["W"], case["tgt"].cuda(), None, rows)
    _fwd_check(spo, case["H"], case["W"], case["tgt"].cuda(), None, rows[:16], inv_temp=1 / 0.7)


def test_ragged_multiturn_workload(spo):
    """32 groups x 8 rollouts x 1-4 turns packed to 65536 tokens, ~40% prompt
    tokens masked, per-turn rewards: selection bit-exact over all tokens, the
    loss over all tokens, log-probs on sampled kept rows."""
    case = inputs.ragged_case(device="cuda")
    cu, mask, tgt = case["cu_seqlens"], case["mask"], case["tgt"]
    lm, n_tok = spo.spo_token_select(cu.cuda(), mask.cuda(), tgt.cuda(), case["window"])
    lm_o, n_o = O.token_select(cu.numpy(), mask.numpy(), tgt.numpy(), case["window"])
    np.testing.assert_array_equal(lm.cpu().numpy(), lm_o)
    np.testing.assert_array_equal(n_tok.cpu().numpy(), n_o)
    assert 0.45 < lm_o.mean() < 0.75
    _loss_check(spo, case, lm, lm_o, 21)
    kept = np.nonzero(lm_o)[0]
    rows = np.sort(np.random.default_rng(5).choice(kept, 32, replace=False))
    logp, *_ = _fwd_check(spo, case["H"], case["W"], tgt.cuda(), lm, rows)
    assert np.all(logp.cpu().numpy()[lm_o == 0] == 0)


def test_large_workload_chunked_backward(spo):
    """131072 tokens: the backward runs in 4 chunks of 32768 rows.  Sampled
    tokens straddle every chunk; dW accumulates across the chunks."""
    case = inputs.large_case(device="cuda")
    H, W, tgt = case["H"], case["W"], case["tgt"].cuda()
    T = case["T"]
    _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
    gen = torch.Generator().manual_seed(6)
    g = torch.where(torch.rand(T, generator=gen) < 0.5, -1e-20, 1e-20).float()
    sel = np.concatenate([_sample(32768, 8, 10 + c) + 32768 * c for c in range(4)] +
                         [np.array([32767, 32768, 65535, 131071])])
    sel = np.unique(sel)
    g[torch.from_numpy(sel)] = (torch.randn(sel.size, generator=gen) * 1e-2).float()
    dH, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, g.cuda())
    torch.cuda.synchronize()
    Wd = W.double().cpu().numpy()
    Hs = H[torch.from_numpy(sel).cuda()].double().cpu().numpy()
    dH_o, dW_o = O.policy_loss_bwd(Hs, Wd, tgt.cpu().numpy()[sel], g.double().numpy()[sel])
    e_dH = P.rel_l2(dH[torch.from_numpy(sel).cuda()].float().cpu().numpy(), dH_o)
    e_dW = P.rel_l2(dW.cpu().numpy(), dW_o)
    print(f"\nlarge bwd (4 chunks): dH rel={e_dH:.2e} dW rel={e_dW:.2e}")
    assert e_dH <= P.TOL_GRAD_REL and e_dW <= P.TOL_GRAD_REL
    # zero-variance groups give exactly zero advantages
    adv = spo.spo_group_advantages(case["rewards"].cuda(), case["group_id"].cuda(), case["n_groups"])
    gid = case["group_id"].numpy()
    zero = np.isin(gid, case["zero_var_groups"])
    assert zero.any() and np.all(adv.cpu().numpy()[zero] == 0)
