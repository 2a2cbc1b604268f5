"""Parity at the ends of the boundary's size ranges (d <= 65536, V <= 2^24,
T <= 2^24): the widest hidden size, a 2^22-row vocabulary and the largest
packed batch, each against the fp64 oracle on outputs it can compute."""

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


def _whole_path(case):
    """The whole path against the oracle.  The loss is a signed sum whose
    advantage-weighted terms cancel within each group, so at these sizes it can
    be far smaller than its terms; its error is bounded by the first-order
    propagation of the log-prob error through g = dL/dlogp (the oracle's), on
    top of the usual relative bar."""
    o = P.run_oracle(case)
    g = P.run_gpu(case, o["old"], o["ref"])
    err_lp = np.abs(g["logp"] - o["logp"]).max()
    err_ent = np.abs(g["entropy"] - o["entropy"]).max()
    d_loss = abs(g["loss"] - o["loss"])
    bound = P.TOL_LOSS_REL * abs(o["loss"]) + 2.0 * np.abs(o["g"]).sum() * err_lp
    e_dH, e_dW = P.rel_l2(g["dH"], o["dH"]), P.rel_l2(g["dW"], o["dW"])
    print(f"\n[{case['name']} d={case['d']} V={case['V']}] |dlogp|={err_lp:.2e} "
          f"|dent|={err_ent:.2e} |dloss|={d_loss:.2e} (loss {o['loss']:.3e}, bound {bound:.2e}) "
          f"dH rel={e_dH:.2e} dW rel={e_dW:.2e}")
    assert err_lp <= P.TOL_LOGP and err_ent <= P.TOL_LOGP
    assert d_loss <= bound
    assert e_dH <= P.TOL_GRAD_REL and e_dW <= P.TOL_GRAD_REL


def test_widest_hidden_size(spo):
    """d = 65536: 1024 k-blocks per tile in the logits GEMMs, 65536-wide dH rows."""
    _whole_path(inputs.tiny_case(seed=1401, T_per_seq=64, n_groups=2, rollouts=2, d=65536, V=512))


def test_large_vocabulary(spo):
    """V = 2^22: 16384 vocabulary tiles merged per row, a 2 GB G chunk, 4M dW rows."""
    _whole_path(inputs.tiny_case(seed=1402, T_per_seq=16, n_groups=2, rollouts=2, d=64,
                                 V=1 << 22))


def test_largest_packed_batch(spo):
    """T = 2^24 tokens (16384 sequences of 1024, groups of 8) at d = 64, V = 256:
    the compaction over 2^24 tokens, the forward on 65536 tile rows, the loss
    over every token and a backward of 512 chunks with dW accumulated across
    them.  Log-probs are checked on sampled rows; the loss on all tokens with
    the oracle run on the same seeded log-prob stand-ins; dH on sampled rows
    and dW from g non-zero on sampled tokens only."""
    T, d, V, L = 1 << 24, 64, 256, 1024
    dev = torch.device("cuda")
    n_seq = T // L
    H, W = inputs._dense_H_W(T, d, V, 1403, "cuda")
    gen = torch.Generator().manual_seed(1404)
    tgt = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32)
    mask = (torch.rand(T, generator=gen) > 0.1).to(torch.uint8)
    cu = torch.arange(0, T + 1, L, dtype=torch.int32)
    gid = (torch.arange(n_seq, dtype=torch.int32) // 8)
    n_groups = n_seq // 8
    rewards = torch.rand(n_seq, generator=gen) * 3.0

    lm, n_tok = spo.spo_token_select(cu.to(dev), mask.to(dev), tgt.to(dev), 1024)
    lm_o, n_o = O.token_select(cu.numpy(), mask.numpy(), tgt.numpy(), 1024)
    np.testing.assert_array_equal(lm.cpu().numpy(), lm_o)
    np.testing.assert_array_equal(n_tok.cpu().numpy(), n_o)

    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt.to(dev), lm)
    rows = np.sort(np.random.default_rng(6).choice(np.nonzero(lm_o)[0], size=256, replace=False))
    Hs = H[torch.from_numpy(rows).to(dev)].double().cpu().numpy()
    Wd = W.double().cpu().numpy()
    lp_o, ent_o, lse_o = O.logprobs(Hs, Wd, tgt.numpy()[rows])
    for gpu, ora in ((logp, lp_o), (ent, ent_o), (lse, lse_o)):
        assert np.abs(gpu.cpu().numpy()[rows] - ora).max() <= P.TOL_LOGP

    # loss over every token on seeded stand-ins for the log-probs (O(T) on both sides)
    lp_in = (-torch.rand(T, generator=gen) * 6).float()
    old = (lp_in + torch.randn(T, generator=gen) * 0.05).float()
    ref = (lp_in + torch.randn(T, generator=gen) * 0.05).float()
    adv = spo.spo_group_advantages(rewards.to(dev), gid.to(dev), n_groups)
    adv32 = O.group_advantages_f32(rewards.numpy(), gid.numpy(), n_groups)
    np.testing.assert_array_equal(adv.cpu().numpy().view(np.uint32), adv32.view(np.uint32))
    loss, g, stats = spo.spo_policy_loss_fwd(lp_in.to(dev), old.to(dev), ref.to(dev), adv,
                                             cu.to(dev), gid.to(dev), n_groups, lm, 0.2, 0.04)
    loss_o, g_o, st_o = O.policy_loss(lp_in.double().numpy(), old.double().numpy(),
                                      ref.double().numpy(), adv32.astype(np.float64), cu.numpy(),
                                      gid.numpy(), n_groups, lm_o, 0.2, 0.04)
    assert abs(loss.item() - loss_o) / abs(loss_o) <= P.TOL_LOSS_REL
    assert P.rel_l2(g.cpu().numpy(), g_o) <= 1e-5
    assert stats[3].item() == st_o["n_loss_tokens"]

    # backward over all 2^24 rows (512 chunks of 32768): g is N(0, 1e-2) on 64
    # sampled tokens and +-1e-20 elsewhere, so every row is active and dW is the
    # sampled tokens' sum to within 2^24 * 1e-20 relative
    sel = np.sort(np.random.default_rng(7).choice(T, size=64, replace=False))
    gb = torch.where(torch.rand(T, generator=gen) < 0.5, -1e-20, 1e-20).float()
    gb[torch.from_numpy(sel)] = (torch.randn(64, generator=gen) * 1e-2).float()
    _, _, lse_all = spo.spo_logprobs_fwd(H, W, tgt.to(dev))
    dH, dW = spo.spo_policy_loss_bwd(H, W, tgt.to(dev), lse_all, gb.to(dev))
    Hsel = H[torch.from_numpy(sel).to(dev)].double().cpu().numpy()
    dH_o, dW_o = O.policy_loss_bwd(Hsel, Wd, tgt.numpy()[sel], gb.double().numpy()[sel])
    assert P.rel_l2(dH[torch.from_numpy(sel).to(dev)].float().cpu().numpy(), dH_o) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), dW_o) <= P.TOL_GRAD_REL
    rest = torch.from_numpy(np.setdiff1d(np.arange(4096), sel)).to(dev)
    assert dH[rest].float().abs().max().item() < 1e-15
    assert spo.spo_device_error() == 0
