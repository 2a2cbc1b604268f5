"""GPU parity of the vocabulary-split form (LM-head rows split into slices,
one per device in a tensor-parallel head).  On one GPU the slices run one
after another: each writes its per-token records, the records are stacked
(what an all-gather would deliver) and merged; the backward's dH parts are
summed (what an all-reduce would deliver) and the slices' dW rows stacked.
Checked against the fp64 oracle's full-vocabulary definitions."""

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


def _case(seed=1201):
    """T = 600 (20 sequences of 30: a ragged last row tile), d = 256, V = 4096;
    ~20 % of tokens masked, two ignored targets, inv_temp 0.8."""
    case = inputs.tiny_case(seed=seed, T_per_seq=30, n_groups=5, rollouts=4)
    gen = torch.Generator().manual_seed(seed + 7)
    case["mask"] = (torch.rand(case["T"], generator=gen) > 0.2).to(torch.uint8)
    case["tgt"][[7, 301]] = -1
    case["inv_temp"] = 0.8
    return case


def _edges(V, cuts):
    e = [0] + list(cuts) + [V]
    return list(zip(e[:-1], e[1:]))


def _gpu_records(spo, H, W, tgt, mask, cuts, inv_temp):
    recs = [spo.spo_logprobs_fwd_slice(H, W[a:b], a, tgt, mask, inv_temp)
            for a, b in _edges(W.shape[0], cuts)]
    return torch.stack(recs)


@pytest.mark.parametrize("cuts", [[], [2048], [1000], [1024, 3072], [256, 1280, 2304]])
def test_merged_slices_match_oracle(spo, cuts):
    """Slices of 1000 / 3096 rows leave a ragged vocabulary tile inside a slice."""
    c = _case()
    H, W = c["H"].cuda(), c["W"].cuda()
    tgt, mask = c["tgt"].cuda(), c["mask"].cuda()
    rec = _gpu_records(spo, H, W, tgt, mask, cuts, c["inv_temp"])
    logp, ent, lse = spo.spo_logprobs_merge_slices(rec)
    torch.cuda.synchronize()
    Ho, Wo = P.oracle_hw(c)
    lp_o, ent_o, lse_o = O.logprobs(Ho, Wo, c["tgt"].numpy(), c["inv_temp"], c["mask"].numpy())
    got = [t.cpu().numpy() for t in (logp, ent, lse)]
    errs = [float(np.abs(g - o).max()) for g, o in zip(got, (lp_o, ent_o, lse_o))]
    assert max(errs) <= P.TOL_LOGP, errs
    skipped = (c["mask"].numpy() == 0) | (c["tgt"].numpy() < 0)
    for g in got:
        assert not g[skipped].any()
    assert np.all(got[0][~skipped] <= 0)


def test_slice_records_match_oracle_records(spo):
    """The exchanged record itself: (max, sumexp, sumexp*z, target logit) per
    slice; the kernel keeps max and the third field in log2 units."""
    c = _case(seed=1202)
    H, W = c["H"].cuda(), c["W"].cuda()
    tgt, mask = c["tgt"].cuda(), c["mask"].cuda()
    Ho, Wo = P.oracle_hw(c)
    for a, b in _edges(c["V"], [1000]):
        rec = spo.spo_logprobs_fwd_slice(H, W[a:b], a, tgt, mask, c["inv_temp"]).cpu().numpy()
        ref = O.logprobs_slice_record(Ho, Wo[a:b], a, c["tgt"].numpy(), c["inv_temp"],
                                      c["mask"].numpy())
        live = ref[:, 1] > 0
        assert not rec[~live].any()
        np.testing.assert_allclose(rec[live, 0] * math.log(2), ref[live, 0], atol=P.TOL_LOGP)
        np.testing.assert_allclose(rec[live, 1], ref[live, 1], rtol=P.TOL_LOGP)
        # third field: sum 2^(u - max u) u with u = z log2 e
        np.testing.assert_allclose(rec[live, 2] * math.log(2), ref[live, 2],
                                   atol=P.TOL_LOGP * np.abs(ref[live, 2]).max())
        fin = np.isfinite(ref[:, 3]) & live
        assert np.array_equal(np.isfinite(rec[:, 3]) & live, fin)
        np.testing.assert_allclose(rec[fin, 3], ref[fin, 3], atol=P.TOL_LOGP)


def test_merged_slices_match_unsplit_kernel_path(spo):
    """Same bf16 products, merged in another order: agreement far inside the
    oracle tolerance."""
    c = _case(seed=1203)
    H, W = c["H"].cuda(), c["W"].cuda()
    tgt, mask = c["tgt"].cuda(), c["mask"].cuda()
    logp, ent, lse = spo.spo_logprobs_merge_slices(
        _gpu_records(spo, H, W, tgt, mask, [1536], c["inv_temp"]))
    lp1, ent1, lse1 = spo.spo_logprobs_fwd(H, W, tgt, mask, c["inv_temp"])
    for a, b in ((logp, lp1), (ent, ent1), (lse, lse1)):
        assert float((a - b).abs().max()) <= 1e-4


@pytest.mark.parametrize("cuts", [[2048], [1000, 2600]])
def test_backward_slices_match_oracle(spo, cuts):
    """dH = sum of the slices' fp32 parts, dW = the slices' rows stacked."""
    c = _case(seed=1204)
    H, W = c["H"].cuda(), c["W"].cuda()
    tgt, mask = c["tgt"].cuda(), c["mask"].cuda()
    _, _, lse = spo.spo_logprobs_merge_slices(
        _gpu_records(spo, H, W, tgt, mask, cuts, c["inv_temp"]))
    gen = torch.Generator().manual_seed(77)
    keep = (c["mask"] == 1) & (c["tgt"] >= 0)
    g = torch.where(keep, torch.randn(c["T"], generator=gen) * 1e-2, torch.zeros(c["T"])).float()
    dH = torch.zeros(c["T"], c["d"], device="cuda")
    dWs = []
    for a, b in _edges(c["V"], cuts):
        part, dw = spo.spo_policy_loss_bwd_slice(H, W[a:b], a, tgt, lse, g.cuda(), c["inv_temp"])
        dH += part
        dWs.append(dw)
    dW = torch.cat(dWs)
    torch.cuda.synchronize()
    Ho, Wo = P.oracle_hw(c)
    dH_o, dW_o = O.policy_loss_bwd(Ho, Wo, c["tgt"].numpy(), g.double().numpy(), c["inv_temp"])
    assert P.rel_l2(dH.cpu().numpy(), dH_o) <= P.TOL_GRAD_REL
    assert P.rel_l2(dW.cpu().numpy(), dW_o) <= P.TOL_GRAD_REL
    assert not dH.cpu().numpy()[~keep.numpy()].any()
    # the unsplit kernel path on the same lse: the fp32 parts sum to its dH
    dH1, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse, g.cuda(), c["inv_temp"])
    assert P.rel_l2(dH.cpu().numpy(), dH1.float().cpu().numpy()) <= 1e-2
    assert P.rel_l2(dW.cpu().numpy(), dW1.cpu().numpy()) <= 1e-5


def test_full_vocabulary_two_slices_sampled_rows(spo):
    """The full workload's head (V = 151936, d = 5120) as two slices of 75968
    rows: every token against the unsplit kernel path, 32 sampled rows against
    the fp64 oracle."""
    case = inputs.full_case(device="cuda")
    H, W, tgt = case["H"], case["W"], case["tgt"].cuda()
    half = case["V"] // 2
    logp, ent, lse = spo.spo_logprobs_merge_slices(_gpu_records(spo, H, W, tgt, None, [half], 1.0))
    lp1, ent1, lse1 = spo.spo_logprobs_fwd(H, W, tgt)
    for a, b in ((logp, lp1), (ent, ent1), (lse, lse1)):
        assert float((a - b).abs().max()) <= 1e-3
    rows = np.sort(np.random.default_rng(5).choice(case["T"], size=32, replace=False))
    Hs = H[torch.from_numpy(rows).cuda()].double().cpu().numpy()
    lp_o, ent_o, lse_o = O.logprobs(Hs, W.double().cpu().numpy(), tgt.cpu().numpy()[rows])
    for gpu, ora in ((logp, lp_o), (ent, ent_o), (lse, lse_o)):
        assert np.abs(gpu.cpu().numpy()[rows] - ora).max() <= P.TOL_LOGP
    del H, W
    torch.cuda.empty_cache()
