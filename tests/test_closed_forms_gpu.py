"""The CUDA path against what the mathematics fixes, with no oracle in between:
properties of the softmax and of Eq. 3 that hold at any size, checked on the
device results at the workloads' vocabulary and hidden sizes.

- equal logits (H = 0): log pi = -ln V, entropy = ln V, lse = ln V for every
  token (tests/golden/uniform_logits.json);
- log-probs are <= 0 and exponentiate to 1 over the vocabulary: each of 16
  tokens is repeated V times with targets 0 .. V-1 and the V probabilities
  of each token are summed;
- ratio 1 (old = current log-probs) and no KL: the loss is minus the average
  of the advantages under Eq. 3's aggregation, the average over groups of
  the average over each group's sequences (random advantages, not
  group-normalised ones, whose average is 0 by construction);
- every row of G sums to 0 over the vocabulary, so the columns of dW sum to 0;
- W with identical rows gives equal logits for every token, and dH = 0.
"""

import json
import os

import numpy as np
import pytest
import torch

from paper_2607_20908_gb300 import inputs

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


@pytest.mark.parametrize("V,d", [(4096, 256), (151936, 5120)])
def test_equal_logits_give_log_v(spo, golden_dir, V, d):
    case = {c["V"]: c for c in json.load(open(os.path.join(golden_dir, "uniform_logits.json")))["cases"]}[V]
    T = 600                                          # three row tiles, the last ragged
    gen = torch.Generator().manual_seed(21)
    H = torch.zeros(T, d, dtype=torch.bfloat16, device="cuda")
    W = (torch.randn(V, d, generator=gen) * 0.02).to(torch.bfloat16).cuda()
    tgt = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32).cuda()
    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt)
    for got, want in ((logp, case["logp"]), (ent, case["entropy"]), (lse, -case["logp"])):
        assert torch.abs(got.double() - want).max().item() <= 4e-6


@pytest.mark.parametrize("inv_temp", [1.0, 1.0 / 0.2])
def test_logprobs_exponentiate_to_one(spo, inv_temp):
    V, d, n_tok = 4096, 256, 16
    gen = torch.Generator().manual_seed(22)
    H0 = torch.randn(n_tok, d, generator=gen).to(torch.bfloat16)
    W = (torch.randn(V, d, generator=gen) * 0.05).to(torch.bfloat16).cuda()
    H = H0.repeat_interleave(V, dim=0).cuda()                       # 65536 rows
    tgt = torch.arange(V, dtype=torch.int32).repeat(n_tok).cuda()   # every target of each token
    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt, None, inv_temp)
    lp = logp.double().view(n_tok, V)
    assert lp.max().item() <= 0.0
    total = torch.exp(lp).sum(dim=1)
    assert torch.abs(total - 1.0).max().item() <= 1e-4
    # the V copies of a token have one lse
    lse = lse.double().view(n_tok, V)
    assert (lse - lse[:, :1]).abs().max().item() <= 1e-5
    # entropy = -sum p log p of the same distribution
    ent_direct = -(torch.exp(lp) * lp).sum(dim=1)
    assert torch.abs(ent.view(n_tok, V)[:, 0].double() - ent_direct).max().item() <= 1e-3


@pytest.mark.parametrize("agg", [0, 1])
def test_ratio_one_no_kl_loss_is_minus_mean_advantage(spo, agg):
    """Sequences of 1-300 tokens in groups of 1-8, a masked prefix in each,
    random advantages; old = logp and kl_beta = 0 make every ratio 1 and every
    clip inactive, so l_t = -A_i and g_t = -c_t A_i."""
    rng = np.random.default_rng(23)
    sizes = rng.integers(1, 9, 40)
    n_seq = int(sizes.sum())
    gid = np.repeat(np.arange(sizes.size), sizes).astype(np.int32)
    lens = rng.integers(1, 301, n_seq)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    lm = np.ones(T, dtype=np.uint8)
    for i in range(n_seq):
        lm[cu[i]:cu[i] + int(rng.integers(0, lens[i]))] = 0   # prompt prefix; >= 1 loss token
    A = rng.normal(size=n_seq).astype(np.float32)
    lp = (-6.0 * rng.random(T)).astype(np.float32)
    dev = lambda a: torch.from_numpy(a).cuda()
    loss, g, stats = spo.spo_policy_loss_fwd(dev(lp), dev(lp), None, dev(A), dev(cu), dev(gid),
                                             sizes.size, dev(lm), 0.2, 0.0, agg)
    n_i = np.array([lm[cu[i]:cu[i + 1]].sum() for i in range(n_seq)], dtype=np.float64)
    if agg == 0:   # mean over groups of the mean over the group's sequences
        want = -np.mean([A[gid == k].astype(np.float64).mean() for k in range(sizes.size)])
    else:          # mean over all loss tokens
        want = -(A.astype(np.float64) * n_i).sum() / n_i.sum()
    assert abs(loss.item() - want) <= 1e-5 * max(1e-3, abs(want))
    assert stats[1].item() == pytest.approx(1.0, abs=1e-6)       # mean ratio
    assert stats[0].item() == 0.0                                # nothing clipped
    # g_t = -c_t A_i, and the weights of a sequence's loss tokens add up to its share
    gt = g.double().cpu().numpy()
    seq_sum = np.array([gt[cu[i]:cu[i + 1]].sum() for i in range(n_seq)])
    share = (1.0 / (sizes.size * sizes[gid])) if agg == 0 else n_i / n_i.sum()
    np.testing.assert_allclose(seq_sum, -share * A, rtol=1e-5, atol=1e-9)
    assert np.all(gt[lm == 0] == 0)


def test_dw_columns_sum_to_zero(spo):
    """Full vocabulary and hidden size, 512 tokens: sum_v G[t, v] = 0 for
    every row, so every column of dW = G^T H sums to 0 (up to G's bf16
    rounding)."""
    T, d, V = 512, 5120, 151936
    H, W = inputs._dense_H_W(T, d, V, 24, "cuda")
    gen = torch.Generator().manual_seed(25)
    tgt = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32).cuda()
    g = (torch.randn(T, generator=gen) * 1e-2).float().cuda()
    _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
    _, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, g)
    col = dW.double().sum(dim=0)
    scale = dW.double().abs().sum(dim=0)
    assert (col.abs() / scale).max().item() <= 2e-3
    # the target rows carry the one-hot part: dW[y_t] holds +g_t H_t (1 - p), far from 0
    assert scale.min().item() > 0


def test_identical_w_rows_give_zero_dh(spo):
    """Every vocabulary row the same: equal logits for every token, so
    p = 1/V, G[t, v] = g_t (1[v = y_t] - 1/V) and dH = G W = g_t (w - w) = 0
    (up to the bf16 rounding of G, far below the size of g_t |w|)."""
    T, d, V = 300, 512, 8192
    gen = torch.Generator().manual_seed(26)
    w = (torch.randn(d, generator=gen) * 0.5).to(torch.bfloat16)
    W = w.repeat(V, 1).cuda()
    H = torch.randn(T, d, generator=gen).to(torch.bfloat16).cuda()
    tgt = torch.randint(0, V, (T,), generator=gen, dtype=torch.int32).cuda()
    g = (torch.rand(T, generator=gen) + 0.5).float().cuda()
    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt)
    assert torch.abs(logp.double() + np.log(V)).max().item() <= 1e-5
    dH, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, g)
    bound = 1e-2 * (g.abs().max() * w.float().abs().max()).item()
    assert dH.float().abs().max().item() <= bound
    # and dW rows are G^T H: target rows gain g_t H_t, every row loses sum_t g_t H_t / V
    assert torch.isfinite(dW).all()
