"""GPU parity of the offline structural ranker (section 2.1): scores and the
pairwise logistic loss with its gradient, against the fp64 oracle."""

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


def _stats(phi):
    """Training-split mean / std of every feature (test-side input preparation)."""
    x = phi.double().numpy()
    return x.mean(axis=0).astype(np.float32), (x.std(axis=0) + 1e-3).astype(np.float32)


def _dev(case, mu, sigma):
    c = lambda t: torch.as_tensor(t).cuda()
    return c(case["phi"]), c(mu), c(sigma), c(case["params"]), c(case["pos"]), c(case["neg"])


def test_ranker_scores(spo):
    case = inputs.ranker_case(n_programs=3001, n_pairs=10)
    mu, sigma = _stats(case["phi"])
    phi, mu_d, sg_d, prm, _, _ = _dev(case, mu, sigma)
    got = spo.spo_ranker_scores(phi, mu_d, sg_d, prm).cpu().numpy()
    want, _ = O.ranker_scores(case["phi"].double().numpy(), mu, sigma, case["params"].double().numpy())
    np.testing.assert_allclose(got, want, atol=1e-4 * max(1.0, np.abs(want).max()))


@pytest.mark.parametrize("n_pairs,dropout", [(1000, False), (997, True), (100003, False)])
def test_ranker_pair_loss_and_grad(spo, n_pairs, dropout):
    case = inputs.ranker_case(n_programs=4096, n_pairs=n_pairs, seed=1006 + n_pairs)
    mu, sigma = _stats(case["phi"])
    phi, mu_d, sg_d, prm, pos, neg = _dev(case, mu, sigma)
    keep1 = keep2 = None
    drop_p = 0.0
    if dropout:
        g = torch.Generator().manual_seed(4)
        drop_p = 0.1
        keep1 = (torch.rand(n_pairs, 2, 64, generator=g) > drop_p).to(torch.uint8)
        keep2 = (torch.rand(n_pairs, 2, 32, generator=g) > drop_p).to(torch.uint8)
    loss, grad = spo.spo_ranker_pair_loss(
        phi, mu_d, sg_d, prm, pos, neg, None if keep1 is None else keep1.cuda(),
        None if keep2 is None else keep2.cuda(), drop_p)
    want_l, want_g = O.ranker_pair_loss(
        case["phi"].double().numpy(), mu, sigma, case["params"].double().numpy(),
        case["pos"].numpy(), case["neg"].numpy(),
        None if keep1 is None else keep1.numpy(), None if keep2 is None else keep2.numpy(), drop_p)
    assert abs(loss.item() - want_l) <= 1e-5 * abs(want_l), (loss.item(), want_l)
    assert P.rel_l2(grad.cpu().numpy(), want_g) <= 1e-4
    # the same call again gives bit-identical results (fixed reduction order)
    loss2, grad2 = spo.spo_ranker_pair_loss(
        phi, mu_d, sg_d, prm, pos, neg, None if keep1 is None else keep1.cuda(),
        None if keep2 is None else keep2.cuda(), drop_p)
    assert torch.equal(grad, grad2) and torch.equal(loss, loss2)


def test_ranker_identical_pair_members(spo):
    case = inputs.ranker_case(n_programs=64, n_pairs=33)
    mu, sigma = _stats(case["phi"])
    phi, mu_d, sg_d, prm, pos, _ = _dev(case, mu, sigma)
    loss, grad = spo.spo_ranker_pair_loss(phi, mu_d, sg_d, prm, pos, pos.clone())
    assert abs(loss.item() - np.log(2.0)) < 1e-6
    assert grad.abs().max().item() < 1e-6
