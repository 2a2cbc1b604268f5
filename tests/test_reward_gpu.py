"""GPU parity of the composite reward (section 2.2 verifiable reward plus the
structural score) against the fp64 oracle, and its use as the input of the
group advantages."""

import json
import os

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spo():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import build
    build.build()
    from paper_2607_20908_gb300 import spo as mod
    return mod


def _cuda(x, dtype):
    return torch.as_tensor(np.asarray(x), dtype=dtype).cuda()


def test_reward_hand_cases(spo, golden_dir):
    with open(os.path.join(golden_dir, "verifiable_reward_hand_cases.json")) as f:
        cs = json.load(f)["cases"]
    r = spo.spo_reward_compose(_cuda([c["compiled"] for c in cs], torch.uint8),
                               _cuda([c["pass_rate"] for c in cs], torch.float32),
                               _cuda([c["speedup"] for c in cs], torch.float32),
                               _cuda([c["cv"] for c in cs], torch.float32),
                               _cuda([c["r_struct"] for c in cs], torch.float32))
    np.testing.assert_allclose(r.cpu().numpy(), [c["reward"] for c in cs], atol=1e-6)


def _random_batch(n, seed):
    rng = np.random.default_rng(seed)
    compiled = (rng.random(n) < 0.8).astype(np.uint8)
    p = np.where(rng.random(n) < 0.5, 1.0, rng.random(n)).astype(np.float32)
    S = np.exp2(rng.uniform(-3, 8, n)).astype(np.float32)
    S[rng.random(n) < 0.01] = 0.0
    S[rng.random(n) < 0.01] = -1.0
    cv = rng.uniform(0, 1, n).astype(np.float32)
    rs = rng.standard_normal(n).astype(np.float32)
    return compiled, p, S, cv, rs


def test_reward_random_batch_matches_oracle(spo):
    n = 100003
    compiled, p, S, cv, rs = _random_batch(n, 1)
    want = O.reward_compose(compiled, p, S, cv, rs)
    got = spo.spo_reward_compose(_cuda(compiled, torch.uint8), _cuda(p, torch.float32),
                                 _cuda(S, torch.float32), _cuda(cv, torch.float32),
                                 _cuda(rs, torch.float32)).cpu().numpy()
    np.testing.assert_allclose(got, want, atol=2e-6, rtol=0)
    got0 = spo.spo_reward_compose(_cuda(compiled, torch.uint8), _cuda(p, torch.float32),
                                  _cuda(S, torch.float32), _cuda(cv, torch.float32)).cpu().numpy()
    np.testing.assert_allclose(got0, O.reward_compose(compiled, p, S, cv), atol=2e-6, rtol=0)


def test_reward_custom_parameters(spo):
    prm = dict(alpha_comp=5.0, alpha_wrong=1.0, alpha_speed=0.5, alpha_cv=2.0, s_min=-1.0, s_max=2.0)
    compiled, p, S, cv, rs = _random_batch(4099, 2)
    got = spo.spo_reward_compose(_cuda(compiled, torch.uint8), _cuda(p, torch.float32),
                                 _cuda(S, torch.float32), _cuda(cv, torch.float32),
                                 _cuda(rs, torch.float32), params=prm).cpu().numpy()
    np.testing.assert_allclose(got, O.reward_compose(compiled, p, S, cv, rs, prm), atol=2e-6)
    with pytest.raises(spo.SpoError):
        spo.spo_reward_compose(_cuda(compiled, torch.uint8), _cuda(p, torch.float32),
                               _cuda(S, torch.float32), _cuda(cv, torch.float32),
                               params=dict(prm, s_min=3.0))


def test_reward_feeds_group_advantages(spo):
    """16 candidates per task (section 3): rewards -> advantages on the device."""
    n_groups, g = 64, 16
    compiled, p, S, cv, rs = _random_batch(n_groups * g, 3)
    gid = np.repeat(np.arange(n_groups), g).astype(np.int32)
    r = spo.spo_reward_compose(_cuda(compiled, torch.uint8), _cuda(p, torch.float32),
                               _cuda(S, torch.float32), _cuda(cv, torch.float32),
                               _cuda(rs, torch.float32))
    adv = spo.spo_group_advantages(r, _cuda(gid, torch.int32), n_groups).cpu().numpy()
    want = O.group_advantages(O.reward_compose(compiled, p, S, cv, rs), gid, n_groups)
    np.testing.assert_allclose(adv, want, atol=1e-5)
