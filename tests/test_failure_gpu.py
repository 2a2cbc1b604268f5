"""Failure detection on the GPU without a fault: a bounded wait is made to run
out (a barrier that nothing arrives on), the host reads the timeout status,
and the context stays usable for the tensor-core path."""

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


def test_expired_wait_is_reported_and_context_survives(spo):
    assert spo.spo_device_error() == 0
    spo.spo_selftest_bounded_wait()
    assert spo.spo_device_error() == 0x1FF          # SPO_ERR_TIMEOUT with the self-test's code
    assert spo.spo_device_error() == 0              # reading clears it

    c = inputs.tiny_case()
    logp, ent, lse = spo.spo_logprobs_fwd(c["H"].cuda(), c["W"].cuda(), c["tgt"].cuda())
    Ho, Wo = P.oracle_hw(c)
    lp_o, _, _ = O.logprobs(Ho, Wo, c["tgt"].numpy())
    assert np.abs(logp.cpu().numpy() - lp_o).max() <= P.TOL_LOGP
    assert spo.spo_device_error() == 0
