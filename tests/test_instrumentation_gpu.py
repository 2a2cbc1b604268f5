"""The library's helper and instrumentation calls on the device: the in-place
scale the data-parallel step applies to g and the loss (host or device
factor), the launch counter and the per-step trace of CUDA-event timings that
the benchmark's roofline is computed from."""

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


@pytest.mark.parametrize("n", [1, 3, 1000, 1 << 20, (1 << 20) + 5])
def test_scale_f32_host_and_device_factor(spo, n):
    gen = torch.Generator().manual_seed(31)
    x0 = torch.randn(n, generator=gen)
    x = x0.clone().cuda()
    spo.spo_scale_f32(x, alpha=0.25)
    assert torch.equal(x.cpu(), x0 * 0.25)         # a power of two: exact
    a = torch.tensor([1.0 / 3.0], dtype=torch.float32, device="cuda")
    y = x0.clone().cuda()
    spo.spo_scale_f32(y, alpha_dev=a)
    want = (x0 * torch.tensor(1.0 / 3.0, dtype=torch.float32))
    assert torch.equal(y.cpu(), want)               # one fp32 multiply per element
    # an offset view (not 16-byte aligned) is scaled the same way
    z = x0.clone().cuda()
    spo.spo_scale_f32(z[1:], alpha=-2.0)
    assert torch.equal(z.cpu()[1:], x0[1:] * -2.0) and z[0].item() == x0[0].item()


def _step(spo, case):
    dev = torch.device("cuda")
    H, W = case["H"].to(dev), case["W"].to(dev)
    tgt, mask = case["tgt"].to(dev), case["mask"].to(dev)
    cu, gid = case["cu_seqlens"].to(dev), case["group_id"].to(dev)
    lm, _ = spo.spo_token_select(cu, mask, tgt, case["window"])
    logp, _, lse = spo.spo_logprobs_fwd(H, W, tgt, lm)
    adv = spo.spo_group_advantages(case["rewards"].to(dev), gid, case["n_groups"])
    _, g, _ = spo.spo_policy_loss_fwd(logp, logp, None, adv, cu, gid, case["n_groups"], lm, 0.2, 0.0)
    g = g + 1e-3 * lm.float()                       # every loss row active in the backward
    spo.spo_policy_loss_bwd(H, W, tgt, lse, g)


def test_trace_and_launch_count_of_one_step(spo):
    """One step traced: the records come back in launch order with one record
    per traced sequence of the path (a1, gather, a2, a3, a4, a5, gather, a6,
    a7, a8), all with positive durations; the launch counter grows by at least
    one kernel per record."""
    case = inputs.tiny_case(seed=1601, T_per_seq=100, n_groups=2, rollouts=4, V=5000)
    _step(spo, case)                                 # warm (module load, descriptors)
    torch.cuda.synchronize()
    spo.spo_trace_read()                             # clear
    spo.spo_trace_enable(True)
    try:
        before = spo.spo_launch_count()
        _step(spo, case)
        torch.cuda.synchronize()
        recs = spo.spo_trace_read()
        launched = spo.spo_launch_count() - before
    finally:
        spo.spo_trace_enable(False)
    kinds = [spo.TRACE_KINDS[k] for k, _ in recs]
    assert kinds[:4] == ["token_select", "select_gather_fwd", "logits_lse_fwd", "lse_combine"]
    for name in ("group_advantages", "policy_loss_fwd", "select_gather_bwd",
                 "logits_grad_recompute", "gemm_dH", "gemm_dW"):
        assert name in kinds, name
    assert kinds.index("logits_grad_recompute") < kinds.index("gemm_dH") < kinds.index("gemm_dW")
    assert all(ms > 0 for _, ms in recs)
    assert launched >= len(recs)
    # tracing off: nothing is recorded
    _step(spo, case)
    torch.cuda.synchronize()
    assert spo.spo_trace_read() == []
    assert spo.spo_device_error() == 0
