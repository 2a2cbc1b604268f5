"""spo_policy_loss_fwd_noalloc: the policy-loss forward for callers that cannot
give the library device scratch memory (a framework pool that owns all device
memory, or a host path that must not call cudaMalloc because it synchronises
the device).  Its scratch is a static array inside libspo that every call
reuses.  It runs the same three kernels in the same fixed order as the
workspace entry point, so on the same inputs the two must agree bit for bit;
here that is checked through the C ABI on three calls in a row, the later
ones on smaller batches with fewer groups (stale group counters or partial
sums left in the array by a larger call would show), and each result is also
checked against the fp64 oracle.  The call must refuse sizes beyond its fixed
scratch.  Collected last on purpose."""

import ctypes

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O
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


def _batch(seed, n_groups, per_group, seq_len, dev):
    g = torch.Generator().manual_seed(seed)
    n_seq = n_groups * per_group
    lens = torch.randint(seq_len // 2, seq_len + 1, (n_seq,), generator=g)
    cu = torch.zeros(n_seq + 1, dtype=torch.int32)
    cu[1:] = torch.cumsum(lens, 0).to(torch.int32)
    T = int(cu[-1])
    logp = -torch.rand(T, generator=g) * 6
    b = dict(
        logp=logp, old=logp + torch.randn(T, generator=g) * 0.2,
        ref=logp + torch.randn(T, generator=g) * 0.05,
        adv=torch.randn(n_seq, generator=g),
        cu=cu, gid=torch.arange(n_groups, dtype=torch.int32).repeat_interleave(per_group),
        mask=(torch.rand(T, generator=g) > 0.25).to(torch.uint8), n_groups=n_groups, T=T,
        n_seq=n_seq)
    return {k: (v.to(dev).contiguous() if isinstance(v, torch.Tensor) else v) for k, v in b.items()}


def _c_call(spo, b, loss, g, stats, agg):
    p = lambda t: ctypes.c_void_p(t.data_ptr())
    stream = ctypes.c_void_p(torch.cuda.current_stream().cuda_stream)
    return spo.lib().spo_policy_loss_fwd_noalloc(
        p(b["logp"]), p(b["old"]), p(b["ref"]), p(b["adv"]), p(b["cu"]), p(b["gid"]), b["n_seq"],
        b["n_groups"], p(b["mask"]), b["T"], 0.2, 0.04, agg, p(loss), p(g), p(stats), stream)


def _oracle(b, agg):
    c = lambda t: t.cpu().numpy()
    return O.policy_loss(c(b["logp"]).astype(np.float64), c(b["old"]).astype(np.float64),
                         c(b["ref"]).astype(np.float64), c(b["adv"]).astype(np.float64), c(b["cu"]),
                         c(b["gid"]), b["n_groups"], c(b["mask"]), 0.2, 0.04, agg)


def test_noalloc_matches_workspace_entry_on_consecutive_calls(spo):
    dev = torch.device("cuda")
    # largest first: each later call has fewer groups and sequences than the one before
    batches = [(_batch(11, 16, 8, 128, dev), 0), (_batch(12, 5, 3, 300, dev), 1),
               (_batch(14, 2, 3, 40, dev), 0)]
    spo.spo_trace_read()
    spo.spo_trace_enable(True)
    try:
        for b, agg in batches:
            want_loss, want_g, want_stats = spo.spo_policy_loss_fwd(
                b["logp"], b["old"], b["ref"], b["adv"], b["cu"], b["gid"], b["n_groups"],
                b["mask"], 0.2, 0.04, agg)
            loss = torch.full((1,), float("nan"), device=dev)
            g = torch.full((b["T"],), float("nan"), device=dev)
            stats = torch.full((4,), float("nan"), device=dev)
            assert _c_call(spo, b, loss, g, stats, agg) == 0
            torch.cuda.synchronize()
            # the same kernels in the same order on the same inputs: the same bits
            assert torch.equal(loss, want_loss), (loss.item(), want_loss.item())
            assert torch.equal(g, want_g)
            assert torch.equal(stats, want_stats)
            # and the definition of Eq. 3 in fp64
            o_loss, o_g, o_st = _oracle(b, agg)
            gl = float(loss.item())
            assert abs(gl - o_loss) <= P.TOL_LOSS_REL * max(abs(o_loss), 1e-12), (gl, o_loss)
            assert P.rel_l2(g.cpu().numpy(), o_g) <= P.TOL_GRAD_REL
            assert int(stats[3].item()) == o_st["n_loss_tokens"]
        recs = spo.spo_trace_read()
    finally:
        spo.spo_trace_enable(False)
    # every loss forward, with or without a workspace, is traced as kind 7
    assert [k for k, _ in recs].count(7) == 2 * len(batches)
    assert spo.spo_device_error() == 0


def test_noalloc_rejects_sizes_beyond_its_scratch(spo):
    dev = torch.device("cuda")
    b = _batch(13, 2, 2, 16, dev)
    b["n_seq"] = 1 << 20        # 1M sequences need ~32 MB of scratch; checked on the host first
    loss = torch.empty(1, device=dev)
    st = _c_call(spo, b, loss, loss, loss, 0)
    assert st == 4
    buf = ctypes.create_string_buffer(512)
    spo.lib().spo_last_error(buf, 512)
    assert b"static scratch" in buf.value
