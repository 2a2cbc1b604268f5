"""The one-call step (spo_grpo_step) and the backward with collective hooks
(spo_policy_loss_bwd_ex), through the C ABI on the GPU.

The step runs a1 -> a8 exactly as the separate calls do, reusing the
forward's compaction of loss tokens in the backward; when no loss token has
g == 0 every output is bit-identical to the separate calls, and in any case
the step matches the fp64 oracle at the path's bars.  The hooked backward
computes dW block by block over the vocabulary with an event per finished
block; the reduction order of every dW element is unchanged, so it is
bit-identical to the plain backward."""

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


def _dev(case, old, ref, dev="cuda"):
    t = lambda x: x.to(dev).contiguous()
    return dict(H=t(case["H"]), W=t(case["W"]), tgt=t(case["tgt"]), mask=t(case["mask"]),
                cu=t(case["cu_seqlens"]), gid=t(case["group_id"]), rewards=t(case["rewards"]),
                old=torch.from_numpy(np.asarray(old, np.float32)).to(dev),
                ref=torch.from_numpy(np.asarray(ref, np.float32)).to(dev))


def _separate(spo, case, b, agg=0, std_mode=0):
    lm, _ = spo.spo_token_select(b["cu"], b["mask"], b["tgt"], case["window"])
    logp, ent, lse = spo.spo_logprobs_fwd(b["H"], b["W"], b["tgt"], lm, case["inv_temp"])
    adv = spo.spo_group_advantages(b["rewards"], b["gid"], case["n_groups"], std_mode, 1e-6)
    loss, g, stats = spo.spo_policy_loss_fwd(logp, b["old"], b["ref"], adv, b["cu"], b["gid"],
                                             case["n_groups"], lm, case["clip_eps"],
                                             case["kl_beta"], agg)
    dH, dW = spo.spo_policy_loss_bwd(b["H"], b["W"], b["tgt"], lse, g, case["inv_temp"])
    return dict(loss_mask=lm, logp=logp, entropy=ent, lse=lse, adv=adv, loss=loss, g=g,
                stats=stats, dH=dH, dW=dW)


def _fused(spo, case, b, agg=0, std_mode=0, **kw):
    return spo.spo_grpo_step(b["H"], b["W"], b["tgt"], b["mask"], b["cu"], b["gid"],
                             case["n_groups"], b["rewards"], b["old"], b["ref"],
                             inv_temp=case["inv_temp"], window=case["window"],
                             clip_eps=case["clip_eps"], kl_beta=case["kl_beta"], agg=agg,
                             std_mode=std_mode, **kw)


def _ragged_case():
    case = inputs.tiny_case(seed=1021, T_per_seq=125, n_groups=2, rollouts=4, d=320, V=5000)
    T = case["T"]
    g = torch.Generator().manual_seed(5)
    mask = (torch.rand(T, generator=g) > 0.3).to(torch.uint8)
    tgt = case["tgt"].clone()
    tgt[torch.rand(T, generator=g) < 0.05] = -100
    case.update(mask=mask, tgt=tgt, window=64)
    return case


@pytest.mark.parametrize("which,agg,std_mode", [("tiny", 0, 0), ("ragged", 0, 0),
                                                ("ragged", 1, 1)])
def test_step_equals_separate_calls_and_oracle(spo, which, agg, std_mode):
    case = inputs.tiny_case() if which == "tiny" else _ragged_case()
    o = P.run_oracle(case, agg=agg, std_mode=std_mode)
    b = _dev(case, o["old"], o["ref"])
    want = _separate(spo, case, b, agg, std_mode)
    got = _fused(spo, case, b, agg, std_mode)
    torch.cuda.synchronize()
    # kl_beta > 0: no loss token has g == 0, so the row sets match and every bit does
    assert bool((got["g"][got["loss_mask"].bool()] != 0).all())
    for k in ("loss_mask", "logp", "entropy", "lse", "adv", "loss", "g", "stats", "dH", "dW"):
        assert torch.equal(got[k], want[k]), k
    # and the fp64 oracle
    lm = o["loss_mask"].astype(bool)
    assert np.abs(got["logp"].cpu().numpy() - o["logp"]).max() <= P.TOL_LOGP
    loss = float(got["loss"].item())
    assert abs(loss - o["loss"]) <= P.TOL_LOSS_REL * max(abs(o["loss"]), 1e-12)
    assert P.rel_l2(got["g"].cpu().numpy(), o["g"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(got["dH"].float().cpu().numpy(), o["dH"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(got["dW"].cpu().numpy(), o["dW"]) <= P.TOL_GRAD_REL
    assert np.all(got["logp"].cpu().numpy()[~lm] == 0)
    assert spo.spo_sync_check() == 0


def test_step_with_zero_gradient_loss_tokens(spo):
    """kl_beta = 0 and a binding clip: many loss tokens have g == 0 exactly.
    The step runs them through the backward with zero gradient rows (the
    separate backward skips them); results still match the oracle, and dH is
    exactly 0 on every row with g == 0."""
    case = inputs.tiny_case(seed=1011, old_noise_std=0.3)
    case["kl_beta"] = 0.0
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    got = _fused(spo, case, b)
    torch.cuda.synchronize()
    g = got["g"].cpu().numpy()
    assert (g == 0).sum() > 10
    assert np.all(got["dH"].float().cpu().numpy()[g == 0] == 0)
    assert abs(float(got["loss"].item()) - o["loss"]) <= P.TOL_LOSS_REL * abs(o["loss"])
    assert P.rel_l2(got["dH"].float().cpu().numpy(), o["dH"]) <= P.TOL_GRAD_REL
    assert P.rel_l2(got["dW"].cpu().numpy(), o["dW"]) <= P.TOL_GRAD_REL


def test_step_outputs_optional_and_loss_scale(spo):
    """Every output but the loss may be omitted (kept in the workspace); a
    device loss scale multiplies the loss and g (a data-parallel weight)."""
    case = inputs.tiny_case(seed=1041)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    full = _fused(spo, case, b)
    bare = _fused(spo, case, b, want=(), want_dH=False, want_dW=False)
    torch.cuda.synchronize()
    assert torch.equal(bare["loss"], full["loss"])
    only_dw = _fused(spo, case, b, want=(), want_dH=False)
    assert torch.equal(only_dw["dW"], full["dW"])
    scale = torch.tensor([0.25], device="cuda")
    sc = _fused(spo, case, b, loss_scale=scale)
    torch.cuda.synchronize()
    np.testing.assert_allclose(sc["loss"].item(), 0.25 * full["loss"].item(), rtol=1e-6)
    np.testing.assert_allclose(sc["g"].cpu().numpy(), 0.25 * full["g"].cpu().numpy(),
                               rtol=1e-6, atol=1e-12)
    assert P.rel_l2(sc["dW"].cpu().numpy(), 0.25 * full["dW"].cpu().numpy()) <= 1e-2
    assert torch.equal(sc["stats"], full["stats"])


def test_step_accumulates_dW(spo):
    case = inputs.tiny_case(seed=1042)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    first = _fused(spo, case, b)
    acc = first["dW"].clone()
    _fused(spo, case, b, dW=acc, accumulate_dW=True, want=())
    torch.cuda.synchronize()
    np.testing.assert_allclose(acc.cpu().numpy(), 2 * first["dW"].cpu().numpy(), rtol=1e-6,
                               atol=1e-12)


@pytest.mark.parametrize("n_blocks,reserve", [(1, 0), (4, 0), (7, 16)])
def test_hooked_backward_bit_identical(spo, n_blocks, reserve):
    """dW by vocabulary blocks with an event per block (and one for dH): the
    same bits as the plain backward; every event completes."""
    case = inputs.tiny_case(seed=1051, d=320, V=5000, T_per_seq=40)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    s = _separate(spo, case, b)
    evs = [torch.cuda.Event() for _ in range(n_blocks)]
    dh_ev = torch.cuda.Event()
    hooks = spo.make_hooks(n_blocks, evs, dh_ev, reserve_sms=reserve)
    dH, dW = spo.spo_policy_loss_bwd_ex(b["H"], b["W"], b["tgt"], s["lse"], s["g"],
                                        case["inv_temp"], hooks=hooks)
    torch.cuda.synchronize()
    assert torch.equal(dH, s["dH"]) and torch.equal(dW, s["dW"])
    assert all(e.query() for e in evs) and dh_ev.query()
    starts = spo.dw_block_starts(case["V"], n_blocks)
    assert starts[0] == 0 and starts[-1] == case["V"]


def test_hooked_slice_backward_bit_identical(spo):
    """The vocabulary-slice form of the hooked call (fp32 dH part) equals
    spo_policy_loss_bwd_slice bit for bit."""
    case = inputs.tiny_case(seed=1052, V=4096)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    s = _separate(spo, case, b)
    off, n = 1024, 2048
    Ws = b["W"][off:off + n]
    want_dH, want_dW = spo.spo_policy_loss_bwd_slice(b["H"], Ws, off, b["tgt"], s["lse"], s["g"])
    ev = torch.cuda.Event()
    hooks = spo.make_hooks(3, [None, torch.cuda.Event(), None], ev)
    dH, dW = spo.spo_policy_loss_bwd_ex(b["H"], Ws, b["tgt"], s["lse"], s["g"], v_offset=off,
                                        dH_fp32=True, hooks=hooks)
    torch.cuda.synchronize()
    assert torch.equal(dH, want_dH) and torch.equal(dW, want_dW) and ev.query()


def test_hooked_step_full_workload_equals_separate_calls(spo):
    """The benchmark's workload (T = 16384, d = 5120, V = 151936) in the
    launch configuration the benchmark times: the one-call step with dW in
    four blocks equals the separate calls bit for bit (their parity against
    the oracle at this size is covered by the full-size tests)."""
    case = inputs.full_case(device="cuda")
    dev = torch.device("cuda")
    b = dict(H=case["H"], W=case["W"], tgt=case["tgt"].to(dev), mask=case["mask"].to(dev),
             cu=case["cu_seqlens"].to(dev), gid=case["group_id"].to(dev),
             rewards=case["rewards"].to(dev))
    lm, _ = spo.spo_token_select(b["cu"], b["mask"], b["tgt"], case["window"])
    logp, _, _ = spo.spo_logprobs_fwd(b["H"], b["W"], b["tgt"], lm)
    b["old"] = logp + case["old_noise"].to(dev)
    b["ref"] = logp + case["ref_noise"].to(dev)
    want = _separate(spo, case, b)
    want = {k: want[k] for k in ("loss", "g", "dH", "dW")}
    torch.cuda.synchronize()
    evs = [torch.cuda.Event() for _ in range(4)]
    got = _fused(spo, case, b, want=("g",), hooks=spo.make_hooks(4, evs, None, reserve_sms=8))
    torch.cuda.synchronize()
    for k in ("loss", "g", "dH", "dW"):
        assert torch.equal(got[k], want[k]), k
    assert all(e.query() for e in evs)
    assert spo.spo_sync_check() == 0


def test_scale_ratio_and_sync_check(spo):
    x = torch.arange(1, 1001, dtype=torch.float32, device="cuda")
    num = torch.tensor([3.0], dtype=torch.float64, device="cuda")
    den = torch.tensor([12.0], dtype=torch.float64, device="cuda")
    y = spo.spo_scale_f32_ratio(x.clone(), num, den)
    assert torch.equal(y, x * 0.25)
    z = spo.spo_scale_f32_ratio(x.clone(), num, torch.zeros(1, dtype=torch.float64, device="cuda"))
    assert torch.equal(z, torch.zeros_like(x))
    # a bounded wait that expires is reported by the next check, then cleared
    spo.spo_selftest_bounded_wait()
    assert spo.spo_sync_check() == 7
    assert spo.spo_sync_check() == 0


def test_k_progress_throttle_changes_no_bit(spo):
    """The k-progress throttle only delays operand loads: with every GEMM kind
    throttled to a tight window the outputs are the same bits."""
    case = inputs.tiny_case(seed=1061, d=512, V=8192, T_per_seq=64)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    want = _separate(spo, case, b)
    try:
        for key in (spo.SPO_TUNE_KSYNC_FWD, spo.SPO_TUNE_KSYNC_GRAD, spo.SPO_TUNE_KSYNC_DH,
                    spo.SPO_TUNE_KSYNC_DW):
            spo.spo_set_tuning(key, 2)
        spo.spo_set_tuning(spo.SPO_TUNE_KSYNC_EPOCH, 1)
        got = _separate(spo, case, b)
        fused = _fused(spo, case, b)
        torch.cuda.synchronize()
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    for k in ("logp", "entropy", "lse", "loss", "g", "dH", "dW"):
        assert torch.equal(got[k], want[k]), k
        assert torch.equal(fused[k], want[k]), k
    assert spo.spo_device_error() == 0


@pytest.mark.parametrize("shape", [dict(d=512, V=8192, T_per_seq=64),
                                   dict(d=320, V=5000, T_per_seq=125, n_groups=2, rollouts=4)])
def test_step_forward_wide_tiles_change_no_bit(spo, shape):
    """Inside the one-call step the forward GEMM takes 256 x 512 tiles (bit 2 of
    SPO_TUNE_LOGITS_WIDE, on by default): the step's outputs are the same bits
    as with 256 x 256 tiles for both logits GEMMs, and as the separate calls
    (whose forward keeps 256 x 256 tiles)."""
    case = inputs.tiny_case(seed=1064, **shape)
    o = P.run_oracle(case)
    b = _dev(case, o["old"], o["ref"])
    try:
        spo.spo_set_tuning(spo.SPO_TUNE_LOGITS_WIDE, 0)
        want = _fused(spo, case, b)
        spo.spo_set_tuning(spo.SPO_TUNE_LOGITS_WIDE, 6)
        got = _fused(spo, case, b)
        sep = _separate(spo, case, b)
        torch.cuda.synchronize()
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    for k in ("logp", "entropy", "lse", "loss", "g", "dH", "dW"):
        assert torch.equal(got[k], want[k]), k
        assert torch.equal(sep[k], want[k]), k
    assert spo.spo_device_error() == 0


def test_step_ragged_workload_two_chunks_equals_separate_calls(spo):
    """The ragged multi-turn workload (65536 packed tokens, ~40% masked, about
    39k loss tokens): the backward runs in two chunks of the forward's
    compaction, reading lse and g at token positions through each chunk's
    offset.  The one-call step equals the separate calls bit for bit."""
    case = inputs.ragged_case(device="cuda")
    dev = torch.device("cuda")
    b = dict(H=case["H"], W=case["W"], tgt=case["tgt"].to(dev), mask=case["mask"].to(dev),
             cu=case["cu_seqlens"].to(dev), gid=case["group_id"].to(dev),
             rewards=case["rewards"].to(dev))
    lm, _ = spo.spo_token_select(b["cu"], b["mask"], b["tgt"], case["window"])
    assert int(lm.sum().item()) > 32768            # more than one backward chunk
    logp, _, _ = spo.spo_logprobs_fwd(b["H"], b["W"], b["tgt"], lm)
    b["old"] = logp + case["old_noise"].to(dev)
    b["ref"] = logp + case["ref_noise"].to(dev)
    want = _separate(spo, case, b)
    want = {k: want[k] for k in ("loss", "g", "logp", "dH", "dW")}
    torch.cuda.synchronize()
    got = _fused(spo, case, b, want=("g", "logp"))
    torch.cuda.synchronize()
    for k in ("loss", "g", "logp", "dH", "dW"):
        assert torch.equal(got[k], want[k]), k
    assert spo.spo_sync_check() == 0


def test_loss_launch_forms_agree_across_the_sequence_threshold(spo):
    """Up to 16384 sequences the loss forward is one cooperative launch (grid
    barriers between its phases); beyond, three launches of the same phases.
    With TOKEN aggregation an empty sequence changes nothing, so the batch of
    16384 sequences and the same batch plus one empty sequence give the same
    bits across the two forms; both match the oracle."""
    dev = torch.device("cuda")
    g = torch.Generator().manual_seed(71)
    n = 16384
    lens = torch.randint(1, 7, (n,), generator=g)
    T = int(lens.sum())
    cu = torch.zeros(n + 2, dtype=torch.int32)
    cu[1:n + 1] = torch.cumsum(lens, 0).to(torch.int32)
    cu[n + 1] = T                                   # the extra sequence is empty
    gid = torch.arange(n + 1, dtype=torch.int32) // 8
    gid[n] = 0
    lp = -torch.rand(T, generator=g) * 6
    old = lp + torch.randn(T, generator=g) * 0.2
    ref = lp + torch.randn(T, generator=g) * 0.05
    adv = torch.randn(n + 1, generator=g)
    lm = (torch.rand(T, generator=g) > 0.2).to(torch.uint8)
    d = lambda t: t.to(dev).contiguous()
    outs = []
    for k in (n, n + 1):
        loss, gg, st = spo.spo_policy_loss_fwd(d(lp), d(old), d(ref), d(adv[:k]), d(cu[:k + 1]),
                                               d(gid[:k]), n // 8, d(lm), 0.2, 0.04, 1)
        torch.cuda.synchronize()
        outs.append((loss, gg, st))
    assert torch.equal(outs[0][0], outs[1][0]) and torch.equal(outs[0][1], outs[1][1])
    assert torch.equal(outs[0][2], outs[1][2])
    o_loss, o_g, o_st = O.policy_loss(lp.double().numpy(), old.double().numpy(),
                                      ref.double().numpy(), adv[:n].double().numpy(),
                                      cu[:n + 1].numpy(), gid[:n].numpy(), n // 8, lm.numpy(),
                                      0.2, 0.04, 1)
    assert abs(outs[0][0].item() - o_loss) <= P.TOL_LOSS_REL * abs(o_loss)
    assert P.rel_l2(outs[0][1].cpu().numpy(), o_g) <= P.TOL_GRAD_REL
    assert int(outs[0][2][3].item()) == o_st["n_loss_tokens"]
    assert spo.spo_sync_check() == 0
