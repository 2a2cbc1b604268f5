"""dH = G W with 256 x 512 tiles per CTA pair (SPO_TUNE_DH_WIDE = 2: forced,
since these vocabularies are below the default's threshold) against the
256 x 256 tiles: every output element sums the same k-steps in the same
order with the same MMA shape, so dH must be the same bits.  The cases cover
whole wide tiles followed by the last round's 256-column halves, a last
column block that ends inside the first half, the fp32 vocabulary-slice
form, the static schedule and solo mode (where the setting is ignored)."""

import pytest
import torch

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spo():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import build
    build.build()
    from paper_2607_20908_gb300 import spo as mod
    return mod


def _inputs(T, d, V, seed):
    g = torch.Generator(device="cuda").manual_seed(seed)
    H = torch.randn(T, d, device="cuda", generator=g).to(torch.bfloat16)
    W = (torch.randn(V, d, device="cuda", generator=g) * 0.02).to(torch.bfloat16)
    tgt = torch.randint(0, V, (T,), device="cuda", generator=g, dtype=torch.int32)
    gv = torch.randn(T, device="cuda", generator=g) * 1e-3
    return H, W, tgt, gv


def _dh(spo, H, W, tgt, gv, wide, slice_form=False):
    _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
    spo.spo_set_tuning(spo.SPO_TUNE_DH_WIDE, wide)
    if slice_form:
        dH, _ = spo.spo_policy_loss_bwd_ex(H, W, tgt, lse, gv, dH_fp32=True, want_dW=False)
    else:
        dH, _ = spo.spo_policy_loss_bwd(H, W, tgt, lse, gv, want_dW=False)
    torch.cuda.synchronize()
    return dH


@pytest.mark.parametrize("T,d,V,slice_form", [
    (2048, 5120, 4096, False),   # 8 x 10 wide tiles: a round of whole tiles, then halves
    (600, 320, 5000, False),     # ragged rows; the columns end inside the first half
    (1024, 1536, 3000, True),    # fp32 slice form; 3 wide column blocks
])
def test_wide_dh_tiles_give_the_same_bits(spo, T, d, V, slice_form):
    H, W, tgt, gv = _inputs(T, d, V, seed=T + d)
    try:
        narrow = _dh(spo, H, W, tgt, gv, 0, slice_form)
        wide = _dh(spo, H, W, tgt, gv, 2, slice_form)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    assert torch.isfinite(narrow.float()).all()
    assert torch.equal(wide, narrow)
    assert spo.spo_device_error() == 0


def test_wide_dh_static_schedule_and_solo_mode(spo):
    H, W, tgt, gv = _inputs(1536, 2048, 2048, seed=77)
    try:
        want = _dh(spo, H, W, tgt, gv, 0)
        spo.spo_set_tuning(spo.SPO_TUNE_DYNAMIC_MASK, 0b1011)   # dH on the static schedule
        static = _dh(spo, H, W, tgt, gv, 2)
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
        spo.spo_set_tuning(spo.SPO_TUNE_PAIR_MMA, 0)            # solo CTAs: the setting is ignored
        solo = _dh(spo, H, W, tgt, gv, 0)
        solo_wide = _dh(spo, H, W, tgt, gv, 2)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    assert torch.equal(static, want)
    assert torch.equal(solo_wide, solo)
    torch.testing.assert_close(solo.float(), want.float(), rtol=2e-2, atol=1e-6)
    assert spo.spo_device_error() == 0


def test_wide_dh_default_threshold(spo):
    """The default (1) takes the wide tile from 32768 vocabulary rows on:
    both sides of the threshold give the 256 x 256 tiles' bits."""
    for V in (32512, 32768):
        H, W, tgt, gv = _inputs(512, 1024, V, seed=V)
        try:
            want = _dh(spo, H, W, tgt, gv, 0)
            got = _dh(spo, H, W, tgt, gv, 1)
        finally:
            spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
        assert torch.equal(got, want), V
    with pytest.raises(spo.SpoError):
        spo.spo_set_tuning(spo.SPO_TUNE_DH_WIDE, 3)


@pytest.mark.parametrize("T,d,V", [
    (2048, 1024, 40960),   # 8 x 40 wide tiles: whole tiles, then the last round's halves
    (600, 320, 4200),      # the vocabulary ends inside a wide tile's first half
    (1000, 512, 5000),     # ... inside its second half
])
def test_logits_wide_tiles_give_the_same_bits(spo, T, d, V):
    """The forward (logsumexp partials per 256-column vocabulary tile) and the
    recompute (G) with 256 x 512 tiles (SPO_TUNE_LOGITS_WIDE): logp, entropy,
    lse, dH and dW are the same bits as with 256 x 256 tiles."""
    H, W, tgt, gv = _inputs(T, d, V, seed=T + V)
    out = {}
    try:
        for wide in (0, 3):
            spo.spo_set_tuning(spo.SPO_TUNE_LOGITS_WIDE, wide)
            logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt)
            dH, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, gv)
            torch.cuda.synchronize()
            out[wide] = (logp, ent, lse, dH, dW)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    assert torch.isfinite(out[0][0]).all()
    for k, (a, b) in enumerate(zip(out[0], out[3])):
        assert torch.equal(a, b), ("logp", "entropy", "lse", "dH", "dW")[k]
    assert spo.spo_device_error() == 0


def test_wide_tiles_on_the_static_schedule(spo):
    """Every GEMM on the static round robin (no tile counter) with all three
    wide-tile GEMMs forced: the same bits as 256 x 256 tiles everywhere on the
    dynamic schedule."""
    H, W, tgt, gv = _inputs(1000, 768, 6000, seed=99)
    try:
        spo.spo_set_tuning(spo.SPO_TUNE_DH_WIDE, 0)
        spo.spo_set_tuning(spo.SPO_TUNE_LOGITS_WIDE, 0)
        _, _, lse0 = spo.spo_logprobs_fwd(H, W, tgt)
        want = spo.spo_policy_loss_bwd(H, W, tgt, lse0, gv)
        spo.spo_set_tuning(spo.SPO_TUNE_DYNAMIC_MASK, 0)
        spo.spo_set_tuning(spo.SPO_TUNE_DH_WIDE, 2)
        spo.spo_set_tuning(spo.SPO_TUNE_LOGITS_WIDE, 3)
        _, _, lse1 = spo.spo_logprobs_fwd(H, W, tgt)
        got = spo.spo_policy_loss_bwd(H, W, tgt, lse1, gv)
        torch.cuda.synchronize()
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
    assert torch.equal(lse1, lse0)
    assert torch.equal(got[0], want[0]) and torch.equal(got[1], want[1])
    assert spo.spo_device_error() == 0
