"""GPU parity: the CUDA path (through the C ABI) against the fp64 oracle on
identical seeded inputs, element by element, at sizes the oracle finishes in
seconds that still span several tiles and a ragged tail."""

import numpy as np
import pytest
import torch

from oracle import spo_oracle as O
from paper_2607_20908_gb300 import inputs
from tests import pipeline as P

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import build
    build.build()


def _compare(case, agg=0, std_mode=0):
    o = P.run_oracle(case, agg=agg, std_mode=std_mode)
    g = P.run_gpu(case, o["old"], o["ref"], agg=agg, std_mode=std_mode)
    lm = o["loss_mask"].astype(bool)
    np.testing.assert_array_equal(g["loss_mask"], o["loss_mask"])
    np.testing.assert_array_equal(g["n_tok"], o["n_tok"])
    err_lp = np.abs(g["logp"] - o["logp"]).max()
    err_ent = np.abs(g["entropy"] - o["entropy"]).max()
    err_lse = np.abs(g["lse"] - o["lse"]).max()
    assert err_lp <= P.TOL_LOGP, err_lp
    assert err_ent <= P.TOL_LOGP, err_ent
    assert err_lse <= P.TOL_LOGP, err_lse
    assert np.all(g["logp"][~lm] == 0) and np.all(g["lse"][~lm] == 0)
    np.testing.assert_allclose(g["adv"], o["adv"], atol=1e-6, rtol=0)
    rel_loss = abs(g["loss"] - o["loss"]) / max(abs(o["loss"]), 1e-12)
    assert rel_loss <= P.TOL_LOSS_REL, (g["loss"], o["loss"])
    assert P.rel_l2(g["g"], o["g"]) <= P.TOL_GRAD_REL
    assert np.all(g["g"][~lm] == 0)
    e_dH = P.rel_l2(g["dH"], o["dH"])
    e_dW = P.rel_l2(g["dW"], o["dW"])
    assert e_dH <= P.TOL_GRAD_REL, e_dH
    assert e_dW <= P.TOL_GRAD_REL, e_dW
    assert abs(g["stats"][3] - o["stats"]["n_loss_tokens"]) == 0
    assert abs(g["stats"][0] - o["stats"]["clip_frac"]) <= 1e-6
    assert abs(g["stats"][1] - o["stats"]["mean_ratio"]) <= 1e-4
    print(f"\n[{case['name']}] |dlogp|={err_lp:.2e} |dent|={err_ent:.2e} "
          f"loss rel={rel_loss:.2e} dH rel={e_dH:.2e} dW rel={e_dW:.2e}")
    return o, g


def test_tiny_workload_fwd_bwd():
    """4 groups x 4 rollouts x 16 tokens, d=256, V=4096 (2 x 16 output tiles)."""
    _compare(inputs.tiny_case())


def test_tiny_workload_clipping_active():
    """Old-policy noise 0.3: a large share of tokens sit on the clipped branch."""
    case = inputs.tiny_case(seed=1011, old_noise_std=0.3)
    o, g = _compare(case)
    assert o["stats"]["clip_frac"] > 0.05


def test_ragged_tails_and_window():
    """T, d and V that are not multiples of the tile (T=1000, d=320, V=5000),
    prompt masks, ignored targets and a window that truncates sequences."""
    case = inputs.tiny_case(seed=1021, T_per_seq=125, n_groups=2, rollouts=4, d=320, V=5000)
    T = case["T"]
    g = torch.Generator().manual_seed(5)
    mask = (torch.rand(T, generator=g) > 0.3).to(torch.uint8)
    tgt = case["tgt"].clone()
    tgt[torch.rand(T, generator=g) < 0.05] = -100
    case.update(mask=mask, tgt=tgt, window=64)
    for agg in (O.AGG_SEQ_GROUP, O.AGG_TOKEN):
        _compare(case, agg=agg)


def test_population_std_and_temperature():
    case = inputs.tiny_case(seed=1031)
    case["inv_temp"] = 1.0 / 0.7
    _compare(case, std_mode=O.STD_POPULATION)


def test_lowest_sampling_temperature():
    """tau = 0.2, the paper's lowest sampling temperature: logits scaled by 5."""
    case = inputs.tiny_case(seed=1032)
    case["inv_temp"] = 1.0 / 0.2
    _compare(case)


def test_peaked_softmax():
    """Logits spread over about +-100 (W ~ N(0, 2^2) at d = 256): most
    exponentials underflow, the softmax is nearly one-hot and the entropy is
    near 0."""
    case = inputs.tiny_case(seed=1033)
    gen = torch.Generator().manual_seed(17)
    case["W"] = (torch.randn(case["V"], case["d"], generator=gen) * 2.0).to(torch.bfloat16)
    o, g = _compare(case)
    assert np.median(o["entropy"]) < 0.5 and np.abs(g["entropy"] - o["entropy"]).max() <= P.TOL_LOGP


def test_advantages_bit_exact_fp32_order():
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(3)
    n, ng = 3000, 200
    r = rng.normal(0.3, 1.0, n).astype(np.float32)
    gid = rng.integers(0, ng, n).astype(np.int32)
    gid[:16] = 7          # one group gets a burst of members
    r[gid == 11] = 1.25   # zero-variance group
    want = O.group_advantages_f32(r, gid, ng)
    got = spo.spo_group_advantages(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(), ng)
    got = got.cpu().numpy()
    np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))
    assert np.all(got[gid == 11] == 0)


@pytest.mark.parametrize("layout", ["contiguous", "scattered", "empty_and_invalid"])
def test_advantages_run_path_bit_exact(layout):
    """The workspace variant: one pass over the runs of equal group ids, then
    each group folded over its own run (contiguous layout) or the per-group
    scan (scattered ids); the same bits as the fp32-order oracle either way."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(4)
    sizes = rng.integers(1, 40, 300)                  # groups of 1..39 sequences
    sizes[[5, 6]] = [1, 64]
    ng = sizes.size
    gid = np.repeat(np.arange(ng), sizes).astype(np.int32)
    n = gid.size
    r = rng.normal(0.3, 1.0, n).astype(np.float32)
    r[gid == 9] = -0.5                                 # zero-variance group
    if layout == "scattered":
        gid = gid[rng.permutation(n)]
    if layout == "empty_and_invalid":
        gid = np.where(gid >= 100, gid + 2, gid).astype(np.int32)   # groups 100, 101 empty
        ng += 2
        gid[[0, n - 1]] = [ng, -1]                      # no group: adv left untouched; every
                                                        # group still one run (the run path)
    want = O.group_advantages_f32(r, np.where((gid >= 0) & (gid < ng), gid, ng), ng + 1)
    adv = torch.full((n,), 7.0, device="cuda")
    got = spo.spo_group_advantages_ws(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(), ng,
                                      adv=adv).cpu().numpy()
    ok = (gid >= 0) & (gid < ng)
    np.testing.assert_array_equal(got[ok].view(np.uint32), want[ok].view(np.uint32))
    assert np.all(got[~ok] == 7.0)
    base = spo.spo_group_advantages(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(), ng)
    np.testing.assert_array_equal(got[ok].view(np.uint32), base.cpu().numpy()[ok].view(np.uint32))


@pytest.mark.parametrize("layout", ["sorted", "reversed"])
def test_advantages_sorted_pass_chunk_edges(layout):
    """Group sizes around the sorted pass's chunks of 4096 sequences: groups
    of one, groups that end exactly on a chunk edge or one before or after it,
    and groups of 4097 and 10000 sequences that run on through two and three
    chunks (one of them with all rewards equal).  "reversed" lays the same
    groups out with their ids in descending order: still one run per group,
    but not sorted, so the call takes the run path.  Bit-exact against the
    fp32-order oracle either way."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(6)
    sizes = np.array([4096, 1, 4095, 2, 4097, 16, 10000, 3, 1, 4094, 5000, 7000]
                     + list(rng.integers(1, 40, 300)))
    ng = sizes.size
    ids = np.arange(ng) if layout == "sorted" else np.arange(ng)[::-1]
    gid = np.repeat(ids, sizes).astype(np.int32)
    r = rng.normal(0.3, 1.0, gid.size).astype(np.float32)
    r[gid == ids[11]] = 2.5                      # 7000 equal rewards across chunk edges
    want = O.group_advantages_f32(r, gid, ng)
    adv = torch.full((gid.size,), 7.0, device="cuda")
    got = spo.spo_group_advantages_ws(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(), ng,
                                      adv=adv).cpu().numpy()
    np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))
    assert np.all(got[gid == ids[11]] == 0) and np.all(got[gid == ids[1]] == 0)


@pytest.mark.parametrize("sizes", [
    [4000, 196],            # the last group runs from chunk 0 to the end of the data, in the halo
    [4000, 1000],           # ... past the halo to the end of the data (folded from memory)
    [3, 4093, 4096, 1],     # groups ending exactly on chunk edges; a last group of one
    [5, 17, 2000],          # one partial chunk
    [1],                    # one sequence
], ids=["tail_in_halo", "tail_past_halo", "exact_edges", "one_chunk", "single"])
def test_advantages_sorted_pass_data_end(sizes):
    """Where the sorted pass's last group meets the end of the data."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(9)
    sizes = np.array(sizes)
    gid = np.repeat(np.arange(sizes.size), sizes).astype(np.int32)
    r = rng.normal(0.3, 1.0, gid.size).astype(np.float32)
    want = O.group_advantages_f32(r, gid, sizes.size)
    adv = torch.full((gid.size,), 7.0, device="cuda")
    got = spo.spo_group_advantages_ws(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(),
                                      sizes.size, adv=adv).cpu().numpy()
    np.testing.assert_array_equal(got.view(np.uint32), want.view(np.uint32))


def test_advantages_sorted_pass_large():
    """2^22 rollouts in sorted groups of 4 to 16 (the enlarged benchmark
    shape): 1025 chunks, every chunk edge inside some group.  The oracle runs
    on 1500 sampled groups (groups are independent, so each sampled group is
    its own small problem)."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(7)
    sizes = rng.integers(4, 17, (1 << 22) // 10)
    sizes = sizes[np.cumsum(sizes) <= (1 << 22) + 1000]
    ng = sizes.size
    gid = np.repeat(np.arange(ng), sizes).astype(np.int32)
    r = rng.normal(0.3, 1.0, gid.size).astype(np.float32)
    got = spo.spo_group_advantages_ws(torch.from_numpy(r).cuda(), torch.from_numpy(gid).cuda(),
                                      ng).cpu().numpy()
    starts = np.concatenate([[0], np.cumsum(sizes)])
    for g in np.sort(rng.choice(ng, 1500, replace=False)):
        seg = slice(starts[g], starts[g + 1])
        want = O.group_advantages_f32(r[seg], np.zeros(sizes[g], dtype=np.int32), 1)
        np.testing.assert_array_equal(got[seg].view(np.uint32), want.view(np.uint32))


@pytest.mark.parametrize("agg", [0, 1])
@pytest.mark.parametrize("max_len", [700, 120])
def test_loss_long_sequences_and_unaligned_mask(agg, max_len):
    """The loss forward on sequences of 1 to 700 tokens (a warp per sequence:
    its first 128 tokens held in registers, the rest reloaded) or of 1 to 120
    (eight lanes per sequence, 32 tokens a pass), groups with a sequence of
    no loss tokens and an empty group, a mask that starts 3 bytes past a
    16-byte boundary (the token mean counts it 16 bytes at a time after a
    ragged head), KL arguments around the switch from the series, and
    stand-in log-probs, against the fp64 oracle."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(8)
    lens = rng.integers(1, max_len + 1, 41 if max_len > 256 else 160)
    lens[[3, 17, 18, 19]] = [128, 129, 32, 33] if max_len > 256 else [31, 32, 33, 120]
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T, n_seq = int(cu[-1]), lens.size
    gid = np.minimum(np.arange(n_seq) // 4, 9).astype(np.int32)
    gid[gid >= 5] += 1                                   # group 5 empty
    ng = int(gid.max()) + 1
    lm = (rng.random(T) < 0.7).astype(np.uint8)
    lm[cu[6]:cu[7]] = 0                                  # a sequence with no loss tokens
    lp = (-6.0 * rng.random(T)).astype(np.float32)
    old = (lp + 0.2 * rng.normal(size=T)).astype(np.float32)
    ref = (lp + 0.05 * rng.normal(size=T)).astype(np.float32)
    # KL arguments on both sides of the series / direct switch at |delta| = 1/2, and far out
    far = rng.choice(np.nonzero(lm)[0], 200, replace=False)
    ref[far] = lp[far] + rng.choice([-0.5001, -0.4999, 0.4999, 0.5001, -3.0, 2.0, 6.0, 1e-4], 200)
    adv = rng.normal(size=n_seq).astype(np.float32)
    buf = torch.zeros(T + 3, dtype=torch.uint8, device="cuda")
    mask = buf[3:]
    mask.copy_(torch.from_numpy(lm))
    dev = lambda a: torch.from_numpy(a).cuda()
    loss, g, stats = spo.spo_policy_loss_fwd(dev(lp), dev(old), dev(ref), dev(adv), dev(cu),
                                             dev(gid), ng, mask, 0.2, 0.04, agg)
    loss_o, g_o, st_o = O.policy_loss(lp.astype(np.float64), old.astype(np.float64),
                                      ref.astype(np.float64), adv.astype(np.float64), cu, gid, ng,
                                      lm, 0.2, 0.04, agg)
    assert abs(loss.item() - loss_o) <= 1e-5 * abs(loss_o)
    assert P.rel_l2(g.cpu().numpy(), g_o) <= 1e-5
    assert np.all(g.cpu().numpy()[lm == 0] == 0)
    assert stats[3].item() == st_o["n_loss_tokens"]
    assert abs(stats[0].item() - st_o["clip_frac"]) <= 1e-6
    assert abs(stats[1].item() - st_o["mean_ratio"]) <= 1e-5 * st_o["mean_ratio"]
    assert abs(stats[2].item() - st_o["mean_kl"]) <= 1e-5 * st_o["mean_kl"]


@pytest.mark.parametrize("window", [-1, 0, 1, 7, 1024])
def test_token_select_windows_and_empty_sequences(window):
    """Loss-token selection, bit-exact against the oracle, for no cap (window
    <= 0), a cap of one token, a small and the paper's 1024-token cap, on
    ragged sequences that include empty ones (equal consecutive cu_seqlens),
    with prompt masks and ignored targets."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(10)
    lens = rng.integers(0, 2000, 60)
    lens[[0, 7, 8, 59]] = 0                           # empty sequences, one at each end
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    mask = (rng.random(T) > 0.4).astype(np.uint8)
    tgt = rng.integers(0, 5000, T).astype(np.int32)
    tgt[rng.random(T) < 0.05] = -100
    lm, n_tok = spo.spo_token_select(torch.from_numpy(cu).cuda(), torch.from_numpy(mask).cuda(),
                                     torch.from_numpy(tgt).cuda(), window)
    lm_o, n_o = O.token_select(cu, mask, tgt, window)
    np.testing.assert_array_equal(lm.cpu().numpy(), lm_o)
    np.testing.assert_array_equal(n_tok.cpu().numpy(), n_o)
    assert np.all(n_tok.cpu().numpy()[lens == 0] == 0)


@pytest.mark.parametrize("agg", [0, 1])
def test_loss_with_empty_sequences(agg):
    """Empty sequences (no tokens) still count in their group's size and add
    nothing to the loss (reading R6); checked against the fp64 oracle."""
    from paper_2607_20908_gb300 import spo
    rng = np.random.default_rng(11)
    lens = rng.integers(1, 300, 48)
    lens[[0, 5, 6, 47]] = 0
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T = int(cu[-1])
    gid = (np.arange(48) // 4).astype(np.int32)
    lm = (rng.random(T) < 0.8).astype(np.uint8)
    lp = (-5.0 * rng.random(T)).astype(np.float32)
    old = (lp + 0.1 * rng.normal(size=T)).astype(np.float32)
    ref = (lp + 0.05 * rng.normal(size=T)).astype(np.float32)
    adv = rng.normal(size=48).astype(np.float32)
    dev = lambda a: torch.from_numpy(a).cuda()
    loss, g, stats = spo.spo_policy_loss_fwd(dev(lp), dev(old), dev(ref), dev(adv), dev(cu),
                                             dev(gid), 12, dev(lm), 0.2, 0.04, agg)
    loss_o, g_o, st_o = O.policy_loss(lp.astype(np.float64), old.astype(np.float64),
                                      ref.astype(np.float64), adv.astype(np.float64), cu, gid, 12,
                                      lm, 0.2, 0.04, agg)
    assert abs(loss.item() - loss_o) <= 1e-5 * abs(loss_o)
    assert P.rel_l2(g.cpu().numpy(), g_o) <= 1e-5
    assert stats[3].item() == st_o["n_loss_tokens"]


def test_no_loss_tokens():
    """Every token masked: log-probs, loss, g, dH and dW are exactly zero."""
    case = inputs.tiny_case(seed=1041)
    case["mask"] = torch.zeros(case["T"], dtype=torch.uint8)
    o = P.run_oracle(case)
    g = P.run_gpu(case, o["old"], o["ref"])
    for k in ("logp", "lse", "entropy", "g", "dH", "dW"):
        assert np.all(g[k] == 0), k
    assert g["loss"] == 0.0


def test_single_loss_token():
    case = inputs.tiny_case(seed=1051)
    m = torch.zeros(case["T"], dtype=torch.uint8)
    m[37] = 1
    case["mask"] = m
    _compare(case)


def test_dw_accumulate_and_skip_outputs():
    from paper_2607_20908_gb300 import spo
    case = inputs.tiny_case(seed=1061)
    H, W, tgt = case["H"].cuda(), case["W"].cuda(), case["tgt"].cuda()
    _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
    g = torch.randn(case["T"], device="cuda") * 1e-2
    _, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse, g, want_dH=False)
    base = torch.randn_like(dW1)
    _, dW2 = spo.spo_policy_loss_bwd(H, W, tgt, lse, g, dW=base.clone(), accumulate_dW=True,
                                     want_dH=False)
    torch.testing.assert_close(dW2, base + dW1, rtol=1e-5, atol=1e-6)
    dH, dWn = spo.spo_policy_loss_bwd(H, W, tgt, lse, g, want_dW=False)
    assert dWn is None and dH is not None


def test_single_cta_mode_matches_oracle():
    """The same kernels with one CTA per 128 x 256 tile (no CTA-pair MMA)."""
    from paper_2607_20908_gb300 import spo
    spo.spo_set_tuning(spo.SPO_TUNE_PAIR_MMA, 0)
    spo.spo_set_tuning(spo.SPO_TUNE_GROUP_M, 3)
    try:
        _compare(inputs.tiny_case(seed=1071))
        case = inputs.tiny_case(seed=1072, T_per_seq=125, n_groups=2, rollouts=4, d=320, V=5000)
        case["mask"] = (torch.rand(case["T"], generator=torch.Generator().manual_seed(9)) > 0.3).to(torch.uint8)
        _compare(case)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)


@pytest.mark.parametrize("mask", [0, 15])
def test_static_and_dynamic_tile_schedules(mask):
    """Every GEMM on the static round robin (mask 0) or on the atomic-counter
    schedule (mask 15), with a small raster group so tiles of several groups
    are in flight at once."""
    from paper_2607_20908_gb300 import spo
    spo.spo_set_tuning(spo.SPO_TUNE_DYNAMIC_MASK, mask)
    spo.spo_set_tuning(spo.SPO_TUNE_GROUP_M, 2)
    try:
        _compare(inputs.tiny_case(seed=1081))
        case = inputs.tiny_case(seed=1082, T_per_seq=125, n_groups=2, rollouts=4, d=320, V=5000)
        _compare(case)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)


def test_validate_inputs_counts_planted_errors():
    from paper_2607_20908_gb300 import spo
    case = inputs.tiny_case(seed=1091)
    T, V = case["T"], case["V"]
    c = lambda t: t.cuda()
    clean = spo.spo_validate_inputs(c(case["tgt"]), V, c(case["cu_seqlens"]), c(case["group_id"]),
                                    case["n_groups"], c(case["rewards"]), c(case["old_noise"]),
                                    c(case["ref_noise"]), c(case["mask"]))
    assert all(v == 0 for v in clean.values()), clean
    tgt = case["tgt"].clone(); tgt[[3, 77]] = V; tgt[5] = -100          # -100 stays valid
    cu = case["cu_seqlens"].clone(); cu[4] = cu[3] - 1; cu[-1] = T + 1   # one decrease, wrong end
    gid = case["group_id"].clone(); gid[0] = case["n_groups"]; gid[1] = -1
    rw = case["rewards"].clone(); rw[2] = float("nan")
    old = case["old_noise"].clone(); old[9] = float("inf")
    mask = case["mask"].clone(); mask[10] = 2
    bad = spo.spo_validate_inputs(c(tgt), V, c(cu), c(gid), case["n_groups"], c(rw), c(old),
                                  c(case["ref_noise"]), c(mask))
    assert bad == dict(tgt_out_of_range=2, bad_cu_seqlens=2, bad_group_id=2, nonfinite_rewards=1,
                       nonfinite_old_ref_logp=1, bad_mask=1), bad


def test_minimum_sizes():
    """T = 1 token, d = 64, V = 256: one partial tile everywhere."""
    case = inputs.tiny_case(seed=1101, T_per_seq=1, n_groups=1, rollouts=1, d=64, V=256)
    _compare(case)


def test_two_rollout_group_and_long_window():
    """Groups of two (the smallest with a non-zero advantage), sequences longer than the window."""
    case = inputs.tiny_case(seed=1111, T_per_seq=300, n_groups=3, rollouts=2, d=128, V=1024)
    case["window"] = 256
    _compare(case)


def test_dw_split_passes():
    """dW reduced over token passes of 256 rows (several reduce-add passes per chunk)."""
    from paper_2607_20908_gb300 import spo
    spo.spo_set_tuning(spo.SPO_TUNE_DW_SPLIT_ROWS, 256)
    try:
        case = inputs.tiny_case(seed=1121, T_per_seq=125, n_groups=2, rollouts=4, d=320, V=5000)
        _compare(case)
    finally:
        spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
