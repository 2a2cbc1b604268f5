"""Shared drivers for the parity tests: run the whole path once through the
C ABI (CUDA) and once through the fp64 oracle on the same seeded inputs."""

from __future__ import annotations

import numpy as np
import torch

from oracle import spo_oracle as O
from paper_2607_20908_gb300 import inputs

# Tolerances (the path's stated bar for bf16 inputs with fp32 accumulation).
TOL_LOGP = 2e-2        # |d logp|, |d entropy|
TOL_LOSS_REL = 1e-3    # relative error of the scalar loss
TOL_GRAD_REL = 2e-2    # relative L2 error of dH, dW (and of g = dL/dlogp)


def rel_l2(a, b) -> float:
    a = np.asarray(a, dtype=np.float64)
    b = np.asarray(b, dtype=np.float64)
    den = np.linalg.norm(b)
    return float(np.linalg.norm(a - b) / (den if den > 0 else 1.0))


def oracle_hw(case):
    return (O.bf16_bits_to_f64(inputs.bf16_bits(case["H"])),
            O.bf16_bits_to_f64(inputs.bf16_bits(case["W"])))


def away_from_clip(noise: np.ndarray, eps: float, margin: float = 2e-3) -> np.ndarray:
    """Shift noise values whose ratio exp(-noise) sits within `margin` of a
    clip bound, so both sides take the same branch of the surrogate."""
    noise = noise.copy()
    for bound in (1.0 + eps, 1.0 - eps):
        for _ in range(4):
            rho = np.exp(-noise)
            near = np.abs(rho - bound) < margin
            if not near.any():
                break
            noise[near] += 4 * margin
    return noise


def run_oracle(case, agg=O.AGG_SEQ_GROUP, std_mode=O.STD_UNBIASED, eps_adv=1e-6):
    """The oracle pipeline; old/ref log-probs = oracle logp + the case's noise."""
    H, W = oracle_hw(case)
    tgt = case["tgt"].numpy()
    cu = case["cu_seqlens"].numpy()
    loss_mask, n_tok = O.token_select(cu, case["mask"].numpy(), tgt, case["window"])
    logp, ent, lse = O.logprobs(H, W, tgt, case["inv_temp"], loss_mask)
    old_noise = away_from_clip(case["old_noise"].double().numpy(), case["clip_eps"])
    old = (logp + old_noise).astype(np.float32)
    ref = (logp + case["ref_noise"].double().numpy()).astype(np.float32)
    adv = O.group_advantages(case["rewards"].numpy(), case["group_id"].numpy(), case["n_groups"],
                             std_mode, eps_adv)
    loss, g, stats = O.policy_loss(logp, old, ref, adv, cu, case["group_id"].numpy(),
                                   case["n_groups"], loss_mask, case["clip_eps"], case["kl_beta"],
                                   agg)
    dH, dW = O.policy_loss_bwd(H, W, tgt, g, case["inv_temp"])
    return dict(loss_mask=loss_mask, n_tok=n_tok, logp=logp, entropy=ent, lse=lse, old=old,
                ref=ref, adv=adv, loss=loss, g=g, stats=stats, dH=dH, dW=dW)


def run_gpu(case, old, ref, agg=0, std_mode=0, eps_adv=1e-6, device="cuda"):
    """The CUDA pipeline through the C ABI, given old/ref log-probs (fp32 numpy)."""
    from paper_2607_20908_gb300 import spo
    dev = torch.device(device)
    H = case["H"].to(dev)
    W = case["W"].to(dev)
    tgt = case["tgt"].to(dev)
    mask = case["mask"].to(dev)
    cu = case["cu_seqlens"].to(dev)
    gid = case["group_id"].to(dev)
    loss_mask, n_tok = spo.spo_token_select(cu, mask, tgt, case["window"])
    logp, ent, lse = spo.spo_logprobs_fwd(H, W, tgt, loss_mask, case["inv_temp"])
    adv = spo.spo_group_advantages(case["rewards"].to(dev), gid, case["n_groups"], std_mode,
                                   eps_adv)
    loss, g, stats = spo.spo_policy_loss_fwd(
        logp, torch.from_numpy(old).to(dev), torch.from_numpy(ref).to(dev), adv, cu, gid,
        case["n_groups"], loss_mask, case["clip_eps"], case["kl_beta"], agg)
    dH, dW = spo.spo_policy_loss_bwd(H, W, tgt, lse, g, case["inv_temp"])
    torch.cuda.synchronize()
    assert spo.spo_device_error() == 0
    cpu = lambda t: t.detach().cpu().numpy() if t is not None else None
    return dict(loss_mask=cpu(loss_mask), n_tok=cpu(n_tok), logp=cpu(logp), entropy=cpu(ent),
                lse=cpu(lse), adv=cpu(adv), loss=float(loss.item()), g=cpu(g),
                stats=cpu(stats), dH=cpu(dH.float()), dW=cpu(dW))
