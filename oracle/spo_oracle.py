"""fp64 CPU oracle for the GRPO log-prob / policy-loss path of CUDAPerf
(arxiv 2607.20908, §3 "Multi-turn RL Training", Eq. 3).

THIS IS TEST INFRASTRUCTURE.  Only ``tests/``, ``__graft_entry__.smoke()`` and
``bench.py``'s CPU-baseline / reference legs may import it.  The product
package (``paper_2607_20908_gb300``) never imports it, and it shares no code,
constants or helpers with the CUDA path; the two meet only at the seeded
inputs of ``paper_2607_20908_gb300.inputs`` (which hold no arithmetic of the
method).

Everything here is the plain definition of what the path computes, in fp64,
written for a reader to check against the paper by eye.  A BLAS matmul is the
only library primitive used (for the logits z = H W^T and the two backward
products).  No blocking, fusion or reordering beyond the definitions.

Notation (the paper's, plus the LM head): a rollout token t of output o_i has
hidden state H[t] (bf16, widened exactly) and next-token id y_t; the policy's
logits are z_t = tau^-1 * H[t] W^T over the full vocabulary V; pi_theta(y_t) is
softmax(z_t)[y_t].  The group-normalised advantage, the clipped surrogate and
the KL term follow Eq. 3 and the sentence under it.

Readings where the paper is silent (each is also listed in the design notes):
  * std in A_hat: unbiased (n-1) by default; population std on request.
  * eps added to std (default 1e-6); groups of size <= 1 or with all rewards
    equal get A_hat = 0 exactly.
  * KL estimator: per-token k3, exp(ref - logp) - (ref - logp) - 1, averaged
    like the surrogate.  beta = 0 (the paper's setting) removes it.
  * aggregation: SEQ_GROUP (Eq. 3: mean over groups of mean over the group's
    outputs of the per-output token mean) or TOKEN (batch token mean).
  * |o_i| = number of loss tokens of output i (mask and window applied);
    outputs with no loss token still count in their group's size.
  * window: the first `window` loss tokens of each sequence (window <= 0: none).
  * the clip bound is inclusive: at rho == 1 +- eps the unclipped branch is
    taken, so the gradient there is rho * A_hat.
  * targets < 0 are ignored tokens (no log-prob, no loss).
"""

from __future__ import annotations

import math

import numpy as np

AGG_SEQ_GROUP = 0
AGG_TOKEN = 1
STD_UNBIASED = 0
STD_POPULATION = 1


# --------------------------------------------------------------------------
# bf16 inputs
# --------------------------------------------------------------------------
def bf16_bits_to_f64(bits) -> np.ndarray:
    """Widen bf16 bit patterns (uint16) to float64 exactly (bf16 is the top
    half of an IEEE binary32)."""
    b = np.ascontiguousarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


# --------------------------------------------------------------------------
# a1: loss-token selection (§3 "Multi-turn RL Training": only unmasked tokens
#     within a 1024-token window of each generation enter the loss)
# --------------------------------------------------------------------------
def token_select(cu_seqlens, mask, tgt, window: int):
    """Loss tokens of every sequence.

    Token t of sequence i (t in [cu[i], cu[i+1])) is a loss token when
    mask[t] == 1, tgt[t] >= 0 and fewer than ``window`` earlier tokens of the
    same sequence were loss tokens (window <= 0: no cap).

    Returns (loss_mask uint8[T], n_tok int64[n_seq]).
    """
    cu = np.asarray(cu_seqlens).astype(np.int64)
    n_seq = cu.size - 1
    eligible = (np.asarray(mask).astype(np.int64) == 1) & (np.asarray(tgt).astype(np.int64) >= 0)
    seq = np.repeat(np.arange(n_seq), np.diff(cu))             # the sequence of every token
    upto = np.cumsum(eligible)                                  # eligible tokens in [0, t]
    at_start = np.concatenate([[0], upto])[cu[:-1]]             # eligible tokens before each sequence
    earlier = upto - eligible - at_start[seq]                   # earlier eligible tokens of t's sequence
    keep = eligible & ((window <= 0) | (earlier < window))
    loss_mask = keep.astype(np.uint8)
    n_tok = np.bincount(seq, weights=keep, minlength=n_seq).astype(np.int64)
    return loss_mask, n_tok


# --------------------------------------------------------------------------
# a2 + a3: per-token policy log-probability and entropy over the full vocab
#          (pi_theta in the ratio of Eq. 3)
# --------------------------------------------------------------------------
def logits(H, W, inv_temp: float = 1.0) -> np.ndarray:
    """z = tau^-1 * H W^T in fp64 (H: [n, d], W: [V, d], both fp64)."""
    return float(inv_temp) * (np.asarray(H, dtype=np.float64) @ np.asarray(W, dtype=np.float64).T)


def logprobs(H, W, tgt, inv_temp: float = 1.0, mask=None):
    """log pi_theta(y_t) = z_t[y_t] - logsumexp_v z_t[v]; entropy of softmax(z_t).

    H, W: fp64 arrays (use bf16_bits_to_f64 on the bf16 bit patterns).
    Tokens with mask == 0 or tgt < 0 are skipped: logp = entropy = lse = 0.
    Returns (logp, entropy, lse) as fp64 arrays of length T.
    """
    T = H.shape[0]
    tgt = np.asarray(tgt).astype(np.int64)
    keep = tgt >= 0
    if mask is not None:
        keep &= np.asarray(mask).astype(np.int64) == 1
    rows = np.nonzero(keep)[0]
    logp = np.zeros(T)
    ent = np.zeros(T)
    lse = np.zeros(T)
    if rows.size == 0:
        return logp, ent, lse
    z = logits(H[rows], W, inv_temp)                       # [n, V]
    m = z.max(axis=1)
    s = np.exp(z - m[:, None]).sum(axis=1)
    lse_r = m + np.log(s)                                  # logsumexp_v z
    p = np.exp(z - lse_r[:, None])                         # softmax(z)
    logp[rows] = z[np.arange(rows.size), tgt[rows]] - lse_r
    ent[rows] = lse_r - (p * z).sum(axis=1)                # -sum p log p
    lse[rows] = lse_r
    return logp, ent, lse


# --------------------------------------------------------------------------
# a2/a3 with the vocabulary split into slices (LM-head rows per device)
# --------------------------------------------------------------------------
def logprobs_slice_record(H, W_slice, v_offset: int, tgt, inv_temp: float = 1.0, mask=None):
    """What one vocabulary slice [v_offset, v_offset + V_slice) knows of each token:
    (max_v z, sum_v exp(z - max), sum_v exp(z - max) z, z[y] if y is in the slice
    else -inf), z over the slice's logits only.  Skipped tokens: (0, 0, 0, 0).
    Returns fp64 [T, 4]."""
    T = H.shape[0]
    tgt = np.asarray(tgt).astype(np.int64)
    keep = tgt >= 0
    if mask is not None:
        keep &= np.asarray(mask).astype(np.int64) == 1
    rows = np.nonzero(keep)[0]
    rec = np.zeros((T, 4))
    if rows.size == 0:
        return rec
    z = logits(H[rows], W_slice, inv_temp)                 # [n, V_slice]
    m = z.max(axis=1)
    w = np.exp(z - m[:, None])
    rec[rows, 0] = m
    rec[rows, 1] = w.sum(axis=1)
    rec[rows, 2] = (w * z).sum(axis=1)
    local = tgt[rows] - v_offset
    hit = (local >= 0) & (local < W_slice.shape[0])
    zt = np.full(rows.size, -np.inf)
    zt[hit] = z[np.nonzero(hit)[0], local[hit]]
    rec[rows, 3] = zt
    return rec


def merge_slice_records(recs):
    """(logp, entropy, lse) from the records of slices that together cover the
    vocabulary once: with M = max_k m_k and S = sum_k s_k exp(m_k - M),
    lse = M + log S; sum_v p_v z_v = (sum_k e_k exp(m_k - M)) / S; the target
    logit is the one finite z[y].  Tokens whose records are all empty get 0."""
    recs = np.asarray(recs, dtype=np.float64)              # [R, T, 4]
    T = recs.shape[1]
    logp, ent, lse = np.zeros(T), np.zeros(T), np.zeros(T)
    live = recs[:, :, 1] > 0
    for t in range(T):
        k = np.nonzero(live[:, t])[0]
        if k.size == 0:
            continue
        m, s, e, zt = recs[k, t, 0], recs[k, t, 1], recs[k, t, 2], recs[k, t, 3]
        M = m.max()
        S = (s * np.exp(m - M)).sum()
        E = (e * np.exp(m - M)).sum()
        lse[t] = M + math.log(S)
        logp[t] = zt.max() - lse[t]
        ent[t] = lse[t] - E / S
    return logp, ent, lse


# --------------------------------------------------------------------------
# a4: group-normalised advantage (the definition of A_hat under Eq. 3)
# --------------------------------------------------------------------------
def group_advantages(rewards, group_id, n_groups: int, std_mode: int = STD_UNBIASED,
                     eps: float = 1e-6) -> np.ndarray:
    """A_hat_i = (r_i - mean(r_g)) / (std(r_g) + eps) over the members of i's group.

    fp64.  Groups of size <= 1, or whose rewards are all equal, give 0.
    """
    r = np.asarray(rewards, dtype=np.float64)
    gid = np.asarray(group_id).astype(np.int64)
    adv = np.zeros(r.size)
    for g in range(n_groups):
        idx = np.nonzero(gid == g)[0]
        n = idx.size
        if n <= 1:
            continue
        rg = r[idx]
        if rg.max() == rg.min():
            continue
        mu = rg.sum() / n
        dof = (n - 1) if std_mode == STD_UNBIASED else n
        sigma = math.sqrt(((rg - mu) ** 2).sum() / dof)
        adv[idx] = (rg - mu) / (sigma + eps)
    return adv


def group_advantages_f32(rewards, group_id, n_groups: int, std_mode: int = STD_UNBIASED,
                         eps: float = 1e-6) -> np.ndarray:
    """The same definition evaluated in IEEE binary32 in one fixed order.

    Each step is a single correctly rounded float32 operation, in this order:
      sum = ((r_0 + r_1) + r_2) + ...          (members in ascending index)
      mu  = sum / n
      ss  = ((d_0*d_0 + d_1*d_1) + ...) with d_j = r_j - mu, each product
            rounded before the add (no fused multiply-add)
      var = ss / (n - 1)   (or / n)
      sig = sqrt(var); den = sig + eps; A_hat_j = d_j / den
    Used to check a device kernel that promises this order bit for bit.
    """
    f = np.float32
    r = np.asarray(rewards, dtype=np.float32)
    gid = np.asarray(group_id).astype(np.int64)
    adv = np.zeros(r.size, dtype=np.float32)
    for g in range(n_groups):
        idx = [int(i) for i in np.nonzero(gid == g)[0]]
        n = len(idx)
        if n <= 1:
            continue
        lo = min(r[i] for i in idx)
        hi = max(r[i] for i in idx)
        if lo == hi:
            continue
        acc = f(0.0)
        for i in idx:
            acc = f(acc + r[i])
        mu = f(acc / f(n))
        ss = f(0.0)
        for i in idx:
            dv = f(r[i] - mu)
            ss = f(ss + f(dv * dv))
        var = f(ss / f(n - 1 if std_mode == STD_UNBIASED else n))
        den = f(f(np.sqrt(var)) + f(eps))
        for i in idx:
            adv[i] = f(f(r[i] - mu) / den)
    return adv


# --------------------------------------------------------------------------
# a5: ratio, clipped surrogate, KL, aggregation (Eq. 3) and dL/dlogp
# --------------------------------------------------------------------------
def _token_weights(cu_seqlens, group_id, n_groups, loss_mask, agg):
    """c_t such that L = sum_t c_t * l_t (Eq. 3's averaging)."""
    cu = np.asarray(cu_seqlens).astype(np.int64)
    n_seq = cu.size - 1
    gid = np.asarray(group_id).astype(np.int64)
    lm = np.asarray(loss_mask).astype(np.int64)
    T = int(cu[-1])
    n_tok = np.array([lm[cu[i]:cu[i + 1]].sum() for i in range(n_seq)], dtype=np.int64)
    c = np.zeros(T)
    if agg == AGG_TOKEN:
        total = n_tok.sum()
        if total > 0:
            c[lm == 1] = 1.0 / total
        return c, n_tok
    size = np.bincount(gid, minlength=n_groups)
    n_nonempty = int((size > 0).sum())
    for i in range(n_seq):
        if n_tok[i] == 0:
            continue
        w = 1.0 / (n_nonempty * size[gid[i]] * n_tok[i])
        seg = slice(cu[i], cu[i + 1])
        c[seg] = np.where(lm[seg] == 1, w, 0.0)
    return c, n_tok


def policy_loss(logp, old_logp, ref_logp, adv_seq, cu_seqlens, group_id, n_groups: int,
                loss_mask, clip_eps: float, kl_beta: float, agg: int = AGG_SEQ_GROUP):
    """Loss to minimise, L = -J_GRPO (Eq. 3), and g_t = dL/dlogp_t.

    Per loss token t of output i:
      rho  = exp(logp - old_logp)                 (pi_theta / pi_theta_old)
      surr = min(rho * A_i, clip(rho, 1-eps, 1+eps) * A_i)
      kl   = exp(ref - logp) - (ref - logp) - 1   (k3 estimate of D_KL(pi_theta || pi_ref))
      l_t  = -(surr - beta * kl)
    L = sum_t c_t l_t with c_t from the aggregation mode.
    g_t = c_t * (-A_i * rho * [unclipped branch taken] + beta * (1 - exp(ref - logp))).
    Returns (loss, g fp64[T], stats dict).
    """
    lp = np.asarray(logp, dtype=np.float64)
    old = np.asarray(old_logp, dtype=np.float64)
    cu = np.asarray(cu_seqlens).astype(np.int64)
    T = int(cu[-1])
    lm = np.asarray(loss_mask).astype(np.int64)
    use_kl = ref_logp is not None and kl_beta != 0.0
    ref = np.asarray(ref_logp, dtype=np.float64) if use_kl else None
    A = np.zeros(T)
    for i in range(cu.size - 1):
        A[cu[i]:cu[i + 1]] = float(adv_seq[i])
    c, n_tok = _token_weights(cu, group_id, n_groups, lm, agg)
    act = lm == 1
    rho = np.where(act, np.exp(lp - old), 0.0)
    clipped = np.clip(rho, 1.0 - clip_eps, 1.0 + clip_eps)
    surr = np.minimum(rho * A, clipped * A)
    # the clip binds (zero gradient through the ratio) when A>0, rho>1+eps or A<0, rho<1-eps
    binds = ((A > 0) & (rho > 1.0 + clip_eps)) | ((A < 0) & (rho < 1.0 - clip_eps))
    if use_kl:
        delta = np.where(act, ref - lp, 0.0)
        kl = np.exp(delta) - delta - 1.0
        dkl = 1.0 - np.exp(delta)                      # d kl / d logp
    else:
        kl = np.zeros(T)
        dkl = np.zeros(T)
    beta = kl_beta if use_kl else 0.0
    ell = np.where(act, -(surr - beta * kl), 0.0)
    loss = float((c * ell).sum())
    g = np.where(act, c * (-A * rho * (~binds) + beta * dkl), 0.0)
    n_loss = int(act.sum())
    stats = dict(
        clip_frac=float(binds[act].mean()) if n_loss else 0.0,
        mean_ratio=float(rho[act].mean()) if n_loss else 0.0,
        mean_kl=float(kl[act].mean()) if n_loss else 0.0,
        n_loss_tokens=n_loss,
    )
    return loss, g, stats


# --------------------------------------------------------------------------
# a6 - a8: backward to H and W (the policy update implied by maximising Eq. 3)
# --------------------------------------------------------------------------
def policy_loss_bwd(H, W, tgt, g, inv_temp: float = 1.0):
    """dH = G W, dW = G^T H with G[t, v] = tau^-1 * g_t * (1[v == y_t] - softmax(z_t)[v]).

    H, W fp64; g = dL/dlogp (fp64).  Rows with g_t == 0 contribute nothing.
    Returns (dH [T, d], dW [V, d]) in fp64.
    """
    T, d = H.shape
    V = W.shape[0]
    tgt = np.asarray(tgt).astype(np.int64)
    g = np.asarray(g, dtype=np.float64)
    rows = np.nonzero(g != 0.0)[0]
    dH = np.zeros((T, d))
    dW = np.zeros((V, d))
    if rows.size == 0:
        return dH, dW
    z = logits(H[rows], W, inv_temp)
    m = z.max(axis=1)
    lse = m + np.log(np.exp(z - m[:, None]).sum(axis=1))
    p = np.exp(z - lse[:, None])
    onehot = np.zeros_like(p)
    onehot[np.arange(rows.size), tgt[rows]] = 1.0
    G = inv_temp * g[rows][:, None] * (onehot - p)
    dH[rows] = G @ W
    dW = G.T @ H[rows]
    return dH, dW


def policy_loss_bwd_slice(H, W_slice, v_offset: int, tgt, lse, g, inv_temp: float = 1.0):
    """One vocabulary slice's share of the backward: G restricted to columns
    [v_offset, v_offset + V_slice), G[t, j] = tau^-1 g_t (1[v_offset + j == y_t]
    - exp(z_t[v_offset + j] - lse_t)) with the full-vocabulary lse.  Returns
    (dH part = G W_slice [T, d], dW rows of the slice = G^T H [V_slice, d]);
    the parts of all slices sum to policy_loss_bwd's dH."""
    T, d = H.shape
    Vs = W_slice.shape[0]
    tgt = np.asarray(tgt).astype(np.int64)
    g = np.asarray(g, dtype=np.float64)
    lse = np.asarray(lse, dtype=np.float64)
    rows = np.nonzero(g != 0.0)[0]
    dH = np.zeros((T, d))
    dW = np.zeros((Vs, d))
    if rows.size == 0:
        return dH, dW
    z = logits(H[rows], W_slice, inv_temp)
    p = np.exp(z - lse[rows][:, None])
    onehot = np.zeros_like(p)
    local = tgt[rows] - v_offset
    hit = np.nonzero((local >= 0) & (local < Vs))[0]
    onehot[hit, local[hit]] = 1.0
    G = inv_temp * g[rows][:, None] * (onehot - p)
    dH[rows] = G @ W_slice
    dW = G.T @ H[rows]
    return dH, dW


# --------------------------------------------------------------------------
# reward composition (§2.2 "Verifiable Reward"; r_i = R_ver(i) + R_str(i), §3)
# --------------------------------------------------------------------------
PAPER_REWARD = dict(alpha_comp=3.0, alpha_wrong=2.0, alpha_speed=1.0, alpha_cv=0.5,
                    s_min=-0.5, s_max=4.0)


def reward_compose(compiled, pass_rate, speedup, cv, r_struct=None, params=None):
    """Composite reward of each candidate program.

    R_comp  = -alpha_comp                         (the program does not compile)
    R_corr  = -alpha_wrong * (1 - p)              (p = fraction of tests passed)
    R_speed = alpha_speed * clip(log2 S, s_min, s_max)   (S = speedup)
    R_cv    = -alpha_cv * cv                       (coefficient of variation)
    R_ver   = R_comp if not compiled; R_corr if p < 1; R_corr + R_speed + R_cv if p == 1
    r       = R_ver + R_str
    A speedup that is not > 0 counts as the lower clip bound.  fp64.
    """
    q = dict(PAPER_REWARD if params is None else params)
    comp = np.asarray(compiled).astype(np.int64)
    p = np.asarray(pass_rate, dtype=np.float64)
    S = np.asarray(speedup, dtype=np.float64)
    c = np.asarray(cv, dtype=np.float64)
    out = np.zeros(p.size)
    for i in range(p.size):
        if comp[i] == 0:
            r = -q["alpha_comp"]
        else:
            r = -q["alpha_wrong"] * (1.0 - p[i])
            if p[i] >= 1.0:
                ls = math.log2(S[i]) if S[i] > 0 else -math.inf
                r += q["alpha_speed"] * min(max(ls, q["s_min"]), q["s_max"])
                r += -q["alpha_cv"] * c[i]
        out[i] = r
    if r_struct is not None:
        out = out + np.asarray(r_struct, dtype=np.float64)
    return out


# --------------------------------------------------------------------------
# offline structural ranker (§2.1 "Structural Reward", appendix "MLP Ranker
# Architecture"): s_psi(phi_hat) with an 11 -> 64 -> 32 -> 1 ReLU MLP and the
# pairwise logistic ranking loss E[softplus(-(s(y+) - s(y-)))]
# --------------------------------------------------------------------------
RANKER_SHAPES = (("W1", (64, 11)), ("b1", (64,)), ("W2", (32, 64)), ("b2", (32,)),
                 ("w3", (32,)), ("b3", (1,)))
RANKER_NPARAMS = sum(int(np.prod(sh)) for _, sh in RANKER_SHAPES)   # 2881


def ranker_unpack(flat):
    """Packed parameter vector -> dict of arrays (row-major, in RANKER_SHAPES order)."""
    flat = np.asarray(flat, dtype=np.float64)
    out, off = {}, 0
    for name, sh in RANKER_SHAPES:
        n = int(np.prod(sh))
        out[name] = flat[off:off + n].reshape(sh)
        off += n
    return out


def ranker_scores(phi, mu, sigma, flat, keep1=None, keep2=None, drop_p=0.0):
    """s_psi(phi_hat) for each row of phi [n, 11]; phi_hat = (phi - mu) / sigma.

    keep1 [n, 64] / keep2 [n, 32]: optional dropout keep flags (0/1) of the two
    hidden layers; kept units are scaled by 1 / (1 - drop_p).
    Returns (scores [n], cache for the backward).
    """
    P = ranker_unpack(flat)
    x = (np.asarray(phi, dtype=np.float64) - np.asarray(mu, dtype=np.float64)) / np.asarray(
        sigma, dtype=np.float64)
    a1 = x @ P["W1"].T + P["b1"]
    h1 = np.maximum(a1, 0.0)
    if keep1 is not None:
        h1 = h1 * np.asarray(keep1, dtype=np.float64) / (1.0 - drop_p)
    a2 = h1 @ P["W2"].T + P["b2"]
    h2 = np.maximum(a2, 0.0)
    if keep2 is not None:
        h2 = h2 * np.asarray(keep2, dtype=np.float64) / (1.0 - drop_p)
    s = h2 @ P["w3"] + P["b3"][0]
    return s, dict(x=x, a1=a1, h1=h1, a2=a2, h2=h2, P=P, keep1=keep1, keep2=keep2, p=drop_p)


def _ranker_backward(c, ds):
    """Gradient of sum_i ds_i * s_i w.r.t. the packed parameters."""
    P = c["P"]
    g = {"w3": c["h2"].T @ ds, "b3": np.array([ds.sum()])}
    dh2 = np.outer(ds, P["w3"])
    if c["keep2"] is not None:
        dh2 = dh2 * np.asarray(c["keep2"], dtype=np.float64) / (1.0 - c["p"])
    da2 = dh2 * (c["a2"] > 0)
    g["W2"] = da2.T @ c["h1"]
    g["b2"] = da2.sum(axis=0)
    dh1 = da2 @ P["W2"]
    if c["keep1"] is not None:
        dh1 = dh1 * np.asarray(c["keep1"], dtype=np.float64) / (1.0 - c["p"])
    da1 = dh1 * (c["a1"] > 0)
    g["W1"] = da1.T @ c["x"]
    g["b1"] = da1.sum(axis=0)
    return np.concatenate([g[name].reshape(-1) for name, _ in RANKER_SHAPES])


def ranker_pair_loss(phi, mu, sigma, flat, pos, neg, keep1=None, keep2=None, drop_p=0.0):
    """L = mean_k softplus(-(s(phi[pos_k]) - s(phi[neg_k]))) and dL/dparams.

    keep1 / keep2 (optional): dropout keep flags per pair member, shaped
    [P, 2, 64] / [P, 2, 32] (index 0 = the y+ member, 1 = the y- member).
    """
    pos = np.asarray(pos).astype(np.int64)
    neg = np.asarray(neg).astype(np.int64)
    Pn = pos.size
    rows = np.concatenate([pos, neg])
    k1 = None if keep1 is None else np.concatenate([np.asarray(keep1)[:, 0], np.asarray(keep1)[:, 1]])
    k2 = None if keep2 is None else np.concatenate([np.asarray(keep2)[:, 0], np.asarray(keep2)[:, 1]])
    s, c = ranker_scores(np.asarray(phi)[rows], mu, sigma, flat, k1, k2, drop_p)
    delta = s[:Pn] - s[Pn:]
    loss = float(np.mean(np.logaddexp(0.0, -delta)))        # softplus(-delta)
    dd = -1.0 / (1.0 + np.exp(delta)) / Pn                   # dL/d delta
    grad = _ranker_backward(c, np.concatenate([dd, -dd]))
    return loss, grad


# --------------------------------------------------------------------------
# the whole step (used for the CPU baseline timing)
# --------------------------------------------------------------------------
def grpo_step(H, W, tgt, mask, cu_seqlens, group_id, n_groups, rewards, old_logp, ref_logp,
              clip_eps, kl_beta, inv_temp=1.0, window=1024, agg=AGG_SEQ_GROUP,
              std_mode=STD_UNBIASED, eps=1e-6):
    """a1 -> a8 in order; returns a dict with every intermediate."""
    loss_mask, n_tok = token_select(cu_seqlens, mask, tgt, window)
    logp, ent, lse = logprobs(H, W, tgt, inv_temp, loss_mask)
    adv = group_advantages(rewards, group_id, n_groups, std_mode, eps)
    loss, g, stats = policy_loss(logp, old_logp, ref_logp, adv, cu_seqlens, group_id, n_groups,
                                 loss_mask, clip_eps, kl_beta, agg)
    dH, dW = policy_loss_bwd(H, W, tgt, g, inv_temp)
    return dict(loss_mask=loss_mask, n_tok=n_tok, logp=logp, entropy=ent, lse=lse, adv=adv,
                loss=loss, g=g, stats=stats, dH=dH, dW=dW)
