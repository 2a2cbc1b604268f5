"""Multi-GPU forms of the GRPO step.

Data-parallel (``DataParallelStep``): whole groups per rank.

Groups (the g candidates of one task and all their turns, section 3) are
independent for the advantages and for every per-token term of Eq. 3, so a
batch shards over ranks by whole groups with no exchange inside the step.
Two things cross ranks:

  * the normaliser of Eq. 3's average.  With SEQ_GROUP aggregation the loss
    is a mean over non-empty groups, so rank r's local loss (a mean over its
    own N_r groups) enters the global loss with weight N_r / N; with TOKEN
    aggregation the weight is the rank's share of loss tokens.  One
    all-reduce of two counts per step gives N (and the token total).
  * dW = sum over ranks of the weighted local dW (an all-reduce of V x d
    fp32).  dH rows stay on the rank that owns the tokens.

Vocabulary-parallel (``VocabParallelStep``): the LM head's V rows split into
contiguous slices, one per rank, the batch replicated.  The softmax
normaliser couples all V logits of a token, so each rank's forward ends in a
16-byte record per token (max, sum-exp, sum-exp*z, target logit of its slice);
one all-gather of T x 16 bytes lets every rank merge the records into the
full-vocabulary logp / entropy / lse, and the loss is then computed
redundantly on every rank.  In the backward each rank forms G for its own
columns: dW stays sharded with W, and dH = sum over ranks of G_k W_k (one
all-reduce of T x d fp32).

The per-rank compute is an engine object (``SpoEngine`` and
``SpoVocabEngine`` run libspo's CUDA kernels); the collectives are
``torch.distributed`` on whatever backend the process group uses (NCCL
between GPUs).
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np
import torch

AGG_SEQ_GROUP = 0
AGG_TOKEN = 1


def shard_groups(tokens_per_group, world: int):
    """Assign every group to one rank, balancing loss tokens (greedy, largest
    first, ties to the lowest rank; deterministic).  Returns sorted group ids
    per rank."""
    if world < 1:
        raise ValueError("world must be >= 1")
    tokens = [int(t) for t in tokens_per_group]
    order = sorted(range(len(tokens)), key=lambda g: (-tokens[g], g))
    loads = [0] * world
    out = [[] for _ in range(world)]
    for g in order:
        r = min(range(world), key=lambda k: (loads[k], k))
        out[r].append(g)
        loads[r] += tokens[g]
    return [sorted(x) for x in out]


@dataclass
class RankBatch:
    seq_index: np.ndarray     # global sequence ids owned by the rank, ascending
    token_index: np.ndarray   # global token ids of those sequences, in order
    cu_seqlens: np.ndarray    # local int32 [n_seq + 1]
    group_id: np.ndarray      # local int32 [n_seq], remapped to 0..n_groups-1
    n_groups: int             # groups owned (each has >= 1 sequence)


def rank_batch(cu_seqlens, group_id, groups) -> RankBatch:
    """The sequences and tokens of the given groups, in their global order."""
    cu = np.asarray(cu_seqlens).astype(np.int64)
    gid = np.asarray(group_id).astype(np.int64)
    remap = {int(g): k for k, g in enumerate(sorted(int(x) for x in groups))}
    seqs = np.array([i for i in range(gid.size) if int(gid[i]) in remap], dtype=np.int64)
    lens = np.array([cu[i + 1] - cu[i] for i in seqs], dtype=np.int64)
    tok = (np.concatenate([np.arange(cu[i], cu[i + 1]) for i in seqs]) if seqs.size
           else np.zeros(0, dtype=np.int64))
    local_cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    local_gid = np.array([remap[int(gid[i])] for i in seqs], dtype=np.int32)
    return RankBatch(seqs, tok, local_cu, local_gid, len(remap))


def dw_block_starts(V: int, n_blocks: int):
    """Row boundaries of dW's vocabulary blocks (libspo's layout: multiples of
    256, the last block ends at V).  Every rank uses the same layout, so the
    per-block collectives match across ranks.  A host computation."""
    from paper_2607_20908_gb300 import spo
    return spo.dw_block_starts(V, n_blocks)


def loss_weight(agg: int, local_groups: float, global_groups: float, local_tokens: float,
                global_tokens: float) -> float:
    """Weight of a rank's local loss (and dL/dlogp) in the global objective."""
    if agg == AGG_SEQ_GROUP:
        return local_groups / global_groups if global_groups > 0 else 0.0
    return local_tokens / global_tokens if global_tokens > 0 else 0.0


class SpoEngine:
    """libspo (CUDA) as the per-rank compute of a data-parallel step."""

    def __init__(self, reserve_sms: int = 0):
        from paper_2607_20908_gb300 import spo
        self.spo = spo
        self.reserve_sms = reserve_sms
        self._side = {}

    def step_local(self, b: dict, agg: int):
        s = self.spo
        lm, _ = s.spo_token_select(b["cu_seqlens"], b["mask"], b["tgt"], b["window"])
        logp, _, lse = s.spo_logprobs_fwd(b["H"], b["W"], b["tgt"], lm, b["inv_temp"])
        adv = s.spo_group_advantages(b["rewards"], b["group_id"], b["n_groups"])
        loss, g, stats = s.spo_policy_loss_fwd(logp, b["old"], b["ref"], adv, b["cu_seqlens"],
                                               b["group_id"], b["n_groups"], lm, b["clip_eps"],
                                               b["kl_beta"], agg)
        return dict(loss=loss, g=g, lse=lse, n_loss_tokens=stats[3:4].to(torch.float64))

    def local_counts(self, b: dict, loc):
        """[groups owned, loss tokens] as a device fp64 tensor (no host read)."""
        groups = torch.full((1,), float(b["n_groups"]), dtype=torch.float64,
                            device=loc["n_loss_tokens"].device)
        return torch.cat([groups, loc["n_loss_tokens"].reshape(1)])

    def zero_counts(self, b: dict):
        return torch.zeros(2, dtype=torch.float64, device=b["W"].device)

    def scale_ratio(self, x, num, den):
        self.spo.spo_scale_f32_ratio(x, num, den)
        return x

    def backward_blocks(self, b: dict, lse, g, n_blocks: int):
        """dH, dW and dW's vocabulary blocks [(first row, end row, event when final)]."""
        s = self.spo
        evs = [torch.cuda.Event() for _ in range(n_blocks)]
        hooks = s.make_hooks(n_blocks, evs, None, reserve_sms=self.reserve_sms)
        dH, dW = s.spo_policy_loss_bwd_ex(b["H"], b["W"], b["tgt"], lse, g, b["inv_temp"],
                                          hooks=hooks)
        starts = dw_block_starts(b["W"].shape[0], n_blocks)
        return dH, dW, [(starts[k], starts[k + 1], evs[k]) for k in range(n_blocks)]

    def step_fused(self, b: dict, weight: float, n_blocks: int):
        """The whole local step in one call (spo_grpo_step) with the loss and g
        scaled by `weight` on the device: (loss, dH, dW, dW blocks)."""
        s = self.spo
        dev = b["W"].device
        scale = torch.full((1,), float(weight), dtype=torch.float32, device=dev)
        evs = [torch.cuda.Event() for _ in range(n_blocks)]
        hooks = s.make_hooks(n_blocks, evs, None, reserve_sms=self.reserve_sms)
        out = s.spo_grpo_step(b["H"], b["W"], b["tgt"], b["mask"], b["cu_seqlens"],
                              b["group_id"], b["n_groups"], b["rewards"], b["old"], b["ref"],
                              inv_temp=b["inv_temp"], window=b["window"], clip_eps=b["clip_eps"],
                              kl_beta=b["kl_beta"], agg=AGG_SEQ_GROUP, loss_scale=scale, want=(),
                              hooks=hooks, dH=b.get("dH_out"), dW=b.get("dW_out"))
        starts = dw_block_starts(b["W"].shape[0], n_blocks)
        return (out["loss"], out["dH"], out["dW"],
                [(starts[k], starts[k + 1], evs[k]) for k in range(n_blocks)])

    def zeros_dW(self, V: int, d: int, like):
        return torch.zeros((V, d), dtype=torch.float32, device=like.device)

    def comm_stream(self, t):
        """Side stream on t's device for the collectives that overlap the GEMMs."""
        dev = t.device
        if dev not in self._side:
            self._side[dev] = torch.cuda.Stream(dev)
        return self._side[dev]


def _overlapped_all_reduce(t, ready, side, group):
    """Sum-all-reduce of t issued once `ready` (a CUDA event, or None: now)
    has fired, from the side stream when there is one, so that it runs while
    the launching stream goes on.  Returns the async work handle."""
    import torch.distributed as dist
    if side is None:
        return dist.all_reduce(t, group=group, async_op=True)
    if ready is not None:
        side.wait_event(ready)
    else:
        side.wait_stream(torch.cuda.current_stream(t.device))
    with torch.cuda.stream(side):
        return dist.all_reduce(t, group=group, async_op=True)


class DataParallelStep:
    """One GRPO step over a process group, whole groups per rank.

    run(b) takes this rank's batch (dict with H, W, tgt, mask, cu_seqlens,
    group_id, n_groups, rewards, old, ref, window, inv_temp, clip_eps,
    kl_beta; n_groups may be 0) and returns (global loss, local dH, global dW).
    Collectives: one all-reduce of [groups, loss tokens] whose result is used
    on the device (the rank's weight is applied by a kernel: the host never
    reads a count), one of the loss, and one per vocabulary block of dW, each
    started as soon as the backward has finished that block, so it runs
    while the GEMMs of the later blocks do.
    """

    def __init__(self, engine, agg: int = AGG_SEQ_GROUP, process_group=None, dw_blocks: int = 4):
        self.engine = engine
        self.agg = agg
        self.pg = process_group
        self.dw_blocks = dw_blocks

    def run(self, b: dict):
        import torch.distributed as dist
        e = self.engine
        V, d = b["W"].shape
        if b["n_groups"] > 0:
            loc = e.step_local(b, self.agg)
            local = e.local_counts(b, loc)
        else:
            loc = None
            local = e.zero_counts(b)
        total = local.clone()
        dist.all_reduce(total, group=self.pg)
        k = 0 if self.agg == AGG_SEQ_GROUP else 1
        if loc is not None:
            # weight of this rank's local average in the global one (Eq. 3)
            e.scale_ratio(loc["g"], local[k:k + 1], total[k:k + 1])
            e.scale_ratio(loc["loss"], local[k:k + 1], total[k:k + 1])
            dH, dW, blocks = e.backward_blocks(b, loc["lse"], loc["g"], self.dw_blocks)
            loss = loc["loss"]
        else:
            dH = None
            dW = e.zeros_dW(V, d, b["W"])
            loss = torch.zeros(1, dtype=dW.dtype, device=dW.device)
            starts = dw_block_starts(V, self.dw_blocks)
            blocks = [(starts[k], starts[k + 1], None) for k in range(self.dw_blocks)]
        return self._exchange(loss, dH, dW, blocks)

    def run_fused(self, b: dict, global_groups: int):
        """The same step for SEQ_GROUP aggregation when every rank knows the
        global number of non-empty groups on the host (each rank owns whole,
        non-empty groups of a sharding plan all ranks share): the rank's
        weight N_r / N is then known before the step, so the local step runs
        as one call (spo_grpo_step) with that weight applied on the device,
        and no count is exchanged.  Collectives: dW per vocabulary block as
        in run(), and the loss."""
        if self.agg != AGG_SEQ_GROUP:
            raise ValueError("run_fused needs SEQ_GROUP aggregation (TOKEN weights need the "
                             "all-reduced token count)")
        e = self.engine
        V, d = b["W"].shape
        starts = dw_block_starts(V, self.dw_blocks)
        if b["n_groups"] > 0:
            weight = b["n_groups"] / global_groups if global_groups > 0 else 0.0
            loss, dH, dW, blocks = e.step_fused(b, weight, self.dw_blocks)
        else:
            dH = None
            dW = e.zeros_dW(V, d, b["W"])
            loss = torch.zeros(1, dtype=dW.dtype, device=dW.device)
            blocks = [(starts[k], starts[k + 1], None) for k in range(self.dw_blocks)]
        return self._exchange(loss, dH, dW, blocks)

    def _exchange(self, loss, dH, dW, blocks):
        import torch.distributed as dist
        side = self.engine.comm_stream(dW)
        works = [_overlapped_all_reduce(dW[r0:r1], ready, side, self.pg)
                 for r0, r1, ready in blocks if r1 > r0]
        dist.all_reduce(loss, group=self.pg)
        for w in works:
            w.wait()          # the launching stream waits for the block sums
        return loss, dH, dW


def vocab_slices(V: int, world: int, align: int = 8):
    """Contiguous [offset, offset + size) slices of V rows, one per rank, sizes
    multiples of `align` (the tensor-map rule for W's rows) and as even as
    that allows; the first slices take the remainder."""
    if world < 1:
        raise ValueError("world must be >= 1")
    if V % align != 0:
        raise ValueError(f"V = {V} is not a multiple of {align}")
    units = V // align
    if units < world:
        raise ValueError(f"V = {V} has fewer than {world} blocks of {align} rows")
    base, extra = divmod(units, world)
    out, off = [], 0
    for r in range(world):
        n = (base + (1 if r < extra else 0)) * align
        out.append((off, n))
        off += n
    return out


class SpoVocabEngine:
    """libspo (CUDA) as the per-rank compute of a vocabulary-parallel step."""

    def __init__(self, reserve_sms: int = 0):
        from paper_2607_20908_gb300 import spo
        self.spo = spo
        self.reserve_sms = reserve_sms
        self._side = {}

    def forward_slice(self, b: dict):
        s = self.spo
        lm, _ = s.spo_token_select(b["cu_seqlens"], b["mask"], b["tgt"], b["window"])
        rec = s.spo_logprobs_fwd_slice(b["H"], b["W_slice"], b["v_offset"], b["tgt"], lm,
                                       b["inv_temp"])
        return lm, rec

    def merge(self, recs):
        return self.spo.spo_logprobs_merge_slices(recs)

    def loss(self, b: dict, lm, logp, agg: int):
        s = self.spo
        adv = s.spo_group_advantages(b["rewards"], b["group_id"], b["n_groups"])
        loss, g, _ = s.spo_policy_loss_fwd(logp, b["old"], b["ref"], adv, b["cu_seqlens"],
                                           b["group_id"], b["n_groups"], lm, b["clip_eps"],
                                           b["kl_beta"], agg)
        return loss, g

    def backward_slice(self, b: dict, lse, g):
        """(fp32 dH part, dW rows of the slice, event recorded once dH is final)."""
        s = self.spo
        ev = torch.cuda.Event()
        hooks = s.make_hooks(1, None, ev, reserve_sms=self.reserve_sms)
        dH, dW = s.spo_policy_loss_bwd_ex(b["H"], b["W_slice"], b["tgt"], lse, g, b["inv_temp"],
                                          v_offset=b["v_offset"], dH_fp32=True, hooks=hooks)
        return dH, dW, ev

    def comm_stream(self, t):
        dev = t.device
        if dev not in self._side:
            self._side[dev] = torch.cuda.Stream(dev)
        return self._side[dev]


class VocabParallelStep:
    """One GRPO step with W's rows split over the ranks of a process group.

    run(b) takes this rank's inputs (dict with the whole batch -- H, tgt,
    mask, cu_seqlens, group_id, n_groups, rewards, old, ref, window,
    inv_temp, clip_eps, kl_beta -- plus W_slice and v_offset of this rank's
    rows) and returns (loss, logp, dH, dW_slice): loss, logp and dH are the
    same on every rank, dW_slice holds the gradient of this rank's rows.
    Collectives: one all-gather of the per-token records, and one all-reduce
    of dH, started as soon as the backward's dH GEMM has finished so that it
    runs while the rank's dW GEMMs do.
    """

    def __init__(self, engine, agg: int = AGG_SEQ_GROUP, process_group=None):
        self.engine = engine
        self.agg = agg
        self.pg = process_group

    def run(self, b: dict):
        import torch.distributed as dist
        e = self.engine
        lm, rec = e.forward_slice(b)
        world = dist.get_world_size(self.pg)
        parts = [torch.empty_like(rec) for _ in range(world)]
        dist.all_gather(parts, rec.contiguous(), group=self.pg)
        logp, _, lse = e.merge(torch.stack(parts))
        loss, g = e.loss(b, lm, logp, self.agg)
        dH, dW, dh_ready = e.backward_slice(b, lse, g)
        work = _overlapped_all_reduce(dH, dh_ready, e.comm_stream(dH), self.pg)
        work.wait()
        return loss, logp, dH, dW
