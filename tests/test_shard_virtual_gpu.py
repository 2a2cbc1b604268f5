"""The multi-GPU step forms through the CUDA kernels, with virtual ranks on
one GPU: ``shard.DataParallelStep`` (whole groups per rank) with
``shard.SpoEngine`` and ``shard.VocabParallelStep`` (W's rows split) with
``shard.SpoVocabEngine`` run unmodified, libspo as every rank's compute, one
host thread and CUDA stream per rank, and their collectives served in-process
(the threads meet at a barrier and add or gather the ranks' tensors in rank
order; nothing on the device waits for another rank).  Each must give the
unsharded step's results."""

import threading

import numpy as np
import pytest
import torch

from paper_2607_20908_gb300 import shard

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def spo():
    if not torch.cuda.is_available():
        pytest.skip("needs a CUDA GPU")
    from paper_2607_20908_gb300 import build
    build.build()
    from paper_2607_20908_gb300 import spo as mod
    return mod


class ThreadCollectives:
    """all_reduce(sum) across n host threads, each registered with its rank."""

    def __init__(self, n):
        self.n = n
        self.bar = threading.Barrier(n, timeout=60)
        self.slots = [None] * n
        self.local = threading.local()

    def get_world_size(self, group=None):
        return self.n

    def all_gather(self, parts, t, group=None):
        if t.is_cuda:
            torch.cuda.current_stream().synchronize()
        self.slots[self.local.rank] = t.detach().clone()
        self.bar.wait()
        for r in range(self.n):
            parts[r].copy_(self.slots[r])
        self.bar.wait()

    def all_reduce(self, t, group=None, async_op=False):
        if t.is_cuda:
            torch.cuda.current_stream().synchronize()
        self.slots[self.local.rank] = t.detach().clone()
        self.bar.wait()
        total = self.slots[0].clone()
        for x in self.slots[1:]:
            total += x.to(total.device)
        self.bar.wait()
        t.copy_(total)
        if async_op:
            return _Done(t.is_cuda)


class _Done:
    """Work handle of a collective served in-process: wait() orders the
    caller's stream after the stream the result was written on."""

    def __init__(self, cuda):
        self.ev = None
        if cuda:
            self.ev = torch.cuda.Event()
            self.ev.record()

    def wait(self):
        if self.ev is not None:
            torch.cuda.current_stream().wait_event(self.ev)


def _batch(seed):
    rng = np.random.default_rng(seed)
    sizes = [3, 5, 2, 4, 6, 1, 8]                 # rollouts per group (variable G, a group of one)
    lens, gid = [], []
    for g, n in enumerate(sizes):
        for _ in range(n):
            lens.append(int(rng.integers(6, 90)))
            gid.append(g)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    T, d, V = int(cu[-1]), 256, 4096
    gen = torch.Generator().manual_seed(seed)
    return dict(H=torch.randn(T, d, generator=gen).to(torch.bfloat16),
                W=(torch.randn(V, d, generator=gen) * 0.05).to(torch.bfloat16),
                tgt=torch.randint(0, V, (T,), generator=gen, dtype=torch.int32),
                mask=torch.from_numpy((rng.random(T) > 0.25).astype(np.uint8)),
                cu=cu, gid=np.array(gid, dtype=np.int32), n_groups=len(sizes),
                rewards=torch.from_numpy(rng.uniform(0, 3, len(lens)).astype(np.float32)),
                old_noise=torch.from_numpy(rng.normal(0, 0.2, T).astype(np.float32)),
                ref_noise=torch.from_numpy(rng.normal(0, 0.05, T).astype(np.float32)))


def _rank_dict(spo, b, rb, old, ref):
    dev = torch.device("cuda")
    tok = torch.from_numpy(rb.token_index).long()
    seq = torch.from_numpy(rb.seq_index).long()
    return dict(H=b["H"][tok].contiguous().to(dev), W=b["W"].to(dev),
                tgt=b["tgt"][tok].contiguous().to(dev), mask=b["mask"][tok].contiguous().to(dev),
                cu_seqlens=torch.from_numpy(rb.cu_seqlens).to(dev),
                group_id=torch.from_numpy(rb.group_id).to(dev), n_groups=rb.n_groups,
                rewards=b["rewards"][seq].contiguous().to(dev),
                old=old[tok].contiguous().to(dev), ref=ref[tok].contiguous().to(dev),
                window=40, inv_temp=1.0, clip_eps=0.2, kl_beta=0.04)


@pytest.mark.parametrize("world", [2, 3])
@pytest.mark.parametrize("agg,fused", [(0, False), (1, False), (0, True)])
def test_virtual_ranks_reproduce_the_unsharded_step(spo, monkeypatch, world, agg, fused):
    import torch.distributed as dist
    b = _batch(40 + world)
    T = b["H"].shape[0]
    # old / ref log-probs around the current policy's, fixed before sharding
    dev = torch.device("cuda")
    lp, _, _ = spo.spo_logprobs_fwd(b["H"].to(dev), b["W"].to(dev), b["tgt"].to(dev))
    old = (lp.cpu() + b["old_noise"]).contiguous()
    ref = (lp.cpu() + b["ref_noise"]).contiguous()

    coll = ThreadCollectives(1)
    monkeypatch.setattr(dist, "all_reduce", coll.all_reduce)
    coll.local.rank = 0
    whole = shard.rank_batch(b["cu"], b["gid"], range(b["n_groups"]))
    loss1, dH1, dW1 = shard.DataParallelStep(shard.SpoEngine(), agg).run(
        _rank_dict(spo, b, whole, old, ref))
    torch.cuda.synchronize()

    tokens_per_group = [int(b["cu"][np.nonzero(b["gid"] == g)[0] + 1].sum()
                            - b["cu"][np.nonzero(b["gid"] == g)[0]].sum())
                        for g in range(b["n_groups"])]
    groups = shard.shard_groups(tokens_per_group, world)
    batches = [shard.rank_batch(b["cu"], b["gid"], groups[r]) for r in range(world)]
    coll = ThreadCollectives(world)
    monkeypatch.setattr(dist, "all_reduce", coll.all_reduce)

    def rank(r):
        step = shard.DataParallelStep(shard.SpoEngine(reserve_sms=8), agg)
        inp = _rank_dict(spo, b, batches[r], old, ref)
        # run_fused: one spo_grpo_step per rank, weight N_r / N known from the plan
        return step.run_fused(inp, b["n_groups"]) if fused else step.run(inp)

    outs = _run_ranks(coll, world, rank)
    for r in range(world):
        loss_r, dH_r, dW_r = outs[r]
        assert abs(loss_r.item() - loss1.item()) <= 1e-5 * abs(loss1.item()) + 1e-7
        rel = ((dW_r - dW1).double().norm() / dW1.double().norm()).item()
        assert rel <= 2e-3, rel
        tok = torch.from_numpy(batches[r].token_index).long().to(dev)
        want = dH1[tok].double()
        rel_h = ((dH_r.double() - want).norm() / want.norm()).item()
        assert rel_h <= 2e-3, rel_h
    assert sum(len(x.token_index) for x in batches) == T
    assert spo.spo_device_error() == 0


def _run_ranks(coll, world, fn):
    outs, errors = [None] * world, []

    def rank(r):
        try:
            coll.local.rank = r
            s = torch.cuda.Stream()
            with torch.cuda.stream(s):
                outs[r] = fn(r)
            s.synchronize()
        except Exception as e:     # reported on the test's thread
            errors.append(e)
            coll.bar.abort()

    threads = [threading.Thread(target=rank, args=(r,)) for r in range(world)]
    for th in threads:
        th.start()
    for th in threads:
        th.join()
    assert not errors, errors
    torch.cuda.synchronize()
    return outs


@pytest.mark.parametrize("world", [2, 3])
def test_virtual_vocab_ranks_reproduce_the_unsplit_step(spo, monkeypatch, world):
    """W's 4096 rows as 2 or 3 slices (3: uneven, with a ragged vocabulary
    tile inside a slice): every rank ends with the unsplit log-probs, loss and
    dH, and its own rows of dW."""
    import torch.distributed as dist
    b = _batch(50 + world)
    dev = torch.device("cuda")
    H, W, tgt = b["H"].to(dev), b["W"].to(dev), b["tgt"].to(dev)
    cu, gid = torch.from_numpy(b["cu"]).to(dev), torch.from_numpy(b["gid"]).to(dev)
    mask, rewards = b["mask"].to(dev), b["rewards"].to(dev)
    lp0, _, _ = spo.spo_logprobs_fwd(H, W, tgt)
    old = (lp0 + b["old_noise"].to(dev)).contiguous()
    ref = (lp0 + b["ref_noise"].to(dev)).contiguous()
    # the unsplit step
    lm, _ = spo.spo_token_select(cu, mask, tgt, 40)
    logp1, _, lse1 = spo.spo_logprobs_fwd(H, W, tgt, lm)
    adv = spo.spo_group_advantages(rewards, gid, b["n_groups"])
    loss1, g1, _ = spo.spo_policy_loss_fwd(logp1, old, ref, adv, cu, gid, b["n_groups"], lm, 0.2,
                                           0.04)
    dH1, dW1 = spo.spo_policy_loss_bwd(H, W, tgt, lse1, g1)
    torch.cuda.synchronize()

    slices = shard.vocab_slices(W.shape[0], world)
    coll = ThreadCollectives(world)
    monkeypatch.setattr(dist, "all_reduce", coll.all_reduce)
    monkeypatch.setattr(dist, "all_gather", coll.all_gather)
    monkeypatch.setattr(dist, "get_world_size", coll.get_world_size)

    def rank(r):
        off, n = slices[r]
        rb = dict(H=H, W_slice=W[off:off + n], v_offset=off, tgt=tgt, mask=mask, cu_seqlens=cu,
                  group_id=gid, n_groups=b["n_groups"], rewards=rewards, old=old, ref=ref,
                  window=40, inv_temp=1.0, clip_eps=0.2, kl_beta=0.04)
        return shard.VocabParallelStep(shard.SpoVocabEngine(), 0).run(rb)

    outs = _run_ranks(coll, world, rank)
    for r, (loss_r, logp_r, dH_r, dW_r) in enumerate(outs):
        assert torch.abs(logp_r - logp1).max().item() <= 1e-5
        assert abs(loss_r.item() - loss1.item()) <= 1e-5 * abs(loss1.item()) + 1e-7
        want = dH1.double()
        assert ((dH_r.double() - want).norm() / want.norm()).item() <= 3e-3
        off, n = slices[r]
        w_rows = dW1[off:off + n].double()
        assert ((dW_r.double() - w_rows).norm() / w_rows.norm()).item() <= 2e-3
    # every rank holds the same merged results
    for loss_r, logp_r, dH_r, _ in outs[1:]:
        assert torch.equal(logp_r, outs[0][1]) and torch.equal(dH_r, outs[0][2])
    assert spo.spo_device_error() == 0

