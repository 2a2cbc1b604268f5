"""Data-parallel shard path on CPU: world-size-2 gloo process groups, with the
fp64 oracle standing in for each rank's compute.  The sharded step (group
assignment, per-rank weights, all-reduces of the counts, loss and dW) must
reproduce the unsharded oracle exactly up to fp64 rounding."""

import os
import socket
import tempfile
from datetime import timedelta

import numpy as np
import pytest
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

from oracle import spo_oracle as O
from paper_2607_20908_gb300 import shard


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _batch(seed=0):
    rng = np.random.default_rng(seed)
    sizes = [3, 5, 2, 4, 6]                       # rollouts per group (variable G)
    lens, gid = [], []
    for g, n in enumerate(sizes):
        for _ in range(n):
            lens.append(int(rng.integers(6, 24)))
            gid.append(g)
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int64)
    T, d, V = int(cu[-1]), 16, 53
    mask = (rng.random(T) > 0.25).astype(np.uint8)
    return dict(H=rng.standard_normal((T, d)), W=0.3 * rng.standard_normal((V, d)),
                tgt=rng.integers(0, V, T), mask=mask, cu=cu, gid=np.array(gid), n_groups=len(sizes),
                rewards=rng.uniform(0, 3, len(lens)), old_noise=rng.normal(0, 0.2, T),
                ref_noise=rng.normal(0, 0.05, T), window=12, eps=0.2, beta=0.04)


def _reference(b, agg):
    lm, _ = O.token_select(b["cu"], b["mask"], b["tgt"], b["window"])
    lp, _, _ = O.logprobs(b["H"], b["W"], b["tgt"], 1.0, lm)
    old, ref = lp + b["old_noise"], lp + b["ref_noise"]
    adv = O.group_advantages(b["rewards"], b["gid"], b["n_groups"])
    loss, g, _ = O.policy_loss(lp, old, ref, adv, b["cu"], b["gid"], b["n_groups"], lm, b["eps"],
                               b["beta"], agg)
    dH, dW = O.policy_loss_bwd(b["H"], b["W"], b["tgt"], g)
    return loss, dH, dW, old, ref


class OracleEngine:
    """The fp64 oracle as a rank's compute (test stand-in for libspo)."""

    def step_local(self, b, agg):
        lm, _ = O.token_select(b["cu_seqlens"], b["mask"], b["tgt"], b["window"])
        lp, _, lse = O.logprobs(b["H"], b["W"], b["tgt"], 1.0, lm)
        adv = O.group_advantages(b["rewards"], b["group_id"], b["n_groups"])
        loss, g, st = O.policy_loss(lp, b["old"], b["ref"], adv, b["cu_seqlens"], b["group_id"],
                                    b["n_groups"], lm, b["clip_eps"], b["kl_beta"], agg)
        return dict(loss=torch.tensor([loss], dtype=torch.float64), g=torch.from_numpy(g),
                    lse=lse, n_loss_tokens=torch.tensor([float(st["n_loss_tokens"])],
                                                        dtype=torch.float64))

    def local_counts(self, b, loc):
        return torch.tensor([float(b["n_groups"]), float(loc["n_loss_tokens"][0])],
                            dtype=torch.float64)

    def zero_counts(self, b):
        return torch.zeros(2, dtype=torch.float64)

    def scale_ratio(self, x, num, den):
        x.mul_(num[0] / den[0] if den[0] != 0 else 0.0)
        return x

    def backward_blocks(self, b, lse, g, n_blocks):
        dH, dW = O.policy_loss_bwd(b["H"], b["W"], b["tgt"], g.numpy())
        starts = shard.dw_block_starts(b["W"].shape[0], n_blocks)
        return (torch.from_numpy(dH), torch.from_numpy(np.ascontiguousarray(dW)),
                [(starts[k], starts[k + 1], None) for k in range(n_blocks)])

    def step_fused(self, b, weight, n_blocks):
        loc = self.step_local(b, O.AGG_SEQ_GROUP)
        g = loc["g"] * weight
        dH, dW, blocks = self.backward_blocks(b, loc["lse"], g, n_blocks)
        return loc["loss"] * weight, dH, dW, blocks

    def zeros_dW(self, V, d, like):
        return torch.zeros((V, d), dtype=torch.float64)

    def comm_stream(self, t):
        return None


def _rank_inputs(b, rb, old, ref):
    t = rb.token_index
    return dict(H=b["H"][t], W=b["W"], tgt=b["tgt"][t], mask=b["mask"][t], cu_seqlens=rb.cu_seqlens,
                group_id=rb.group_id, n_groups=rb.n_groups, rewards=b["rewards"][rb.seq_index],
                old=old[t], ref=ref[t], window=b["window"], inv_temp=1.0, clip_eps=b["eps"],
                kl_beta=b["beta"])


def _worker(rank, world, port, outdir, agg, groups_override, dw_blocks=4, fused=False):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=timedelta(seconds=60))
    b = _batch()
    _, _, _, old, ref = _reference(b, agg)
    lm, _ = O.token_select(b["cu"], b["mask"], b["tgt"], b["window"])
    tokens = [int(sum(lm[b["cu"][i]:b["cu"][i + 1]].sum() for i in np.nonzero(b["gid"] == g)[0]))
              for g in range(b["n_groups"])]
    groups = groups_override or shard.shard_groups(tokens, world)
    rb = shard.rank_batch(b["cu"], b["gid"], groups[rank])
    step = shard.DataParallelStep(OracleEngine(), agg, dw_blocks=dw_blocks)
    if fused:   # every rank knows the plan: all n_groups groups are non-empty
        loss, dH, dW = step.run_fused(_rank_inputs(b, rb, old, ref), b["n_groups"])
    else:
        loss, dH, dW = step.run(_rank_inputs(b, rb, old, ref))
    np.save(os.path.join(outdir, f"loss{rank}.npy"), loss.numpy())
    np.save(os.path.join(outdir, f"dW{rank}.npy"), dW.numpy())
    np.save(os.path.join(outdir, f"tok{rank}.npy"), rb.token_index)
    np.save(os.path.join(outdir, f"dH{rank}.npy"), np.zeros((0, 16)) if dH is None else dH.numpy())
    dist.destroy_process_group()


def test_shard_groups_covers_and_balances():
    tokens = [50, 10, 30, 30, 5, 70, 20]
    for world in (1, 2, 3, 4, 9):
        parts = shard.shard_groups(tokens, world)
        flat = sorted(g for p in parts for g in p)
        assert flat == list(range(len(tokens)))
        loads = [sum(tokens[g] for g in p) for p in parts]
        if world <= len(tokens):
            assert max(loads) - min(loads) <= max(tokens)
    assert shard.shard_groups(tokens, 2) == shard.shard_groups(tokens, 2)


def test_rank_batch_selects_whole_groups():
    cu = np.array([0, 3, 5, 9, 10])
    gid = np.array([2, 0, 2, 1])
    rb = shard.rank_batch(cu, gid, [2])
    assert rb.seq_index.tolist() == [0, 2]
    assert rb.token_index.tolist() == [0, 1, 2, 5, 6, 7, 8]
    assert rb.cu_seqlens.tolist() == [0, 3, 7] and rb.group_id.tolist() == [0, 0]
    assert rb.n_groups == 1
    empty = shard.rank_batch(cu, gid, [])
    assert empty.n_groups == 0 and empty.token_index.size == 0


@pytest.mark.parametrize("agg,override", [(O.AGG_SEQ_GROUP, None), (O.AGG_TOKEN, None),
                                          (O.AGG_SEQ_GROUP, [[0, 1, 2, 3, 4], []])])
def test_data_parallel_step_matches_unsharded(agg, override):
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_worker, args=(world, _free_port(), d, agg, override), nprocs=world,
                           join=True, start_method="spawn")
        b = _batch()
        loss, dH, dW, _, _ = _reference(b, agg)
        for r in range(world):
            assert abs(float(np.load(os.path.join(d, f"loss{r}.npy"))[0]) - loss) < 1e-12
            np.testing.assert_allclose(np.load(os.path.join(d, f"dW{r}.npy")), dW, atol=1e-13)
            tok = np.load(os.path.join(d, f"tok{r}.npy"))
            if tok.size:
                np.testing.assert_allclose(np.load(os.path.join(d, f"dH{r}.npy")), dH[tok], atol=1e-13)


@pytest.mark.parametrize("override", [None, [[0, 1, 2, 3, 4], []]])
def test_fused_data_parallel_step_matches_unsharded(override):
    """run_fused: one local call per rank with its weight N_r / N applied before
    the backward, then the per-block dW and loss all-reduces."""
    world = 2
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_worker, args=(world, _free_port(), d, O.AGG_SEQ_GROUP, override, 4,
                                          True), nprocs=world, join=True, start_method="spawn")
        b = _batch()
        loss, dH, dW, _, _ = _reference(b, O.AGG_SEQ_GROUP)
        for r in range(world):
            assert abs(float(np.load(os.path.join(d, f"loss{r}.npy"))[0]) - loss) < 1e-12
            np.testing.assert_allclose(np.load(os.path.join(d, f"dW{r}.npy")), dW, atol=1e-13)
            tok = np.load(os.path.join(d, f"tok{r}.npy"))
            if tok.size:
                np.testing.assert_allclose(np.load(os.path.join(d, f"dH{r}.npy")), dH[tok], atol=1e-13)


def test_block_by_block_dW_reduction_equals_one_reduction():
    """dW summed across ranks as one all-reduce, or as one all-reduce per
    vocabulary block (each issued as its block is final), gives the same
    bits; the blocks tile the vocabulary (V = 53: one 256-row block holds it
    all, the others are empty and skipped)."""
    world = 2
    outs = {}
    for blocks in (1, 3):
        with tempfile.TemporaryDirectory() as d:
            mp.start_processes(_worker, args=(world, _free_port(), d, O.AGG_SEQ_GROUP, None, blocks),
                               nprocs=world, join=True, start_method="spawn")
            outs[blocks] = [np.load(os.path.join(d, f"dW{r}.npy")) for r in range(world)]
    for r in range(world):
        np.testing.assert_array_equal(outs[1][r], outs[3][r])
    assert shard.dw_block_starts(53, 3) == [0, 0, 0, 53]


def _wide_worker(rank, world, port, outdir, n_blocks):
    """dW rows summed block by block over a vocabulary of 1000 rows (blocks of
    0, 256, 512 and 744 rows... as the library lays them out)."""
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=timedelta(seconds=60))
    V, d = 1000, 3
    dW = torch.from_numpy(np.random.default_rng(rank).standard_normal((V, d)))
    starts = shard.dw_block_starts(V, n_blocks)
    works = [shard._overlapped_all_reduce(dW[starts[k]:starts[k + 1]], None, None, None)
             for k in range(n_blocks) if starts[k + 1] > starts[k]]
    for w in works:
        w.wait()
    np.save(os.path.join(outdir, f"w{rank}.npy"), dW.numpy())
    dist.destroy_process_group()


def test_overlapped_block_reductions_sum_every_row():
    world = 3
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_wide_worker, args=(world, _free_port(), d, 4), nprocs=world, join=True,
                           start_method="spawn")
        want = sum(np.random.default_rng(r).standard_normal((1000, 3)) for r in range(world))
        for r in range(world):
            np.testing.assert_allclose(np.load(os.path.join(d, f"w{r}.npy")), want, atol=1e-12)
    assert shard.dw_block_starts(1000, 4) == [0, 0, 256, 512, 1000]


def _failing_worker(rank, world, port, outdir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=timedelta(seconds=4))
    if rank == 1:
        os._exit(0)            # the rank leaves between steps, before its next collective
    t = torch.ones(2, dtype=torch.float64)
    try:
        dist.all_reduce(t)
        status = "completed"
    except Exception as e:     # gloo reports the lost peer or the timeout
        status = "error: " + type(e).__name__
    with open(os.path.join(outdir, "rank0.txt"), "w") as f:
        f.write(status)
    os._exit(0)


def test_lost_rank_ends_the_next_collective_with_an_error():
    with tempfile.TemporaryDirectory() as d:
        ctx = mp.start_processes(_failing_worker, args=(2, _free_port(), d), nprocs=2, join=False,
                                 start_method="spawn")
        for p in ctx.processes:
            p.join(60)
        status = open(os.path.join(d, "rank0.txt")).read()
        assert status.startswith("error"), status


# ---------------------------------------------------------------- vocabulary-parallel form
class OracleVocabEngine:
    """The fp64 oracle as a rank's compute for the vocabulary split."""

    def forward_slice(self, b):
        lm, _ = O.token_select(b["cu_seqlens"], b["mask"], b["tgt"], b["window"])
        rec = O.logprobs_slice_record(b["H"], b["W_slice"], b["v_offset"], b["tgt"], b["inv_temp"],
                                      lm)
        return lm, torch.from_numpy(rec)

    def merge(self, recs):
        return tuple(torch.from_numpy(x) for x in O.merge_slice_records(recs.numpy()))

    def loss(self, b, lm, logp, agg):
        adv = O.group_advantages(b["rewards"], b["group_id"], b["n_groups"])
        loss, g, _ = O.policy_loss(logp.numpy(), b["old"], b["ref"], adv, b["cu_seqlens"],
                                   b["group_id"], b["n_groups"], lm, b["clip_eps"], b["kl_beta"], agg)
        return torch.tensor([loss], dtype=torch.float64), torch.from_numpy(g)

    def backward_slice(self, b, lse, g):
        dH, dW = O.policy_loss_bwd_slice(b["H"], b["W_slice"], b["v_offset"], b["tgt"],
                                         lse.numpy(), g.numpy(), b["inv_temp"])
        return torch.from_numpy(dH), torch.from_numpy(dW), None

    def comm_stream(self, t):
        return None


def _vocab_batch():
    b = _batch(seed=3)
    rng = np.random.default_rng(4)
    V = 72
    b["W"] = 0.3 * rng.standard_normal((V, b["H"].shape[1]))
    b["tgt"] = rng.integers(0, V, b["H"].shape[0])
    b["tgt"][[4, 17]] = -1
    return b


def _vocab_worker(rank, world, port, outdir, agg):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world, timeout=timedelta(seconds=60))
    b = _vocab_batch()
    _, _, _, old, ref = _reference(b, agg)
    off, n = shard.vocab_slices(b["W"].shape[0], world)[rank]
    inp = dict(H=b["H"], W_slice=b["W"][off:off + n], v_offset=off, tgt=b["tgt"], mask=b["mask"],
               cu_seqlens=b["cu"], group_id=b["gid"], n_groups=b["n_groups"],
               rewards=b["rewards"], old=old, ref=ref, window=b["window"], inv_temp=1.0,
               clip_eps=b["eps"], kl_beta=b["beta"])
    loss, logp, dH, dW = shard.VocabParallelStep(OracleVocabEngine(), agg).run(inp)
    np.save(os.path.join(outdir, f"loss{rank}.npy"), loss.numpy())
    np.save(os.path.join(outdir, f"logp{rank}.npy"), logp.numpy())
    np.save(os.path.join(outdir, f"dH{rank}.npy"), dH.numpy())
    np.save(os.path.join(outdir, f"dW{rank}.npy"), dW.numpy())
    dist.destroy_process_group()


@pytest.mark.parametrize("world,agg", [(2, O.AGG_SEQ_GROUP), (3, O.AGG_TOKEN)])
def test_vocab_parallel_step_matches_unsplit(world, agg):
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_vocab_worker, args=(world, _free_port(), d, agg), nprocs=world,
                           join=True, start_method="spawn")
        b = _vocab_batch()
        loss, dH, dW, _, _ = _reference(b, agg)
        lm, _ = O.token_select(b["cu"], b["mask"], b["tgt"], b["window"])
        lp, _, _ = O.logprobs(b["H"], b["W"], b["tgt"], 1.0, lm)
        rows = []
        for r in range(world):
            assert abs(float(np.load(os.path.join(d, f"loss{r}.npy"))[0]) - loss) < 1e-12
            np.testing.assert_allclose(np.load(os.path.join(d, f"logp{r}.npy")), lp, atol=1e-12)
            np.testing.assert_allclose(np.load(os.path.join(d, f"dH{r}.npy")), dH, atol=1e-13)
            rows.append(np.load(os.path.join(d, f"dW{r}.npy")))
        np.testing.assert_allclose(np.concatenate(rows), dW, atol=1e-13)


def test_vocab_slices_cover_the_vocabulary():
    for V, world in ((151936, 2), (151936, 3), (151936, 7), (4096, 8), (72, 9)):
        sl = shard.vocab_slices(V, world)
        assert len(sl) == world and sl[0][0] == 0
        assert all(o1 + n1 == o2 for (o1, n1), (o2, _) in zip(sl[:-1], sl[1:]))
        assert sl[-1][0] + sl[-1][1] == V
        assert all(n % 8 == 0 and n > 0 for _, n in sl)
        assert max(n for _, n in sl) - min(n for _, n in sl) <= 8
    with pytest.raises(ValueError):
        shard.vocab_slices(4100, 2)
    with pytest.raises(ValueError):
        shard.vocab_slices(16, 3)
