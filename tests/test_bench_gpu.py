"""bench.py's data-parallel step wiring on one GPU: rank 0 of two identical
ranks (the collectives stand in for the second rank by doubling each
tensor, with work handles ordered by events like NCCL's).  The rank weighs
its loss and g by 1/2 on the device and sums dW block by block, so its loss
and dW must be the one-GPU step's bits (every scale is a power of two) and
its dH half of it."""

import types

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


class _Work:
    def __init__(self):
        self.ev = torch.cuda.Event()
        self.ev.record()

    def wait(self):
        torch.cuda.current_stream().wait_event(self.ev)


def test_data_parallel_bench_step_on_two_identical_ranks(spo, monkeypatch):
    import torch.distributed as dist

    import bench
    calls = []

    def all_reduce(t, group=None, async_op=False):
        calls.append(t.numel())
        t.mul_(2)
        return _Work() if async_op else None

    monkeypatch.setattr(dist, "all_reduce", all_reduce)
    dev = torch.device("cuda")
    case = inputs.tiny_case(seed=1401, d=320, V=5000, T_per_seq=40)
    one = bench.Step(case, dev, None, mode="fused")
    one.prepare_old_ref()
    one.run()
    torch.cuda.synchronize()
    fake = types.SimpleNamespace(world=2, rank=0, pg=dist)
    two = bench.Step(case, dev, fake, mode="fused")
    two.old.copy_(one.old)
    two.ref.copy_(one.ref)
    two.run()
    torch.cuda.synchronize()
    assert torch.equal(two.loss, one.loss)
    assert torch.equal(two.dW, one.dW)
    assert torch.equal(two.dH.float() * 2, one.dH.float())
    # one all-reduce per dW vocabulary block (rows 0, 1024, 2304, 3584, 5000), then the loss
    starts = spo.dw_block_starts(case["V"], 4)
    assert calls == [(b - a) * case["d"] for a, b in zip(starts[:-1], starts[1:]) if b > a] + [1]
    assert spo.spo_sync_check() == 0


def test_end_to_end_pipeline_copies_each_output_after_its_event(spo):
    """bench.py's end-to-end pipeline copies dH and each dW vocabulary block
    out when the step's hook event marks it final.  Every step first poisons
    dH and dW with NaN on the compute stream, so a copy that ran ahead of its
    event would bring back NaN or a partial block."""
    import bench
    dev = torch.device("cuda")
    case = inputs.tiny_case(seed=1402, d=320, V=5000, T_per_seq=40)
    st = bench.Step(case, dev, None, mode="fused")
    st.prepare_old_ref()
    st.run()
    torch.cuda.synchronize()
    names = ("loss", "stats", "logp", "ent", "dH", "dW")
    want = {k: getattr(st, k).cpu() for k in names}
    hio = bench.HostIO(st, sets=2, dw_blocks=4)
    assert hio.blocks is not None and len(hio.starts) == 5
    for x in hio.sets:
        def poisoned(x=x, run=x.run):
            x.dW.fill_(float("nan"))
            x.dH.fill_(float("nan"))
            run()
        x.run = poisoned
    for _ in range(5):
        hio.step()
    torch.cuda.synchronize()
    for host in hio.host_out:
        for k, h in zip(names, host):
            assert torch.equal(h, want[k]), k
    assert spo.spo_sync_check() == 0
