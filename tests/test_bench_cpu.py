"""bench.py's multi-rank plumbing on CPU: two gloo ranks join the process
group, pass the barrier and agree on the maximum of their step times (the
timing rule is the max over ranks)."""

import os
import socket
import tempfile

import torch.multiprocessing as mp


def _free_port():
    s = socket.socket()
    s.bind(("127.0.0.1", 0))
    p = s.getsockname()[1]
    s.close()
    return p


def _worker(rank, port, outdir):
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port), WORLD_SIZE="2",
                      RANK=str(rank), LOCAL_RANK=str(rank))
    import torch

    import bench
    dist = bench.Dist()
    dist.init("gloo", torch.device("cpu"))
    dist.barrier()
    ms = dist.max(10.0 + rank, torch.device("cpu"))
    with open(os.path.join(outdir, f"r{rank}"), "w") as f:
        f.write(repr((dist.world, dist.rank, ms)))
    dist.close()


def test_two_ranks_agree_on_the_slowest_time():
    with tempfile.TemporaryDirectory() as d:
        mp.start_processes(_worker, args=(_free_port(), d), nprocs=2, join=True,
                           start_method="spawn")
        got = [eval(open(os.path.join(d, f"r{r}")).read()) for r in range(2)]
    assert got == [(2, 0, 11.0), (2, 1, 11.0)]


def test_single_process_needs_no_group():
    import torch

    import bench
    dist = bench.Dist()
    dist.init("nccl", torch.device("cpu"))   # world size 1: no process group is created
    dist.barrier()
    assert dist.pg is None and dist.max(3.5, torch.device("cpu")) == 3.5
