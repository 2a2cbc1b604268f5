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


ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _run_bench(args, env_extra=None, timeout=600):
    import subprocess
    import sys
    env = dict(os.environ)
    env.update(env_extra or {})
    return subprocess.run([sys.executable, os.path.join(ROOT, "bench.py"), *args], cwd=ROOT, env=env,
                          capture_output=True, text=True, timeout=timeout)


def test_reference_arm_prints_one_json_line():
    """`bench.py --impl reference` runs the fp64 oracle on a bounded sample of
    the full workload and prints one JSON line with the GPU arm's metric, unit
    and config, plus the reference arm's own keys."""
    import json

    import bench
    r = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3"])
    assert r.returncode == 0, r.stderr[-2000:]
    lines = [ln for ln in r.stdout.splitlines() if ln.strip().startswith("{")]
    assert len(lines) == 1, r.stdout
    d = json.loads(lines[0])
    assert d["impl"] == "reference" and d["metric"] == bench.METRIC and d["unit"] == bench.UNIT
    assert d["higher_is_better"] is True and d["steps"] == 1 and d["warmup"] == 3
    assert d["value"] > 0 and d["ms_per_step"] > 0 and d["n_gpus"] == 1
    assert d["config"]["workload"].startswith("full loss fwd+bwd") and d["config"]["T"] == 16384
    cb = d["cpu_baseline"]
    assert cb["kind"] == "oracle" and cb["value"] == d["value"] and cb["cores"] >= 1 and cb["sample"]
    assert d["e2e"] == {"value": d["value"], "unit": bench.UNIT, "h2d_bytes_per_step": 0,
                        "d2h_bytes_per_step": 0}


def test_reference_arm_other_ranks_exit_quietly():
    """Under torchrun only rank 0 runs the reference arm; the others print
    nothing and exit 0 without joining a process group."""
    r = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "3"],
                   {"RANK": "1", "LOCAL_RANK": "1", "WORLD_SIZE": "2"}, timeout=300)
    assert r.returncode == 0, r.stderr[-2000:]
    assert r.stdout.strip() == ""


def test_warmup_below_three_is_refused():
    r = _run_bench(["--impl", "reference", "--steps", "1", "--warmup", "2"], timeout=300)
    assert r.returncode != 0 and "--warmup must be >= 3" in r.stderr
