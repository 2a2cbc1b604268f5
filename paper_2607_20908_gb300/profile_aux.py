"""Runs the bandwidth-bound calls of the path at an enlarged size, as a target
for ncu captures: the group advantages (spo_group_advantages_ws; 2^n
rollouts in sorted contiguous groups of 16) and the loss forward
(spo_policy_loss_fwd; 2^n tokens as sequences of 128, groups of 8, every
token a loss token, KL on), with the inputs bench.py's `aux` measurement
uses; or the forward at the full workload's T = 16384 and V = 151936 with a
hidden size of 256 ("combine"), whose split-vocabulary combine reads the
same 117 MB of partials as the full workload's while the device holds under
1 GB.

    python -m paper_2607_20908_gb300.profile_aux --which adv --reps 6
    python -m paper_2607_20908_gb300.profile_aux --which loss --reps 6
    python -m paper_2607_20908_gb300.profile_aux --which combine --reps 6

Each rep follows a 256 MB write that evicts L2 and is timed with CUDA events;
prints the sorted per-call times in microseconds.
"""

import argparse
import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--which", choices=["adv", "loss", "both", "combine"], default="both")
    ap.add_argument("--log2n", type=int, default=24)
    ap.add_argument("--reps", type=int, default=6)
    a = ap.parse_args()
    from paper_2607_20908_gb300 import spo
    dev = torch.device("cuda")
    n = 1 << a.log2n
    gen = torch.Generator(device=dev).manual_seed(5)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    calls = {}
    if a.which in ("adv", "both"):
        groups = n // 16
        gid = torch.arange(n, device=dev, dtype=torch.int32) // 16
        r = torch.randn(n, device=dev, generator=gen)
        adv = torch.empty(n, device=dev)
        ws = torch.empty(spo.group_advantages_workspace_size(n, groups), dtype=torch.uint8,
                         device=dev)
        calls["adv"] = lambda: spo.spo_group_advantages_ws(r, gid, groups, adv=adv, ws=ws)
    if a.which in ("loss", "both"):
        L = 128
        ns = n // L
        ng = ns // 8
        cu = torch.arange(0, n + 1, L, device=dev, dtype=torch.int32)
        gid2 = torch.arange(ns, device=dev, dtype=torch.int32) // 8
        lp = -8.0 * torch.rand(n, device=dev, generator=gen)
        old = lp + 0.05 * torch.randn(n, device=dev, generator=gen)
        ref = lp + 0.05 * torch.randn(n, device=dev, generator=gen)
        a_seq = torch.randn(ns, device=dev, generator=gen)
        lm = torch.ones(n, dtype=torch.uint8, device=dev)
        ws2 = torch.empty(spo.policy_loss_workspace_size(ns, ng), dtype=torch.uint8, device=dev)
        calls["loss"] = lambda: spo.spo_policy_loss_fwd(lp, old, ref, a_seq, cu, gid2, ng, lm, 0.2,
                                                        0.04, ws=ws2)
    if a.which == "combine":
        T, d, V = 16384, 256, 151936
        H = torch.randn(T, d, device=dev, generator=gen).to(torch.bfloat16)
        W = (torch.randn(V, d, device=dev, generator=gen) * 0.02).to(torch.bfloat16)
        tgt = torch.randint(0, V, (T,), device=dev, generator=gen, dtype=torch.int32)
        ws3 = torch.empty(spo.logprobs_workspace_size(T, d, V), dtype=torch.uint8, device=dev)
        calls["fwd_d256"] = lambda: spo.spo_logprobs_fwd(H, W, tgt, ws=ws3)
    for name, fn in calls.items():
        times = []
        for i in range(a.reps):
            flush.fill_(i & 0xFF)
            t0 = torch.cuda.Event(enable_timing=True)
            t1 = torch.cuda.Event(enable_timing=True)
            t0.record()
            fn()
            t1.record()
            torch.cuda.synchronize(dev)
            times.append(t0.elapsed_time(t1) * 1e3)
        print(name, "us", [round(t, 1) for t in sorted(times)])


if __name__ == "__main__":
    main()
