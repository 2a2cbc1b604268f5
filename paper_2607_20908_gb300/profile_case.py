"""Runs the whole path a few times on a reduced, profiler-friendly case.

    python -m paper_2607_20908_gb300.profile_case --T 16384 --d 5120 --V 8192 --iters 3

Used as the target of ncu captures: the same kernels as the full workload
with the same reduction lengths (K = d = 5120 for the logits and their
recompute, K = T = 16384 tokens for dW), but a vocabulary cut to 8192 so one
launch takes about a millisecond and the device holds about 1 GB.  The
streamed operands of dW (G = 268 MB, H = 168 MB) stay larger than the
129 MB L2.  Prints per-GEMM CUDA-event times of the last iteration.
"""

import argparse
import ctypes
import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--T", type=int, default=16384)
    ap.add_argument("--d", type=int, default=5120)
    ap.add_argument("--V", type=int, default=8192)
    ap.add_argument("--iters", type=int, default=3)
    a = ap.parse_args()
    from paper_2607_20908_gb300 import spo
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(7)
    H = torch.randn(a.T, a.d, device=dev, generator=g).to(torch.bfloat16)
    W = (torch.randn(a.V, a.d, device=dev, generator=g) * 0.02).to(torch.bfloat16)
    tgt = torch.randint(0, a.V, (a.T,), device=dev, generator=g, dtype=torch.int32)
    gl = torch.randn(a.T, device=dev, generator=g) * 1e-4
    for i in range(a.iters):
        spo.spo_trace_enable(i == a.iters - 1)
        _, _, lse = spo.spo_logprobs_fwd(H, W, tgt)
        spo.spo_policy_loss_bwd(H, W, tgt, lse, gl)
    torch.cuda.synchronize()
    for kind, ms in spo.spo_trace_read():
        print(f"{spo.TRACE_KINDS[kind]:24s} {ms:8.3f} ms  {2.0 * a.T * a.d * a.V / ms / 1e9:8.1f} TFLOP/s")
    assert spo.spo_device_error() == 0


if __name__ == "__main__":
    main()
