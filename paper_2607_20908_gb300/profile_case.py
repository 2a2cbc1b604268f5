"""Runs the GEMM part of the path (logits + logsumexp forward, then the
backward) on a chosen size, as a target for ncu captures and launch-tuning
sweeps.

    python -m paper_2607_20908_gb300.profile_case --T 16384 --d 5120 --V 8192 --iters 3
    python -m paper_2607_20908_gb300.profile_case --V 151936 --iters 1 \\
        --configs "1,16,0;1,8,0;0,16,0"

--configs is a ';'-separated list of launch tunings (spo_set_tuning), each
either "pair,group,raster[,dynamic_mask[,dw_split_rows]]" applied to every
GEMM, or '|'-separated "key=value" settings (spo_tune_key numbers, e.g.
"7=4|11=0" for dH's raster group and direction) applied after the defaults;
each is run for --iters iterations of fwd + bwd.  --no-dW leaves dW out, so a
case with the full vocabulary and a reduced token count (e.g. --T 8192) holds
a few GB on the device.  The default reduced size keeps the reduction lengths of the full workload
(K = d = 5120 for the logits and their recompute, K = T = 16384 tokens for
dW) with a vocabulary cut to 8192, so one launch takes about a millisecond
and the device holds about 1 GB; the streamed operands of dW (G = 268 MB,
H = 168 MB) stay larger than the 129 MB L2.  Prints per-GEMM CUDA-event
times of the last iteration of each configuration.
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
    ap.add_argument("--T", type=int, default=16384)
    ap.add_argument("--d", type=int, default=5120)
    ap.add_argument("--V", type=int, default=8192)
    ap.add_argument("--iters", type=int, default=3)
    ap.add_argument("--configs", type=str, default="", help='e.g. "1,16,0;0,16,0"')
    ap.add_argument("--no-dW", action="store_true",
                    help="backward without dW (the forward, the recompute and dH only)")
    a = ap.parse_args()
    from paper_2607_20908_gb300 import spo
    dev = torch.device("cuda")
    g = torch.Generator(device=dev).manual_seed(7)
    H = torch.randn(a.T, a.d, device=dev, generator=g).to(torch.bfloat16)
    W = (torch.randn(a.V, a.d, device=dev, generator=g) * 0.02).to(torch.bfloat16)
    tgt = torch.randint(0, a.V, (a.T,), device=dev, generator=g, dtype=torch.int32)
    gl = torch.randn(a.T, device=dev, generator=g) * 1e-4
    ws_f = torch.empty(spo.logprobs_workspace_size(a.T, a.d, a.V), dtype=torch.uint8, device=dev)
    ws_b = torch.empty(spo.policy_loss_bwd_workspace_size(a.T, a.d, a.V), dtype=torch.uint8,
                       device=dev)
    dH = torch.empty(a.T, a.d, dtype=torch.bfloat16, device=dev)
    dW = None if a.no_dW else torch.empty(a.V, a.d, dtype=torch.float32, device=dev)
    configs = [c if "=" in c else tuple(int(x) for x in c.split(","))
               for c in a.configs.split(";") if c] or [None]
    for cfg in configs:
        if isinstance(cfg, str):
            spo.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0)
            for kv in cfg.split("|"):
                key, value = kv.split("=")
                spo.spo_set_tuning(int(key), int(value))
        elif cfg is not None:
            pair, group, raster = cfg[:3]
            spo.spo_set_tuning(spo.SPO_TUNE_PAIR_MMA, pair)
            spo.spo_set_tuning(spo.SPO_TUNE_GROUP_M, group)
            spo.spo_set_tuning(spo.SPO_TUNE_RASTER, raster)
            if len(cfg) > 3:
                spo.spo_set_tuning(spo.SPO_TUNE_DYNAMIC_MASK, cfg[3])
            if len(cfg) > 4:
                spo.spo_set_tuning(spo.SPO_TUNE_DW_SPLIT_ROWS, cfg[4])
        for i in range(a.iters):
            spo.spo_trace_enable(i == a.iters - 1)
            _, _, lse = spo.spo_logprobs_fwd(H, W, tgt, ws=ws_f)
            spo.spo_policy_loss_bwd(H, W, tgt, lse, gl, dH=dH, dW=dW, ws=ws_b,
                                    want_dW=dW is not None)
        torch.cuda.synchronize()
        label = ("default" if cfg is None else cfg if isinstance(cfg, str)
                 else "pair,group,raster,dynamic=" + ",".join(map(str, cfg)))
        print(f"--- {label}")
        recs = [(k, ms) for k, ms in spo.spo_trace_read() if k <= 3]
        per_kind = {k: sum(1 for kk, _ in recs if kk == k) for k, _ in recs}
        for kind, ms in recs:
            # a GEMM run as several launches (dW passes) splits its FLOPs evenly
            tflops = 2.0 * a.T * a.d * a.V / per_kind[kind] / ms / 1e9
            print(f"{spo.TRACE_KINDS[kind]:24s} {ms:8.3f} ms  {tflops:8.1f} TFLOP/s")
    assert spo.spo_device_error() == 0


if __name__ == "__main__":
    main()
