#!/usr/bin/env python
"""Throughput of the GRPO log-prob + policy-loss path (fwd + bwd) on GB300.

    python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

One step = one pass of the whole path over one batch held in HBM:
token selection -> log-probs over the full vocabulary (tensor-core logits +
online logsumexp) -> group advantages -> clipped surrogate + KL loss ->
backward (logit recompute, dH = G W, dW = G^T H).  Workload: 16 groups x 8
rollouts x 128 tokens = 16384 tokens, d = 5120, V = 151936, bf16.

Prints one JSON line (rank 0).  `value` is loss tokens per second over all
GPUs; `e2e` is the same metric with host<->device copies of every input and
output inside the timed region; `roofline` is the dominant kernel's
algorithmic TFLOP/s (from CUDA events recorded around each launch on its
stream) against the measured bf16 peak; `cpu_baseline` is the fp64 oracle on
a bounded sample of the same workload on this machine's host cores.

The step is one C-ABI call (spo_grpo_step); --separate-calls times the
individual calls in turn instead.  --impl reference times the fp64 oracle
itself (host cores) on bounded samples of the same workload and prints the
same line with impl=reference.  Under torchrun every rank owns 16 whole
groups of a data-parallel batch (weak scaling): its loss and dL/dlogp carry
weight 1/N (applied on the device) and dW is summed across ranks by NCCL in
four vocabulary blocks, each started as soon as the backward has finished
it; with --workload vocab-split the ranks instead split W's rows over one
shared batch (strong scaling).  The timing adds a barrier and a max over
ranks.
"""

from __future__ import annotations

import os

_CORES = len(os.sched_getaffinity(0)) if hasattr(os, "sched_getaffinity") else (os.cpu_count() or 1)
os.environ.setdefault("OPENBLAS_NUM_THREADS", str(_CORES))
os.environ.setdefault("OMP_NUM_THREADS", str(_CORES))

import argparse  # noqa: E402
import ctypes  # noqa: E402
import json  # noqa: E402
import statistics  # noqa: E402
import subprocess  # noqa: E402
import sys  # noqa: E402
import threading  # noqa: E402
import time  # noqa: E402

import numpy as np  # noqa: E402
import torch  # noqa: E402

ROOT = os.path.dirname(os.path.abspath(__file__))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

from paper_2607_20908_gb300 import inputs  # noqa: E402

METRIC = "tokens/s fused logprob+PG loss fwd+bwd (d=5120,V=151936); % BF16 tensor peak"
METRIC_FWD = "tokens/s forward logprobs + entropy (d=4096,V=151936); % BF16 tensor peak"
UNIT = "tokens/s"
WORKLOAD = ("full loss fwd+bwd: T=16384 tokens (16 groups x 8 rollouts x 128 tokens), d=5120, "
            "V=151936, bf16 H/W, fp32 accumulate, rewards correctness+log-speedup+structural, "
            "clip eps=0.2, KL beta=0.04, window 1024, SEQ_GROUP aggregation")
# Supplementary workloads (--workload); the default is the one the metric is quoted on.
WORKLOADS = {
    "full": WORKLOAD,
    "forward": "forward logprobs only: T=8192 tokens (8 rollouts x 1024), d=4096, V=151936, bf16; "
               "outputs fp32 per-token logprob and entropy",
    "ragged": "multi-turn ragged: 32 groups x 8 rollouts x 1-4 turns packed to 65536 tokens, ~40% "
              "prompt/feedback tokens masked, per-turn rewards, d=5120, V=151936, bf16 fwd+bwd",
    "large": "large batch: T=131072 packed tokens, groups of 4/8/16, 5% of rollouts in zero-variance "
             "groups, KL to reference log-probs, d=5120, V=151936, bf16 fwd+bwd (4 backward chunks)",
    "kept": WORKLOAD + "; kept-exponential form: the forward also keeps exp(z - tile max) in bf16 "
            "(5 GB) and the backward forms G from it instead of recomputing the logits",
    "vocab-split": WORKLOAD + "; vocabulary-split form: the head's rows as slices (one per GPU; "
                   "on one GPU 2 slices of 75968 run in turn, fp32 dH parts summed on the device "
                   "where ranks all-reduce), per-slice log-prob records merged, dW written per slice",
}

KERNEL_NAMES = {0: "logits_lse_fwd", 1: "logits_grad_recompute", 2: "gemm_dH", 3: "gemm_dW",
                4: "lse_combine", 5: "select_gather_fwd", 6: "select_gather_bwd",
                7: "policy_loss_fwd", 8: "group_advantages", 9: "token_select",
                10: "reward_compose", 12: "merge_slices", 13: "form_g"}
GEMM_KINDS = ("logits_lse_fwd", "logits_grad_recompute", "gemm_dH", "gemm_dW")
SAMPLE_SEQS, SAMPLE_TOKENS = 8, 8   # CPU sample: one group of 8 rollouts, first 8 tokens each


# DRAM bytes (read + write) per launch of each tensor-core kernel at this workload, valid only for
# the kernel sources they were taken on.  Derived from one-pass ncu captures
# (dram__bytes_read.sum + dram__bytes_write.sum, the GEMM kernels only) of two reduced cases of the
# same kernels, scaled by the units a launch processes: 8192 tokens with the full vocabulary and no
# dW (the logits GEMMs and dH: x 2 tokens) and the full 16384 tokens with 8192 vocabulary rows (dW:
# x 151936 / 8192 rows, the mean of its two passes).  The logits GEMMs' traffic is proportional to
# the tokens (checked against full-size captures: 6.88 and 13.57 GB); dH's grows faster than its
# waves (its CTA pairs drift further apart over more waves), so its figure is a lower estimate.
TRAFFIC = {"sources_sha256_16": "a941936797edddb8",
           "bytes": {"logits_lse_fwd": 8.889e9, "logits_grad_recompute": 16.62e9,
                     "gemm_dH": 29.00e9, "gemm_dW": 17.03e9},
           "derivation": "reduced-case captures, every GEMM in the tile form the one-call step "
                         "uses, scaled by tokens (T = 8192 -> 16384) or vocabulary rows "
                         "(V = 8192 -> 151936); dH a lower estimate (23-35 GB over nine captures "
                         "of the same kernel)"}
KERNEL_SOURCES = ["paper_2607_20908_gb300/csrc/gemm.cu", "paper_2607_20908_gb300/csrc/tc.cuh",
                  "paper_2607_20908_gb300/csrc/gemm.h"]


def kernel_traffic(name):
    """ncu DRAM bytes per launch for `name`, or None if the kernel sources changed since."""
    import hashlib
    h = hashlib.sha256()
    for f in KERNEL_SOURCES:
        with open(os.path.join(ROOT, f), "rb") as fh:
            h.update(fh.read())
    if h.hexdigest()[:16] != TRAFFIC["sources_sha256_16"]:
        return None
    return TRAFFIC["bytes"].get(name)


def peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        with open(p) as f:
            j = json.load(f)
        return dict(bf16_burst=float(j["bf16_tflops"]), bf16_sustained=float(j["bf16_tflops_sustained"]),
                    hbm=float(j["hbm_gbs"]), source="measured (MEASURED_PEAKS.json)")
    return dict(bf16_burst=1900.0, bf16_sustained=1700.0, hbm=6800.0,
                source="fallback (no MEASURED_PEAKS.json)")


# ----------------------------------------------------------------- distributed
class Dist:
    def __init__(self):
        self.world = int(os.environ.get("WORLD_SIZE", "1"))
        self.rank = int(os.environ.get("RANK", "0"))
        self.local = int(os.environ.get("LOCAL_RANK", "0"))
        self.pg = None
        self.device = None

    def init(self, backend, device=None):
        """Joins the process group; with NCCL the group is bound to this rank's
        GPU (set as the current device first) so no collective guesses GPU 0."""
        self.device = device
        if self.world > 1:
            import torch.distributed as dist
            if device is not None and device.type == "cuda":
                torch.cuda.set_device(device)
                dist.init_process_group(backend, device_id=device)
            else:
                dist.init_process_group(backend)
            self.pg = dist

    def barrier(self):
        if self.pg:
            if self.device is not None and self.device.type == "cuda":
                self.pg.barrier(device_ids=[self.device.index])
            else:
                self.pg.barrier()

    def max(self, x: float, device) -> float:
        if not self.pg:
            return x
        t = torch.tensor([x], dtype=torch.float64, device=device)
        self.pg.all_reduce(t, op=self.pg.ReduceOp.MAX)
        return float(t.item())

    def close(self):
        if self.pg:
            self.pg.destroy_process_group()


# ----------------------------------------------------------------- clocks
class ClockSampler:
    """Samples nvidia-smi clocks / throttle reasons in the background."""
    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.hw_slowdown,"
              "clocks_event_reasons.hw_thermal_slowdown,clocks_event_reasons.sw_thermal_slowdown,"
              "clocks_event_reasons.sw_power_cap")
    NAMES = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device):
        self.samples = []
        self.proc = None
        try:
            uuid = str(torch.cuda.get_device_properties(device).uuid)
            sel = uuid if uuid.startswith("GPU-") else "GPU-" + uuid
        except Exception:
            sel = str(device.index or 0)
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", "-i", sel, f"--query-gpu={self.FIELDS}", "--format=csv,noheader,nounits",
                 "-lms", "100"], stdout=subprocess.PIPE, stderr=subprocess.DEVNULL, text=True)
            threading.Thread(target=self._read, daemon=True).start()
        except Exception:
            self.proc = None

    def _read(self):
        for line in self.proc.stdout:
            parts = [p.strip() for p in line.split(",")]
            if len(parts) >= 7:
                self.samples.append((time.time(), parts))

    def stop(self):
        if self.proc:
            self.proc.terminate()
            try:
                self.proc.wait(timeout=5)
            except Exception:
                self.proc.kill()

    def summary(self, t0, t1):
        win = [p for (t, p) in self.samples if t0 <= t <= t1]
        scope = "timed region"
        if len(win) < 3:
            win = [p for (_, p) in self.samples]
            scope = "warm-up + timed region"
        if not win:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": [], "samples": 0}
        def num(x):
            try:
                return float(x)
            except ValueError:
                return None
        sm = [num(p[0]) for p in win if num(p[0]) is not None]
        reasons = sorted({self.NAMES[i] for p in win for i in range(4) if p[3 + i].lower() == "active"})
        return {"sm_mhz": statistics.median(sm) if sm else None,
                "sm_max_mhz": num(win[0][1]), "power_w_max": max((num(p[2]) or 0) for p in win),
                "reasons": reasons, "samples": len(win), "scope": scope}


# ----------------------------------------------------------------- the GPU step
class Step:
    """Device buffers + workspaces for one batch, driven through the C ABI.

    Modes: "fused" (the default: spo_grpo_step, the whole path in one call;
    with several ranks, shard.DataParallelStep.run_fused: each rank's step
    weighted by 1/N on the device, dW all-reduced block by block while the
    backward's later blocks run), "separate" (the individual calls in turn),
    "kept" (the kept-exponential form), "vocab" (W's rows as slices: in turn
    on one GPU, or one slice per rank through shard.VocabParallelStep) and
    "forward" (log-probs and entropy only)."""

    def __init__(self, case, dev, dist=None, own_inputs=False, mode="fused", reserve_sms=8):
        from paper_2607_20908_gb300 import shard, spo
        self.spo = spo
        self.forward_only = case.get("forward_only", "cu_seqlens" not in case)
        self.mode = "forward" if self.forward_only else mode
        # data parallel over whole groups: every rank owns the same number of groups, so each
        # rank's share of Eq. 3's group average is exactly 1 / world
        self.dist = dist if dist is not None and dist.world > 1 else None
        self.world = dist.world if self.dist else 1
        self.rank = dist.rank if self.dist else 0
        self.L = spo.lib()
        self.dev = dev
        self.case = case
        T, d, V = case["T"], case["d"], case["V"]
        self.T, self.d, self.V = T, d, V
        # own_inputs: fresh device copies even where the case already sits on the device
        to = lambda t: t.to(dev, copy=own_inputs).contiguous()
        self.H, self.W = to(case["H"]), to(case["W"])
        self.tgt, self.mask = to(case["tgt"]), to(case["mask"])
        f32 = dict(dtype=torch.float32, device=dev)
        if self.forward_only:
            case = dict(case, cu_seqlens=torch.tensor([0, T], dtype=torch.int32),
                        group_id=torch.zeros(1, dtype=torch.int32), n_groups=1,
                        rewards=torch.zeros(1), old_noise=torch.zeros(T), ref_noise=torch.zeros(T),
                        window=0, clip_eps=0.2, kl_beta=0.0, forward_only=True)
            self.case = case
        self.n_seq = case["cu_seqlens"].numel() - 1
        self.n_groups = case["n_groups"]
        self.cu, self.gid = to(case["cu_seqlens"]), to(case["group_id"])
        self.rewards = to(case["rewards"])
        self.loss_mask = self.mask if self.forward_only else torch.empty(T, dtype=torch.uint8, device=dev)
        self.n_tok = torch.empty(self.n_seq, dtype=torch.int32, device=dev)
        self.logp, self.ent, self.lse = (torch.empty(T, **f32) for _ in range(3))
        self.adv = torch.empty(self.n_seq, **f32)
        self.loss, self.stats = torch.empty(1, **f32), torch.empty(4, **f32)
        self.g = torch.empty(T, **f32)
        self.dH = torch.empty((T, d), dtype=torch.bfloat16, device=dev)
        self.old = torch.empty(T, **f32)
        self.ref = torch.empty(T, **f32)
        self.ws_f = torch.empty(spo.logprobs_workspace_size(T, d, V), dtype=torch.uint8, device=dev)
        self.ws_l = self.ws_b = self.ws_s = self.keep = None
        self.slices = []
        if self.mode == "vocab":
            # one slice per rank (the rank's rows only), or every slice in turn on one GPU
            self.slices = shard.vocab_slices(V, max(2, self.world))
            if self.dist:
                off, n = self.slices[self.rank]
                self.v_offset = off
                self.W = self.W[off:off + n].contiguous()
                self.vstep = shard.VocabParallelStep(shard.SpoVocabEngine(reserve_sms), 0)
                self.dW = torch.empty((n, d), **f32)
            else:
                self.rec = torch.empty((len(self.slices), T, 4), **f32)
                self.dH_parts = [torch.empty((T, d), **f32) for _ in self.slices]
                self.dW = torch.empty((V, d), **f32)
            self.dH = torch.empty((T, d), **f32)   # the sum of the parts (fp32)
        elif not self.forward_only:
            self.dW = torch.empty((V, d), **f32)
        if self.mode == "kept":   # the forward keeps exp(z - tile max) for the backward
            self.keep = torch.empty(spo.logprobs_keep_size(T, V), dtype=torch.uint8, device=dev)
        if self.mode in ("separate", "kept", "vocab"):
            self.ws_l = torch.empty(max(256, spo.policy_loss_workspace_size(self.n_seq, self.n_groups)),
                                    dtype=torch.uint8, device=dev)
        if self.mode in ("separate", "vocab") and not self.dist:
            self.ws_b = torch.empty(spo.policy_loss_bwd_workspace_size(T, d, V), dtype=torch.uint8,
                                    device=dev)
        if self.mode == "fused":
            if self.dist:
                self.dp = shard.DataParallelStep(shard.SpoEngine(reserve_sms), 0, dw_blocks=4)
            else:
                self.ws_s = torch.empty(spo.grpo_workspace_size(T, d, V, self.n_seq, self.n_groups),
                                        dtype=torch.uint8, device=dev)
                self._structs()
        self.stream = torch.cuda.current_stream(dev)
        self.c_hooks = None   # spo_bwd_hooks for the one-call step (set by the end-to-end pipeline)

    def _structs(self):
        """The one-call step's argument blocks, built once (device pointers stay fixed)."""
        spo, c, p = self.spo, self.case, lambda t: ctypes.c_void_p(t.data_ptr())
        self.c_batch = spo.GrpoBatch(p(self.H), p(self.W), p(self.tgt), p(self.mask), p(self.cu),
                                     p(self.gid), p(self.rewards), p(self.old), p(self.ref), self.T,
                                     self.d, self.V, self.n_seq, self.n_groups)
        self.c_params = spo.GrpoParams(c["inv_temp"], c["window"], c["clip_eps"], c["kl_beta"], 0, 0,
                                       1e-6, None)
        self.c_out = spo.GrpoOutputs(p(self.loss), p(self.stats), p(self.logp), p(self.ent),
                                     p(self.lse), p(self.g), p(self.adv), p(self.loss_mask),
                                     p(self.dH), p(self.dW), 0)

    def prepare_old_ref(self):
        """Old / reference log-probs = current log-probs + noise (one forward, untimed)."""
        if self.forward_only:
            return
        L, p, c = self.L, lambda t: ctypes.c_void_p(t.data_ptr()), self.case
        s = ctypes.c_void_p(self.stream.cuda_stream)
        W, V = (self.case["W"].to(self.dev), self.V) if self.mode == "vocab" else (self.W, self.V)
        self.spo._check(L.spo_logprobs_fwd(p(self.H), p(W), p(self.tgt), p(self.mask), self.T,
                                           self.d, V, c["inv_temp"], p(self.logp), None, None,
                                           p(self.ws_f), self.ws_f.numel(), s))
        torch.cuda.synchronize(self.dev)
        self.old.copy_(self.logp + self.case["old_noise"].to(self.dev))
        self.ref.copy_(self.logp + self.case["ref_noise"].to(self.dev))

    def _rank_batch(self):
        c = self.case
        return dict(H=self.H, W=self.W, tgt=self.tgt, mask=self.mask, cu_seqlens=self.cu,
                    group_id=self.gid, n_groups=self.n_groups, rewards=self.rewards, old=self.old,
                    ref=self.ref, window=c["window"], inv_temp=c["inv_temp"],
                    clip_eps=c["clip_eps"], kl_beta=c["kl_beta"], dH_out=self.dH, dW_out=self.dW)

    def run(self):
        L, p, c = self.L, lambda t: ctypes.c_void_p(t.data_ptr()), self.case
        s = ctypes.c_void_p(self.stream.cuda_stream)
        chk = self.spo._check
        if self.forward_only:   # log-probs and entropy only (old-policy / rescoring pass)
            chk(L.spo_logprobs_fwd(p(self.H), p(self.W), p(self.tgt), p(self.mask), self.T, self.d,
                                   self.V, c["inv_temp"], p(self.logp), p(self.ent), p(self.lse),
                                   p(self.ws_f), self.ws_f.numel(), s))
            return
        if self.mode == "fused":
            if self.dist:       # whole groups per rank; the plan gives every rank 1/N of them
                self.loss, _, _ = self.dp.run_fused(self._rank_batch(), self.n_groups * self.world)
            else:
                R = ctypes.byref
                hooks = R(self.c_hooks) if self.c_hooks is not None else None
                chk(L.spo_grpo_step(R(self.c_batch), R(self.c_params), R(self.c_out), hooks,
                                    p(self.ws_s), self.ws_s.numel(), s))
            return
        if self.mode == "vocab" and self.dist:
            b = self._rank_batch()
            b.update(W_slice=self.W, v_offset=self.v_offset)
            self.loss, self.logp, self.dH, self.dW = self.vstep.run(b)
            return
        chk(L.spo_token_select(p(self.cu), p(self.mask), p(self.tgt), self.n_seq, self.T, c["window"],
                               p(self.loss_mask), p(self.n_tok), s))
        if self.slices:
            for k, (off, n) in enumerate(self.slices):
                chk(L.spo_logprobs_fwd_slice(p(self.H), p(self.W[off:off + n]), p(self.tgt),
                                             p(self.loss_mask), self.T, self.d, n, off, c["inv_temp"],
                                             p(self.rec[k]), p(self.ws_f), self.ws_f.numel(), s))
            chk(L.spo_logprobs_merge_slices(p(self.rec), len(self.slices), self.T, p(self.logp),
                                            p(self.ent), p(self.lse), s))
        elif self.keep is not None:
            chk(L.spo_logprobs_fwd_keep(p(self.H), p(self.W), p(self.tgt), p(self.loss_mask),
                                        self.T, self.d, self.V, c["inv_temp"], p(self.logp),
                                        p(self.ent), p(self.lse), p(self.keep), self.keep.numel(),
                                        p(self.ws_f), self.ws_f.numel(), s))
        else:
            chk(L.spo_logprobs_fwd(p(self.H), p(self.W), p(self.tgt), p(self.loss_mask), self.T,
                                   self.d, self.V, c["inv_temp"], p(self.logp), p(self.ent),
                                   p(self.lse), p(self.ws_f), self.ws_f.numel(), s))
        chk(L.spo_group_advantages(p(self.rewards), p(self.gid), self.n_seq, self.n_groups, 0, 1e-6,
                                   p(self.adv), s))
        chk(L.spo_policy_loss_fwd(p(self.logp), p(self.old), p(self.ref), p(self.adv), p(self.cu),
                                  p(self.gid), self.n_seq, self.n_groups, p(self.loss_mask), self.T,
                                  c["clip_eps"], c["kl_beta"], 0, p(self.loss), p(self.g),
                                  p(self.stats), p(self.ws_l), self.ws_l.numel(), s))
        if self.slices:
            for k, (off, n) in enumerate(self.slices):
                chk(L.spo_policy_loss_bwd_slice(p(self.H), p(self.W[off:off + n]), p(self.tgt),
                                                p(self.lse), p(self.g), self.T, self.d, n, off,
                                                c["inv_temp"], p(self.dH_parts[k]),
                                                p(self.dW[off:off + n]), 0, p(self.ws_b),
                                                self.ws_b.numel(), s))
            # stands in for the ranks' all-reduce of their dH parts
            with torch.cuda.stream(self.stream):
                torch.add(self.dH_parts[0], self.dH_parts[1], out=self.dH)
                for part in self.dH_parts[2:]:
                    self.dH.add_(part)
        elif self.keep is not None:
            chk(L.spo_policy_loss_bwd_kept(p(self.W), p(self.lse), p(self.g), self.T, self.d,
                                           self.V, c["inv_temp"], p(self.keep), self.keep.numel(),
                                           p(self.ws_f), self.ws_f.numel(), p(self.dH), p(self.dW),
                                           0, s))
        else:
            chk(L.spo_policy_loss_bwd(p(self.H), p(self.W), p(self.tgt), p(self.lse), p(self.g),
                                      self.T, self.d, self.V, c["inv_temp"], p(self.dH),
                                      p(self.dW), 0, p(self.ws_b), self.ws_b.numel(), s))


class HostIO:
    """End-to-end step from host buffers: every input copied host -> device and
    every output copied device -> host, pipelined over `sets` device buffer
    sets so that the copies of one step overlap the compute of its neighbours
    (H2D and D2H each on their own stream, compute on the step's stream).  A
    set is reused `sets` steps later, which is the time its copies have: host
    copies on this platform stall now and then for tens of milliseconds, and
    four sets give a step's copies three steps of compute to land in.  With
    the one-call step on one GPU, dH and each dW vocabulary block leave as soon
    as the step's hook events mark them final."""

    def __init__(self, st: "Step", sets: int = 4, set_bytes: int = 0, reserve_sms: int = 8,
                 dw_blocks: int = 4):
        # at most what fits in 70 % of the free device memory (a set of the large
        # workload in the kept form holds ~60 GB), never fewer than two
        if set_bytes > 0:
            free, _ = torch.cuda.mem_get_info(st.dev)
            sets = max(2, min(sets, 1 + int(0.7 * free) // set_bytes))
        self.n = sets
        # every set owns its inputs: a step's copies in must not land in a buffer
        # another step's kernels are reading
        self.sets = [st] + [Step(st.case, st.dev, st.dist, own_inputs=True, mode=st.mode,
                                 reserve_sms=reserve_sms) for _ in range(sets - 1)]
        for x in self.sets[1:]:
            x.old.copy_(st.old)
            x.ref.copy_(st.ref)
        pinned = lambda t: torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        if st.forward_only:
            ins = lambda x: (x.H, x.W, x.tgt, x.mask)
            outs = lambda x: (x.logp, x.ent, x.lse)
        else:
            ins = lambda x: (x.H, x.W, x.tgt, x.mask, x.cu, x.gid, x.rewards, x.old, x.ref)
            if st.dist and st.mode == "vocab":       # the rank's results
                outs = lambda x: (x.loss, x.logp, x.dH, x.dW)
            elif st.dist:
                outs = lambda x: (x.loss, x.dH, x.dW)
            else:
                outs = lambda x: (x.loss, x.stats, x.logp, x.ent, x.dH, x.dW)
        # outputs are looked up after each step: a multi-rank step may hand back new tensors
        self.outs = outs
        self.host_in = [pinned(t).copy_(t) for t in ins(st)]
        self.host_out = [[pinned(t) for t in outs(st)] for _ in self.sets]
        self.dev_in = [ins(x) for x in self.sets]
        self.h2d = sum(t.numel() * t.element_size() for t in self.host_in)
        self.d2h = sum(t.numel() * t.element_size() for t in self.host_out[0])
        self.compute = st.stream
        self.s_in = torch.cuda.Stream(st.dev)
        self.s_out = torch.cuda.Stream(st.dev)
        for x in self.sets:
            x.stream = self.compute
        mk = lambda: [torch.cuda.Event() for _ in range(sets)]
        self.in_done, self.comp_done, self.out_done = mk(), mk(), mk()
        self.i = 0
        # One GPU, one-call step: the step records an event when dH is final and
        # one per vocabulary block of dW (spo_bwd_hooks), and each slice is copied
        # out as soon as its event fires, while the rest of the backward runs.
        # Only the last block's copy is left after the last step's compute.
        self.blocks = None
        if st.mode == "fused" and not st.dist and not st.forward_only and dw_blocks > 0:
            spo = st.spo
            self.starts = spo.dw_block_starts(st.V, dw_blocks)
            self.blocks = []
            for x in self.sets:
                dh_ev, dw_ev = torch.cuda.Event(), [torch.cuda.Event() for _ in range(dw_blocks)]
                x.c_hooks = spo.make_hooks(dw_blocks, dw_ev, dh_ev, reserve_sms=0)
                self.blocks.append((dh_ev, dw_ev))

    def step(self):
        b = self.i % self.n
        x = self.sets[b]
        if self.i >= self.n:
            self.s_in.wait_event(self.comp_done[b])     # set b's inputs no longer read
        with torch.cuda.stream(self.s_in):
            for d, h in zip(self.dev_in[b], self.host_in):
                d.copy_(h, non_blocking=True)
            self.in_done[b].record(self.s_in)
        self.compute.wait_event(self.in_done[b])
        if self.i >= self.n:
            self.compute.wait_event(self.out_done[b])   # set b's outputs already copied out
        x.run()
        self.comp_done[b].record(self.compute)
        outs, host = self.outs(x), self.host_out[b]
        with torch.cuda.stream(self.s_out):
            if self.blocks is not None:   # (loss, stats, logp, ent, dH, dW): dH and dW early
                dh_ev, dw_ev = self.blocks[b]
                self.s_out.wait_event(dh_ev)
                host[4].copy_(outs[4], non_blocking=True)
                for k, ev in enumerate(dw_ev):
                    v0, v1 = self.starts[k], self.starts[k + 1]
                    if v1 > v0:
                        self.s_out.wait_event(ev)
                        host[5][v0:v1].copy_(outs[5][v0:v1], non_blocking=True)
                outs, host = outs[:4], host[:4]
            self.s_out.wait_event(self.comp_done[b])
            for d, h in zip(outs, host):
                h.copy_(d, non_blocking=True)
            self.out_done[b].record(self.s_out)
        self.i += 1


def timed_e2e(hio: HostIO, K, dist, dev):
    """Times K end-to-end steps: from before the first copy in to after the last copy out."""
    dist.barrier()
    torch.cuda.synchronize(dev)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    a.record(hio.s_in)
    hio.compute.wait_event(a)
    hio.s_out.wait_event(a)
    for _ in range(K):
        hio.step()
    hio.s_in.wait_stream(hio.s_out)
    hio.s_in.wait_stream(hio.compute)
    b.record(hio.s_in)
    torch.cuda.synchronize(dev)
    dist.barrier()
    return dist.max(a.elapsed_time(b), dev)


def timed(fn, K, dist, dev, stream):
    dist.barrier()
    torch.cuda.synchronize(dev)
    a, b = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    t0 = time.time()
    a.record(stream)
    for _ in range(K):
        fn()
    b.record(stream)
    torch.cuda.synchronize(dev)
    t1 = time.time()
    dist.barrier()
    return dist.max(a.elapsed_time(b), dev), t0, t1


# ----------------------------------------------------------------- CPU sample (oracle)
def cpu_sample(H, W, tgt, cu, rewards, old, ref, case):
    """One group of SAMPLE_SEQS rollouts, the first SAMPLE_TOKENS tokens of each (full d, V)."""
    rows = np.concatenate([np.arange(int(cu[i]), int(cu[i]) + SAMPLE_TOKENS) for i in range(SAMPLE_SEQS)])
    n = rows.size
    return dict(
        H=H[rows], W=W, tgt=tgt[rows], mask=np.ones(n, np.uint8),
        cu=np.arange(0, n + 1, SAMPLE_TOKENS, dtype=np.int64), gid=np.zeros(SAMPLE_SEQS, np.int64),
        rewards=rewards[:SAMPLE_SEQS], old=old[rows], ref=ref[rows],
        eps=case["clip_eps"], beta=case["kl_beta"], tau=case["inv_temp"], n=n)


def oracle_step(O, s):
    return O.grpo_step(s["H"], s["W"], s["tgt"], s["mask"], s["cu"], s["gid"], 1, s["rewards"],
                       s["old"], s["ref"], s["eps"], s["beta"], s["tau"], 1024)


def sample_description(n):
    return (f"one group of {SAMPLE_SEQS} rollouts x first {SAMPLE_TOKENS} tokens = {n} loss tokens of "
            f"the same workload, full d=5120 and V=151936, whole path (a1-a8) in fp64 numpy/BLAS; "
            f"tokens/s extrapolated linearly in tokens")


def host_inputs_from_device(st: Step):
    """fp64 host copies of the step's inputs (exact bf16 widening done by torch)."""
    return (st.H.double().cpu().numpy(), st.W.double().cpu().numpy(), st.tgt.cpu().numpy(),
            st.cu.cpu().numpy(), st.rewards.double().cpu().numpy(), st.old.double().cpu().numpy(),
            st.ref.double().cpu().numpy())


def run_cpu_baseline(st: Step, budget_s: float = 12.0):
    from oracle import spo_oracle as O
    H, W, tgt, cu, rew, old, ref = host_inputs_from_device(st)
    s = cpu_sample(H, W, tgt, cu, rew, old, ref, st.case)
    oracle_step(O, s)  # warm (page-in, BLAS threads)
    reps, t0 = 0, time.perf_counter()
    while True:
        oracle_step(O, s)
        reps += 1
        el = time.perf_counter() - t0
        if el >= budget_s or reps >= 20:
            break
    return {"value": s["n"] * reps / el, "unit": UNIT, "cores": int(os.environ["OPENBLAS_NUM_THREADS"]),
            "kind": "oracle", "sample": sample_description(s["n"]) + f"; {reps} reps in {el:.1f} s"}


def read_ceiling_gbs(dev, nbytes, reps=15):
    """Achievable DRAM rate for one transfer of nbytes: a library copy
    (torch's vectorised copy kernel) that reads nbytes / 2 and writes
    nbytes / 2 -- the same kind of transfer as the measured copy peak, at the
    size a small HBM-bound step actually moves.  Each rep follows a 256 MB
    write that evicts L2; CUDA events as for the library's own launches.
    The copy peak itself is reached only by multi-GB transfers."""
    n = max(1, nbytes // 8)
    x = torch.rand(n, device=dev)
    y = torch.empty_like(x)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)
    ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
          for _ in range(reps)]
    for i, (a, b) in enumerate(ev):
        flush.fill_(i & 0xFF)
        a.record()
        y.copy_(x)
        b.record()
    torch.cuda.synchronize(dev)
    ms = sorted(a.elapsed_time(b) for a, b in ev[3:])[(reps - 3) // 2]
    return 2 * n * 4 / (ms / 1e3) / 1e9


def aux_measurements(dev, pk):
    """HBM-bound steps at enlarged synthetic sizes, outside the timed loop:
    the reward composition (section 2.2; 2^24 candidates, 21 algorithmic bytes
    each), the group advantages (2^24 rollouts in contiguous groups of 16,
    12 algorithmic bytes each: group id, reward, advantage) and the loss
    forward (2^24 tokens, 17 bytes each).  Each rep runs
    after a 256 MB write that evicts L2 and is timed on its own with CUDA
    events; the median is reported."""
    from paper_2607_20908_gb300 import spo
    n = 1 << 24
    gen = torch.Generator(device=dev).manual_seed(5)
    flush = torch.empty(256 << 20, dtype=torch.uint8, device=dev)

    def median_ms(fn, reps=12):
        for _ in range(3):
            fn()
        ev = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
              for _ in range(reps)]
        for i, (a, b) in enumerate(ev):
            flush.fill_(i & 0xFF)
            a.record()
            fn()
            b.record()
        torch.cuda.synchronize(dev)
        return sorted(a.elapsed_time(b) for a, b in ev)[reps // 2]

    compiled = (torch.rand(n, device=dev, generator=gen) < 0.8).to(torch.uint8)
    p = torch.where(torch.rand(n, device=dev, generator=gen) < 0.5, 1.0,
                    torch.rand(n, device=dev, generator=gen))
    S = torch.exp2(torch.rand(n, device=dev, generator=gen) * 11 - 3)
    cv = torch.rand(n, device=dev, generator=gen)
    rs = torch.randn(n, device=dev, generator=gen)
    out = torch.empty(n, device=dev)
    ms = median_ms(lambda: spo.spo_reward_compose(compiled, p, S, cv, rs, out=out))
    gbs = 21 * n / (ms / 1e3) / 1e9
    res = {"reward_compose": {"candidates": n, "ms": ms, "gbs": gbs, "frac_of_hbm": gbs / pk["hbm"],
                              "bound": "hbm",
                              "note": "enlarged synthetic size; the workload itself has 128 rollouts"}}
    del compiled, p, S, cv, rs, out

    groups = n // 16
    gid = torch.arange(n, device=dev, dtype=torch.int32) // 16
    r = torch.randn(n, device=dev, generator=gen)
    adv = torch.empty(n, device=dev)
    ws = torch.empty(spo.group_advantages_workspace_size(n, groups), dtype=torch.uint8, device=dev)
    ms = median_ms(lambda: spo.spo_group_advantages_ws(r, gid, groups, adv=adv, ws=ws))
    gbs = 12 * n / (ms / 1e3) / 1e9
    res["group_advantages"] = {"rollouts": n, "groups": groups, "ms": ms, "gbs": gbs,
                               "frac_of_hbm": gbs / pk["hbm"], "bound": "issue",
                               "note": "enlarged synthetic size, sorted contiguous groups of 16 "
                                       "(spo_group_advantages_ws); issue- and latency-bound block "
                                       "program (stage, search, fold in the fp32 order, store); "
                                       "a step has 128-640 sequences"}
    del gid, r, adv, ws

    # a5 at 2^24 loss tokens (131072 sequences of 128, groups of 8): per token
    # logp, old, ref (fp32), the loss mask (u8) in and g (fp32) out = 17 bytes
    L = 128
    ns = n // L
    ng = ns // 8
    cu = torch.arange(0, n + 1, L, device=dev, dtype=torch.int32)
    gid = torch.arange(ns, device=dev, dtype=torch.int32) // 8
    lp = -8.0 * torch.rand(n, device=dev, generator=gen)
    old = lp + 0.05 * torch.randn(n, device=dev, generator=gen)
    ref = lp + 0.05 * torch.randn(n, device=dev, generator=gen)
    a_seq = torch.randn(ns, device=dev, generator=gen)
    lm = torch.ones(n, dtype=torch.uint8, device=dev)
    ws = torch.empty(spo.policy_loss_workspace_size(ns, ng), dtype=torch.uint8, device=dev)
    ms = median_ms(lambda: spo.spo_policy_loss_fwd(lp, old, ref, a_seq, cu, gid, ng, lm, 0.2, 0.04,
                                                   ws=ws))
    alg = 17 * n + 12 * ns
    gbs = alg / (ms / 1e3) / 1e9
    res["policy_loss_fwd"] = {"tokens": n, "sequences": ns, "groups": ng, "ms": ms, "gbs": gbs,
                              "frac_of_hbm": gbs / pk["hbm"], "bound": "hbm",
                              "note": "enlarged synthetic size; a step has 16384-131072 tokens"}
    del cu, gid, lp, old, ref, a_seq, lm, ws

    # a3 at the large workload's 131072 rows x 594 vocabulary tiles (936 MB of partials), timed
    # by the library's own events around the combine launch inside a forward at d = 256
    T2, d2, V2 = 131072, 256, 151936
    H2 = torch.randn(T2, d2, device=dev, generator=gen).to(torch.bfloat16)
    W2 = (torch.randn(V2, d2, device=dev, generator=gen) * 0.02).to(torch.bfloat16)
    tgt2 = torch.randint(0, V2, (T2,), device=dev, generator=gen, dtype=torch.int32)
    ws2 = torch.empty(spo.logprobs_workspace_size(T2, d2, V2), dtype=torch.uint8, device=dev)
    fwd = lambda: spo.spo_logprobs_fwd(H2, W2, tgt2, ws=ws2)
    for _ in range(2):
        fwd()
    torch.cuda.synchronize(dev)
    spo.spo_trace_read()
    spo.spo_trace_enable(True)
    try:
        for i in range(6):
            flush.fill_(i & 0xFF)
            fwd()
        torch.cuda.synchronize(dev)
        recs = spo.spo_trace_read()
    finally:
        spo.spo_trace_enable(False)
    comb = sorted(t for k, t in recs if KERNEL_NAMES.get(k) == "lse_combine")
    ms = comb[len(comb) // 2]
    nbytes = T2 * (12 * ((V2 + 255) // 256) + 20)
    gbs = nbytes / (ms / 1e3) / 1e9
    res["lse_combine"] = {"rows": T2, "vocab_tiles": (V2 + 255) // 256, "ms": ms, "gbs": gbs,
                          "frac_of_hbm": gbs / pk["hbm"], "bound": "hbm",
                          "note": "the large workload's row count (the full workload's 16384 rows "
                                  "move 117 MB, where launch and ramp weigh); partials written by "
                                  "the forward just before, so part of them may sit in L2"}
    return res


# ----------------------------------------------------------------- arms
def config_block(case, T_L, world, workload="full", mode="fused", tunings=()):
    cfg = {"workload": WORKLOADS[workload], "T": case["T"], "loss_tokens": T_L, "d": case["d"],
           "V": case["V"]}
    if workload == "full":
        cfg.update(groups=case["n_groups"], rollouts_per_group=8, tokens_per_rollout=128)
    elif workload != "forward":
        cfg.update(groups=case["n_groups"], sequences=int(case["cu_seqlens"].numel() - 1))
    if workload != "forward":
        cfg.update(clip_eps=case["clip_eps"], kl_beta=case["kl_beta"], window=case["window"])
    if case.get("vocab_slices"):
        cfg["vocab_slices"] = case["vocab_slices"]
    if case.get("keep"):
        cfg["kept_exponentials"] = "forward keeps exp(z - tile max) in bf16; backward forms G from it"
    cfg["l2"] = "inputs larger than L2 (W alone is 1.2-1.56 GB and is streamed every step)"
    if tunings:
        cfg["tunings"] = {str(k): v for k, v in tunings}
    cfg["call"] = {"fused": "spo_grpo_step: the whole path (a1-a8) in one C-ABI call per step",
                   "separate": "spo_token_select, spo_logprobs_fwd, spo_group_advantages, "
                               "spo_policy_loss_fwd, spo_policy_loss_bwd in turn",
                   "kept": "the kept-exponential forward and backward calls",
                   "vocab": "per-slice forward, record merge, loss, per-slice backward",
                   "forward": "spo_logprobs_fwd"}[mode]
    if world == 1:
        cfg["parallelism"] = "1 GPU"
    elif workload == "vocab-split":
        cfg["parallelism"] = (f"tp{world}: W's rows split over the GPUs, the batch on every GPU; "
                              "per-token records all-gathered (NCCL), dH all-reduced while the "
                              "rank's dW GEMMs run")
    else:
        cfg["parallelism"] = (f"dp{world}: whole groups per GPU, each rank's loss and g weighted "
                              "1/N on the device; dW all-reduced (NCCL) in 4 vocabulary blocks, "
                              "each as soon as the backward has finished it, while the later "
                              "blocks' GEMMs run; loss all-reduced")
    return cfg


def ours(args):
    dist = Dist()
    dev = torch.device("cuda", dist.local)
    torch.cuda.set_device(dev)
    dist.init("nccl", dev)
    from paper_2607_20908_gb300 import build, spo
    if dist.rank == 0 and not os.path.exists(spo.LIB_PATH):
        build.build()
    dist.barrier()
    maker = {"full": inputs.full_case, "forward": inputs.forward_case, "ragged": inputs.ragged_case,
             "large": inputs.large_case, "vocab-split": inputs.full_case,
             "kept": inputs.full_case}[args.workload]
    seed0 = {"full": 1003, "forward": 1002, "ragged": 1004, "large": 1005,
             "vocab-split": 1003, "kept": 1003}[args.workload]
    # data parallel: every rank its own batch (weak scaling); vocabulary split: one batch, W's
    # rows split over the ranks (strong scaling)
    vocab_ranks = args.workload == "vocab-split" and dist.world > 1
    case = maker(seed=seed0 + (0 if vocab_ranks else dist.rank), device=str(dev))
    mode = "fused"
    if args.workload == "vocab-split":
        case["vocab_slices"] = max(2, dist.world)
        mode = "vocab"
    if args.workload == "kept" or args.keep:
        if args.workload in ("forward", "vocab-split"):
            raise SystemExit(f"--keep does not apply to --workload {args.workload}")
        case["keep"] = True
        mode = "kept"
    if args.separate_calls and mode == "fused":
        mode = "separate"
    if dist.world > 1 and (args.workload == "forward" or mode in ("kept", "separate")):
        raise SystemExit(f"--workload {args.workload} ({mode}) runs on one GPU")
    tunings = [tuple(int(x) for x in kv.split("=")) for kv in args.tune.split(",") if kv]
    for key, value in tunings:
        spo.spo_set_tuning(key, value)
    base_bytes = torch.cuda.memory_allocated(dev)
    st = Step(case, dev, dist, mode=mode, reserve_sms=args.reserve_sms)
    step_bytes = (torch.cuda.memory_allocated(dev) - base_bytes      # one buffer set:
                  + sum(t.numel() * t.element_size() for t in (st.H, st.W)))  # + its own H, W
    st.prepare_old_ref()
    torch.cuda.synchronize(dev)
    if st.forward_only:
        T_L = int(st.mask.sum().item())
    else:   # loss tokens: the same selection the step makes (untimed)
        lm, _ = spo.spo_token_select(st.cu, st.mask, st.tgt, case["window"])
        T_L = int(lm.sum().item())
    V_rank = st.W.shape[0]                       # this rank's vocabulary rows
    flop_gemm = 2.0 * T_L * st.d * V_rank        # one GEMM-equivalent on this GPU (algorithmic)
    # fwd + dH + dW (the backward's recompute is not counted); the forward-only workload: fwd
    flop_metric = (1.0 if st.forward_only else 3.0) * flop_gemm
    pk = peaks()

    for _ in range(args.warmup):
        st.run()
    torch.cuda.synchronize(dev)
    assert spo.spo_device_error(dev) == 0, "device wait expired during warm-up"

    clocks = ClockSampler(dev)
    time.sleep(0.3)
    for _ in range(2):             # keep the GPU loaded while the sampler starts
        st.run()
    spo.spo_trace_enable(True)
    n0 = spo.spo_launch_count()
    ms, t0, t1 = timed(st.run, args.steps, dist, dev, st.stream)
    n_launch = spo.spo_launch_count() - n0
    spo.spo_trace_enable(False)
    clocks.stop()
    trace = spo.spo_trace_read()
    err = spo.spo_device_error(dev)
    assert err == 0, f"device wait expired (code {err:#x})"

    tokens_s = (1 if vocab_ranks else dist.world) * T_L * args.steps / (ms / 1e3)
    kern = {}
    for kind, t in trace:
        k = kern.setdefault(KERNEL_NAMES.get(kind, str(kind)), {"launches": 0, "total_ms": 0.0})
        k["launches"] += 1
        k["total_ms"] += t
    nsplit = (V_rank + 255) // 256
    hbm_bytes = {   # algorithmic bytes per call of the HBM-bound steps
        "lse_combine": 12 * nsplit * T_L + 8 * T_L + 12 * st.T,
        "select_gather_fwd": 4 * T_L * st.d + 5 * st.T + 8 * T_L,
        "select_gather_bwd": 4 * T_L * st.d + 12 * st.T + 16 * T_L,
        "form_g": 4 * T_L * st.V + 12 * T_L,   # kept form: E read, G written (bf16)
    }
    for name, k in kern.items():
        k["avg_ms"] = k["total_ms"] / k["launches"]
        k["share_of_step"] = k["total_ms"] / ms
        if name in GEMM_KINDS:
            # a GEMM may run as several launches per step (token chunks, dW passes)
            k["launches_per_step"] = k["launches"] / args.steps
            k["flop_per_launch"] = flop_gemm / k["launches_per_step"]
            k["tflops"] = k["flop_per_launch"] / (k["avg_ms"] / 1e3) / 1e12
        elif name in hbm_bytes:
            k["gbs"] = hbm_bytes[name] / (k["avg_ms"] / 1e3) / 1e9
            k["frac_of_hbm"] = k["gbs"] / pk["hbm"]
            k["algorithmic_bytes"] = hbm_bytes[name]
        else:
            k["bound"] = "latency"
            k["avg_us"] = k["avg_ms"] * 1e3
    dom_name, dom = max(((n, k) for n, k in kern.items() if n in GEMM_KINDS),
                        key=lambda kv: kv[1]["total_ms"])
    achieved = dom["tflops"]
    roofline = {"bound": "tensor", "kernel": dom_name, "achieved": achieved,
                "peak": pk["bf16_sustained"], "unit": "TFLOP/s", "frac": achieved / pk["bf16_sustained"],
                "peak_kind": f"bf16 dense sustained, {pk['source']}",
                "frac_of_burst": achieved / pk["bf16_burst"],
                "flop_per_launch": dom["flop_per_launch"], "traffic": kernel_traffic(dom_name),
                "traffic_unit": "bytes per launch (ncu dram__bytes_read.sum + dram__bytes_write.sum)",
                "traffic_source": TRAFFIC["derivation"],
                "algorithmic_bytes": None}
    Vr = V_rank   # the vocabulary rows this GPU's GEMMs cover
    alg = {"logits_lse_fwd": 2 * T_L * st.d + 2 * Vr * st.d + 12 * T_L * nsplit,
           "logits_grad_recompute": 2 * T_L * st.d + 2 * Vr * st.d + 2 * T_L * Vr,
           "gemm_dH": 2 * T_L * Vr + 2 * Vr * st.d + 2 * T_L * st.d,
           "gemm_dW": 2 * T_L * Vr + 2 * T_L * st.d + 4 * Vr * st.d}
    # per launch: a step's operand and output bytes spread over its launches of that GEMM
    roofline["algorithmic_bytes"] = alg[dom_name] / dom["launches_per_step"]
    for name, k in kern.items():
        if name in alg:
            k["dram_bytes_ncu"] = kernel_traffic(name)
            k["algorithmic_bytes"] = alg[name] / k["launches_per_step"]

    for name, k in kern.items():
        if name in hbm_bytes:
            k["read_ceiling_gbs"] = read_ceiling_gbs(dev, hbm_bytes[name])
            k["frac_of_read_ceiling"] = k["gbs"] / k["read_ceiling_gbs"]

    # e2e: host buffers, H2D + step + D2H inside the timed region
    hio = HostIO(st, sets=args.e2e_sets, set_bytes=step_bytes, reserve_sms=args.reserve_sms,
                 dw_blocks=args.e2e_dw_blocks)
    for _ in range(hio.n):
        hio.step()
    ms_e2e = timed_e2e(hio, args.steps, dist, dev)
    e2e = {"value": (1 if vocab_ranks else dist.world) * T_L * args.steps / (ms_e2e / 1e3),
           "unit": UNIT,
           "h2d_bytes_per_step": hio.h2d, "d2h_bytes_per_step": hio.d2h,
           "ms_per_step": ms_e2e / args.steps,
           "path": ("pinned host -> device copies of every input (H, W, targets, mask), the C-ABI "
                    "call, device -> host copies of logp, entropy, lse"
                    if st.forward_only else
                    "pinned host -> device copies of every input (H, W, ids, masks, rewards, old/ref "
                    "log-probs), the C-ABI calls, device -> host copies of loss, stats, logp, "
                    "entropy, dH, dW")
                   + f"; {hio.n} buffer sets so a step's copies overlap the compute of the steps "
                     "around it"
                   + (f"; dH and each of {len(hio.starts) - 1} vocabulary blocks of dW copied out "
                      "as soon as the step's hook events mark them final"
                      if hio.blocks is not None else "")}

    line = {
        "metric": METRIC_FWD if st.forward_only else METRIC, "value": tokens_s, "unit": UNIT,
        "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": ms / args.steps, "higher_is_better": True,
        "scaling": "strong" if vocab_ranks else "weak", "vs_baseline": None, "dtype": "bf16",
        "data": "synthetic (seeded; H~N(0,1), W~N(0,0.02^2) rounded to bf16: random-init stand-in for "
                "the policy's final hidden states and LM head)",
        "config": config_block(case, T_L, dist.world, args.workload, mode, tunings),
        "tensor_peak_frac": {"metric_tflops": flop_metric * args.steps / (ms / 1e3) / 1e12,
                             "of_burst": flop_metric * args.steps / (ms / 1e3) / 1e12 / pk["bf16_burst"],
                             "of_sustained": flop_metric * args.steps / (ms / 1e3) / 1e12 / pk["bf16_sustained"],
                             "flop_per_step": flop_metric,
                             "note": ("algorithmic 2*T*d*V per step (forward only)" if st.forward_only else
                                      "algorithmic 3 x 2*T*d*V per step; the backward's logit "
                                      "recompute is done but not counted")},
        "roofline": roofline,
        "kernels": kern,
        "e2e": e2e,
        "gpu_launches": n_launch,
        "launches_per_step": n_launch / args.steps,
        "clocks": clocks.summary(t0, t1),
    }
    if args.workload == "full":
        line["aux"] = aux_measurements(dev, pk)
    if dist.rank == 0 and dist.world == 1 and not args.no_cpu_baseline and args.workload == "full":
        line["cpu_baseline"] = run_cpu_baseline(st)
    if dist.rank == 0:
        print(json.dumps(line), flush=True)
    dist.close()


def reference(args):
    dist = Dist()
    if dist.rank != 0:
        return
    from oracle import spo_oracle as O
    dev = torch.device("cuda", dist.local) if torch.cuda.is_available() else torch.device("cpu")
    case = inputs.full_case(seed=1003, device=str(dev))
    # inputs (H, W on the device when there is one, else on the host); old/ref = noise around a
    # reference log-prob level, since the sample never sees the GPU path
    H = case["H"].double().cpu().numpy()
    W = case["W"].double().cpu().numpy()
    del case["H"], case["W"]
    tgt, cu = case["tgt"].numpy(), case["cu_seqlens"].numpy()
    s0 = cpu_sample(H, W, tgt, cu, case["rewards"].double().numpy(), np.zeros(case["T"]),
                    np.zeros(case["T"]), case)
    lp, _, _ = O.logprobs(s0["H"], s0["W"], s0["tgt"], s0["tau"])
    rows_noise_old = case["old_noise"].double().numpy()[:s0["n"]]
    rows_noise_ref = case["ref_noise"].double().numpy()[:s0["n"]]
    s0["old"], s0["ref"] = lp + rows_noise_old, lp + rows_noise_ref
    for _ in range(args.warmup):
        oracle_step(O, s0)
    t0 = time.perf_counter()
    for _ in range(args.steps):
        oracle_step(O, s0)
    el = time.perf_counter() - t0
    val = s0["n"] * args.steps / el
    line = {
        "metric": METRIC, "value": val, "unit": UNIT, "n_gpus": dist.world, "steps": args.steps,
        "warmup": args.warmup, "ms_per_step": el * 1e3 / args.steps, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": "f64", "impl": "reference",
        "data": "synthetic (same seeded workload as the GPU arm)",
        "config": config_block(case, case["T"], 1),
        "cpu_baseline": {"value": val, "unit": UNIT, "cores": int(os.environ["OPENBLAS_NUM_THREADS"]),
                         "kind": "oracle", "sample": sample_description(s0["n"]) + " per step"},
        "e2e": {"value": val, "unit": UNIT, "h2d_bytes_per_step": 0, "d2h_bytes_per_step": 0},
    }
    print(json.dumps(line), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=30)
    ap.add_argument("--warmup", type=int, default=3)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--no-cpu-baseline", action="store_true", help="skip the oracle timing")
    ap.add_argument("--e2e-sets", type=int, default=4,
                    help="device buffer sets the end-to-end pipeline rotates through")
    ap.add_argument("--e2e-dw-blocks", type=int, default=4,
                    help="one GPU, one-call step: vocabulary blocks of dW copied out as each becomes "
                         "final (spo_bwd_hooks events); 0 = every output after the step")
    ap.add_argument("--keep", action="store_true",
                    help="kept-exponential form (spo_logprobs_fwd_keep / spo_policy_loss_bwd_kept) "
                         "for a forward + backward workload")
    ap.add_argument("--workload", choices=sorted(WORKLOADS), default="full",
                    help="supplementary workloads; the default is the one the metric is quoted on")
    ap.add_argument("--separate-calls", action="store_true",
                    help="run the step as the separate C-ABI calls instead of spo_grpo_step")
    ap.add_argument("--tune", type=str, default="",
                    help="launch tunings applied first, 'key=value' pairs (spo_tune_key numbers) "
                         "separated by ','; results do not depend on them")
    ap.add_argument("--reserve-sms", type=int, default=8,
                    help="with several GPUs: SMs the GEMMs that overlap a collective leave free")
    args = ap.parse_args()
    if args.warmup < 3:
        ap.error("--warmup must be >= 3")
    if args.impl == "reference":
        reference(args)
    else:
        ours(args)


if __name__ == "__main__":
    main()
