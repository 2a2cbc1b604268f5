"""Thin Python binding of libspo (include/spo.h) over PyTorch tensors.

Argument marshalling only: every function checks dtypes / devices /
contiguity, allocates the outputs and the workspace with torch (the library
itself never allocates), and forwards raw device pointers plus the current
CUDA stream to the C entry point of the same name.  All computation happens
in libspo's CUDA kernels; there is no fallback path.  If the shared library
is not built, every call raises.
"""

from __future__ import annotations

import ctypes
import os

import torch

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "lib", "libspo.so")

SPO_AGG_SEQ_GROUP = 0
SPO_AGG_TOKEN = 1
SPO_STD_UNBIASED = 0
SPO_STD_POPULATION = 1

_lib = None

_c_size = ctypes.c_size_t
_vp = ctypes.c_void_p
_i32 = ctypes.c_int32
_i64 = ctypes.c_int64
_f32 = ctypes.c_float

_SIGS = {
    "spo_version": ([], ctypes.c_int),
    "spo_status_string": ([ctypes.c_int], ctypes.c_char_p),
    "spo_last_error": ([ctypes.c_char_p, _c_size], ctypes.c_int),
    "spo_device_error": ([ctypes.POINTER(ctypes.c_int), _vp], ctypes.c_int),
    "spo_token_select": ([_vp, _vp, _vp, _i32, _i64, _i32, _vp, _vp, _vp], ctypes.c_int),
    "spo_logprobs_workspace_size": ([_i64, _i64, _i64, ctypes.POINTER(_c_size)], ctypes.c_int),
    "spo_logprobs_fwd": ([_vp, _vp, _vp, _vp, _i64, _i64, _i64, _f32, _vp, _vp, _vp, _vp, _c_size,
                          _vp], ctypes.c_int),
    "spo_group_advantages": ([_vp, _vp, _i32, _i32, ctypes.c_int, _f32, _vp, _vp], ctypes.c_int),
    "spo_policy_loss_workspace_size": ([_i32, _i32, ctypes.POINTER(_c_size)], ctypes.c_int),
    "spo_policy_loss_fwd": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _i64, _f32, _f32,
                             ctypes.c_int, _vp, _vp, _vp, _vp, _c_size, _vp], ctypes.c_int),
    "spo_policy_loss_bwd_workspace_size": ([_i64, _i64, _i64, ctypes.POINTER(_c_size)],
                                           ctypes.c_int),
    "spo_policy_loss_bwd": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i64, _f32, _vp, _vp,
                             ctypes.c_int, _vp, _c_size, _vp], ctypes.c_int),
    "spo_trace_enable": ([ctypes.c_int], ctypes.c_int),
    "spo_trace_read": ([ctypes.POINTER(ctypes.c_int), ctypes.POINTER(ctypes.c_float), ctypes.c_int,
                        ctypes.POINTER(ctypes.c_int)], ctypes.c_int),
    "spo_launch_count": ([], ctypes.c_longlong),
    "spo_set_tuning": ([ctypes.c_int, ctypes.c_int64], ctypes.c_int),
    "spo_reward_compose": ([_vp, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp], ctypes.c_int),
    "spo_ranker_scores": ([_vp, _vp, _vp, _i32, _vp, _vp, _vp], ctypes.c_int),
    "spo_scale_f32": ([_vp, _i64, _f32, _vp, _vp], ctypes.c_int),
    "spo_validate_inputs": ([_vp, _i64, _i64, _vp, _i32, _vp, _i32, _vp, _vp, _vp, _vp, _vp, _vp],
                            ctypes.c_int),
    "spo_ranker_workspace_size": ([_i32, ctypes.POINTER(_c_size)], ctypes.c_int),
    "spo_ranker_pair_loss": ([_vp, _vp, _vp, _vp, _vp, _i32, _vp, _vp, _vp, _f32, _vp, _vp, _vp,
                              _c_size, _vp], ctypes.c_int),
    "spo_policy_loss_fwd_noalloc": ([_vp, _vp, _vp, _vp, _vp, _vp, _i32, _i32, _vp, _i64, _f32,
                                     _f32, ctypes.c_int, _vp, _vp, _vp, _vp], ctypes.c_int),
    "spo_selftest_bounded_wait": ([_vp], ctypes.c_int),
    "spo_logprobs_keep_size": ([_i64, _i64, ctypes.POINTER(_c_size)], ctypes.c_int),
    "spo_logprobs_fwd_keep": ([_vp, _vp, _vp, _vp, _i64, _i64, _i64, _f32, _vp, _vp, _vp, _vp,
                               _c_size, _vp, _c_size, _vp], ctypes.c_int),
    "spo_policy_loss_bwd_kept": ([_vp, _vp, _vp, _i64, _i64, _i64, _f32, _vp, _c_size, _vp,
                                  _c_size, _vp, _vp, ctypes.c_int, _vp], ctypes.c_int),
    "spo_group_advantages_workspace_size": ([_i32, _i32, ctypes.POINTER(_c_size)], ctypes.c_int),
    "spo_group_advantages_ws": ([_vp, _vp, _i32, _i32, ctypes.c_int, _f32, _vp, _vp, _c_size, _vp],
                                ctypes.c_int),
    "spo_logprobs_fwd_slice": ([_vp, _vp, _vp, _vp, _i64, _i64, _i64, _i64, _f32, _vp, _vp,
                                _c_size, _vp], ctypes.c_int),
    "spo_logprobs_merge_slices": ([_vp, _i32, _i64, _vp, _vp, _vp, _vp], ctypes.c_int),
    "spo_policy_loss_bwd_slice": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i64, _i64, _f32, _vp,
                                   _vp, ctypes.c_int, _vp, _c_size, _vp], ctypes.c_int),
    "spo_last_error_detail": ([ctypes.c_char_p, _c_size], ctypes.c_int),
    "spo_sync_check": ([_vp], ctypes.c_int),
    "spo_scale_f32_ratio": ([_vp, _i64, _vp, _vp, _vp], ctypes.c_int),
    "spo_dw_block_starts": ([_i64, _i32, ctypes.POINTER(_i64)], ctypes.c_int),
    "spo_policy_loss_bwd_ex": ([_vp, _vp, _vp, _vp, _vp, _i64, _i64, _i64, _i64, _f32, _vp,
                                ctypes.c_int, _vp, ctypes.c_int, _vp, _vp, _c_size, _vp],
                               ctypes.c_int),
    "spo_grpo_workspace_size": ([_i64, _i64, _i64, _i32, _i32, ctypes.POINTER(_c_size)],
                                ctypes.c_int),
    "spo_grpo_step": ([_vp, _vp, _vp, _vp, _vp, _c_size, _vp], ctypes.c_int),
    "spo_workspace_size": ([_i64, _i64, _i64, _i32, ctypes.POINTER(_c_size)], ctypes.c_int),
}

TRACE_KINDS = {0: "logits_lse_fwd", 1: "logits_grad_recompute", 2: "gemm_dH", 3: "gemm_dW",
               4: "lse_combine", 5: "select_gather_fwd", 6: "select_gather_bwd",
               7: "policy_loss_fwd", 8: "group_advantages", 9: "token_select",
               10: "reward_compose", 11: "ranker", 12: "merge_slices", 13: "form_g"}


class SpoError(RuntimeError):
    def __init__(self, status: int, text: str):
        super().__init__(f"{status_string(status)}: {text}")
        self.status = status


def lib() -> ctypes.CDLL:
    """The loaded libspo.so (raises if it has not been built)."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"libspo.so not found at {LIB_PATH}: build it with "
                "`python -m paper_2607_20908_gb300.build` (the CUDA path has no fallback)")
        handle = ctypes.CDLL(LIB_PATH)
        for name, (args, res) in _SIGS.items():
            fn = getattr(handle, name)
            fn.argtypes = args
            fn.restype = res
        _lib = handle
    return _lib


def exported_symbols():
    return list(_SIGS)


def status_string(status: int) -> str:
    return lib().spo_status_string(int(status)).decode()


def _check(status: int):
    if status != 0:
        buf = ctypes.create_string_buffer(512)
        lib().spo_last_error(buf, 512)
        raise SpoError(status, buf.value.decode())


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _stream(device) -> ctypes.c_void_p:
    return ctypes.c_void_p(torch.cuda.current_stream(device).cuda_stream)


def _need(t, name, dtype, numel=None, device=None):
    if not isinstance(t, torch.Tensor):
        raise TypeError(f"{name} must be a torch.Tensor")
    if t.dtype != dtype:
        raise TypeError(f"{name} must be {dtype}, got {t.dtype}")
    if not t.is_cuda:
        raise ValueError(f"{name} must be on a CUDA device")
    if device is not None and t.device != device:
        raise ValueError(f"{name} is on {t.device}, expected {device}")
    if not t.is_contiguous():
        raise ValueError(f"{name} must be contiguous")
    if numel is not None and t.numel() != numel:
        raise ValueError(f"{name} has {t.numel()} elements, expected {numel}")
    return t


def _workspace(nbytes: int, device, ws=None):
    if ws is not None:
        if ws.numel() < nbytes or ws.dtype != torch.uint8:
            raise ValueError(f"workspace needs {nbytes} uint8 bytes")
        return ws
    return torch.empty(max(int(nbytes), 256), dtype=torch.uint8, device=device)


def spo_device_error(device=None) -> int:
    """Reads and clears the device error word (synchronises the current stream)."""
    device = torch.device(device or torch.cuda.current_device())
    code = ctypes.c_int(0)
    st = lib().spo_device_error(ctypes.byref(code), _stream(device))
    if st not in (0, 7):
        _check(st)
    return code.value


def spo_token_select(cu_seqlens, mask, tgt, window: int = 1024):
    """a1: loss-token mask and per-sequence loss-token counts."""
    dev = tgt.device
    T = tgt.numel()
    n_seq = cu_seqlens.numel() - 1
    _need(cu_seqlens, "cu_seqlens", torch.int32, device=dev)
    _need(tgt, "tgt", torch.int32)
    if mask is not None:
        _need(mask, "mask", torch.uint8, T, dev)
    loss_mask = torch.empty(T, dtype=torch.uint8, device=dev)
    n_tok = torch.empty(n_seq, dtype=torch.int32, device=dev)
    _check(lib().spo_token_select(_ptr(cu_seqlens), _ptr(mask), _ptr(tgt), n_seq, T, int(window),
                                  _ptr(loss_mask), _ptr(n_tok), _stream(dev)))
    return loss_mask, n_tok


def logprobs_workspace_size(T: int, d: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_logprobs_workspace_size(T, d, V, ctypes.byref(n)))
    return n.value


def spo_logprobs_fwd(H, W, tgt, mask=None, inv_temp: float = 1.0, ws=None, want_entropy=True):
    """a2+a3: returns (logp, entropy or None, lse), fp32[T]."""
    dev = H.device
    T, d = H.shape
    V = W.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W, "W", torch.bfloat16, device=dev)
    if W.shape[1] != d:
        raise ValueError(f"W has {W.shape[1]} columns, H has {d}")
    _need(tgt, "tgt", torch.int32, T, dev)
    if mask is not None:
        _need(mask, "mask", torch.uint8, T, dev)
    logp = torch.empty(T, dtype=torch.float32, device=dev)
    ent = torch.empty(T, dtype=torch.float32, device=dev) if want_entropy else None
    lse = torch.empty(T, dtype=torch.float32, device=dev)
    nbytes = logprobs_workspace_size(T, d, V)
    w = _workspace(nbytes, dev, ws)
    _check(lib().spo_logprobs_fwd(_ptr(H), _ptr(W), _ptr(tgt), _ptr(mask), T, d, V,
                                  float(inv_temp), _ptr(logp), _ptr(ent), _ptr(lse), _ptr(w),
                                  w.numel(), _stream(dev)))
    return logp, ent, lse


def logprobs_keep_size(T: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_logprobs_keep_size(T, V, ctypes.byref(n)))
    return n.value


def spo_logprobs_fwd_keep(H, W, tgt, mask=None, inv_temp: float = 1.0, keep=None, ws=None):
    """Kept-exponential forward: returns (logp, entropy, lse, keep, ws); pass
    keep and ws unchanged to spo_policy_loss_bwd_kept."""
    dev = H.device
    T, d = H.shape
    V = W.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W, "W", torch.bfloat16, device=dev)
    _need(tgt, "tgt", torch.int32, T, dev)
    if mask is not None:
        _need(mask, "mask", torch.uint8, T, dev)
    logp, ent, lse = (torch.empty(T, dtype=torch.float32, device=dev) for _ in range(3))
    kb = logprobs_keep_size(T, V)
    if keep is None:
        keep = torch.empty(kb, dtype=torch.uint8, device=dev)
    w = _workspace(logprobs_workspace_size(T, d, V), dev, ws)
    _check(lib().spo_logprobs_fwd_keep(_ptr(H), _ptr(W), _ptr(tgt), _ptr(mask), T, d, V,
                                       float(inv_temp), _ptr(logp), _ptr(ent), _ptr(lse),
                                       _ptr(keep), keep.numel() * keep.element_size(), _ptr(w),
                                       w.numel(), _stream(dev)))
    return logp, ent, lse, keep, w


def spo_policy_loss_bwd_kept(W, lse, g, keep, fwd_ws, T: int, d: int, inv_temp: float = 1.0,
                             dH=None, dW=None, accumulate_dW: bool = False, want_dH=True,
                             want_dW=True):
    """Backward from a kept forward: returns (dH bf16[T, d] or None, dW fp32[V, d] or None)."""
    dev = W.device
    V = W.shape[0]
    _need(W, "W", torch.bfloat16, device=dev)
    _need(lse, "lse", torch.float32, T, dev)
    _need(g, "g", torch.float32, T, dev)
    if want_dH and dH is None:
        dH = torch.empty((T, d), dtype=torch.bfloat16, device=dev)
    if want_dW and dW is None:
        dW = (torch.zeros if accumulate_dW else torch.empty)((V, d), dtype=torch.float32,
                                                             device=dev)
    _check(lib().spo_policy_loss_bwd_kept(_ptr(W), _ptr(lse), _ptr(g), T, d, V, float(inv_temp),
                                          _ptr(keep), keep.numel() * keep.element_size(),
                                          _ptr(fwd_ws), fwd_ws.numel() * fwd_ws.element_size(),
                                          _ptr(dH), _ptr(dW), int(bool(accumulate_dW)),
                                          _stream(dev)))
    return dH, dW


def spo_group_advantages(rewards, group_id, n_groups: int, std_mode: int = SPO_STD_UNBIASED,
                         eps: float = 1e-6):
    """a4: per-sequence group-normalised advantages, fp32[n_seq]."""
    dev = rewards.device
    n = rewards.numel()
    _need(rewards, "rewards", torch.float32, device=dev)
    _need(group_id, "group_id", torch.int32, n, dev)
    adv = torch.empty(n, dtype=torch.float32, device=dev)
    _check(lib().spo_group_advantages(_ptr(rewards), _ptr(group_id), n, int(n_groups),
                                      int(std_mode), float(eps), _ptr(adv), _stream(dev)))
    return adv


def group_advantages_workspace_size(n_seq: int, n_groups: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_group_advantages_workspace_size(n_seq, n_groups, ctypes.byref(n)))
    return n.value


def spo_group_advantages_ws(rewards, group_id, n_groups: int, std_mode: int = SPO_STD_UNBIASED,
                            eps: float = 1e-6, adv=None, ws=None):
    """a4 in O(n_seq + n_groups) for contiguous groups (same bits as
    spo_group_advantages); fp32[n_seq]."""
    dev = rewards.device
    n = rewards.numel()
    _need(rewards, "rewards", torch.float32, device=dev)
    _need(group_id, "group_id", torch.int32, n, dev)
    if adv is None:
        adv = torch.empty(n, dtype=torch.float32, device=dev)
    _need(adv, "adv", torch.float32, n, dev)
    w = _workspace(group_advantages_workspace_size(n, int(n_groups)), dev, ws)
    _check(lib().spo_group_advantages_ws(_ptr(rewards), _ptr(group_id), n, int(n_groups),
                                         int(std_mode), float(eps), _ptr(adv), _ptr(w), w.numel(),
                                         _stream(dev)))
    return adv


def policy_loss_workspace_size(n_seq: int, n_groups: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_policy_loss_workspace_size(n_seq, n_groups, ctypes.byref(n)))
    return n.value


def spo_policy_loss_fwd(logp, old_logp, ref_logp, adv, cu_seqlens, group_id, n_groups: int,
                        loss_mask, clip_eps: float = 0.2, kl_beta: float = 0.0,
                        agg: int = SPO_AGG_SEQ_GROUP, ws=None):
    """a5: returns (loss fp32[1], g fp32[T], stats fp32[4])."""
    dev = logp.device
    T = logp.numel()
    n_seq = adv.numel()
    _need(logp, "logp", torch.float32, device=dev)
    _need(old_logp, "old_logp", torch.float32, T, dev)
    if ref_logp is not None:
        _need(ref_logp, "ref_logp", torch.float32, T, dev)
    _need(adv, "adv", torch.float32, device=dev)
    _need(cu_seqlens, "cu_seqlens", torch.int32, n_seq + 1, dev)
    _need(group_id, "group_id", torch.int32, n_seq, dev)
    _need(loss_mask, "loss_mask", torch.uint8, T, dev)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    g = torch.empty(T, dtype=torch.float32, device=dev)
    stats = torch.empty(4, dtype=torch.float32, device=dev)
    w = _workspace(policy_loss_workspace_size(n_seq, n_groups), dev, ws)
    _check(lib().spo_policy_loss_fwd(_ptr(logp), _ptr(old_logp), _ptr(ref_logp), _ptr(adv),
                                     _ptr(cu_seqlens), _ptr(group_id), n_seq, int(n_groups),
                                     _ptr(loss_mask), T, float(clip_eps), float(kl_beta), int(agg),
                                     _ptr(loss), _ptr(g), _ptr(stats), _ptr(w), w.numel(),
                                     _stream(dev)))
    return loss, g, stats


def policy_loss_bwd_workspace_size(T: int, d: int, V: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_policy_loss_bwd_workspace_size(T, d, V, ctypes.byref(n)))
    return n.value


def spo_policy_loss_bwd(H, W, tgt, lse, g, inv_temp: float = 1.0, dH=None, dW=None,
                        accumulate_dW: bool = False, want_dH=True, want_dW=True, ws=None):
    """a6-a8: returns (dH bf16[T, d] or None, dW fp32[V, d] or None)."""
    dev = H.device
    T, d = H.shape
    V = W.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W, "W", torch.bfloat16, device=dev)
    _need(tgt, "tgt", torch.int32, T, dev)
    _need(lse, "lse", torch.float32, T, dev)
    _need(g, "g", torch.float32, T, dev)
    if want_dH and dH is None:
        dH = torch.empty((T, d), dtype=torch.bfloat16, device=dev)
    if want_dW and dW is None:
        dW = (torch.zeros if accumulate_dW else torch.empty)((V, d), dtype=torch.float32,
                                                             device=dev)
    if dH is not None:
        _need(dH, "dH", torch.bfloat16, T * d, dev)
    if dW is not None:
        _need(dW, "dW", torch.float32, V * d, dev)
    w = _workspace(policy_loss_bwd_workspace_size(T, d, V), dev, ws)
    _check(lib().spo_policy_loss_bwd(_ptr(H), _ptr(W), _ptr(tgt), _ptr(lse), _ptr(g), T, d, V,
                                     float(inv_temp), _ptr(dH), _ptr(dW), int(bool(accumulate_dW)),
                                     _ptr(w), w.numel(), _stream(dev)))
    return dH, dW


def spo_logprobs_fwd_slice(H, W_slice, v_offset: int, tgt, mask=None, inv_temp: float = 1.0,
                           rec=None, ws=None):
    """Vocabulary-split a2+a3 over rows [v_offset, v_offset + V_slice) of the
    head: returns this slice's per-token records, fp32[T, 4]."""
    dev = H.device
    T, d = H.shape
    V = W_slice.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W_slice, "W_slice", torch.bfloat16, device=dev)
    if W_slice.shape[1] != d:
        raise ValueError(f"W_slice has {W_slice.shape[1]} columns, H has {d}")
    _need(tgt, "tgt", torch.int32, T, dev)
    if mask is not None:
        _need(mask, "mask", torch.uint8, T, dev)
    if rec is None:
        rec = torch.empty((T, 4), dtype=torch.float32, device=dev)
    _need(rec, "rec", torch.float32, T * 4, dev)
    w = _workspace(logprobs_workspace_size(T, d, V), dev, ws)
    _check(lib().spo_logprobs_fwd_slice(_ptr(H), _ptr(W_slice), _ptr(tgt), _ptr(mask), T, d, V,
                                        int(v_offset), float(inv_temp), _ptr(rec), _ptr(w),
                                        w.numel(), _stream(dev)))
    return rec


def spo_logprobs_merge_slices(rec, want_entropy=True):
    """rec fp32[n_slices, T, 4] (the slices' records stacked) -> (logp, entropy or None, lse)."""
    dev = rec.device
    if rec.dim() != 3 or rec.shape[2] != 4:
        raise ValueError("rec must have shape [n_slices, T, 4]")
    n, T = rec.shape[0], rec.shape[1]
    _need(rec, "rec", torch.float32, n * T * 4, dev)
    logp = torch.empty(T, dtype=torch.float32, device=dev)
    ent = torch.empty(T, dtype=torch.float32, device=dev) if want_entropy else None
    lse = torch.empty(T, dtype=torch.float32, device=dev)
    _check(lib().spo_logprobs_merge_slices(_ptr(rec), n, T, _ptr(logp), _ptr(ent), _ptr(lse),
                                           _stream(dev)))
    return logp, ent, lse


def spo_policy_loss_bwd_slice(H, W_slice, v_offset: int, tgt, lse, g, inv_temp: float = 1.0,
                              dH_part=None, dW_slice=None, accumulate_dW: bool = False,
                              want_dH=True, want_dW=True, ws=None):
    """Vocabulary-split a6-a8: returns (this slice's fp32 part of dH [T, d] or
    None, dW rows of the slice fp32[V_slice, d] or None)."""
    dev = H.device
    T, d = H.shape
    V = W_slice.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W_slice, "W_slice", torch.bfloat16, device=dev)
    _need(tgt, "tgt", torch.int32, T, dev)
    _need(lse, "lse", torch.float32, T, dev)
    _need(g, "g", torch.float32, T, dev)
    if want_dH and dH_part is None:
        dH_part = torch.empty((T, d), dtype=torch.float32, device=dev)
    if want_dW and dW_slice is None:
        dW_slice = (torch.zeros if accumulate_dW else torch.empty)((V, d), dtype=torch.float32,
                                                                   device=dev)
    if dH_part is not None:
        _need(dH_part, "dH_part", torch.float32, T * d, dev)
    if dW_slice is not None:
        _need(dW_slice, "dW_slice", torch.float32, V * d, dev)
    w = _workspace(policy_loss_bwd_workspace_size(T, d, V), dev, ws)
    _check(lib().spo_policy_loss_bwd_slice(_ptr(H), _ptr(W_slice), _ptr(tgt), _ptr(lse), _ptr(g),
                                           T, d, V, int(v_offset), float(inv_temp), _ptr(dH_part),
                                           _ptr(dW_slice), int(bool(accumulate_dW)), _ptr(w),
                                           w.numel(), _stream(dev)))
    return dH_part, dW_slice


class BwdHooks(ctypes.Structure):
    """spo_bwd_hooks: dW in vocabulary blocks with an event per finished block."""
    _fields_ = [("n_dw_blocks", _i32), ("reserve_sms", _i32), ("dw_block_events", _vp),
                ("dh_event", _vp)]


def _event_handle(ev) -> int:
    """The cudaEvent_t of a torch.cuda.Event (created by recording it once)."""
    if ev.cuda_event == 0:
        ev.record()
    return int(ev.cuda_event)


def make_hooks(n_dw_blocks: int = 1, dw_events=None, dh_event=None, reserve_sms: int = 0):
    """A spo_bwd_hooks for the C call; keep the returned object alive until the call returns."""
    h = BwdHooks()
    h.n_dw_blocks = int(n_dw_blocks)
    h.reserve_sms = int(reserve_sms)
    # the events must outlive the call that records them: the hooks hold them
    h._events = (list(dw_events) if dw_events is not None else [], dh_event)
    if dw_events is not None:
        if len(dw_events) != n_dw_blocks:
            raise ValueError("one event per dW block")
        arr = (_vp * n_dw_blocks)(*[_event_handle(e) if e is not None else None for e in dw_events])
        h._arr = arr
        h.dw_block_events = ctypes.cast(arr, _vp)
    h.dh_event = _event_handle(dh_event) if dh_event is not None else None
    return h


def dw_block_starts(V: int, n_blocks: int):
    """First dW row of each of n_blocks vocabulary blocks, plus V (host computation)."""
    out = (_i64 * (n_blocks + 1))()
    _check(lib().spo_dw_block_starts(int(V), int(n_blocks), out))
    return [int(x) for x in out]


def spo_policy_loss_bwd_ex(H, W, tgt, lse, g, inv_temp: float = 1.0, v_offset: int = 0,
                           dH=None, dW=None, dH_fp32: bool = False, accumulate_dW: bool = False,
                           hooks=None, want_dH=True, want_dW=True, ws=None):
    """a6-a8 with hooks: returns (dH, dW).  With v_offset / dH_fp32 the vocabulary-slice form."""
    dev = H.device
    T, d = H.shape
    V = W.shape[0]
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W, "W", torch.bfloat16, device=dev)
    _need(tgt, "tgt", torch.int32, T, dev)
    _need(lse, "lse", torch.float32, T, dev)
    _need(g, "g", torch.float32, T, dev)
    dh_type = torch.float32 if dH_fp32 else torch.bfloat16
    if want_dH and dH is None:
        dH = torch.empty((T, d), dtype=dh_type, device=dev)
    if want_dW and dW is None:
        dW = (torch.zeros if accumulate_dW else torch.empty)((V, d), dtype=torch.float32,
                                                             device=dev)
    if dH is not None:
        _need(dH, "dH", dh_type, T * d, dev)
    if dW is not None:
        _need(dW, "dW", torch.float32, V * d, dev)
    w = _workspace(policy_loss_bwd_workspace_size(T, d, V), dev, ws)
    _check(lib().spo_policy_loss_bwd_ex(_ptr(H), _ptr(W), _ptr(tgt), _ptr(lse), _ptr(g), T, d, V,
                                        int(v_offset), float(inv_temp), _ptr(dH), int(bool(dH_fp32)),
                                        _ptr(dW), int(bool(accumulate_dW)),
                                        None if hooks is None else ctypes.byref(hooks), _ptr(w),
                                        w.numel(), _stream(dev)))
    return dH, dW


class GrpoBatch(ctypes.Structure):
    _fields_ = [("H", _vp), ("W", _vp), ("tgt", _vp), ("mask", _vp), ("cu_seqlens", _vp),
                ("group_id", _vp), ("rewards", _vp), ("old_logp", _vp), ("ref_logp", _vp),
                ("T", _i64), ("d", _i64), ("V", _i64), ("n_seq", _i32), ("n_groups", _i32)]


class GrpoParams(ctypes.Structure):
    _fields_ = [("inv_temp", _f32), ("window", _i32), ("clip_eps", _f32), ("kl_beta", _f32),
                ("agg", _i32), ("std_mode", _i32), ("adv_eps", _f32), ("loss_scale", _vp)]


class GrpoOutputs(ctypes.Structure):
    _fields_ = [("loss", _vp), ("stats", _vp), ("logp", _vp), ("entropy", _vp), ("lse", _vp),
                ("g", _vp), ("adv", _vp), ("loss_mask", _vp), ("dH", _vp), ("dW", _vp),
                ("accumulate_dW", _i32)]


def grpo_workspace_size(T: int, d: int, V: int, n_seq: int, n_groups: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_grpo_workspace_size(T, d, V, n_seq, n_groups, ctypes.byref(n)))
    return n.value


def workspace_size(T: int, d: int, V: int, n_seq: int) -> int:
    n = ctypes.c_size_t(0)
    _check(lib().spo_workspace_size(T, d, V, n_seq, ctypes.byref(n)))
    return n.value


def spo_grpo_step(H, W, tgt, mask, cu_seqlens, group_id, n_groups: int, rewards, old_logp,
                  ref_logp=None, inv_temp: float = 1.0, window: int = 1024, clip_eps: float = 0.2,
                  kl_beta: float = 0.0, agg: int = SPO_AGG_SEQ_GROUP,
                  std_mode: int = SPO_STD_UNBIASED, adv_eps: float = 1e-6, loss_scale=None,
                  want=("logp", "entropy", "lse", "g", "adv", "loss_mask", "stats"),
                  want_dH=True, want_dW=True, dH=None, dW=None, accumulate_dW=False, hooks=None,
                  ws=None):
    """The whole step a1 -> a8 in one call.  Returns a dict of the outputs
    asked for (loss always; dH, dW unless switched off)."""
    dev = H.device
    T, d = H.shape
    V = W.shape[0]
    n_seq = cu_seqlens.numel() - 1
    _need(H, "H", torch.bfloat16, device=dev)
    _need(W, "W", torch.bfloat16, device=dev)
    _need(tgt, "tgt", torch.int32, T, dev)
    if mask is not None:
        _need(mask, "mask", torch.uint8, T, dev)
    _need(cu_seqlens, "cu_seqlens", torch.int32, n_seq + 1, dev)
    _need(group_id, "group_id", torch.int32, n_seq, dev)
    _need(rewards, "rewards", torch.float32, n_seq, dev)
    _need(old_logp, "old_logp", torch.float32, T, dev)
    if ref_logp is not None:
        _need(ref_logp, "ref_logp", torch.float32, T, dev)
    if loss_scale is not None:
        _need(loss_scale, "loss_scale", torch.float32, 1, dev)
    f32 = dict(dtype=torch.float32, device=dev)
    out = {"loss": torch.empty(1, **f32)}
    shapes = {"stats": (4, torch.float32), "logp": (T, torch.float32),
              "entropy": (T, torch.float32), "lse": (T, torch.float32), "g": (T, torch.float32),
              "adv": (n_seq, torch.float32), "loss_mask": (T, torch.uint8)}
    for k in want:
        n, dt = shapes[k]
        out[k] = torch.empty(n, dtype=dt, device=dev)
    if want_dH:
        out["dH"] = dH if dH is not None else torch.empty((T, d), dtype=torch.bfloat16, device=dev)
        _need(out["dH"], "dH", torch.bfloat16, T * d, dev)
    if want_dW:
        out["dW"] = dW if dW is not None else (torch.zeros if accumulate_dW else torch.empty)(
            (V, d), **f32)
        _need(out["dW"], "dW", torch.float32, V * d, dev)
    b = GrpoBatch(_ptr(H), _ptr(W), _ptr(tgt), _ptr(mask), _ptr(cu_seqlens), _ptr(group_id),
                  _ptr(rewards), _ptr(old_logp), _ptr(ref_logp), T, d, V, n_seq, int(n_groups))
    q = GrpoParams(float(inv_temp), int(window), float(clip_eps), float(kl_beta), int(agg),
                   int(std_mode), float(adv_eps), _ptr(loss_scale))
    o = GrpoOutputs(*[_ptr(out.get(k)) for k in ("loss", "stats", "logp", "entropy", "lse", "g",
                                                  "adv", "loss_mask", "dH", "dW")],
                    int(bool(accumulate_dW)))
    w = _workspace(grpo_workspace_size(T, d, V, n_seq, int(n_groups)), dev, ws)
    _check(lib().spo_grpo_step(ctypes.byref(b), ctypes.byref(q), ctypes.byref(o),
                               None if hooks is None else ctypes.byref(hooks), _ptr(w), w.numel(),
                               _stream(dev)))
    return out


def spo_sync_check(device=None) -> int:
    """Synchronises the current stream; the status (0, SPO_ERR_TIMEOUT or SPO_ERR_CUDA)."""
    device = torch.device(device or torch.cuda.current_device())
    return int(lib().spo_sync_check(_stream(device)))


def spo_scale_f32_ratio(x, num, den):
    """In place x *= num[0] / den[0] (device fp64 scalars; 0 when den[0] is 0)."""
    _need(x, "x", torch.float32, device=x.device)
    _need(num, "num", torch.float64, 1, x.device)
    _need(den, "den", torch.float64, 1, x.device)
    _check(lib().spo_scale_f32_ratio(_ptr(x), x.numel(), _ptr(num), _ptr(den), _stream(x.device)))
    return x


def spo_selftest_bounded_wait(device=None):
    """Enqueue the bounded-wait self-test on the current stream (returns at once;
    the kernel gives up after about a second and records code 0x1ff)."""
    dev = torch.device("cuda", torch.cuda.current_device()) if device is None else device
    _check(lib().spo_selftest_bounded_wait(_stream(dev)))


def spo_trace_enable(on: bool = True):
    _check(lib().spo_trace_enable(1 if on else 0))


def spo_trace_read(max_records: int = 65536):
    """[(kind, ms)] for every traced GEMM launch since the last read (synchronises)."""
    kinds = (ctypes.c_int * max_records)()
    ms = (ctypes.c_float * max_records)()
    n = ctypes.c_int(0)
    _check(lib().spo_trace_read(kinds, ms, max_records, ctypes.byref(n)))
    return [(int(kinds[i]), float(ms[i])) for i in range(min(n.value, max_records))]


def spo_launch_count() -> int:
    return int(lib().spo_launch_count())


def spo_policy_loss_fwd_noalloc(logp, old_logp, ref_logp, adv, cu_seqlens, group_id,
                                n_groups: int, loss_mask, loss, g, stats=None,
                                clip_eps: float = 0.2, kl_beta: float = 0.0,
                                agg: int = SPO_AGG_SEQ_GROUP):
    """a5 without a workspace: writes into the caller's loss / g / stats tensors and
    allocates nothing (scratch is the library's static 1 MiB device array)."""
    dev = logp.device
    T = logp.numel()
    n_seq = adv.numel()
    _need(logp, "logp", torch.float32, device=dev)
    _need(old_logp, "old_logp", torch.float32, T, dev)
    if ref_logp is not None:
        _need(ref_logp, "ref_logp", torch.float32, T, dev)
    _need(adv, "adv", torch.float32, device=dev)
    _need(cu_seqlens, "cu_seqlens", torch.int32, n_seq + 1, dev)
    _need(group_id, "group_id", torch.int32, n_seq, dev)
    _need(loss_mask, "loss_mask", torch.uint8, T, dev)
    _need(loss, "loss", torch.float32, 1, dev)
    _need(g, "g", torch.float32, T, dev)
    if stats is not None:
        _need(stats, "stats", torch.float32, 4, dev)
    # the library uses the current device's copy of its static scratch
    with torch.cuda.device(dev):
        _check(lib().spo_policy_loss_fwd_noalloc(
            _ptr(logp), _ptr(old_logp), _ptr(ref_logp), _ptr(adv), _ptr(cu_seqlens),
            _ptr(group_id), n_seq, int(n_groups), _ptr(loss_mask), T, float(clip_eps),
            float(kl_beta), int(agg), _ptr(loss), _ptr(g), _ptr(stats), _stream(dev)))


SPO_TUNE_PAIR_MMA = 0
SPO_TUNE_GROUP_M = 1
SPO_TUNE_RASTER = 2
SPO_TUNE_DYNAMIC_MASK = 3
SPO_TUNE_DW_SPLIT_ROWS = 4
SPO_TUNE_GROUP_M_FWD, SPO_TUNE_GROUP_M_GRAD, SPO_TUNE_GROUP_M_DH, SPO_TUNE_GROUP_M_DW = 5, 6, 7, 8
SPO_TUNE_RASTER_FWD, SPO_TUNE_RASTER_GRAD, SPO_TUNE_RASTER_DH, SPO_TUNE_RASTER_DW = 9, 10, 11, 12
SPO_TUNE_DEFAULTS = 13
SPO_TUNE_KSYNC_FWD, SPO_TUNE_KSYNC_GRAD, SPO_TUNE_KSYNC_DH, SPO_TUNE_KSYNC_DW = 14, 15, 16, 17
SPO_TUNE_KSYNC_EPOCH = 18
SPO_TUNE_DH_WIDE = 19
SPO_TUNE_LOGITS_WIDE = 20


def spo_set_tuning(key: int, value: int):
    """Host-global launch tuning (results do not depend on it)."""
    _check(lib().spo_set_tuning(int(key), int(value)))


class RewardParams(ctypes.Structure):
    """spo_reward_params (section 2.2 constants; the defaults are the paper's)."""
    _fields_ = [("alpha_comp", ctypes.c_float), ("alpha_wrong", ctypes.c_float),
                ("alpha_speed", ctypes.c_float), ("alpha_cv", ctypes.c_float),
                ("s_min", ctypes.c_float), ("s_max", ctypes.c_float)]


def spo_reward_compose(compiled, pass_rate, speedup, cv, r_struct=None, params=None, out=None):
    """Composite reward r = R_ver + R_str per candidate, fp32[n]."""
    dev = pass_rate.device
    n = pass_rate.numel()
    _need(compiled, "compiled", torch.uint8, n, dev)
    _need(pass_rate, "pass_rate", torch.float32, n, dev)
    _need(speedup, "speedup", torch.float32, n, dev)
    _need(cv, "cv", torch.float32, n, dev)
    if r_struct is not None:
        _need(r_struct, "r_struct", torch.float32, n, dev)
    out = torch.empty(n, dtype=torch.float32, device=dev) if out is None else out
    _need(out, "rewards", torch.float32, n, dev)
    prm = None
    if params is not None:
        prm = ctypes.byref(RewardParams(**params) if isinstance(params, dict) else params)
    _check(lib().spo_reward_compose(_ptr(compiled), _ptr(pass_rate), _ptr(speedup), _ptr(cv),
                                    _ptr(r_struct), n, prm, _ptr(out), _stream(dev)))
    return out


RANKER_FEATURES = 11
RANKER_PARAMS = 2881


def spo_ranker_scores(phi, mu, sigma, params):
    """Structural score s_psi(phi_hat) per program, fp32[n]."""
    dev = phi.device
    n = phi.shape[0]
    _need(phi, "phi", torch.float32, n * RANKER_FEATURES, dev)
    _need(mu, "mu", torch.float32, RANKER_FEATURES, dev)
    _need(sigma, "sigma", torch.float32, RANKER_FEATURES, dev)
    _need(params, "params", torch.float32, RANKER_PARAMS, dev)
    out = torch.empty(n, dtype=torch.float32, device=dev)
    _check(lib().spo_ranker_scores(_ptr(phi), _ptr(mu), _ptr(sigma), n, _ptr(params), _ptr(out),
                                   _stream(dev)))
    return out


def spo_ranker_pair_loss(phi, mu, sigma, params, pos, neg, keep1=None, keep2=None,
                         drop_p: float = 0.0, want_grad=True, ws=None):
    """Pairwise logistic ranking loss and its gradient: (loss fp32[1], grad fp32[2881])."""
    dev = phi.device
    n_pairs = pos.numel()
    _need(phi, "phi", torch.float32, phi.shape[0] * RANKER_FEATURES, dev)
    _need(mu, "mu", torch.float32, RANKER_FEATURES, dev)
    _need(sigma, "sigma", torch.float32, RANKER_FEATURES, dev)
    _need(params, "params", torch.float32, RANKER_PARAMS, dev)
    _need(pos, "pos", torch.int32, n_pairs, dev)
    _need(neg, "neg", torch.int32, n_pairs, dev)
    if keep1 is not None:
        _need(keep1, "keep1", torch.uint8, n_pairs * 2 * 64, dev)
    if keep2 is not None:
        _need(keep2, "keep2", torch.uint8, n_pairs * 2 * 32, dev)
    loss = torch.empty(1, dtype=torch.float32, device=dev)
    grad = torch.empty(RANKER_PARAMS, dtype=torch.float32, device=dev) if want_grad else None
    n = ctypes.c_size_t(0)
    _check(lib().spo_ranker_workspace_size(n_pairs, ctypes.byref(n)))
    w = _workspace(n.value, dev, ws)
    _check(lib().spo_ranker_pair_loss(_ptr(phi), _ptr(mu), _ptr(sigma), _ptr(pos), _ptr(neg),
                                      n_pairs, _ptr(params), _ptr(keep1), _ptr(keep2),
                                      float(drop_p), _ptr(loss), _ptr(grad), _ptr(w), w.numel(),
                                      _stream(dev)))
    return loss, grad


def spo_scale_f32(x, alpha=None, alpha_dev=None):
    """In place x *= alpha (host float) or x *= alpha_dev[0] (device fp32 scalar)."""
    _need(x, "x", torch.float32, device=x.device)
    if alpha_dev is not None:
        _need(alpha_dev, "alpha_dev", torch.float32, 1, x.device)
    _check(lib().spo_scale_f32(_ptr(x), x.numel(), float(alpha if alpha is not None else 1.0),
                               _ptr(alpha_dev), _stream(x.device)))
    return x


VALIDATION_FIELDS = ("tgt_out_of_range", "bad_cu_seqlens", "bad_group_id", "nonfinite_rewards",
                     "nonfinite_old_ref_logp", "bad_mask")


def spo_validate_inputs(tgt=None, V=0, cu_seqlens=None, group_id=None, n_groups=0, rewards=None,
                        old_logp=None, ref_logp=None, mask=None, T=None, sync=True):
    """Counts of invalid device inputs (see include/spo.h); a dict when sync, else the
    device int32[6] counts tensor."""
    ref = next(t for t in (tgt, cu_seqlens, group_id, rewards, old_logp, ref_logp, mask)
               if t is not None)
    dev = ref.device
    if T is None:
        T = (tgt if tgt is not None else old_logp if old_logp is not None else
             mask if mask is not None else torch.empty(0)).numel()
    n_seq = (cu_seqlens.numel() - 1 if cu_seqlens is not None else
             group_id.numel() if group_id is not None else
             rewards.numel() if rewards is not None else 0)
    counts = torch.empty(6, dtype=torch.int32, device=dev)
    _check(lib().spo_validate_inputs(_ptr(tgt), T, V, _ptr(cu_seqlens), n_seq, _ptr(group_id),
                                     n_groups, _ptr(rewards), _ptr(old_logp), _ptr(ref_logp),
                                     _ptr(mask), _ptr(counts), _stream(dev)))
    if not sync:
        return counts
    return dict(zip(VALIDATION_FIELDS, counts.cpu().tolist()))
