"""The C-ABI library loads, exports every symbol include/spo.h declares, and
rejects bad arguments on the host before touching a GPU.  CPU only: no call
here reaches a kernel."""

import ctypes
import os
import re

import pytest

from paper_2607_20908_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    B.build()
    from paper_2607_20908_gb300 import spo
    return spo.lib()


def _declared():
    text = open(os.path.join(ROOT, "include", "spo.h")).read()
    return sorted(set(re.findall(r"SPO_API\s+[^;(]*?\b(spo_\w+)\s*\(", text)))


def test_every_declared_symbol_is_exported(lib):
    names = _declared()
    assert len(names) >= 12
    from paper_2607_20908_gb300 import spo
    for n in names:
        assert hasattr(lib, n), n
        assert n in spo.exported_symbols(), f"binding misses {n}"


def test_status_strings(lib):
    from paper_2607_20908_gb300 import spo
    assert spo.status_string(0) == "SPO_OK"
    assert spo.status_string(4) == "SPO_ERR_WORKSPACE"
    assert spo.status_string(99) == "SPO_ERR_UNKNOWN"
    assert lib.spo_version() >= 1


def test_workspace_sizes_are_host_only(lib):
    from paper_2607_20908_gb300 import spo
    small = spo.logprobs_workspace_size(256, 256, 4096)
    big = spo.logprobs_workspace_size(16384, 5120, 151936)
    assert 0 < small < big
    # partials (ceil(V/256) x T_pad x 16 B) dominate at the full vocabulary
    assert big >= 594 * 16384 * 16
    bwd = spo.policy_loss_bwd_workspace_size(16384, 5120, 151936)
    assert bwd >= 16384 * 151936 * 2          # one bf16 G chunk
    assert spo.policy_loss_bwd_workspace_size(131072, 5120, 151936) < 131072 * 151936 * 2
    assert spo.policy_loss_workspace_size(128, 16) > 0


def _err(lib):
    buf = ctypes.create_string_buffer(256)
    st = lib.spo_last_error(buf, 256)
    return st, buf.value.decode()


def test_host_validation_without_gpu(lib):
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    nul = ctypes.c_void_p(0)
    f = lib.spo_logprobs_fwd
    st = f(nul, p, p, nul, 256, 256, 4096, 1.0, p, nul, nul, p, 1 << 30, nul)
    assert st == 1 and "non-NULL" in _err(lib)[1]
    st = f(p, p, p, nul, 256, 100, 4096, 1.0, p, nul, nul, p, 1 << 30, nul)
    assert st == 2 and "multiple of 64" in _err(lib)[1]
    st = f(p, p, p, nul, 256, 256, 4100, 1.0, p, nul, nul, p, 1 << 30, nul)
    assert st == 2
    st = f(ctypes.c_void_p(4097), p, p, nul, 256, 256, 4096, 1.0, p, nul, nul, p, 1 << 30, nul)
    assert st == 3
    st = f(p, p, p, nul, 256, 256, 4096, -1.0, p, nul, nul, p, 1 << 30, nul)
    assert st == 1
    st = f(p, p, p, nul, 256, 256, 4096, 1.0, p, nul, nul, p, 16, nul)
    assert st == 4 and "workspace" in _err(lib)[1]
    g = lib.spo_group_advantages
    assert g(p, p, 16, 4, 7, 1e-6, p, nul) == 1
    assert g(p, p, 0, 4, 0, 1e-6, p, nul) == 2
    lf = lib.spo_policy_loss_fwd
    assert lf(p, p, nul, p, p, p, 4, 2, p, 64, 0.2, 0.0, 5, p, p, nul, p, 1 << 20, nul) == 1
    assert lf(p, p, nul, p, p, p, 4, 2, p, 64, 1.5, 0.0, 0, p, p, nul, p, 1 << 20, nul) == 1
    assert lf(p, p, nul, p, p, p, 4, 2, p, 64, 0.2, 0.0, 0, p, p, nul, p, 8, nul) == 4
    bw = lib.spo_policy_loss_bwd
    assert bw(p, p, p, nul, p, 256, 256, 4096, 1.0, p, p, 0, p, 1 << 40, nul) == 1
    assert bw(p, p, p, p, p, 256, 256, 4096, 1.0, ctypes.c_void_p(4098), p, 0, p, 1 << 40, nul) == 3


def test_vocab_split_host_validation_without_gpu(lib):
    p = ctypes.c_void_p(4096)  # never dereferenced: validation fails first
    nul = ctypes.c_void_p(0)
    fs = lib.spo_logprobs_fwd_slice
    assert fs(p, p, p, nul, 256, 256, 2048, 1024, 1.0, nul, p, 1 << 30, nul) == 1
    assert fs(p, p, p, nul, 256, 256, 2048, 1024, 1.0, ctypes.c_void_p(4100), p, 1 << 30, nul) == 3
    assert fs(p, p, p, nul, 256, 256, 2048, -8, 1.0, p, p, 1 << 30, nul) == 2
    assert "v_offset" in _err(lib)[1]
    assert fs(p, p, p, nul, 256, 256, 128, 0, 1.0, p, p, 1 << 30, nul) == 2
    assert fs(p, p, p, nul, 256, 256, 2048, 0, 1.0, p, p, 64, nul) == 4
    mg = lib.spo_logprobs_merge_slices
    assert mg(p, 0, 256, p, nul, nul, nul) == 2
    assert mg(p, 2, 0, p, nul, nul, nul) == 2
    assert mg(ctypes.c_void_p(4104), 2, 256, p, nul, nul, nul) == 3
    assert mg(p, 2, 256, nul, nul, nul, nul) == 1
    bs = lib.spo_policy_loss_bwd_slice
    assert bs(p, p, p, p, p, 256, 256, 2048, -1, 1.0, p, p, 0, p, 1 << 40, nul) == 2
    assert bs(p, p, p, nul, p, 256, 256, 2048, 0, 1.0, p, p, 0, p, 1 << 40, nul) == 1
    assert bs(p, p, p, p, p, 256, 256, 2048, 0, 1.0, ctypes.c_void_p(4100), p, 0, p, 1 << 40,
              nul) == 3


def test_token_and_loss_size_limits(lib):
    """T above 2^30 is refused on the host (the kernels index tokens in 32-bit)."""
    p = ctypes.c_void_p(4096)
    nul = ctypes.c_void_p(0)
    assert lib.spo_token_select(p, nul, p, 4, (1 << 30) + 1, 1024, p, p, nul) == 2
    assert lib.spo_policy_loss_fwd(p, p, nul, p, p, p, 4, 2, p, (1 << 30) + 1, 0.2, 0.0, 0, p, p,
                                   nul, p, 1 << 20, nul) == 2


def test_scale_host_validation(lib):
    p = ctypes.c_void_p(4096)
    nul = ctypes.c_void_p(0)
    f = lib.spo_scale_f32
    assert f(nul, 0, 2.0, nul, nul) == 0                    # nothing to scale: no launch
    assert f(nul, 5, 2.0, nul, nul) == 1                    # data needed
    assert f(p, -1, 2.0, nul, nul) == 2
    assert f(p, 5, float("inf"), nul, nul) == 1             # host factor must be finite


def test_group_advantages_ws_host_validation(lib):
    from paper_2607_20908_gb300 import spo
    p = ctypes.c_void_p(4096)
    nul = ctypes.c_void_p(0)
    assert spo.group_advantages_workspace_size(1 << 24, 1 << 20) >= 4 * 3 * (1 << 20)
    f = lib.spo_group_advantages_ws
    assert f(p, p, 16, 4, 0, 1e-6, p, p, 16, nul) == 4
    assert f(p, p, 16, 4, 0, 1e-6, p, ctypes.c_void_p(4100), 1 << 20, nul) == 3
    assert f(p, p, 16, 4, 5, 1e-6, p, p, 1 << 20, nul) == 1
    assert f(p, nul, 16, 4, 0, 1e-6, p, p, 1 << 20, nul) == 1
    assert f(p, p, 0, 4, 0, 1e-6, p, p, 1 << 20, nul) == 2


def test_kept_form_host_validation(lib):
    from paper_2607_20908_gb300 import spo
    p = ctypes.c_void_p(4096)
    nul = ctypes.c_void_p(0)
    assert spo.logprobs_keep_size(16384, 151936) == 16384 * 151936 * 2
    assert spo.logprobs_keep_size(300, 4096) == 512 * 4096 * 2      # rows padded to 256
    fk = lib.spo_logprobs_fwd_keep
    ok_ws = 1 << 30
    assert fk(p, p, p, nul, 256, 256, 4096, 1.0, p, nul, nul, p, 1 << 30, p, ok_ws, nul) == 1  # lse
    assert fk(p, p, p, nul, 256, 256, 4096, 1.0, p, nul, p, p, 1024, p, ok_ws, nul) == 4      # keep
    assert fk(p, p, p, nul, 256, 256, 4096, 1.0, p, nul, p, ctypes.c_void_p(4100), 1 << 30, p,
              ok_ws, nul) == 3
    bk = lib.spo_policy_loss_bwd_kept
    assert bk(nul, p, p, 256, 256, 4096, 1.0, p, 1 << 30, p, ok_ws, p, p, 0, nul) == 1
    assert bk(p, p, p, 256, 100, 4096, 1.0, p, 1 << 30, p, ok_ws, p, p, 0, nul) == 2
    assert bk(p, p, p, 256, 256, 4096, 1.0, p, 1 << 30, p, 64, p, p, 0, nul) == 4            # fwd ws


def test_boundary_names_and_step_sizes(lib):
    """The boundary's named entry points: the error text under both names,
    one workspace size for a whole step, and the dW block layout (host only)."""
    from paper_2607_20908_gb300 import spo
    nul = ctypes.c_void_p(0)
    assert lib.spo_grpo_step(nul, nul, nul, nul, nul, 0, nul) == 1
    b1 = ctypes.create_string_buffer(256)
    b2 = ctypes.create_string_buffer(256)
    assert lib.spo_last_error(b1, 256) == 1 and lib.spo_last_error_detail(b2, 256) == 1
    assert b1.value == b2.value and b"non-NULL" in b1.value
    T, d, V, n_seq = 16384, 5120, 151936, 128
    step = spo.grpo_workspace_size(T, d, V, n_seq, 16)
    one = spo.workspace_size(T, d, V, n_seq)
    assert one >= step >= spo.logprobs_workspace_size(T, d, V) + T * V * 2
    for part in (spo.logprobs_workspace_size(T, d, V), spo.policy_loss_bwd_workspace_size(T, d, V),
                 spo.policy_loss_workspace_size(n_seq, n_seq),
                 spo.group_advantages_workspace_size(n_seq, n_seq),
                 spo.grpo_workspace_size(T, d, V, n_seq, n_seq)):
        assert one >= part
    starts = spo.dw_block_starts(V, 4)
    assert starts == [0, 37888, 75776, 113920, V]
    assert spo.dw_block_starts(V, 1) == [0, V]
    small = spo.dw_block_starts(256, 4)                 # blocks may be empty
    assert small[0] == 0 and small[-1] == 256 and all(x % 256 == 0 for x in small[:-1])
    out = (ctypes.c_int64 * 2)()
    assert lib.spo_dw_block_starts(V, 0, out) == 1


def test_step_and_hooks_host_validation(lib):
    from paper_2607_20908_gb300 import spo
    p = ctypes.c_void_p(4096)
    nul = ctypes.c_void_p(0)
    T, d, V, n_seq, n_groups = 64, 128, 1024, 8, 2
    b = spo.GrpoBatch(p, p, p, nul, p, p, p, p, nul, T, d, V, n_seq, n_groups)
    q = spo.GrpoParams(1.0, 1024, 0.2, 0.04, 0, 0, 1e-6, nul)
    o = spo.GrpoOutputs(p, nul, nul, nul, nul, nul, nul, nul, nul, nul, 0)
    need = spo.grpo_workspace_size(T, d, V, n_seq, n_groups)
    R = ctypes.byref
    f = lib.spo_grpo_step
    assert f(R(b), R(q), R(o), nul, p, need - 1, nul) == 4
    assert f(R(b), R(q), R(o), nul, ctypes.c_void_p(4368), need, nul) == 3
    o.loss = None
    assert f(R(b), R(q), R(o), nul, p, need, nul) == 1 and "loss" in _err(lib)[1]
    o.loss = p
    for field, bad, code in (("agg", 3, 1), ("std_mode", 2, 1), ("clip_eps", 1.0, 1),
                             ("adv_eps", -1.0, 1), ("inv_temp", 0.0, 1)):
        old = getattr(q, field)
        setattr(q, field, bad)
        assert f(R(b), R(q), R(o), nul, p, need, nul) == code, field
        setattr(q, field, old)
    b.n_groups = 0
    assert f(R(b), R(q), R(o), nul, p, need, nul) == 2
    b.n_groups = n_groups
    b.d = 100
    assert f(R(b), R(q), R(o), nul, p, need, nul) == 2
    b.d = d
    o.dH = ctypes.c_void_p(4098)
    assert f(R(b), R(q), R(o), nul, p, need, nul) == 3
    bx = lib.spo_policy_loss_bwd_ex
    assert bx(p, p, p, p, p, 256, 256, 2048, -1, 1.0, p, 1, p, 0, nul, p, 1 << 40, nul) == 2
    assert bx(p, p, p, nul, p, 256, 256, 2048, 0, 1.0, p, 0, p, 0, nul, p, 1 << 40, nul) == 1
    sr = lib.spo_scale_f32_ratio
    assert sr(nul, 0, nul, nul, nul) == 0
    assert sr(p, 4, p, nul, nul) == 1
    assert sr(p, -1, p, p, nul) == 2


def test_tuning_keys_host_validation(lib):
    """spo_set_tuning checks each value on the host (no device involved)."""
    from paper_2607_20908_gb300 import spo
    ok = [(spo.SPO_TUNE_DH_WIDE, 0), (spo.SPO_TUNE_DH_WIDE, 1), (spo.SPO_TUNE_DH_WIDE, 2),
          (spo.SPO_TUNE_LOGITS_WIDE, 0), (spo.SPO_TUNE_LOGITS_WIDE, 7),
          (spo.SPO_TUNE_PAIR_MMA, 0), (spo.SPO_TUNE_GROUP_M_DH, 8), (spo.SPO_TUNE_KSYNC_DH, 64),
          (spo.SPO_TUNE_DW_SPLIT_ROWS, 4096)]
    bad = [(spo.SPO_TUNE_DH_WIDE, 3), (spo.SPO_TUNE_DH_WIDE, -1), (spo.SPO_TUNE_PAIR_MMA, 2),
           (spo.SPO_TUNE_LOGITS_WIDE, 8),
           (spo.SPO_TUNE_GROUP_M_DH, 0), (spo.SPO_TUNE_DW_SPLIT_ROWS, 100),
           (spo.SPO_TUNE_KSYNC_EPOCH, 0), (99, 0)]
    try:
        for key, value in ok:
            assert lib.spo_set_tuning(key, value) == 0, (key, value)
        for key, value in bad:
            assert lib.spo_set_tuning(key, value) == 1, (key, value)   # SPO_ERR_INVALID_ARG
    finally:
        assert lib.spo_set_tuning(spo.SPO_TUNE_DEFAULTS, 0) == 0
