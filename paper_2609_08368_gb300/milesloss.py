"""Thin Python binding of libmilesloss (ctypes).

Argument marshalling only: every step of the loss runs in the CUDA library.
torch.Tensors go in by ``data_ptr()`` and calls are enqueued on the current
torch CUDA stream. There is no fallback: if the library is missing the
import of this module's functions fails loudly.
"""

from __future__ import annotations

import ctypes
import os
import struct

from . import build as _build

RL_OK = 0
RL_BF16, RL_F32 = 0, 1
RL_PHASE_BEGIN, RL_PHASE_ROWS, RL_PHASE_END, RL_PHASE_ALL = 1, 2, 4, 7
RL_SHARD_COUNT, RL_SHARD_SWEEP, RL_SHARD_FINISH, RL_SHARD_SEQ = 1, 2, 4, 8
RL_VSHARD_COUNT, RL_VSHARD_PARTIAL, RL_VSHARD_SWEEP, RL_VSHARD_FINISH, RL_VSHARD_SEQ = 1, 2, 3, 4, 5
PARTIALS_SUMS = 14   # rl_loss_partials: sum[9] and count[5], combined by addition
PARTIALS_DOUBLES = 16  # ... then max[2], combined by maximum
CORRECTIONS = {"none": 0, "tis": 1, "clip_or_pop": 2}
ESTIMATORS = {"grpo": 0, "reinforcepp": 1, "reinforcepp_baseline": 2, "gspo": 3}
STATS_BYTES = 128


class RlLossParams(ctypes.Structure):
    _fields_ = [
        ("temperature", ctypes.c_float),
        ("eps_lo", ctypes.c_float),
        ("eps_hi", ctypes.c_float),
        ("dual_clip_c", ctypes.c_float),
        ("kl_coef", ctypes.c_float),
        ("entropy_coef", ctypes.c_float),
        ("std_floor", ctypes.c_float),
        ("normalize_std", ctypes.c_int32),
        ("unbiased_std", ctypes.c_int32),
        ("correction", ctypes.c_int32),
        ("corr_lo", ctypes.c_float),
        ("corr_hi", ctypes.c_float),
        ("opd_coef", ctypes.c_float),
        ("estimator", ctypes.c_int32),
        ("opd_topk", ctypes.c_int32),
        ("opd_topk_ids", ctypes.c_void_p),
        ("opd_topk_teacher", ctypes.c_void_p),
    ]


def make_params(temperature=1.0, eps_lo=0.2, eps_hi=0.2, dual_clip_c=0.0, kl_coef=0.0,
                entropy_coef=0.0, std_floor=1e-6, normalize_std=True, unbiased_std=True,
                correction="none", corr_lo=0.0, corr_hi=2.0, opd_coef=0.0, estimator="grpo",
                opd_topk=0, opd_topk_ids=None, opd_topk_teacher=None) -> RlLossParams:
    """One rl_loss_params. ``opd_topk_ids`` / ``opd_topk_teacher`` are device
    tensors ([n_rows, K] int32 / fp32); the caller keeps them alive."""
    return RlLossParams(temperature, eps_lo, eps_hi, dual_clip_c, kl_coef, entropy_coef,
                        std_floor, int(bool(normalize_std)), int(bool(unbiased_std)),
                        CORRECTIONS[correction] if isinstance(correction, str) else int(correction),
                        corr_lo, corr_hi, opd_coef,
                        ESTIMATORS[estimator] if isinstance(estimator, str) else int(estimator),
                        int(opd_topk),
                        None if opd_topk_ids is None else opd_topk_ids.data_ptr(),
                        None if opd_topk_teacher is None else opd_topk_teacher.data_ptr())


class RlLaunchOverrides(ctypes.Structure):
    _fields_ = [
        ("sweep_kernel", ctypes.c_int32),
        ("cluster_size", ctypes.c_int32),
        ("cluster_stages", ctypes.c_int32),
        ("cluster_threads", ctypes.c_int32),
        ("cluster_ctas_per_sm", ctypes.c_int32),
        ("stream_chunk_bytes", ctypes.c_int32),
        ("stream_slots", ctypes.c_int32),
        ("stream_hold", ctypes.c_int32),
        ("stream_split_first", ctypes.c_int32),
        ("stream_prefetch_bytes", ctypes.c_int32),
        ("stream_ctas_per_sm", ctypes.c_int32),
        ("stall_first_wait_ns", ctypes.c_int64),
        ("stream_cluster", ctypes.c_int32),
    ]


SWEEP_KERNELS = {"cluster": 0, "stream": 1}


class MilesLossError(RuntimeError):
    def __init__(self, status: int, where: str):
        super().__init__(f"{where}: {status_string(status)} (status {status})")
        self.status = status


_lib = None


def library_path() -> str:
    return _build.LIB


def load(build_if_missing: bool = True) -> ctypes.CDLL:
    """Load libmilesloss.so (building it first if it is missing)."""
    global _lib
    if _lib is not None:
        return _lib
    path = _build.LIB
    if not os.path.exists(path):
        if not build_if_missing:
            raise RuntimeError(f"libmilesloss is not built ({path}); run build()")
        _build.build()
    lib = ctypes.CDLL(path)
    P, I64, I32, F32, SZ = (ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float,
                            ctypes.c_size_t)
    PP = ctypes.POINTER(RlLossParams)
    lib.rl_loss_workspace_size.argtypes = [I64, I32, I32, ctypes.POINTER(SZ)]
    fwd_common = [P, I32, I64, I64, I64, P, P, P, P, P, P, P, P, I32, I32, P, PP, P, P, P, P, P]
    lib.rl_loss_fwd.argtypes = fwd_common + [P, SZ, P]
    lib.rl_loss_fwd_bwd.argtypes = fwd_common + [F32, P, P, I32, I64, P, SZ, P]
    lib.rl_loss_fwd_bwd_rows.argtypes = [I32, I64, I64] + fwd_common + [F32, P, P, I32, I64, P,
                                                                        SZ, P]
    lib.rl_loss_bwd.argtypes = [P, I32, I64, I64, I64, P, P, PP, F32, P, P, SZ, P, I32, I64, P]
    lib.rl_loss_check_device_error.argtypes = [P]
    lib.rl_status_string.argtypes = [I32]
    lib.rl_status_string.restype = ctypes.c_char_p
    lib.rl_set_sweep_events.argtypes = [P, P]
    lib.rl_launch_overrides_init.argtypes = [ctypes.POINTER(RlLaunchOverrides)]
    lib.rl_set_launch_overrides.argtypes = [ctypes.POINTER(RlLaunchOverrides)]
    lib.rl_loss_fwd_bwd_noalloc.argtypes = fwd_common + [F32, P, P, I32, I64, P]
    lib.rl_loss_shard_fwd_bwd.argtypes = ([I32, I64, I64] + fwd_common[:-1] + [P, P, P, P] +
                                          [F32, P, P, I32, I64, P, SZ, P])
    lib.rl_loss_vocab_shard_fwd_bwd.argtypes = (
        [I32, I32, I32, P, I64, I64, P, I32, I64, I64] + fwd_common[5:-1] + [P, P, P, P, P, P] +
        [F32, P, P, I32, I64, P, SZ, P])
    lib.rl_loss_noalloc_check_device_error.argtypes = []
    for name in ("rl_loss_workspace_size", "rl_loss_fwd", "rl_loss_fwd_bwd", "rl_loss_fwd_bwd_rows",
                 "rl_loss_bwd", "rl_loss_fwd_bwd_noalloc", "rl_loss_noalloc_check_device_error",
                 "rl_loss_shard_fwd_bwd", "rl_loss_vocab_shard_fwd_bwd",
                 "rl_launch_overrides_init", "rl_set_launch_overrides",
                 "rl_loss_check_device_error", "rl_set_sweep_events", "rl_loss_abi_version"):
        getattr(lib, name).restype = ctypes.c_int32
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().rl_status_string(int(status)).decode()


def _check(status: int, where: str):
    if status != RL_OK:
        raise MilesLossError(status, where)


def _ptr(t):
    return None if t is None else ctypes.c_void_p(t.data_ptr())


def _dtype_code(t) -> int:
    import torch
    if t.dtype == torch.bfloat16:
        return RL_BF16
    if t.dtype == torch.float32:
        return RL_F32
    raise TypeError(f"unsupported dtype {t.dtype}")


def _stream(stream):
    import torch
    s = torch.cuda.current_stream() if stream is None else stream
    return ctypes.c_void_p(s.cuda_stream)


def rl_loss_workspace_size(n_rows: int, n_traj: int, n_groups: int) -> int:
    out = ctypes.c_size_t(0)
    _check(load().rl_loss_workspace_size(n_rows, n_traj, n_groups, ctypes.byref(out)),
           "rl_loss_workspace_size")
    return int(out.value)


def _params(p) -> RlLossParams:
    if isinstance(p, RlLossParams):
        return p
    return make_params(**(p or {}))


def _fwd_args(logits, vocab, targets, rollout_logprobs, ref_logprobs, old_logprobs,
              teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask, params,
              token_logprobs, entropy, advantages, group_sizes, stats):
    n_rows = int(logits.shape[0])
    V = int(logits.shape[1]) if vocab is None else int(vocab)
    n_traj = int(rewards.shape[0]) if rewards is not None else 0
    return [_ptr(logits), _dtype_code(logits), n_rows, V, int(logits.stride(0)), _ptr(targets),
            _ptr(rollout_logprobs), _ptr(ref_logprobs), _ptr(old_logprobs),
            _ptr(teacher_logprobs), _ptr(rewards), _ptr(group_id), _ptr(cu_seqlens), n_traj,
            int(n_groups), _ptr(loss_mask), ctypes.byref(_params(params)), _ptr(token_logprobs),
            _ptr(entropy), _ptr(advantages), _ptr(group_sizes), _ptr(stats)]


def rl_loss_fwd(logits, targets, rollout_logprobs, ref_logprobs, old_logprobs, teacher_logprobs,
                rewards, group_id, cu_seqlens, n_groups, loss_mask, params, token_logprobs,
                entropy, advantages, group_sizes, stats, workspace, vocab=None, stream=None):
    args = _fwd_args(logits, vocab, targets, rollout_logprobs, ref_logprobs, old_logprobs,
                     teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask, params,
                     token_logprobs, entropy, advantages, group_sizes, stats)
    _check(load().rl_loss_fwd(*args, _ptr(workspace), workspace.numel() * workspace.element_size(),
                              _stream(stream)), "rl_loss_fwd")


def rl_loss_fwd_bwd(logits, targets, rollout_logprobs, ref_logprobs, old_logprobs,
                    teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask, params,
                    token_logprobs, entropy, advantages, group_sizes, stats, dlogits, workspace,
                    grad_loss=1.0, grad_loss_device=None, vocab=None, stream=None):
    args = _fwd_args(logits, vocab, targets, rollout_logprobs, ref_logprobs, old_logprobs,
                     teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask, params,
                     token_logprobs, entropy, advantages, group_sizes, stats)
    _check(load().rl_loss_fwd_bwd(*args, float(grad_loss), _ptr(grad_loss_device), _ptr(dlogits),
                                  _dtype_code(dlogits), int(dlogits.stride(0)), _ptr(workspace),
                                  workspace.numel() * workspace.element_size(), _stream(stream)),
           "rl_loss_fwd_bwd")


def rl_loss_fwd_bwd_rows(phase, row_begin, row_end, n_rows, logits, targets, rollout_logprobs,
                         ref_logprobs, old_logprobs, teacher_logprobs, rewards, group_id,
                         cu_seqlens, n_groups, loss_mask, params, token_logprobs, entropy,
                         advantages, group_sizes, stats, dlogits, workspace, vocab,
                         logits_dtype=None, grad_loss=1.0, grad_loss_device=None, stream=None):
    """One phase (or several) of the chunked call. ``logits`` / ``dlogits``
    hold rows [row_begin, row_end) (their row 0 is row row_begin) or are None
    outside the ROWS phase (``dlogits`` None: forward only); every other
    per-row tensor covers all n_rows."""
    import torch
    n_traj = int(rewards.shape[0]) if rewards is not None else 0
    if logits is not None:
        ldt, ld = _dtype_code(logits), int(logits.stride(0))
    else:
        ldt = _dtype_code(torch.empty(0, dtype=logits_dtype or torch.bfloat16))
        ld = int(vocab)
    if dlogits is not None:
        ddt, ld_out = _dtype_code(dlogits), int(dlogits.stride(0))
    else:
        ddt, ld_out = ldt, int(vocab)
    _check(load().rl_loss_fwd_bwd_rows(
        int(phase), int(row_begin), int(row_end), _ptr(logits), ldt, int(n_rows), int(vocab), ld,
        _ptr(targets), _ptr(rollout_logprobs), _ptr(ref_logprobs), _ptr(old_logprobs),
        _ptr(teacher_logprobs), _ptr(rewards), _ptr(group_id), _ptr(cu_seqlens), n_traj,
        int(n_groups), _ptr(loss_mask), ctypes.byref(_params(params)), _ptr(token_logprobs),
        _ptr(entropy), _ptr(advantages), _ptr(group_sizes), _ptr(stats), float(grad_loss),
        _ptr(grad_loss_device), _ptr(dlogits), ddt, ld_out, _ptr(workspace),
        workspace.numel() * workspace.element_size(), _stream(stream)), "rl_loss_fwd_bwd_rows")


def rl_loss_bwd(logits, targets, loss_mask, params, workspace, dlogits, grad_loss=1.0,
                grad_loss_device=None, vocab=None, stream=None):
    V = int(logits.shape[1]) if vocab is None else int(vocab)
    _check(load().rl_loss_bwd(_ptr(logits), _dtype_code(logits), int(logits.shape[0]), V,
                              int(logits.stride(0)), _ptr(targets), _ptr(loss_mask),
                              ctypes.byref(_params(params)), float(grad_loss),
                              _ptr(grad_loss_device), _ptr(workspace),
                              workspace.numel() * workspace.element_size(), _ptr(dlogits),
                              _dtype_code(dlogits), int(dlogits.stride(0)), _stream(stream)),
           "rl_loss_bwd")


def rl_loss_check_device_error(workspace) -> int:
    return int(load().rl_loss_check_device_error(_ptr(workspace)))


def set_launch_overrides(**fields) -> None:
    """Install process-wide launch-plan overrides (rl_set_launch_overrides);
    no arguments removes them. ``sweep_kernel`` may be given as "cluster" or
    "stream"; any other field as in the header."""
    lib = load()
    if not fields:
        _check(lib.rl_set_launch_overrides(None), "rl_set_launch_overrides")
        return
    o = RlLaunchOverrides()
    _check(lib.rl_launch_overrides_init(ctypes.byref(o)), "rl_launch_overrides_init")
    for k, v in fields.items():
        if k == "sweep_kernel" and isinstance(v, str):
            v = SWEEP_KERNELS[v]
        if not hasattr(o, k):
            raise TypeError(f"unknown launch override {k!r}")
        setattr(o, k, int(v))
    _check(lib.rl_set_launch_overrides(ctypes.byref(o)), "rl_set_launch_overrides")


class launch_overrides:
    """Context manager: the given overrides while the block runs, none after."""

    def __init__(self, **fields):
        self.fields = fields

    def __enter__(self):
        set_launch_overrides(**self.fields)
        return self

    def __exit__(self, *exc):
        set_launch_overrides()
        return False


def rl_loss_fwd_bwd_noalloc(logits, targets, rollout_logprobs, ref_logprobs, old_logprobs,
                            teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask,
                            params, token_logprobs, entropy, advantages, group_sizes, stats,
                            dlogits, grad_loss=1.0, grad_loss_device=None, vocab=None,
                            stream=None):
    """rl_loss_fwd_bwd without a workspace (the library's fixed array)."""
    args = _fwd_args(logits, vocab, targets, rollout_logprobs, ref_logprobs, old_logprobs,
                     teacher_logprobs, rewards, group_id, cu_seqlens, n_groups, loss_mask, params,
                     token_logprobs, entropy, advantages, group_sizes, stats)
    _check(load().rl_loss_fwd_bwd_noalloc(*args, float(grad_loss), _ptr(grad_loss_device),
                                          _ptr(dlogits), _dtype_code(dlogits),
                                          int(dlogits.stride(0)), _stream(stream)),
           "rl_loss_fwd_bwd_noalloc")


def rl_loss_shard_fwd_bwd(phase, row_offset, n_rows_total, logits, targets, rollout_logprobs,
                          ref_logprobs, old_logprobs, teacher_logprobs, rewards, group_id,
                          cu_seqlens, n_groups, loss_mask, params, token_logprobs, entropy,
                          advantages, group_sizes, traj_counts, partials, stats, dlogits,
                          workspace, vocab, n_rows=None, logits_dtype=None, grad_loss=1.0,
                          grad_loss_device=None, stream=None, traj_sums=None):
    """One phase of a shard's part of a row-sharded call. Per-row tensors
    hold the shard's rows; ``traj_counts`` is int32 [n_traj], ``partials``
    float64 [16] (one rl_loss_partials) and ``traj_sums`` (GSPO) float64
    [n_traj, 2], all on the device."""
    import torch
    n_traj = int(rewards.shape[0]) if rewards is not None else 0
    if logits is not None:
        ldt, ld, R = _dtype_code(logits), int(logits.stride(0)), int(logits.shape[0])
    else:
        ldt = _dtype_code(torch.empty(0, dtype=logits_dtype or torch.bfloat16))
        ld, R = int(vocab), int(n_rows if n_rows is not None else targets.shape[0])
    if dlogits is not None:
        ddt, ld_out = _dtype_code(dlogits), int(dlogits.stride(0))
    else:
        ddt, ld_out = ldt, int(vocab)
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().rl_loss_shard_fwd_bwd(
        int(phase), int(row_offset), int(n_rows_total), _ptr(logits), ldt, R, int(vocab), ld,
        _ptr(targets), _ptr(rollout_logprobs), _ptr(ref_logprobs), _ptr(old_logprobs),
        _ptr(teacher_logprobs), _ptr(rewards), _ptr(group_id), _ptr(cu_seqlens), n_traj,
        int(n_groups), _ptr(loss_mask), ctypes.byref(_params(params)), _ptr(token_logprobs),
        _ptr(entropy), _ptr(advantages), _ptr(group_sizes), _ptr(traj_counts), _ptr(traj_sums),
        _ptr(partials), _ptr(stats), float(grad_loss), _ptr(grad_loss_device), _ptr(dlogits), ddt,
        ld_out, _ptr(workspace), ws_bytes, _stream(stream)), "rl_loss_shard_fwd_bwd")


def rl_loss_vocab_shard_fwd_bwd(phase, col_shard, col_starts, row_offset, n_rows_total, logits,
                                targets, rollout_logprobs, ref_logprobs, old_logprobs,
                                teacher_logprobs, rewards, group_id, cu_seqlens, n_groups,
                                loss_mask, params, token_logprobs, entropy, advantages,
                                group_sizes, traj_counts, row_partials, row_partials_all,
                                partials, stats, dlogits, workspace, n_rows=None,
                                logits_dtype=None, grad_loss=1.0, grad_loss_device=None,
                                stream=None, traj_sums=None):
    """One phase of a column shard's part of a vocabulary-sharded call.
    ``col_starts`` is a host sequence of n_col_shards + 1 vocabulary ids;
    ``logits`` / ``dlogits`` hold this shard's columns of its rows;
    ``row_partials`` is float32 [n_rows, 8] and ``row_partials_all`` float32
    [n_col_shards, n_rows, 8] (device)."""
    import torch
    cs = [int(c) for c in col_starts]
    n_shards = len(cs) - 1
    c_arr = (ctypes.c_int64 * len(cs))(*cs)
    V = cs[col_shard + 1] - cs[col_shard] if 0 <= col_shard < n_shards else 1
    n_traj = int(rewards.shape[0]) if rewards is not None else 0
    if logits is not None:
        ldt, ld, R = _dtype_code(logits), int(logits.stride(0)), int(logits.shape[0])
    else:
        ldt = _dtype_code(torch.empty(0, dtype=logits_dtype or torch.bfloat16))
        ld, R = V, int(n_rows if n_rows is not None else targets.shape[0])
    if dlogits is not None:
        ddt, ld_out = _dtype_code(dlogits), int(dlogits.stride(0))
    else:
        ddt, ld_out = ldt, V
    ws_bytes = 0 if workspace is None else workspace.numel() * workspace.element_size()
    _check(load().rl_loss_vocab_shard_fwd_bwd(
        int(phase), int(col_shard), n_shards, ctypes.cast(c_arr, ctypes.c_void_p),
        int(row_offset), int(n_rows_total), _ptr(logits), ldt, R, ld, _ptr(targets),
        _ptr(rollout_logprobs), _ptr(ref_logprobs), _ptr(old_logprobs), _ptr(teacher_logprobs),
        _ptr(rewards), _ptr(group_id), _ptr(cu_seqlens), n_traj, int(n_groups), _ptr(loss_mask),
        ctypes.byref(_params(params)), _ptr(token_logprobs), _ptr(entropy), _ptr(advantages),
        _ptr(group_sizes), _ptr(traj_counts), _ptr(traj_sums), _ptr(row_partials),
        _ptr(row_partials_all),
        _ptr(partials), _ptr(stats), float(grad_loss), _ptr(grad_loss_device), _ptr(dlogits), ddt,
        ld_out, _ptr(workspace), ws_bytes, _stream(stream)), "rl_loss_vocab_shard_fwd_bwd")


def rl_loss_noalloc_check_device_error() -> int:
    return int(load().rl_loss_noalloc_check_device_error())


def rl_set_sweep_events(begin=None, end=None):
    _check(load().rl_set_sweep_events(None if begin is None else ctypes.c_void_p(begin.cuda_event),
                                      None if end is None else ctypes.c_void_p(end.cuda_event)),
           "rl_set_sweep_events")


_STATS_FMT = "<9d2f5q"
STATS_FIELDS = ("loss", "pg_loss_mean", "kl_mean", "entropy_mean", "ratio_mean",
                "ratio_absdev_mean", "logprob_absdiff_mean", "corr_ratio_mean",
                "corr_absdev_mean", "ratio_min", "ratio_max", "n_tokens", "n_clip_hi",
                "n_clip_lo", "n_dual_clip", "n_corr_clip")
assert struct.calcsize(_STATS_FMT) == 120


def parse_stats(raw: bytes) -> dict:
    """Decode one rl_loss_stats (bytes copied back from the device)."""
    return dict(zip(STATS_FIELDS, struct.unpack(_STATS_FMT, bytes(raw)[:120])))
