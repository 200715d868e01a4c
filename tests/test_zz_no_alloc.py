"""The allocation-free entry point, rl_loss_fwd_bwd_noalloc.

It exists for callers that cannot allocate device memory when they compute
the loss (a framework that has reserved nearly all of HBM for its own pool,
a plain-C host or plugin without access to the allocator, code whose memory
footprint is fixed after start-up): it takes the inputs and outputs of
rl_loss_fwd_bwd but uses a fixed array inside the library instead of a
caller-provided workspace. These tests call it through the C ABI: after a
call of another shape, twice in a row against rl_loss_fwd_bwd with a
caller-provided workspace, within the tolerances the parity tests use; its
device-side errors read back with rl_loss_noalloc_check_device_error; and an
oversized call rejected before anything runs. It is collected last so
that a stop at its first failure has already run every other test.
"""

import ctypes

import numpy as np
import pytest
import torch

import _parity as P
from paper_2609_08368_gb300 import api, workloads as wl
from paper_2609_08368_gb300 import milesloss as ml

pytestmark = pytest.mark.gpu

RL_ERR_WORKSPACE_TOO_SMALL = 3


def _noalloc_fn():
    lib = ml.load()
    fn = lib.rl_loss_fwd_bwd_noalloc
    Pt, I64, I32, F32 = ctypes.c_void_p, ctypes.c_int64, ctypes.c_int32, ctypes.c_float
    fn.argtypes = [Pt, I32, I64, I64, I64, Pt, Pt, Pt, Pt, Pt, Pt, Pt, Pt, I32, I32, Pt,
                   ctypes.POINTER(ml.RlLossParams), Pt, Pt, Pt, Pt, Pt, F32, Pt, Pt, I32, I64, Pt]
    fn.restype = ctypes.c_int32
    return fn


def _call(fn, w, buf, n_rows=None):
    ptr = ml._ptr
    params = ml.make_params(**w.params)
    return fn(ptr(w.logits), ml._dtype_code(w.logits), w.n_rows if n_rows is None else n_rows,
              w.vocab, int(w.logits.stride(0)), ptr(w.targets), ptr(w.rollout_logprobs),
              ptr(w.ref_logprobs), ptr(w.old_logprobs), ptr(w.teacher_logprobs),
              ptr(w.rewards), ptr(w.group_id), ptr(w.cu_seqlens), int(w.rewards.shape[0]),
              w.n_groups, ptr(w.loss_mask), ctypes.byref(params), ptr(buf.token_logprobs),
              ptr(buf.entropy), ptr(buf.advantages), ptr(buf.group_sizes), ptr(buf.stats), 1.0,
              None, ptr(buf.dlogits), ml._dtype_code(buf.dlogits), int(buf.dlogits.stride(0)),
              ctypes.c_void_p(torch.cuda.current_stream().cuda_stream))


def _compare(out, ref, w):
    tol = P.logp_tol(w)
    np.testing.assert_allclose(out.token_logprobs.cpu().numpy(),
                               ref.token_logprobs.cpu().numpy(), atol=tol, rtol=0)
    np.testing.assert_allclose(out.entropy.cpu().numpy(), ref.entropy.cpu().numpy(),
                               atol=tol, rtol=0)
    np.testing.assert_allclose(out.advantages.cpu().numpy(), ref.advantages.cpu().numpy(),
                               rtol=1e-6, atol=1e-6)
    assert torch.equal(out.group_sizes, ref.group_sizes)
    P.assert_dlogits_close(out.dlogits.float().cpu().numpy(), ref.dlogits.double().cpu().numpy())
    st, rs = out.read_stats(), ref.read_stats()
    assert st["n_tokens"] == rs["n_tokens"]
    for k in ("n_clip_hi", "n_clip_lo", "n_dual_clip", "n_corr_clip"):
        assert st[k] == rs[k]
    P.assert_loss_close(st["loss"], rs["loss"], what="no-alloc loss")


def _workload(**kw):
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=64, vocab=20480,
                    rho_noise=0.35, ref_noise=0.3)
    return wl.make(wl.shrink(rec, **kw) if kw else rec, "cuda")


def _alloc(w):
    return api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, "cuda", vocab=w.vocab,
                     dlogits_dtype=torch.bfloat16, fill_nan=True)


def test_noalloc_matches_the_workspace_entry_point_twice():
    fn = _noalloc_fn()
    # The array keeps the previous call's contents: first a call of another
    # shape (more rows, trajectories and groups, with statistics, so that the
    # reduction ticket and the group tables move), then the checked calls.
    other = _workload(n_prompts=5, group_size=3, traj_len=40, vocab=12000, seed=77)
    assert _call(fn, other, _alloc(other)) == 0
    w = _workload()
    ref = _alloc(w)
    api.fwd_bwd(w, ref)
    torch.cuda.synchronize()
    assert ml.rl_loss_check_device_error(ref.workspace) == 0
    for _ in range(2):
        out = _alloc(w)
        assert _call(fn, w, out) == 0
        torch.cuda.synchronize()
        assert ml.rl_loss_noalloc_check_device_error() == 0
        _compare(out, ref, w)


def test_noalloc_reports_its_device_errors():
    """The data-dependent errors of a no-alloc call are read back with
    rl_loss_noalloc_check_device_error; the next clean call reads RL_OK."""
    fn = _noalloc_fn()
    w = _workload()
    w.targets[5] = w.vocab                 # target outside [0, vocab)
    out = _alloc(w)
    assert _call(fn, w, out) == 0
    torch.cuda.synchronize()
    assert ml.rl_loss_noalloc_check_device_error() == 5   # RL_ERR_TARGET_OUT_OF_RANGE
    assert out.token_logprobs[5].item() == 0.0 and (out.dlogits[5] == 0).all()
    w = _workload()
    w.group_id[2] = w.n_groups + 3         # group id outside [0, n_groups)
    assert _call(fn, w, _alloc(w)) == 0
    torch.cuda.synchronize()
    assert ml.rl_loss_noalloc_check_device_error() == 6   # RL_ERR_GROUP_OUT_OF_RANGE
    w = _workload()
    assert _call(fn, w, _alloc(w)) == 0
    torch.cuda.synchronize()
    assert ml.rl_loss_noalloc_check_device_error() == 0


def test_noalloc_rejects_calls_beyond_its_array():
    fn = _noalloc_fn()
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=1, group_size=2, traj_len=8, vocab=256)
    w = wl.make(rec, "cuda")
    buf = api.alloc(w.n_rows, 2, 1, "cuda", vocab=256, dlogits_dtype=torch.bfloat16)
    # 10 million rows need far more than the 8 MiB array: rejected on the
    # host before anything is enqueued (the pointers are never read).
    assert _call(fn, w, buf, n_rows=10_000_000) == RL_ERR_WORKSPACE_TOO_SMALL
