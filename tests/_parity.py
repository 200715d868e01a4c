"""Helpers of the GPU parity tests: run the CUDA library on a seeded
workload, run the float64 oracle on the same inputs (copied to the host),
and compare with the tolerances of the target:
  token log-probs / entropy   2e-3 absolute for bf16 logits, 1e-5 for fp32
  scalar loss                 1e-4 relative to the oracle's loss
  dLogits                     1e-2 relative or 1e-5 absolute
  integer outputs             exact (clip counts: exact outside a 1e-5
                              relative guard band around each threshold)
"""

from __future__ import annotations

import json
import os

import numpy as np
import torch

import oracle
from paper_2609_08368_gb300 import api
from paper_2609_08368_gb300 import milesloss as ml

GUARD = 1e-5


def oracle_params(params: dict) -> oracle.LossParams:
    return oracle.LossParams(**{k: v for k, v in params.items()
                                if k not in ("opd_topk_ids", "opd_topk_teacher")})


def gpu_params(w, params=None) -> dict:
    """The call's parameters with the top-K OPD inputs attached when used."""
    p = dict(w.params if params is None else params)
    if p.get("opd_topk", 0) > 0:
        p.update(opd_topk_ids=w.topk_ids, opd_topk_teacher=w.topk_teacher)
    return p


def host_logits(w, rows=None) -> np.ndarray:
    z = w.logits[:, :w.vocab] if rows is None else w.logits[rows, :w.vocab]
    z = z.cpu()
    if z.dtype == torch.bfloat16:
        return z.contiguous().view(torch.int16).numpy().view(np.uint16)
    return z.numpy()


def np_(t):
    return None if t is None else t.cpu().numpy()


def run_gpu(w, mode="fused", dl_dtype=None, grad_loss=1.0, ld_out=None, params=None):
    """mode: 'fused' (rl_loss_fwd_bwd), 'split' (rl_loss_fwd then rl_loss_bwd)
    or 'fwd' (rl_loss_fwd only)."""
    R, n_traj = w.n_rows, int(w.rewards.shape[0])
    if dl_dtype is None:
        dl_dtype = w.logits.dtype
    buf = api.alloc(R, n_traj, w.n_groups, w.logits.device, vocab=w.vocab,
                    dlogits_dtype=None if mode == "fwd" else dl_dtype, ld_out=ld_out,
                    fill_nan=True)
    params = gpu_params(w, params)
    if mode == "fused":
        api.fwd_bwd(w, buf, params=params, grad_loss=grad_loss)
    else:
        api.fwd(w, buf, params=params)
        if mode == "split":
            api.bwd(w, buf, params=params, grad_loss=grad_loss)
    torch.cuda.synchronize()
    out = dict(logp=np_(buf.token_logprobs), H=np_(buf.entropy), A=np_(buf.advantages),
               group_sizes=np_(buf.group_sizes), stats=buf.read_stats(),
               err=ml.rl_loss_check_device_error(buf.workspace), buf=buf)
    if buf.dlogits is not None:
        out["dlogits_t"] = buf.dlogits
    return out


def run_oracle(w, grad_loss=1.0, want_dlogits=True, params=None):
    p = oracle_params(params if params is not None else w.params)
    return oracle.rl_loss(host_logits(w), np_(w.targets), np_(w.rollout_logprobs),
                          np_(w.ref_logprobs), np_(w.rewards), np_(w.group_id),
                          np_(w.cu_seqlens), w.n_groups, np_(w.loss_mask), p,
                          grad_loss=grad_loss, old=np_(w.old_logprobs),
                          teacher=np_(w.teacher_logprobs), want_dlogits=want_dlogits,
                          topk_ids=np_(w.topk_ids), topk_teacher=np_(w.topk_teacher))


def logp_tol(w) -> float:
    return 2e-3 if w.logits.dtype == torch.bfloat16 else 1e-5


def assert_dlogits_close(got: np.ndarray, ref: np.ndarray, rel=1e-2, abs_=1e-5):
    got = got.astype(np.float64)
    err = np.abs(got - ref)
    bound = np.maximum(rel * np.abs(ref), abs_)
    bad = err > bound
    assert np.isfinite(got).all(), "non-finite dLogits"
    if bad.any():
        i = np.argwhere(bad)[0]
        raise AssertionError(f"dLogits mismatch at {tuple(i)}: got {got[tuple(i)]!r} "
                             f"ref {ref[tuple(i)]!r} ({int(bad.sum())} entries)")


def assert_rel_on_large(got: np.ndarray, ref: np.ndarray, terms: np.ndarray | None = None,
                        floor=1e-6, rel=1e-2, cancel=1e-4):
    """Relative error on every entry with |ref| >= floor (entries of O(p)).

    ``terms`` is the magnitude of the summands of each entry,
    |scale| p_j (|G| + gamma |log p_j + H|): where G and the entropy term
    nearly cancel, fp32 evaluation can only be accurate relative to them, so
    the bound is rel |ref| + cancel * terms."""
    got = got.astype(np.float64)
    sel = np.abs(ref) >= floor
    err = np.zeros_like(ref)
    denom = np.abs(ref) if terms is None else np.abs(ref) + (cancel / rel) * terms
    err[sel] = np.abs(got[sel] - ref[sel]) / denom[sel]
    assert sel.any()
    i = np.unravel_index(np.argmax(err), err.shape)
    assert err[i] <= rel, (f"max rel err {err[i]:.3g} at {i}: got {got[i]!r} ref {ref[i]!r} "
                           f"({int(sel.sum())} entries checked)")


def summand_magnitude(w, o, grad_loss, params=None):
    """|scale| p_j (|G| + gamma |log p_j + H|) for every entry (oracle values)."""
    p = oracle_params(params if params is not None else w.params)
    z = oracle.widen_bf16(host_logits(w)) if w.logits.dtype == torch.bfloat16 else \
        host_logits(w).astype(np.float64)
    logp_all = z / p.temperature - o["lse"][:, None]
    pj = np.exp(logp_all)
    m = np_(w.loss_mask).astype(np.float64)
    scale = grad_loss * m / max(o["N"], 1) / p.temperature
    return np.abs(scale)[:, None] * pj * (np.abs(o["G"])[:, None]
                                          + p.entropy_coef * np.abs(logp_all + o["H"][:, None]))


def clip_counts(p: oracle.LossParams, logp, rho, q, A_row, H, mask, old=None):
    """Clip counts of the oracle's decision rule applied to given log-probs,
    and the number of training tokens within the guard band of a threshold."""
    o = oracle.token_objective(logp, rho, q, A_row, H, p, old=old)
    m = np.asarray(mask).astype(bool)
    th = [1 - p.eps_lo, 1 + p.eps_hi] + ([p.dual_clip_c] if p.dual_clip_c else [])
    near = np.zeros_like(m)
    for t in th:
        near |= np.abs(o["r"] - t) <= GUARD * t
    if p.correction != "none":
        for t in (p.corr_lo, p.corr_hi):
            near |= np.abs(o["rc"] - t) <= GUARD * max(t, 1e-30)
    counts = dict(n_clip_hi=int(o["clip_hi"][m].sum()), n_clip_lo=int(o["clip_lo"][m].sum()),
                  n_dual_clip=int(o["dual"][m].sum()), n_corr_clip=int(o["corr_clip"][m].sum()))
    return counts, int((near & m).sum())


def fp32_logp_loss_floor(w, o, params=None) -> float:
    """The part of the loss error that fp32 log-probs cannot avoid when rows
    have large |lse|: the kernels form logp = z_y / T - lse in fp32, so a
    row's log-prob carries an error of a few ulp of max(|lse|, |z_y / T|)
    (8 eps (|lse| + |z_y / T|) with eps = 2^-24), and its entropy the same.
    Through l = pg + beta k3 - gamma H that moves the loss by at most
    sum m (|G| + gamma) * that / N. It matters only when |lse| is large (logits
    shifted to -1000, or divided by a small temperature); on ordinary rows it
    is far below 1e-4 |L| and is not used."""
    p = oracle_params(params if params is not None else w.params)
    z = host_logits(w)
    zw = oracle.widen_bf16(z) if z.dtype == np.uint16 else z.astype(np.float64)
    zy = zw[np.arange(w.n_rows), np_(w.targets).astype(np.int64)] / p.temperature
    m = np_(w.loss_mask).astype(bool)
    if not m.any():
        return 0.0
    row = 8 * 2.0 ** -24 * (np.abs(o["lse"]) + np.abs(zy))
    return float(((np.abs(o["G"]) + p.entropy_coef) * row)[m].sum() / m.sum())


def compare_forward(w, g, o, params=None, loss_floor=0.0):
    """Per-row outputs, advantages, group sizes, counts and the loss (to
    1e-4 relative, plus ``loss_floor`` where a test names one)."""
    p = oracle_params(params if params is not None else w.params)
    tol = logp_tol(w)
    np.testing.assert_allclose(g["logp"], o["logp"], atol=tol, rtol=0)
    np.testing.assert_allclose(g["H"], o["H"], atol=tol, rtol=0)
    np.testing.assert_allclose(g["A"], o["A_traj"], rtol=1e-6, atol=1e-6)
    np.testing.assert_array_equal(g["group_sizes"], o["group_sizes"])
    st = g["stats"]
    assert st["n_tokens"] == o["N"]
    # clip counts: the oracle's rule on the GPU's own log-probs reproduces the
    # GPU counts exactly (up to tokens in the guard band); against the
    # oracle's float64 log-probs they differ only inside the band.
    old = np_(w.old_logprobs)
    if p.estimator == "gspo":
        # sequence-level decisions: every training token of a trajectory
        # carries its sequence's flags; tokens of sequences whose ratio lies in
        # the guard band of a threshold may fall either way
        m = np_(w.loss_mask).astype(bool)
        th = [1 - p.eps_lo, 1 + p.eps_hi] + ([p.dual_clip_c] if p.dual_clip_c else [])
        band = int(sum(((np.abs(o["r"] - t) <= GUARD * t) & m).sum() for t in th))
        for k in ("n_clip_hi", "n_clip_lo", "n_dual_clip", "n_corr_clip"):
            assert abs(st[k] - o["stats"][k]) <= band, (k, st[k], o["stats"][k], band)
    else:
        c_gpu, band_g = clip_counts(p, g["logp"].astype(np.float64), np_(w.rollout_logprobs),
                                    np_(w.ref_logprobs), o["A_row"], g["H"], np_(w.loss_mask),
                                    old)
        c_ora, band_o = clip_counts(p, o["logp"], np_(w.rollout_logprobs), np_(w.ref_logprobs),
                                    o["A_row"], o["H"], np_(w.loss_mask), old)
        for k in c_gpu:
            assert abs(st[k] - c_gpu[k]) <= band_g, (k, st[k], c_gpu[k], band_g)
            assert abs(st[k] - c_ora[k]) <= band_g + band_o, (k, st[k], c_ora[k])
    os_ = o["stats"]
    assert_loss_close(st["loss"], os_["loss"], atol=loss_floor)
    # The metrics are functions of the row log-probs and entropies, which were
    # compared above at their own tolerance. Evaluated by the oracle on the
    # GPU's own log-probs and entropies, they must match the GPU's metrics to
    # 1e-4 (this checks the per-row objective and the reduction). Against the
    # oracle's float64 log-probs they would also carry the log-prob's fp32
    # evaluation error, a few ulp of |lse| (6e-5 at |lse| ~ 1e3), propagated.
    own = stats_on_gpu_logp(w, g, o, p)
    for k in ("ratio_mean", "ratio_absdev_mean", "logprob_absdiff_mean", "entropy_mean",
              "kl_mean", "pg_loss_mean", "corr_ratio_mean", "corr_absdev_mean",
              "ratio_min", "ratio_max"):
        assert abs(st[k] - own[k]) <= 1e-4 * max(abs(own[k]), 1e-3), (k, st[k], own[k], os_[k])


LOSS_RTOL = 1e-4
LOSS_ATOL = 1e-12  # only for losses that are exactly 0 (no training token)


def assert_loss_close(got: float, ref: float, what: str = "loss", atol: float = 0.0):
    """The scalar loss within 1e-4 of the oracle's, relative: |got - ref| <=
    1e-4 |ref| (+1e-12 for a loss of exactly 0, + ``atol`` where a test names
    an fp32 floor). The measured relative error is appended to the file named
    by LOSS_ERROR_LOG, when set."""
    err = abs(got - ref)
    rel = err / abs(ref) if ref != 0 else (0.0 if err == 0 else float("inf"))
    path = os.environ.get("LOSS_ERROR_LOG")
    if path:
        test = os.environ.get("PYTEST_CURRENT_TEST", "?").split(" ")[0]
        with open(path, "a") as f:
            f.write(json.dumps({"test": test, "what": what, "gpu": got, "oracle": ref,
                                "rel": rel, "floor": atol}) + "\n")
    assert err <= LOSS_RTOL * abs(ref) + LOSS_ATOL + atol, \
        f"{what}: gpu {got!r} oracle {ref!r} (relative error {rel:.3g} > {LOSS_RTOL})"


def stats_on_gpu_logp(w, g, o, p):
    """The oracle's objective and metrics evaluated on the GPU's row log-probs
    and entropies (the advantages are the oracle's)."""
    lp = g["logp"].astype(np.float64)
    H = g["H"].astype(np.float64)
    m = np_(w.loss_mask).astype(bool)
    rho, q, old = np_(w.rollout_logprobs), np_(w.ref_logprobs), np_(w.old_logprobs)
    if p.estimator == "gspo":
        obj = oracle.sequence_objective(lp, rho, q, o["A_traj"], H, np_(w.cu_seqlens), m, p,
                                        old=old)
    else:
        obj = oracle.token_objective(lp, rho, q, o["A_row"], H, p, old=old)
    return oracle.loss_stats(obj, lp, rho, H, m)
