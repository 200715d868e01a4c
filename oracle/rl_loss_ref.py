"""Float64 CPU oracle of the per-token RL loss over the vocabulary.

TEST INFRASTRUCTURE ONLY: imported by ``tests/``, ``__graft_entry__.smoke()``
and the CPU-baseline leg of ``bench.py``; never by the library.

Every function is the plain definition, written in numpy float64 in the order
the method states it, with no fusion, blocking or reordering beyond chunking
rows (which changes no arithmetic of any row). Inputs in bf16 or fp32 are
widened exactly to float64 first.

What the paper fixes (Miles v0.1, arxiv 2609.08368):
  * the importance ratio r = exp(log pi_train - log pi_rollout)      (Sec. 3.4)
  * GRPO: a trajectory is scored against the other trajectories of the same
    prompt, i.e. rewards are centred within their group                (Sec. 2, Sec. 9.1)
  * a group whose attempts all got the same reward carries no signal  (Sec. 2.2, Table 2)
  * tokens the model did not generate are loss-masked                 (Sec. 2.4)
  * truncated importance sampling (TIS): clamp the ratio
    exp(log pi_train - log pi_rollout) to an interval, default [0, 2], and
    use it as a per-token weight on the PG loss (log pi_train: given old
    log-probs, or the trainer's own log-prob of this pass, held constant);
    clip-or-pop: weight 0 outside the interval, the unclipped ratio inside;
    reported metrics: pre-clamp ratio, clipped fraction, mean |r - 1|  (Sec. 3.4)
  * OPD shaping: subtract coef * (log pi_student - log pi_teacher) of the
    sampled token from each token's advantage; both are fixed inputs   (Sec. 5.2)

What the paper leaves unwritten, and the reading taken here (each is listed
with its reason in the design notes): the PPO clipped surrogate with asymmetric
clip and dual clip (PPO, Schulman et al. 2017, cited in Sec. 3.4), the k3 KL
estimator exp(d) - d - 1 with d = log pi_ref - log pi, an entropy bonus, a
temperature dividing the logits, sample (n-1) standard deviation with a floor
max(sigma, floor), one global masked token-mean, strict inequalities at every
clip threshold.

Parity status: every function here is pinned by the CPU tests in
``tests/test_oracle_pins.py`` (closed forms, invariants, library special
cases, finite differences, brute force); the paper prints no worked example.
"""

from __future__ import annotations

from dataclasses import dataclass

import numpy as np

CORRECTIONS = ("none", "tis", "clip_or_pop")
ESTIMATORS = ("grpo", "reinforcepp", "reinforcepp_baseline", "gspo")


@dataclass(frozen=True)
class LossParams:
    """Scalar knobs of the loss (one set per call)."""

    temperature: float = 1.0
    eps_lo: float = 0.2
    eps_hi: float = 0.2
    dual_clip_c: float = 0.0      # 0 = off, else > 1
    kl_coef: float = 0.0          # beta
    entropy_coef: float = 0.0     # gamma: loss -= gamma * H
    std_floor: float = 1e-6
    normalize_std: bool = True    # GRPO divides by the group std
    unbiased_std: bool = True     # Bessel (n - 1)
    correction: str = "none"      # "none" | "tis" | "clip_or_pop"   (Sec. 3.4)
    corr_lo: float = 0.0
    corr_hi: float = 2.0
    opd_coef: float = 0.0         # lambda of Sec. 5.2
    estimator: str = "grpo"       # "grpo" | "reinforcepp" | "reinforcepp_baseline" | "gspo" (Sec. 3.4)
    opd_topk: int = 0             # K of the top-K OPD variant (Sec. 5.2), 0 = off


# --------------------------------------------------------------------------
# input widening
# --------------------------------------------------------------------------

def widen_bf16(bits: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) -> exact float64 values.

    A bf16 number is the upper half of the fp32 number with the same bits, so
    shifting the 16 bits into the top of a 32-bit word gives the fp32 value
    exactly, and fp32 -> fp64 is exact.
    """
    b = np.asarray(bits, dtype=np.uint16).astype(np.uint32) << np.uint32(16)
    return b.view(np.float32).astype(np.float64)


def _widen(z: np.ndarray) -> np.ndarray:
    if z.dtype == np.uint16:
        return widen_bf16(z)
    return np.asarray(z, dtype=np.float64)


# --------------------------------------------------------------------------
# (a2) log-softmax, gathered log-prob and entropy of each row
# --------------------------------------------------------------------------

def row_log_softmax(z: np.ndarray, y: np.ndarray, temperature: float):
    """Tempered log-softmax of each row, the sampled token's log-prob and the
    entropy of the row's distribution.

    s_j = z_j / T;  lse = log sum_j exp(s_j) (taken as M + log sum exp(s - M)
    with M = max s, the textbook stable form);  log p_j = s_j - lse;
    logp = log p_y;  H = -sum_j p_j log p_j.

    The ratio of Sec. 3.4 needs log pi_train of the sampled token; the
    trainer computes it for the same tokens the rollout sampled (Sec. 9.2).
    Returns (logp [r], H [r], lse [r]) in float64.
    """
    s = _widen(z) / float(temperature)
    m = s.max(axis=1, keepdims=True)
    lse = m[:, 0] + np.log(np.exp(s - m).sum(axis=1))
    logp_all = s - lse[:, None]
    p = np.exp(logp_all)
    rows = np.arange(s.shape[0])
    logp = logp_all[rows, np.asarray(y, dtype=np.int64)]
    H = -_p_log_p(p, logp_all).sum(axis=1)
    return logp, H, lse


def _p_log_p(p, logp_all):
    """p log p with the limit 0 log 0 = 0 for a category of probability zero
    (a logit of -inf): such a category contributes nothing, as if it were
    absent from the vocabulary."""
    zero = np.isneginf(logp_all)
    return np.where(zero, 0.0, p * np.where(zero, 0.0, logp_all))


# --------------------------------------------------------------------------
# (a1) GRPO group-relative advantages
# --------------------------------------------------------------------------

def group_advantages(w: np.ndarray, gid: np.ndarray, n_groups: int, p: LossParams):
    """Per-trajectory GRPO advantages.

    Each trajectory is scored against the other trajectories for the same
    prompt (Sec. 2): with the members i of group g,
        mu = mean(w_i),  sigma = std(w_i) (n-1 if unbiased, n otherwise),
        A_i = (w_i - mu) / max(sigma, floor)      if normalize_std
        A_i =  w_i - mu                           otherwise.
    A group whose members all received the same reward carries no advantage
    signal (Sec. 2.2, Table 2): its A_i are exactly 0. A one-member group is
    such a group.
    Returns (A [n_traj] float64, n_g [n_groups] int64).
    """
    w = np.asarray(w, dtype=np.float64)
    gid = np.asarray(gid, dtype=np.int64)
    A = np.zeros(w.shape[0], dtype=np.float64)
    n_g = np.zeros(n_groups, dtype=np.int64)
    for g in range(n_groups):
        idx = np.nonzero(gid == g)[0]
        n_g[g] = idx.size
        if idx.size == 0:
            continue
        wg = w[idx]
        if wg.max() == wg.min():
            continue  # equal rewards: no signal, A stays exactly 0
        mu = wg.mean()
        if not p.normalize_std:
            A[idx] = wg - mu
            continue
        ddof = 1 if p.unbiased_std else 0
        sigma = float(np.sqrt(((wg - mu) ** 2).sum() / (idx.size - ddof)))
        A[idx] = (wg - mu) / max(sigma, p.std_floor)
    return A, n_g


def row_advantages(A_traj: np.ndarray, cu_seqlens: np.ndarray, n_rows: int) -> np.ndarray:
    """Broadcast each trajectory's advantage to its rows.

    Trajectory i owns rows [cu[i], cu[i+1]) of the packed layout; an outcome
    reward gives every token of the trajectory the same advantage.
    """
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    A_row = np.zeros(n_rows, dtype=np.float64)
    for i in range(cu.shape[0] - 1):
        A_row[cu[i]:cu[i + 1]] = A_traj[i]
    return A_row


def shape_advantages_opd(A_row: np.ndarray, student_lp: np.ndarray,
                         teacher_lp: np.ndarray, coef: float) -> np.ndarray:
    """On-policy distillation shaping (Sec. 5.2): after the estimator, each
    token's advantage loses coef * (log pi_student(x_t) - log pi_teacher(x_t)).
    Both log-probs are fixed inputs (recorded at rollout / by a teacher pass);
    the student's is the rollout-recorded one."""
    return np.asarray(A_row, np.float64) - coef * (
        np.asarray(student_lp, np.float64) - np.asarray(teacher_lp, np.float64))


def training_tokens_per_trajectory(cu_seqlens, mask) -> np.ndarray:
    """n_i = number of training tokens (mask 1) in trajectory i."""
    cu = np.asarray(cu_seqlens, dtype=np.int64)
    m = np.asarray(mask).astype(bool)
    return np.array([int(m[cu[i]:cu[i + 1]].sum()) for i in range(cu.shape[0] - 1)],
                    dtype=np.int64)


def estimator_advantages(w, gid, n_groups, cu_seqlens, mask, p: LossParams):
    """Per-row advantages of the configured estimator (Sec. 3.4 names GRPO,
    GSPO and REINFORCE++ in plain and baseline-relative forms).

    grpo, gspo: the GRPO advantage of the row's trajectory.
    reinforcepp: the trajectory's outcome reward is the return of each of its
        tokens; reinforcepp_baseline: the reward minus its group's mean reward.
        Either return is then normalised over all training tokens of the
        batch: A = (b - mu) / max(sigma, floor) with mu, sigma the mean and std
        (n - 1 if unbiased) of b over the tokens with mask 1 (centred only when
        normalize_std is off); A = 0 everywhere when those returns are all
        equal or no token trains.
    Returns (A_traj [n_traj], A_row [n_rows], group sizes)."""
    if p.estimator not in ESTIMATORS:
        raise ValueError(p.estimator)
    n_rows = int(np.asarray(mask).shape[0])
    A_grpo, n_g = group_advantages(w, gid, n_groups, p)
    if p.estimator in ("grpo", "gspo"):
        return A_grpo, row_advantages(A_grpo, cu_seqlens, n_rows), n_g
    w = np.asarray(w, np.float64)
    gid = np.asarray(gid, np.int64)
    b = w.copy()
    if p.estimator == "reinforcepp_baseline":
        for g in range(n_groups):
            idx = gid == g
            if idx.any():
                b[idx] = w[idx] - w[idx].mean()
    b_row = row_advantages(b, cu_seqlens, n_rows)
    m = np.asarray(mask).astype(bool)
    N = int(m.sum())
    A = np.zeros_like(b)
    if N > 0 and b_row[m].max() != b_row[m].min():
        mu = b_row[m].mean()
        A = b - mu
        if p.normalize_std:
            ddof = 1 if p.unbiased_std else 0
            sigma = float(np.sqrt(((b_row[m] - mu) ** 2).sum() / (N - ddof))) if N > ddof else 0.0
            A = A / max(sigma, p.std_floor)
    return A, row_advantages(A, cu_seqlens, n_rows), n_g


def opd_topk_estimate(z_rows, temperature, lse, cand_ids, teacher_lp):
    """Top-K on-policy distillation signal (Sec. 5.2): the teacher scores a
    candidate set per position; the estimate is the weighted sum, over the
    set, of log pi_student - log pi_teacher, weighted by the student's
    probabilities renormalised over the set (the reverse KL restricted to
    the set). The student's log-probs are the trainer's, from the logits;
    the estimate is a fixed per-token signal (no gradient flows through it).
    A candidate id outside [0, V) is an input error (raised, never wrapped
    around to another column)."""
    s = _widen(z_rows) / float(temperature)
    ids = np.asarray(cand_ids, np.int64)
    if ids.size and (ids.min() < 0 or ids.max() >= s.shape[1]):
        raise ValueError("top-K candidate id outside [0, vocab)")
    rows = np.arange(s.shape[0])[:, None]
    lps = s[rows, ids] - np.asarray(lse, np.float64)[:, None]
    ps = np.exp(lps)
    wts = ps / ps.sum(axis=1, keepdims=True)
    return (wts * (lps - np.asarray(teacher_lp, np.float64))).sum(axis=1)


# --------------------------------------------------------------------------
# (a3) per-token objective
# --------------------------------------------------------------------------

def correction_ratio(logp, rho, old=None):
    """The train/rollout ratio the corrections act on (Sec. 3.4):
    rc = exp(log pi_train - log pi_rollout). log pi_train is ``old`` when the
    caller gives the trainer's log-probs from a separate pass, else the
    trainer's own log-prob of the token in this pass. Either way the ratio
    is a constant per-token weight: no gradient flows through it."""
    train = np.asarray(logp if old is None else old, np.float64)
    return np.exp(train - np.asarray(rho, np.float64))


def token_objective(logp, rho, q, A_row, H, p: LossParams, old=None):
    """Per-token loss terms and the derivative of the token loss w.r.t. logp.

    ratio (Sec. 3.4):  r = exp(logp - base), base = old if given else rho.
    PPO clip:          u = -A r;  c = -A clip(r, 1-eps_lo, 1+eps_hi);
                       pg = max(u, c); clipped iff c > u (strict);
                       clip_hi iff clipped and r > 1+eps_hi; clip_lo iff
                       clipped and r < 1-eps_lo.
    dual clip:         if c_dual > 0 and A < 0: d = -A c_dual; if d < pg
                       (strict) then pg = d and the token is dual-clipped.
    correction (Sec. 3.4): rc = correction_ratio(logp, rho, old), the
                       train/rollout ratio (exp(old - rho), or without old
                       exp(logp - rho) of this pass), a constant weight:
                       TIS wt = min(max(rc, lo), hi);
                       clip-or-pop wt = rc if lo <= rc <= hi else 0;
                       pg <- wt * pg.
    k3 KL:             dlt = q - logp; k3 = exp(dlt) - dlt - 1.
    token loss:        l = pg + beta k3 - gamma H.
    G = dl/dlogp:      wt * (-A r if neither clipped nor dual-clipped else 0)
                       + beta (1 - exp(dlt)).
    """
    logp = np.asarray(logp, np.float64)
    rho = np.asarray(rho, np.float64)
    A = np.asarray(A_row, np.float64)
    H = np.asarray(H, np.float64)
    base = rho if old is None else np.asarray(old, np.float64)
    r = np.exp(logp - base)
    u = -A * r
    c = -A * np.clip(r, 1.0 - p.eps_lo, 1.0 + p.eps_hi)
    pg = np.maximum(u, c)
    clipped = c > u
    clip_hi = clipped & (r > 1.0 + p.eps_hi)
    clip_lo = clipped & (r < 1.0 - p.eps_lo)
    dual = np.zeros_like(clipped)
    if p.dual_clip_c > 0.0:
        d = -A * p.dual_clip_c
        dual = (A < 0.0) & (d < pg)
        pg = np.where(dual, d, pg)
    g_pg = np.where(clipped | dual, 0.0, -A * r)

    wt = np.ones_like(r)
    rc = np.ones_like(r)
    corr_clip = np.zeros_like(clipped)
    if p.correction != "none":
        if p.correction not in CORRECTIONS:
            raise ValueError(p.correction)
        rc = correction_ratio(logp, rho, old)
        outside = (rc < p.corr_lo) | (rc > p.corr_hi)
        corr_clip = outside
        if p.correction == "tis":
            wt = np.minimum(np.maximum(rc, p.corr_lo), p.corr_hi)
        else:
            wt = np.where(outside, 0.0, rc)
        pg = wt * pg
        g_pg = wt * g_pg

    if q is None:
        dlt = np.zeros_like(logp)
        k3 = np.zeros_like(logp)
        g_kl = np.zeros_like(logp)
    else:
        dlt = np.asarray(q, np.float64) - logp
        k3 = np.exp(dlt) - dlt - 1.0
        g_kl = 1.0 - np.exp(dlt)
    ell = pg + p.kl_coef * k3 - p.entropy_coef * H
    G = g_pg + p.kl_coef * g_kl
    return dict(r=r, pg=pg, k3=k3, ell=ell, G=G, clip_hi=clip_hi, clip_lo=clip_lo,
                dual=dual, wt=wt, rc=rc, corr_clip=corr_clip)


def sequence_objective(logp, rho, q, A_traj, H, cu_seqlens, mask, p: LossParams, old=None):
    """GSPO (Sec. 3.4 lists it among the estimators; Zheng et al. 2025): the
    importance ratio of trajectory i is the length-normalised sequence ratio
        s_i = exp( (1/n_i) sum_{t in i, m_t = 1} (logp_t - base_t) ),
    clipped at the sequence level with the trajectory's GRPO advantage A_i:
        pg_i = max(-A_i s_i, -A_i clip(s_i, 1-eps_lo, 1+eps_hi)), dual clip for
        A_i < 0 as in the token objective;
    the policy term is the mean of pg_i over the n_seq trajectories that have
    training tokens, the k3 and entropy terms stay token means. Written per
    row so that sum m l / N is that loss: a training token of trajectory i
    carries l_t = (N / (n_seq n_i)) pg_i + beta k3_t - gamma H_t and
    G_t = dl/dlogp_t = (N / (n_seq n_i)) (-A_i s_i if unclipped else 0)
    + beta (1 - exp(q_t - logp_t)). A ratio correction (Sec. 3.4) weights each
    token's share by its constant weight w_t; since s_i depends on every
    token of the trajectory, the policy part of G_t then carries the mean of
    w over the trajectory's training tokens. Every row of trajectory i
    reports r = s_i and the sequence's clip flags."""
    logp = np.asarray(logp, np.float64)
    rho = np.asarray(rho, np.float64)
    H = np.asarray(H, np.float64)
    base = rho if old is None else np.asarray(old, np.float64)
    cu = np.asarray(cu_seqlens, np.int64)
    m = np.asarray(mask).astype(bool)
    N = int(m.sum())
    n_i = training_tokens_per_trajectory(cu, m)
    n_seq = int((n_i > 0).sum())
    R = logp.shape[0]
    # ratio correction (Sec. 3.4): a constant weight on each token's share
    wt = np.ones(R)
    rc = np.ones(R)
    corr_clip = np.zeros(R, bool)
    if p.correction != "none":
        rc = correction_ratio(logp, rho, old)
        outside = (rc < p.corr_lo) | (rc > p.corr_hi)
        corr_clip = outside
        wt = (np.minimum(np.maximum(rc, p.corr_lo), p.corr_hi) if p.correction == "tis"
              else np.where(outside, 0.0, rc))
    r = np.ones(R)
    pg = np.zeros(R)
    g_pg = np.zeros(R)
    clip_hi = np.zeros(R, bool)
    clip_lo = np.zeros(R, bool)
    dual = np.zeros(R, bool)
    for i in range(cu.shape[0] - 1):
        if n_i[i] == 0:
            continue
        rows = slice(cu[i], cu[i + 1])
        mm = m[rows]
        s_i = float(np.exp((logp[rows][mm] - base[rows][mm]).sum() / n_i[i]))
        A = float(A_traj[i])
        u = -A * s_i
        c = -A * min(max(s_i, 1.0 - p.eps_lo), 1.0 + p.eps_hi)
        pgi = max(u, c)
        clipped = c > u
        du = False
        if p.dual_clip_c > 0.0 and A < 0.0:
            d = -A * p.dual_clip_c
            if d < pgi:
                pgi, du = d, True
        scale = N / (n_seq * n_i[i])
        r[rows] = s_i
        pg[rows] = scale * pgi * wt[rows]
        # every token's logp moves s_i, which every share of the trajectory
        # carries: the gradient takes the trajectory's mean weight
        mean_wt = float(wt[rows][mm].mean())
        g_pg[rows] = 0.0 if (clipped or du) else scale * mean_wt * (-A * s_i)
        clip_hi[rows] = clipped and s_i > 1.0 + p.eps_hi
        clip_lo[rows] = clipped and s_i < 1.0 - p.eps_lo
        dual[rows] = du
    if q is None:
        k3 = np.zeros(R)
        g_kl = np.zeros(R)
    else:
        dlt = np.asarray(q, np.float64) - logp
        k3 = np.exp(dlt) - dlt - 1.0
        g_kl = 1.0 - np.exp(dlt)
    ell = pg + p.kl_coef * k3 - p.entropy_coef * H
    G = g_pg + p.kl_coef * g_kl
    return dict(r=r, pg=pg, k3=k3, ell=ell, G=G, clip_hi=clip_hi, clip_lo=clip_lo, dual=dual,
                wt=wt, rc=rc, corr_clip=corr_clip)


# --------------------------------------------------------------------------
# (a4) masked token-mean and the reported metrics
# --------------------------------------------------------------------------

def masked_token_mean(ell: np.ndarray, mask: np.ndarray):
    """One global token mean over the tokens that train: L = sum m l / N,
    N = sum m (L = 0 when N = 0). Returns (L, N)."""
    m = np.asarray(mask).astype(bool)
    N = int(m.sum())
    if N == 0:
        return 0.0, 0
    return float(np.asarray(ell, np.float64)[m].sum() / N), N


def loss_stats(obj: dict, logp, rho, H, mask) -> dict:
    """Metrics over the tokens that train (m = 1): means of r, |r - 1|,
    |logp - rho| (the train/rollout divergence of Sec. 9.2), k3, H and the PG
    term; min / max of r; counts of clip_hi / clip_lo / dual-clipped tokens;
    for a correction (Sec. 3.4) the mean pre-clamp ratio rc, the number of
    tokens whose weight was changed, and mean |rc - 1|. All zero when N = 0."""
    m = np.asarray(mask).astype(bool)
    N = int(m.sum())
    L, _ = masked_token_mean(obj["ell"], m)
    out = dict(loss=L, n_tokens=N,
               n_clip_hi=int(obj["clip_hi"][m].sum()),
               n_clip_lo=int(obj["clip_lo"][m].sum()),
               n_dual_clip=int(obj["dual"][m].sum()),
               n_corr_clip=int(obj["corr_clip"][m].sum()))
    if N == 0:
        out.update(pg_loss_mean=0.0, kl_mean=0.0, entropy_mean=0.0, ratio_mean=0.0,
                   ratio_absdev_mean=0.0, logprob_absdiff_mean=0.0, ratio_min=0.0,
                   ratio_max=0.0, corr_ratio_mean=0.0, corr_absdev_mean=0.0)
        return out
    r = obj["r"][m]
    out.update(
        pg_loss_mean=float(obj["pg"][m].sum() / N),
        kl_mean=float(obj["k3"][m].sum() / N),
        entropy_mean=float(np.asarray(H, np.float64)[m].sum() / N),
        ratio_mean=float(r.sum() / N),
        ratio_absdev_mean=float(np.abs(r - 1.0).sum() / N),
        logprob_absdiff_mean=float(np.abs(np.asarray(logp, np.float64)[m]
                                          - np.asarray(rho, np.float64)[m]).sum() / N),
        ratio_min=float(r.min()),
        ratio_max=float(r.max()),
        corr_ratio_mean=float(obj["rc"][m].sum() / N),
        corr_absdev_mean=float(np.abs(obj["rc"][m] - 1.0).sum() / N),
    )
    return out


# --------------------------------------------------------------------------
# (a5) dLogits
# --------------------------------------------------------------------------

def dlogits_rows(z, y, temperature, lse, H, G, mask, N, grad_loss, entropy_coef):
    """Gradient of g * L with respect to the logits of the given rows.

    With p_j = exp(s_j - lse), d logp / d s_j = 1[j = y] - p_j and
    d H / d s_j = -p_j (log p_j + H); the chain rule through l = pg + beta k3
    - gamma H and L = sum m l / N gives
        dZ_j = g (m / N) (1 / T) [ G (1[j = y] - p_j) + gamma p_j (log p_j + H) ].
    """
    s = _widen(z) / float(temperature)
    logp_all = s - np.asarray(lse, np.float64)[:, None]
    pj = np.exp(logp_all)
    onehot = np.zeros_like(s)
    onehot[np.arange(s.shape[0]), np.asarray(y, np.int64)] = 1.0
    m = np.asarray(mask).astype(np.float64)
    scale = (grad_loss * m / N / float(temperature)) if N > 0 else np.zeros_like(m)
    Gc = np.asarray(G, np.float64)[:, None]
    Hc = np.asarray(H, np.float64)[:, None]
    # the entropy term p_j (log p_j + H) vanishes with p_j (a logit of -inf)
    ent = np.where(np.isneginf(logp_all), 0.0, pj * (np.where(np.isneginf(logp_all), 0.0, logp_all) + Hc))
    return scale[:, None] * (Gc * (onehot - pj) + entropy_coef * ent)


# --------------------------------------------------------------------------
# whole pipeline
# --------------------------------------------------------------------------

def rl_loss_rows(z, y, rho, q, A_row, mask, N, p: LossParams, grad_loss=1.0,
                 old=None, want_dlogits=True):
    """Every per-row output for a set of rows, given the call-wide values
    (their advantages and the masked count N of the whole call)."""
    logp, H, lse = row_log_softmax(z, y, p.temperature)
    obj = token_objective(logp, rho, q, A_row, H, p, old=old)
    out = dict(logp=logp, H=H, lse=lse, **obj)
    if want_dlogits:
        out["dlogits"] = dlogits_rows(z, y, p.temperature, lse, H, obj["G"], mask, N,
                                      grad_loss, p.entropy_coef)
    return out


def rl_loss(z, y, rho, q, w, gid, cu_seqlens, n_groups, mask, p: LossParams,
            grad_loss=1.0, old=None, teacher=None, want_dlogits=True, chunk=256,
            topk_ids=None, topk_teacher=None):
    """The whole loss for one call: advantages, per-row outputs, the loss,
    the metrics, and (optionally) dLogits as a float64 array.

    Order (Sec. 5.2: the estimator first, then the OPD shaping): estimator
    advantages; row log-softmax statistics; OPD shaping (one-sample from the
    rollout / teacher log-probs, or top-K from the candidate sets); the token
    objective (or GSPO's sequence objective); masked mean and metrics;
    dLogits. Rows are processed in chunks of ``chunk`` rows; each row's
    arithmetic is independent of the chunking."""
    R = int(np.asarray(y).shape[0])
    m = np.asarray(mask).astype(bool)
    N = int(m.sum())
    A_traj, A_row, n_g = estimator_advantages(w, gid, n_groups, cu_seqlens, m, p)
    V = np.asarray(z).shape[1] if R else 0
    logp = np.zeros(R)
    H = np.zeros(R)
    lse = np.zeros(R)
    for lo in range(0, R, chunk):
        hi = min(R, lo + chunk)
        logp[lo:hi], H[lo:hi], lse[lo:hi] = row_log_softmax(z[lo:hi], np.asarray(y)[lo:hi],
                                                            p.temperature)
    if p.opd_coef != 0.0:
        if p.opd_topk > 0:
            est = np.zeros(R)
            for lo in range(0, R, chunk):
                hi = min(R, lo + chunk)
                est[lo:hi] = opd_topk_estimate(z[lo:hi], p.temperature, lse[lo:hi],
                                               np.asarray(topk_ids)[lo:hi],
                                               np.asarray(topk_teacher)[lo:hi])
            A_row = A_row - p.opd_coef * est
        else:
            A_row = shape_advantages_opd(A_row, rho, teacher, p.opd_coef)
    q_ = None if q is None else np.asarray(q)
    if p.estimator == "gspo":
        obj = sequence_objective(logp, rho, q_, A_traj, H, cu_seqlens, m, p, old=old)
    else:
        obj = token_objective(logp, rho, q_, A_row, H, p, old=old)
    cat = dict(obj, logp=logp, H=H, lse=lse)
    stats = loss_stats(cat, logp, rho, H, m)
    out = dict(cat, A_traj=A_traj, group_sizes=n_g, A_row=A_row, N=N, stats=stats,
               loss=stats["loss"])
    if want_dlogits:
        dz = [dlogits_rows(z[lo:min(R, lo + chunk)], np.asarray(y)[lo:min(R, lo + chunk)],
                           p.temperature, lse[lo:lo + chunk], H[lo:lo + chunk],
                           obj["G"][lo:lo + chunk], m[lo:lo + chunk], N, grad_loss,
                           p.entropy_coef)
              for lo in range(0, R, chunk)]
        out["dlogits"] = np.concatenate(dz) if dz else np.zeros((0, V))
    return out
