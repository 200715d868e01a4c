"""Mutation check of the oracle's pins (CPU): each planted mistake below,
applied to a temporary copy of oracle/rl_loss_ref.py (the tracked file is
never touched), must make tests/test_oracle_pins.py fail. The mistakes are the
plausible ones: a sign flipped, a term dropped, a transposed operand, a wrong
estimator convention, a strict comparison made loose."""

import os
import shutil
import subprocess
import sys
from concurrent.futures import ThreadPoolExecutor

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
SRC = os.path.join(ROOT, "oracle", "rl_loss_ref.py")

# (what the mistake is, text in the oracle, its replacement)
MUTANTS = [
    ("dLogits sign of the policy-gradient term",
     "scale[:, None] * (Gc * (onehot - pj)", "scale[:, None] * (Gc * (pj - onehot)"),
    ("entropy term of dLogits loses + H",
     "np.where(np.isneginf(logp_all), 0.0, logp_all) + Hc))",
     "np.where(np.isneginf(logp_all), 0.0, logp_all)))"),
    ("k3 gradient sign", "g_kl = 1.0 - np.exp(dlt)", "g_kl = np.exp(dlt) - 1.0"),
    ("dual clip comparison reversed", "dual = (A < 0.0) & (d < pg)", "dual = (A < 0.0) & (d > pg)"),
    ("std estimator swapped", "ddof = 1 if p.unbiased_std else 0", "ddof = 0 if p.unbiased_std else 1"),
    ("1/T dropped from dLogits", "(grad_loss * m / N / float(temperature))", "(grad_loss * m / N)"),
    ("correction weight dropped from the gradient", "        g_pg = wt * g_pg\n", "\n"),
    ("OPD shaping sign", "coef * (\n", "-coef * (\n"),
    ("clip test made loose", "clipped = c > u", "clipped = c >= u"),
    ("k3 loses its -1", "k3 = np.exp(dlt) - dlt - 1.0", "k3 = np.exp(dlt) - dlt"),
    ("entropy sign", "H = -_p_log_p(p, logp_all).sum(axis=1)", "H = _p_log_p(p, logp_all).sum(axis=1)"),
    ("0 log 0 limit dropped", "return np.where(zero, 0.0, p * np.where(zero, 0.0, logp_all))",
     "return p * logp_all"),
    ("REINFORCE++ baseline dropped", "b[idx] = w[idx] - w[idx].mean()", "b[idx] = w[idx]"),
    ("REINFORCE++ floor made additive", "A = A / max(sigma, p.std_floor)", "A = A / (sigma + p.std_floor)"),
    ("REINFORCE++ mean over all rows instead of training tokens", "mu = b_row[m].mean()", "mu = b.mean()"),
    ("GSPO 1/n_i dropped", "(logp[rows][mm] - base[rows][mm]).sum() / n_i[i]",
     "(logp[rows][mm] - base[rows][mm]).sum()"),
    ("GSPO mean correction weight dropped", "mean_wt = float(wt[rows][mm].mean())", "mean_wt = 1.0"),
    ("top-K weights unnormalised", "wts = ps / ps.sum(axis=1, keepdims=True)", "wts = ps"),
    ("top-K signal sign", "(wts * (lps - np.asarray(teacher_lp, np.float64)))",
     "(wts * (np.asarray(teacher_lp, np.float64) - lps))"),
    ("clip-or-pop keeps the weight 1", "wt = np.where(outside, 0.0, rc)", "wt = np.where(outside, 0.0, 1.0)"),
    ("GRPO floor made additive", "A[idx] = (wg - mu) / max(sigma, p.std_floor)",
     "A[idx] = (wg - mu) / (sigma + p.std_floor)"),
    ("entropy bonus sign", "ell = pg + p.kl_coef * k3 - p.entropy_coef * H",
     "ell = pg + p.kl_coef * k3 + p.entropy_coef * H"),
    ("ratio inverted", "r = np.exp(logp - base)", "r = np.exp(base - logp)"),
    ("lse drops its max", "lse = m[:, 0] + np.log(np.exp(s - m).sum(axis=1))",
     "lse = np.log(np.exp(s - m).sum(axis=1))"),
    ("temperature ignored in the log-softmax", "s = _widen(z) / float(temperature)\n    m = s.max",
     "s = _widen(z)\n    m = s.max"),
    ("first row of each trajectory without advantage", "A_row[cu[i]:cu[i + 1]] = A_traj[i]",
     "A_row[cu[i] + 1:cu[i + 1]] = A_traj[i]"),
    ("token mean over all rows", "return float(np.asarray(ell, np.float64)[m].sum() / N), N",
     "return float(np.asarray(ell, np.float64)[m].sum() / m.size), N"),
    ("ratio deviation metric without the absolute value",
     "ratio_absdev_mean=float(np.abs(r - 1.0).sum() / N)", "ratio_absdev_mean=float((r - 1.0).sum() / N)"),
    ("TIS lower clamp dropped", "wt = np.minimum(np.maximum(rc, p.corr_lo), p.corr_hi)",
     "wt = np.minimum(rc, p.corr_hi)"),
    ("clip_hi tests eps_lo", "clip_hi = clipped & (r > 1.0 + p.eps_hi)",
     "clip_hi = clipped & (r > 1.0 + p.eps_lo)"),
    ("clip_lo tests eps_hi", "clip_lo = clipped & (r < 1.0 - p.eps_lo)",
     "clip_lo = clipped & (r < 1.0 - p.eps_hi)"),
    ("clip interval with the eps swapped", "np.clip(r, 1.0 - p.eps_lo, 1.0 + p.eps_hi)",
     "np.clip(r, 1.0 - p.eps_hi, 1.0 + p.eps_lo)"),
    ("KL gradient subtracted", "G = g_pg + p.kl_coef * g_kl", "G = g_pg - p.kl_coef * g_kl"),
    ("top-K log-probs miss the lse", "lps = s[rows, ids] - np.asarray(lse, np.float64)[:, None]",
     "lps = s[rows, ids]"),
    ("GSPO ratio over masked tokens too",
     "s_i = float(np.exp((logp[rows][mm] - base[rows][mm]).sum() / n_i[i]))",
     "s_i = float(np.exp((logp[rows] - base[rows]).sum() / n_i[i]))"),
    ("GSPO share without 1/n_i", "scale = N / (n_seq * n_i[i])", "scale = N / n_seq"),
    ("GSPO clip_hi tests eps_lo", "clip_hi[rows] = clipped and s_i > 1.0 + p.eps_hi",
     "clip_hi[rows] = clipped and s_i > 1.0 + p.eps_lo"),
    ("GSPO dual clip for A > 0",
     "        if p.dual_clip_c > 0.0 and A < 0.0:\n            d = -A * p.dual_clip_c\n            if d < pgi:",
     "        if p.dual_clip_c > 0.0 and A > 0.0:\n            d = -A * p.dual_clip_c\n            if d < pgi:"),
    ("dLogits entropy term subtracted", "+ entropy_coef * ent)", "- entropy_coef * ent)"),
    ("dual clip for A > 0", "dual = (A < 0.0) & (d < pg)", "dual = (A > 0.0) & (d < pg)"),
    ("REINFORCE++ std over all rows",
     "sigma = float(np.sqrt(((b_row[m] - mu) ** 2).sum() / (N - ddof))) if N > ddof else 0.0",
     "sigma = float(np.sqrt(((b_row - mu) ** 2).sum() / (N - ddof))) if N > ddof else 0.0"),
    ("clip-or-pop lower bound exclusive", "outside = (rc < p.corr_lo) | (rc > p.corr_hi)",
     "outside = (rc <= p.corr_lo) | (rc > p.corr_hi)"),
    ("entropy from unnormalised probabilities", "    p = np.exp(logp_all)\n", "    p = np.exp(s - m)\n"),
    ("ratio minimum over masked rows too", "ratio_min=float(r.min()),", "ratio_min=float(obj['r'].min()),"),
    ("divergence metric signed",
     "logprob_absdiff_mean=float(np.abs(np.asarray(logp, np.float64)[m]",
     "logprob_absdiff_mean=float((np.asarray(logp, np.float64)[m]"),
]


def _pins_pass(workdir, source):
    """Run the pins against a copy of the oracle whose main module is
    `source`; True if they pass."""
    shutil.copytree(os.path.join(ROOT, "oracle"), os.path.join(workdir, "oracle"),
                    ignore=shutil.ignore_patterns("__pycache__"))
    with open(os.path.join(workdir, "oracle", "rl_loss_ref.py"), "w") as f:
        f.write(source)
    tests = os.path.join(workdir, "tests")
    os.makedirs(tests)
    shutil.copy(os.path.join(ROOT, "tests", "conftest.py"), tests)
    shutil.copy(os.path.join(ROOT, "tests", "test_oracle_pins.py"), tests)
    shutil.copytree(os.path.join(ROOT, "tests", "golden"), os.path.join(tests, "golden"))
    # the copy's conftest puts the copy first on sys.path: its oracle is the
    # one imported
    env = dict(os.environ, PYTHONPATH=ROOT, PYTHONDONTWRITEBYTECODE="1")
    r = subprocess.run([sys.executable, "-m", "pytest", "-x", "-q", "-p", "no:cacheprovider",
                        os.path.join(tests, "test_oracle_pins.py")],
                       cwd=workdir, env=env, capture_output=True, text=True, timeout=600)
    return r.returncode == 0


def test_every_planted_mistake_fails_the_pins(tmp_path):
    with open(SRC) as f:
        orig = f.read()
    for name, a, _ in MUTANTS:  # (a site found more than once is mutated at its first)
        assert a in orig, f"mutation site not found: {name}"
    jobs = [("unmutated", orig)] + [(name, orig.replace(a, b, 1)) for name, a, b in MUTANTS]
    with ThreadPoolExecutor(max_workers=min(16, os.cpu_count() or 1)) as ex:
        passed = list(ex.map(lambda j: _pins_pass(str(tmp_path / f"m{j[0]}"), j[1]),
                             enumerate(s for _, s in jobs)))
    assert passed[0], "the unmutated copy must pass its pins"
    missed = [jobs[i][0] for i in range(1, len(jobs)) if passed[i]]
    assert not missed, f"mutants not caught by the pins: {missed}"
