"""Pins of the float64 oracle against facts that do not come from the oracle:
hand-derived closed forms, invariants, library routines that compute the same
quantity (torch.log_softmax, torch.nn.functional.cross_entropy, torch.std,
Categorical entropy), arbitrary-precision brute force (mpmath), and central
finite differences of the loss. CPU only.
"""

import json
import math
import os

import numpy as np
import pytest
import torch

import oracle
from oracle import LossParams

HERE = os.path.dirname(os.path.abspath(__file__))


def _ev(x):
    return float(eval(x, {"math": math})) if isinstance(x, str) else float(x)


def _golden():
    with open(os.path.join(HERE, "golden", "hand_cases.json")) as f:
        return {c["name"]: c for c in json.load(f)["cases"]}


# ---------------------------------------------------------------- log-softmax

@pytest.mark.parametrize("name", ["two_point_row", "tempered_row"])
def test_row_golden(name):
    c = _golden()[name]
    z = np.array([[_ev(v) for v in row] for row in c["z"]])
    logp, H, lse = oracle.row_log_softmax(z, np.array(c["y"]), _ev(c["T"]))
    for key, got in (("logp", logp), ("lse", lse), ("H", H)):
        want = np.array([_ev(v) for v in c["expect"][key]])
        np.testing.assert_allclose(got, want, rtol=0, atol=1e-14)


def test_log_softmax_matches_torch_library():
    rng = np.random.default_rng(1)
    z = rng.normal(0, 3, size=(17, 301))
    y = rng.integers(0, 301, size=17)
    for T in (1.0, 0.7, 1.9):
        logp, H, lse = oracle.row_log_softmax(z, y, T)
        zt = torch.from_numpy(z) / T
        ref = torch.log_softmax(zt, dim=1)
        np.testing.assert_allclose(logp, ref[torch.arange(17), torch.from_numpy(y)].numpy(),
                                   atol=1e-12, rtol=0)
        np.testing.assert_allclose(lse, torch.logsumexp(zt, dim=1).numpy(), atol=1e-12, rtol=0)
        ent = torch.distributions.Categorical(logits=zt).entropy().numpy()
        np.testing.assert_allclose(H, ent, atol=1e-12, rtol=0)


def test_probabilities_sum_to_one_and_shift_invariance():
    rng = np.random.default_rng(2)
    z = rng.normal(0, 5, size=(9, 1000))
    y = rng.integers(0, 1000, size=9)
    logp, H, lse = oracle.row_log_softmax(z, y, 1.0)
    assert np.all(np.abs(np.exp(z - lse[:, None]).sum(1) - 1.0) < 1e-12)
    # adding a constant to a row changes nothing but lse
    logp2, H2, lse2 = oracle.row_log_softmax(z + 1000.0, y, 1.0)
    np.testing.assert_allclose(logp2, logp, atol=1e-9)
    np.testing.assert_allclose(H2, H, atol=1e-9)
    np.testing.assert_allclose(lse2 - lse, 1000.0, atol=1e-9)


def test_entropy_extremes():
    for V in (1, 2, 7, 4096):
        z = np.zeros((1, V))
        logp, H, _ = oracle.row_log_softmax(z, np.array([0]), 1.0)
        assert abs(H[0] - math.log(V)) < 1e-12
        assert abs(logp[0] + math.log(V)) < 1e-12
    z = np.zeros((1, 50))
    z[0, 3] = 200.0
    logp, H, _ = oracle.row_log_softmax(z, np.array([3]), 1.0)
    assert H[0] < 1e-80 and abs(logp[0]) < 1e-80


def test_minus_inf_logits_are_absent_categories():
    """A logit of -inf is a category of probability zero: the log-prob,
    entropy and lse equal those of the row with that category removed, its
    own dLogit is 0 (the limit 0 log 0 = 0), and the other dLogits equal the
    reduced row's. A row with one live category has H = 0 and log p = 0."""
    rng = np.random.default_rng(11)
    V = 37
    z = rng.normal(0.0, 2.0, size=(3, V))
    dead = np.zeros((3, V), dtype=bool)
    dead[0, [1, 5, 30]] = True
    dead[1, 10:36] = True
    dead[2, 0] = True
    y = np.array([0, 3, 7])
    zi = np.where(dead, -np.inf, z)
    G = rng.normal(size=3)
    mask = np.ones(3, dtype=np.uint8)
    for T, gamma in ((1.0, 0.0), (0.7, 0.05)):
        lp, H, lse = oracle.row_log_softmax(zi, y, T)
        d = oracle.dlogits_rows(zi, y, T, lse, H, G, mask, 3, 1.0, gamma)
        assert np.all(np.isfinite(d)) and np.all(d[dead] == 0.0)
        for r in range(3):
            keep = ~dead[r]
            yr = np.array([int(keep[:y[r]].sum())])
            lp_r, H_r, lse_r = oracle.row_log_softmax(z[r:r + 1, keep], yr, T)
            assert abs(lp[r] - lp_r[0]) < 1e-13 and abs(H[r] - H_r[0]) < 1e-13
            assert abs(lse[r] - lse_r[0]) < 1e-13
            d_r = oracle.dlogits_rows(z[r:r + 1, keep], yr, T, lse_r, H_r, G[r:r + 1],
                                      mask[r:r + 1], 3, 1.0, gamma)
            assert np.allclose(d[r, keep], d_r[0], rtol=1e-13, atol=1e-16)
    one = np.full((1, 9), -np.inf)
    one[0, 4] = 1.5
    lp, H, _ = oracle.row_log_softmax(one, np.array([4]), 1.0)
    assert lp[0] == 0.0 and H[0] == 0.0


def test_log_softmax_mpmath_brute_force():
    mpmath = pytest.importorskip("mpmath")
    mpmath.mp.dps = 50
    rng = np.random.default_rng(3)
    for V in (2, 3, 5, 8):
        z = rng.normal(0, 4, size=(4, V))
        y = rng.integers(0, V, size=4)
        T = 0.8
        logp, H, lse = oracle.row_log_softmax(z, y, T)
        for i in range(4):
            s = [mpmath.mpf(float(v)) / mpmath.mpf(T) for v in z[i]]
            L = mpmath.log(mpmath.fsum(mpmath.exp(v) for v in s))
            ps = [mpmath.exp(v - L) for v in s]
            Hm = -mpmath.fsum(p * mpmath.log(p) for p in ps)
            assert abs(float(L) - lse[i]) < 1e-13
            assert abs(float(s[y[i]] - L) - logp[i]) < 1e-13
            assert abs(float(Hm) - H[i]) < 1e-13


def test_widen_bf16_exact():
    x = torch.tensor([1.0, -2.5, 3.140625, 1e-30, 65504.0, -0.0], dtype=torch.bfloat16)
    bits = x.view(torch.int16).numpy().view(np.uint16)
    np.testing.assert_array_equal(oracle.widen_bf16(bits), x.double().numpy())


# ---------------------------------------------------------------- advantages

@pytest.mark.parametrize("name", ["grpo_two_members", "grpo_three_members"])
def test_group_advantages_golden(name):
    c = _golden()[name]
    w = np.array([_ev(v) for v in c["w"]])
    gid = np.array(c["gid"])
    A, n = oracle.group_advantages(w, gid, c["n_groups"], LossParams())
    np.testing.assert_allclose(A, [_ev(v) for v in c["expect_unbiased"]], atol=1e-15, rtol=0)
    A, _ = oracle.group_advantages(w, gid, c["n_groups"], LossParams(unbiased_std=False))
    np.testing.assert_allclose(A, [_ev(v) for v in c["expect_population"]], atol=1e-15, rtol=0)
    assert n.tolist() == [len(w)]


def test_group_advantages_match_torch_std_and_sum_to_zero():
    rng = np.random.default_rng(4)
    n_groups, gsz = 11, 7
    w = rng.random(n_groups * gsz)
    gid = rng.permutation(np.repeat(np.arange(n_groups), gsz))  # scattered members
    A, n = oracle.group_advantages(w, gid, n_groups, LossParams())
    assert n.tolist() == [gsz] * n_groups
    for g in range(n_groups):
        idx = gid == g
        wt = torch.from_numpy(w[idx])
        ref = ((wt - wt.mean()) / wt.std()).numpy()  # torch.std is the n-1 std
        np.testing.assert_allclose(A[idx], ref, atol=1e-13, rtol=0)
        assert abs(A[idx].sum()) < 1e-12 * gsz
    A0, _ = oracle.group_advantages(w, gid, n_groups, LossParams(normalize_std=False))
    for g in range(n_groups):
        idx = gid == g
        np.testing.assert_allclose(A0[idx], w[idx] - w[idx].mean(), atol=1e-15)


def test_group_advantages_equal_rewards_floor_and_empty_groups():
    p = LossParams(std_floor=1e-6)
    w = np.array([0.5, 0.5, 0.5, 0.0, 1e-9, 3.0])
    gid = np.array([0, 0, 0, 1, 1, 3])  # group 2 empty, group 3 single member
    A, n = oracle.group_advantages(w, gid, 4, p)
    assert A[0] == 0.0 and A[1] == 0.0 and A[2] == 0.0  # equal rewards: exactly 0
    assert A[5] == 0.0
    assert n.tolist() == [3, 2, 0, 1]
    # sigma = 1e-9/sqrt(2) < floor -> divide by the floor
    np.testing.assert_allclose(A[3:5], [-0.5e-9 / 1e-6, 0.5e-9 / 1e-6], rtol=1e-12)


def test_row_advantages_and_opd_shaping():
    A = np.array([1.0, -2.0, 3.0])
    cu = np.array([0, 2, 2, 5])
    np.testing.assert_array_equal(oracle.row_advantages(A, cu, 5), [1, 1, 3, 3, 3])
    s = oracle.shape_advantages_opd(np.array([1.0, 1.0]), np.array([-1.0, -3.0]),
                                    np.array([-2.0, -1.0]), 0.5)
    # student favoured token 0 more than the teacher (+1) -> penalised;
    # teacher favoured token 1 more (-2) -> encouraged
    np.testing.assert_allclose(s, [0.5, 2.0], atol=1e-15)


# ---------------------------------------------------------------- objective

@pytest.mark.parametrize("name", ["ppo_tokens", "ppo_tokens_asymmetric_lo", "ppo_tokens_asymmetric_hi"])
def test_ppo_tokens_golden(name):
    """Hand-derived PPO tokens: symmetric clip with dual clip, and both
    asymmetric intervals (each bound and each flag tied to its own eps)."""
    c = _golden()[name]
    A = np.array([_ev(v) for v in c["A"]])
    logp = np.array([_ev(v) for v in c["log_r"]])
    o = oracle.token_objective(logp, np.zeros_like(logp), None, A, np.zeros_like(A),
                               LossParams(**c["params"]))
    np.testing.assert_allclose(o["pg"], [_ev(v) for v in c["expect"]["pg"]], atol=1e-14)
    np.testing.assert_allclose(o["G"], [_ev(v) for v in c["expect"]["G"]], atol=1e-14)
    for k in ("clip_hi", "clip_lo", "dual"):
        assert o[k].astype(int).tolist() == c["expect"][k]


def test_k3_golden():
    c = _golden()["k3_token"]
    logp = np.array([_ev(v) for v in c["logp"]])
    q = np.array([_ev(v) for v in c["q"]])
    o = oracle.token_objective(logp, logp, q, np.array([0.0]), np.zeros(1),
                               LossParams(kl_coef=c["kl_coef"]))
    for k in ("k3", "ell", "G"):
        np.testing.assert_allclose(o[k], [_ev(v) for v in c["expect"][k]], atol=1e-15)
    # q == logp: k3 and its gradient vanish
    o = oracle.token_objective(logp, logp, logp, np.array([0.0]), np.zeros(1),
                               LossParams(kl_coef=1.0))
    assert o["k3"][0] == 0.0 and o["G"][0] == 0.0


def _threshold_probe(approx):
    """A float64 d, the ratio t = exp(d) it gives (the threshold), and the
    neighbouring doubles d_up / d_dn whose exp lies strictly above / below t."""
    d = math.log(approx)
    t = math.exp(d)
    up = np.nextafter(d, math.inf)
    while math.exp(up) <= t:
        up = np.nextafter(up, math.inf)
    dn = np.nextafter(d, -math.inf)
    while math.exp(dn) >= t:
        dn = np.nextafter(dn, -math.inf)
    return d, t, up, dn


def test_clip_engages_exactly_past_the_threshold():
    d_hi, t_hi, up_hi, _ = _threshold_probe(1.25)
    d_lo, t_lo, _, dn_lo = _threshold_probe(0.75)
    d_c, t_c, up_c, _ = _threshold_probe(3.0)
    # eps chosen so that 1 + eps_hi == t_hi and 1 - eps_lo == t_lo exactly
    # (Sterbenz: t - 1 and 1 - t are exact for t in [0.5, 2])
    p = LossParams(eps_lo=1.0 - t_lo, eps_hi=t_hi - 1.0, dual_clip_c=t_c)
    assert 1.0 + p.eps_hi == t_hi and 1.0 - p.eps_lo == t_lo
    logp = np.array([d_hi, up_hi, d_lo, dn_lo, d_c, up_c])
    A = np.array([1.0, 1.0, -1.0, -1.0, -1.0, -1.0])
    o = oracle.token_objective(logp, np.zeros(6), None, A, np.zeros(6), p)
    assert o["r"][0] == t_hi and o["r"][2] == t_lo and o["r"][4] == t_c
    assert o["clip_hi"].tolist() == [False, True, False, False, False, False]
    assert o["clip_lo"].tolist() == [False, False, False, True, False, False]
    assert o["dual"].tolist() == [False, False, False, False, False, True]
    # at the threshold the gradient flows through the unclipped branch
    assert o["G"][0] == -t_hi and o["G"][2] == t_lo and o["G"][4] == t_c
    assert o["G"][1] == 0.0 and o["G"][3] == 0.0 and o["G"][5] == 0.0


def test_ratio_one_gives_minus_mean_advantage():
    rng = np.random.default_rng(5)
    R = 64
    logp = -rng.random(R) * 5
    A = rng.normal(size=R)
    m = rng.random(R) < 0.6
    o = oracle.token_objective(logp, logp.copy(), None, A, np.zeros(R),
                               LossParams(dual_clip_c=3.0))
    assert np.all(o["r"] == 1.0)
    L, N = oracle.masked_token_mean(o["ell"], m)
    assert N == int(m.sum())
    assert abs(L - (-(A[m]).sum() / N)) < 1e-14
    assert not o["clip_hi"].any() and not o["clip_lo"].any() and not o["dual"].any()


def test_corrections_tis_and_clip_or_pop():
    rho = np.zeros(5)
    old = np.log(np.array([3.0, 0.5, 2.0, 1.0, 2.5]))
    logp = old.copy()                 # PPO ratio against old is exactly 1
    A = np.ones(5)
    base = oracle.token_objective(logp, rho, None, A, np.zeros(5), LossParams(), old=old)
    tis = oracle.token_objective(logp, rho, None, A, np.zeros(5),
                                 LossParams(correction="tis", corr_lo=0.0, corr_hi=2.0), old=old)
    pop = oracle.token_objective(logp, rho, None, A, np.zeros(5),
                                 LossParams(correction="clip_or_pop", corr_lo=0.0, corr_hi=2.0),
                                 old=old)
    rc = np.exp(old - rho)
    np.testing.assert_allclose(tis["wt"], [2.0, 0.5, rc[2], 1.0, 2.0], rtol=1e-15)
    np.testing.assert_allclose(pop["wt"], [0.0, 0.5, rc[2], 1.0, 0.0], rtol=1e-15)
    assert tis["corr_clip"].tolist() == [True, False, False, False, True]
    assert pop["corr_clip"].tolist() == [True, False, False, False, True]
    np.testing.assert_allclose(tis["pg"], tis["wt"] * base["pg"], rtol=1e-15)
    np.testing.assert_allclose(pop["G"], pop["wt"] * base["G"], rtol=1e-15)


@pytest.mark.parametrize("correction", ["tis", "clip_or_pop"])
def test_correction_without_old_logprobs_golden(correction):
    """Without old log-probs the correction ratio is the trainer's own
    log-prob of this pass against the rollout's (a constant weight), and the
    PPO ratio is taken against the rollout log-prob (hand-derived)."""
    c = _golden()["tis_own_ratio"]
    logp = np.array([_ev(v) for v in c["log_r"]])
    A = np.array([float(v) for v in c["A"]])
    o = oracle.token_objective(logp, np.zeros(4), None, A, np.zeros(4),
                               LossParams(correction=correction, **c["params"]))
    e = c["expect"][correction]
    for k in ("wt", "pg", "G"):
        np.testing.assert_allclose(o[k], [_ev(v) for v in e[k]], atol=1e-14, err_msg=k)
    assert o["corr_clip"].astype(int).tolist() == e["corr_clip"]
    assert o["clip_hi"].astype(int).tolist() == e["clip_hi"]
    np.testing.assert_allclose(o["rc"], o["r"], rtol=0, atol=0)


def test_tis_lower_clamp_golden():
    c = _golden()["tis_lower_clamp"]
    old = np.array([math.log(_ev(c["rc"]))])
    o = oracle.token_objective(old.copy(), np.zeros(1), None, np.ones(1), np.zeros(1),
                               LossParams(**c["params"]), old=old)
    for k in ("wt", "pg", "G"):
        assert abs(o[k][0] - _ev(c["expect"][k])) < 1e-15, k
    assert int(o["corr_clip"][0]) == c["expect"]["corr_clip"]


def test_clip_or_pop_bounds_are_inclusive():
    """A correction ratio exactly at either bound keeps its weight; the next
    double outside pops the token (weight 0)."""
    for lo, hi in ((0.5, 2.0), (0.8, 1.25)):
        for bound in (lo, hi):
            d, t, up, dn = _threshold_probe(bound)
            assert float(np.exp(np.float64(d))) == t  # the double the oracle forms from d
            outer = dn if bound == lo else up
            p = LossParams(correction="clip_or_pop", corr_lo=t if bound == lo else lo,
                           corr_hi=t if bound == hi else hi)
            old = np.array([d, outer])
            o = oracle.token_objective(old.copy(), np.zeros(2), None, np.ones(2), np.zeros(2), p,
                                       old=old)
            assert o["wt"][0] == t and o["corr_clip"][0] == 0
            assert o["wt"][1] == 0.0 and o["corr_clip"][1] == 1


def test_metrics_golden():
    """The reported metrics are means, minima and maxima over the tokens that
    train, of absolute deviations where the definition says so."""
    c = _golden()["metrics_over_training_tokens"]
    lr = np.array([_ev(v) for v in c["log_r"]])
    logp = np.array([-0.5, -1.0, -2.0])
    rho = logp - lr
    H = np.array([_ev(v) for v in c["H"]])
    mask = np.array(c["mask"])
    p = LossParams(entropy_coef=c["entropy_coef"])
    obj = oracle.token_objective(logp, rho, None, np.zeros(3), H, p)
    st = oracle.loss_stats(obj, logp, rho, H, mask)
    for k, v in c["expect"].items():
        assert abs(st[k] - _ev(v)) < 1e-14, (k, st[k])


def test_metrics_with_correction_kl_clip_golden():
    """Counts and means over the training tokens, with a masked row that would
    be clipped, corrected and carry KL."""
    c = _golden()["metrics_with_correction_kl_clip"]
    logp = np.full(3, -1.0)
    old = logp - np.array([_ev(v) for v in c["log_r"]])
    rho = old - np.array([_ev(v) for v in c["log_rc"]])
    q = logp + np.array([_ev(v) for v in c["delta"]])
    A = np.array([_ev(v) for v in c["A"]])
    mask = np.array(c["mask"])
    H = np.zeros(3)
    obj = oracle.token_objective(logp, rho, q, A, H, LossParams(**c["params"]), old=old)
    st = oracle.loss_stats(obj, logp, rho, H, mask)
    for k, v in c["expect"].items():
        assert abs(st[k] - _ev(v)) < 1e-14, (k, st[k])


def test_masked_mean_edge_cases():
    assert oracle.masked_token_mean(np.array([1.0, 2.0]), np.array([0, 0])) == (0.0, 0)
    L, N = oracle.masked_token_mean(np.array([1.0, 2.0, 4.0]), np.array([1, 0, 1]))
    assert N == 2 and L == 2.5


# ---------------------------------------------------------------- gradient

@pytest.mark.parametrize("name", ["full_two_tokens"])
def test_full_pipeline_golden(name):
    c = _golden()[name]
    z = np.array([[_ev(v) for v in row] for row in c["z"]])
    out = oracle.rl_loss(z, np.array(c["y"]), np.array([_ev(v) for v in c["rho"]]), None,
                         np.array([_ev(v) for v in c["w"]]), np.array(c["gid"]),
                         np.array(c["cu"]), c["n_groups"], np.array(c["mask"]), LossParams())
    assert abs(out["loss"] - _ev(c["expect"]["loss"])) < 1e-14
    want = np.array([[_ev(v) for v in row] for row in c["expect"]["dlogits"]])
    np.testing.assert_allclose(out["dlogits"], want, atol=1e-14, rtol=0)


def _call_inputs(c):
    z = np.array([[_ev(v) for v in row] for row in c["z"]])
    return (z, np.array(c["y"]), np.array([_ev(v) for v in c["rho"]]),
            np.array([_ev(v) for v in c["w"]]), np.array(c["gid"]), np.array(c["cu"]),
            c["n_groups"], np.array(c["mask"]))


def test_full_call_kl_opd_golden():
    """The whole call wires the KL reference and the one-sample OPD teacher
    into the advantages, the objective and dLogits."""
    c = _golden()["full_call_kl_opd"]
    z, y, rho, w, gid, cu, n_groups, mask = _call_inputs(c)
    q = rho + np.array([_ev(v) for v in c["delta"]])  # rho = logp here
    out = oracle.rl_loss(z, y, rho, q, w, gid, cu, n_groups, mask, LossParams(**c["params"]),
                         teacher=np.array([_ev(v) for v in c["teacher"]]))
    e = c["expect"]
    np.testing.assert_allclose(out["A_row"], [_ev(v) for v in e["A_row"]], atol=1e-14, rtol=0)
    np.testing.assert_allclose(out["G"], [_ev(v) for v in e["G"]], atol=1e-14, rtol=0)
    assert abs(out["loss"] - _ev(e["loss"])) < 1e-14
    want = np.array([[_ev(v) for v in row] for row in e["dlogits"]])
    np.testing.assert_allclose(out["dlogits"], want, atol=1e-14, rtol=0)


def test_full_call_topk_opd_golden():
    """The whole call shapes the advantages with the top-K signal of each
    row's own statistics (one row per chunk)."""
    c = _golden()["full_call_topk_opd"]
    z, y, rho, w, gid, cu, n_groups, mask = _call_inputs(c)
    ids = np.array(c["topk_ids"])
    tt = np.array([[_ev(v) for v in row] for row in c["topk_teacher"]])
    out = oracle.rl_loss(z, y, rho, None, w, gid, cu, n_groups, mask, LossParams(**c["params"]),
                         chunk=1, topk_ids=ids, topk_teacher=tt)
    np.testing.assert_allclose(out["A_row"], [_ev(v) for v in c["expect"]["A_row"]], atol=1e-14,
                               rtol=0)
    assert abs(out["loss"] - _ev(c["expect"]["loss"])) < 1e-14


def test_full_call_gspo_golden():
    """The whole call gives GSPO each trajectory's advantage."""
    c = _golden()["full_call_gspo_two_row_trajectories"]
    z, y, rho, w, gid, cu, n_groups, mask = _call_inputs(c)
    out = oracle.rl_loss(z, y, rho, None, w, gid, cu, n_groups, mask, LossParams(**c["params"]))
    np.testing.assert_allclose(out["G"], [_ev(v) for v in c["expect"]["G"]], atol=1e-14, rtol=0)
    assert abs(out["loss"] - _ev(c["expect"]["loss"])) < 1e-14


def test_cross_entropy_special_case():
    """A = 1, rho = logp, beta = gamma = 0, T = 1, all tokens train: r = 1,
    L = -1 and dZ = (p - onehot)/N, the gradient of the mean cross-entropy."""
    rng = np.random.default_rng(6)
    R, V = 12, 37
    z = rng.normal(0, 2, size=(R, V))
    y = rng.integers(0, V, size=R)
    logp, H, lse = oracle.row_log_softmax(z, y, 1.0)
    o = oracle.rl_loss_rows(z, y, logp, None, np.ones(R), np.ones(R, bool), R, LossParams())
    assert np.all(o["r"] == 1.0) and abs(o["ell"].mean() + 1.0) < 1e-15
    zt = torch.from_numpy(z).requires_grad_(True)
    torch.nn.functional.cross_entropy(zt, torch.from_numpy(y), reduction="mean").backward()
    np.testing.assert_allclose(o["dlogits"], zt.grad.numpy(), atol=1e-15, rtol=0)


def _near_kink(out, p, guard=1e-4):
    r = out["r"]
    th = [1 - p.eps_lo, 1 + p.eps_hi] + ([p.dual_clip_c] if p.dual_clip_c else [])
    if p.correction != "none":
        th += [p.corr_lo, p.corr_hi]
        r = np.concatenate([r, out["rc"]])
    return any(np.any(np.abs(r - t) < guard * max(1.0, t)) for t in th)


@pytest.mark.parametrize("V", [2, 3, 5, 8])
@pytest.mark.parametrize("variant", ["ppo_dual_kl_ent_T", "tis", "clip_or_pop", "opd",
                                     "tis_own", "clip_or_pop_own"])
def test_dlogits_central_finite_differences(V, variant, monkeypatch):
    rng = np.random.default_rng(100 + V)
    n_traj, L_ = 4, 2
    R = n_traj * L_
    p = LossParams(temperature=0.8, eps_lo=0.15, eps_hi=0.25, dual_clip_c=2.5,
                   kl_coef=0.3, entropy_coef=0.07)
    own = variant.endswith("_own")  # the correction ratio from this pass's own log-prob
    if variant in ("tis", "clip_or_pop", "tis_own", "clip_or_pop_own"):
        p = LossParams(temperature=1.3, eps_lo=0.2, eps_hi=0.2, kl_coef=0.1,
                       entropy_coef=0.02, correction=variant.replace("_own", ""), corr_lo=0.5,
                       corr_hi=1.5)
    if variant == "opd":
        p = LossParams(temperature=1.0, eps_lo=0.2, eps_hi=0.2, opd_coef=0.7)
    for attempt in range(50):
        z = rng.normal(0, 1.5, size=(R, V))
        y = rng.integers(0, V, size=R)
        logp, _, _ = oracle.row_log_softmax(z, y, p.temperature)
        rho = logp + rng.normal(0, 0.6, size=R)
        q = logp + rng.normal(0, 0.5, size=R)
        old = logp + rng.normal(0, 0.3, size=R) if (p.correction != "none" and not own) else None
        if own:
            rho = logp + rng.normal(0, 0.25, size=R)
        teacher = logp + rng.normal(0, 0.5, size=R)
        w = rng.random(n_traj)
        gid = np.array([0, 0, 1, 1])
        cu = np.arange(n_traj + 1) * L_
        m = np.array([1, 1, 0, 1, 1, 1, 1, 0], dtype=bool)
        args = (y, rho, q, w, gid, cu, 2, m, p)
        out = oracle.rl_loss(z, *args, grad_loss=1.7, old=old, teacher=teacher)
        if not _near_kink(out, p):
            break
    else:
        pytest.fail("no draw away from the kinks")
    if variant == "ppo_dual_kl_ent_T":
        assert out["clip_hi"].any() or out["clip_lo"].any() or out["dual"].any()
    if own:
        # the weight is a constant: hold the correction ratio at its value
        frozen = out["rc"].copy()
        monkeypatch.setattr(oracle.rl_loss_ref, "correction_ratio", lambda *a, **k: frozen)
    h = 1e-6
    num = np.zeros_like(z)
    for i in range(R):
        for j in range(V):
            zp = z.copy(); zp[i, j] += h
            zm = z.copy(); zm[i, j] -= h
            lp = oracle.rl_loss(zp, *args, old=old, teacher=teacher, want_dlogits=False)["loss"]
            lm = oracle.rl_loss(zm, *args, old=old, teacher=teacher, want_dlogits=False)["loss"]
            num[i, j] = 1.7 * (lp - lm) / (2 * h)
    scale = np.abs(out["dlogits"]).max()
    np.testing.assert_allclose(out["dlogits"], num, atol=1e-6 * max(scale, 1e-3), rtol=1e-6)
    assert np.all(out["dlogits"][~m] == 0.0)


def test_chunking_changes_nothing():
    rng = np.random.default_rng(7)
    R, V = 40, 33
    z = rng.normal(0, 2, size=(R, V))
    y = rng.integers(0, V, size=R)
    rho = rng.normal(-3, 0.1, size=R)
    w = rng.random(8)
    gid = np.repeat(np.arange(2), 4)
    cu = np.arange(9) * 5
    m = rng.random(R) < 0.7
    p = LossParams(dual_clip_c=3.0)
    a = oracle.rl_loss(z, y, rho, None, w, gid, cu, 2, m, p, chunk=1)
    b = oracle.rl_loss(z, y, rho, None, w, gid, cu, 2, m, p, chunk=256)
    assert a["loss"] == b["loss"]
    np.testing.assert_array_equal(a["dlogits"], b["dlogits"])


def test_no_training_tokens():
    z = np.zeros((3, 4))
    out = oracle.rl_loss(z, np.array([0, 1, 2]), np.zeros(3), None, np.array([0.0, 1.0]),
                         np.array([0, 0]), np.array([0, 2, 3]), 1, np.zeros(3), LossParams())
    assert out["loss"] == 0.0 and out["N"] == 0
    assert np.all(out["dlogits"] == 0.0)
    # every metric of an empty call is 0 (none is a mean, extreme or count
    # over rows that do not train)
    for k, v in out["stats"].items():
        assert v == 0, (k, v)


# ---------------------------------------------------------------- estimators

def test_reinforcepp_golden():
    c = _golden()["reinforcepp_two_trajectories"]
    w = np.array([_ev(v) for v in c["w"]])
    for est in ("reinforcepp", "reinforcepp_baseline"):
        A, A_row, _ = oracle.estimator_advantages(w, np.array(c["gid"]), c["n_groups"],
                                                  np.array(c["cu"]), np.array(c["mask"]),
                                                  LossParams(estimator=est))
        np.testing.assert_allclose(A, [_ev(v) for v in c["expect"]], atol=1e-15)


def test_reinforcepp_global_normalisation_invariants():
    rng = np.random.default_rng(11)
    n_traj, n_groups = 12, 3
    w = rng.normal(size=n_traj)
    gid = rng.permutation(np.repeat(np.arange(n_groups), 4))
    lens = rng.integers(1, 9, size=n_traj)
    cu = np.concatenate([[0], np.cumsum(lens)])
    mask = rng.random(cu[-1]) < 0.7
    for est in ("reinforcepp", "reinforcepp_baseline"):
        p = LossParams(estimator=est)
        A, A_row, _ = oracle.estimator_advantages(w, gid, n_groups, cu, mask, p)
        Am = A_row[mask]
        assert abs(Am.sum()) < 1e-12
        assert abs((Am ** 2).sum() - (mask.sum() - 1)) < 1e-9
        # the token-level z-score of the returns, by the library's std
        b = w.copy()
        if est == "reinforcepp_baseline":
            for g in range(n_groups):
                b[gid == g] -= w[gid == g].mean()
        bt = torch.from_numpy(oracle.row_advantages(b, cu, cu[-1])[mask])
        np.testing.assert_allclose(Am, ((bt - bt.mean()) / bt.std()).numpy(), atol=1e-12)
    # baseline-relative returns ignore a constant added to a group's rewards
    p = LossParams(estimator="reinforcepp_baseline")
    w2 = w.copy()
    w2[gid == 1] += 5.0
    a1 = oracle.estimator_advantages(w, gid, n_groups, cu, mask, p)[0]
    a2 = oracle.estimator_advantages(w2, gid, n_groups, cu, mask, p)[0]
    np.testing.assert_allclose(a1, a2, atol=1e-12)
    # plain returns: a positive affine map of the rewards changes nothing
    p = LossParams(estimator="reinforcepp")
    a3 = oracle.estimator_advantages(3.0 * w - 7.0, gid, n_groups, cu, mask, p)[0]
    np.testing.assert_allclose(oracle.estimator_advantages(w, gid, n_groups, cu, mask, p)[0],
                               a3, atol=1e-12)
    # equal returns: exactly zero
    z = oracle.estimator_advantages(np.full(n_traj, 0.25), gid, n_groups, cu, mask, p)[0]
    assert np.all(z == 0.0)


def test_opd_topk_estimate_pins():
    rng = np.random.default_rng(12)
    R, V = 5, 9
    z = rng.normal(0, 2, size=(R, V))
    T = 0.9
    _, _, lse = oracle.row_log_softmax(z, np.zeros(R, np.int64), T)
    t_logits = rng.normal(0, 2, size=(R, V))
    log_t = torch.log_softmax(torch.from_numpy(t_logits), dim=1).numpy()
    # the full vocabulary as the candidate set: the reverse KL(student || teacher)
    ids = np.tile(np.arange(V), (R, 1))
    est = oracle.opd_topk_estimate(z, T, lse, ids, log_t)
    log_s = torch.log_softmax(torch.from_numpy(z) / T, dim=1)
    kl = torch.nn.functional.kl_div(torch.from_numpy(log_t), log_s, log_target=True,
                                    reduction="none").sum(1).numpy()
    np.testing.assert_allclose(est, kl, atol=1e-12)
    # one candidate: the one-sample difference at that token
    c = rng.integers(0, V, size=(R, 1))
    est1 = oracle.opd_topk_estimate(z, T, lse, c, log_t[np.arange(R)[:, None], c])
    np.testing.assert_allclose(est1, (log_s.numpy() - log_t)[np.arange(R), c[:, 0]], atol=1e-12)
    # a candidate outside [0, V) is rejected, not wrapped to another column
    for bad in (-1, V):
        ids_bad = ids.copy()
        ids_bad[2, 4] = bad
        with pytest.raises(ValueError):
            oracle.opd_topk_estimate(z, T, lse, ids_bad, log_t)


def test_gspo_golden():
    c = _golden()["gspo_one_trajectory"]
    lr = np.array([_ev(v) for v in c["log_ratio"]])
    logp = np.array([-1.0, -2.0])
    rho = logp - lr
    o = oracle.sequence_objective(logp, rho, None, np.array([_ev(c["A"])]), np.zeros(2),
                                  np.array([0, 2]), np.array([1, 1]),
                                  LossParams(estimator="gspo"))
    L, _ = oracle.masked_token_mean(o["ell"], np.array([1, 1]))
    assert abs(L - _ev(c["expect"]["loss"])) < 1e-14
    np.testing.assert_allclose(o["G"], [_ev(v) for v in c["expect"]["G"]], atol=1e-14)
    np.testing.assert_allclose(o["r"], _ev(c["expect"]["r"]), atol=1e-15)


@pytest.mark.parametrize("name", ["gspo_asymmetric_clip", "gspo_asymmetric_clip_lo"])
def test_gspo_asymmetric_clip_golden(name):
    c = _golden()[name]
    lr = np.array([_ev(v) for v in c["log_ratio"]])
    logp = np.array([-1.0, -2.0])
    rho = logp - lr
    o = oracle.sequence_objective(logp, rho, None, np.array([_ev(c["A"])]), np.zeros(2),
                                  np.array([0, 2]), np.array([1, 1]), LossParams(**c["params"]))
    L, _ = oracle.masked_token_mean(o["ell"], np.array([1, 1]))
    assert abs(L - _ev(c["expect"]["loss"])) < 1e-14
    np.testing.assert_allclose(o["G"], [_ev(v) for v in c["expect"]["G"]], atol=1e-14)
    np.testing.assert_allclose(o["r"], _ev(c["expect"]["r"]), atol=1e-14)
    for k in ("clip_hi", "clip_lo"):
        assert o[k].astype(int).tolist() == c["expect"][k]


def test_gspo_with_an_untrained_trajectory_golden():
    c = _golden()["gspo_with_an_untrained_trajectory"]
    lr = np.array([_ev(v) for v in c["log_ratio"]])
    logp = np.array([-1.0, -2.0, -0.5])
    rho = logp - lr
    mask = np.array(c["mask"])
    o = oracle.sequence_objective(logp, rho, None, np.array([_ev(v) for v in c["A"]]), np.zeros(3),
                                  np.array(c["cu"]), mask, LossParams(estimator="gspo"))
    L, _ = oracle.masked_token_mean(o["ell"], mask)
    assert abs(L - _ev(c["expect"]["loss"])) < 1e-14
    np.testing.assert_allclose(o["G"], [_ev(v) for v in c["expect"]["G"]], atol=1e-14)
    np.testing.assert_allclose(o["r"], [_ev(v) for v in c["expect"]["r"]], atol=1e-14)


def test_gspo_on_one_token_trajectories_is_token_ppo():
    rng = np.random.default_rng(13)
    R = 16
    logp = -rng.random(R) * 3
    rho = logp + rng.normal(0, 0.3, size=R)
    q = logp + rng.normal(0, 0.2, size=R)
    A = rng.normal(size=R)
    H = rng.random(R)
    cu = np.arange(R + 1)
    m = np.ones(R, bool)
    p = LossParams(estimator="gspo", dual_clip_c=2.0, kl_coef=0.1, entropy_coef=0.05)
    seq = oracle.sequence_objective(logp, rho, q, A, H, cu, m, p)
    tok = oracle.token_objective(logp, rho, q, A, H, p)
    for k in ("r", "pg", "ell", "G", "clip_hi", "clip_lo", "dual"):
        np.testing.assert_allclose(seq[k], tok[k], atol=1e-13)


@pytest.mark.parametrize("variant", ["gspo", "gspo_tis", "topk", "reinforcepp_baseline",
                                     "gspo_tis_own"])
def test_dlogits_fd_estimators(variant, monkeypatch):
    rng = np.random.default_rng(200 + len(variant))
    V, n_traj, L_ = 6, 4, 3
    R = n_traj * L_
    base = dict(temperature=0.9, eps_lo=0.2, eps_hi=0.25, kl_coef=0.2, entropy_coef=0.03)
    extra = dict(gspo=dict(estimator="gspo", dual_clip_c=2.0),
                 gspo_tis=dict(estimator="gspo", correction="tis", corr_lo=0.5, corr_hi=1.5),
                 topk=dict(opd_coef=0.6, opd_topk=3),
                 reinforcepp_baseline=dict(estimator="reinforcepp_baseline"),
                 gspo_tis_own=dict(estimator="gspo", correction="tis", corr_lo=0.5,
                                   corr_hi=1.1))[variant]
    p = LossParams(**base, **extra)
    gid = np.array([0, 0, 1, 1])
    cu = np.arange(n_traj + 1) * L_
    m = np.array([1, 1, 0, 1, 1, 1, 0, 1, 1, 1, 1, 1], dtype=bool)
    for attempt in range(60):
        z = rng.normal(0, 1.5, size=(R, V))
        y = rng.integers(0, V, size=R)
        logp, _, _ = oracle.row_log_softmax(z, y, p.temperature)
        rho = logp + rng.normal(0, 0.5, size=R)
        q = logp + rng.normal(0, 0.4, size=R)
        own = variant.endswith("_own")
        old = logp + rng.normal(0, 0.3, size=R) if (p.correction != "none" and not own) else None
        w = rng.random(n_traj)
        ids = np.stack([rng.choice(V, 3, replace=False) for _ in range(R)])
        tlp = np.log(rng.dirichlet(np.ones(V), size=R))[np.arange(R)[:, None], ids]
        kw = dict(old=old, topk_ids=ids, topk_teacher=tlp)
        out = oracle.rl_loss(z, y, rho, q, w, gid, cu, 2, m, p, grad_loss=1.3, **kw)
        if not _near_kink(out, p):
            break
    else:
        pytest.fail("no draw away from the kinks")
    if own:
        # the correction weight is a constant: hold the ratio at its value
        frozen_rc = oracle.correction_ratio(out["logp"], rho)
        assert (np.minimum(np.maximum(frozen_rc, 0.5), 1.1) != frozen_rc).any()
        monkeypatch.setattr(oracle.rl_loss_ref, "correction_ratio", lambda *a, **k: frozen_rc)
    if variant == "topk":
        # the top-K signal is a fixed per-token reward: hold it at its value
        frozen = oracle.opd_topk_estimate(z, p.temperature, out["lse"], ids, tlp)
        monkeypatch.setattr(oracle.rl_loss_ref, "opd_topk_estimate",
                            lambda *a, **k: frozen[:a[0].shape[0]] if a[0].shape[0] == R else None)
    h = 1e-6
    num = np.zeros_like(z)
    for i in range(R):
        for j in range(V):
            zp = z.copy(); zp[i, j] += h
            zm = z.copy(); zm[i, j] -= h
            lp = oracle.rl_loss(zp, y, rho, q, w, gid, cu, 2, m, p, want_dlogits=False,
                                chunk=R, **kw)["loss"]
            lm = oracle.rl_loss(zm, y, rho, q, w, gid, cu, 2, m, p, want_dlogits=False,
                                chunk=R, **kw)["loss"]
            num[i, j] = 1.3 * (lp - lm) / (2 * h)
    scale = np.abs(out["dlogits"]).max()
    np.testing.assert_allclose(out["dlogits"], num, atol=1e-6 * max(scale, 1e-3), rtol=1e-6)
