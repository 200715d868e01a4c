"""GPU parity of vocabulary-sharded calls (rl_loss_vocab_shard_fwd_bwd): the
vocabulary of one call split over column shards (tensor parallelism), alone
and with its rows split as well (context / data parallelism), every shard run
on one GPU one after the other with the exchanges done by stacks, sums and
maxima over the shards' small arrays. The assembled outputs are compared with
the float64 oracle at the library's tolerances; every column shard of a row
must hold the same log-prob and entropy bits."""

import numpy as np
import pytest
import torch

import _parity as P
from paper_2609_08368_gb300 import api, workloads as wl
from paper_2609_08368_gb300 import milesloss as ml

pytestmark = pytest.mark.gpu

DEV = "cuda"


@pytest.fixture(autouse=True)
def ov():
    """Launch-plan overrides for one test; none are left installed afterwards."""
    fields = {}

    def set_(**kw):
        fields.update(kw)
        ml.set_launch_overrides(**fields)
    ml.set_launch_overrides()
    yield set_
    ml.set_launch_overrides()


def _view(w, r0, r1, c0, c1):
    """Rows [r0, r1) and vocabulary columns [c0, c1) of a workload as one
    shard's workload: the logits are a strided view (the row stride stays the
    whole call's), the per-trajectory inputs stay the whole call's."""
    sl = slice(r0, r1)

    def rows(t):
        return None if t is None else t[sl].contiguous()
    return wl.Workload(w.recipe, w.logits[sl, c0:c1], rows(w.targets), rows(w.rollout_logprobs),
                       rows(w.ref_logprobs), rows(w.old_logprobs), rows(w.teacher_logprobs),
                       w.rewards, w.group_id, w.cu_seqlens, rows(w.loss_mask), w.n_groups,
                       dict(w.params), rows(w.topk_ids), rows(w.topk_teacher))


def run_sharded(w, col_starts, row_cuts, params, dl_dtype=None, drive=True):
    """shards[i][k]: column shard k of row shard i, each with its own buffers
    (NaN-filled), driven through every phase unless drive is False."""
    R, n_traj = w.n_rows, int(w.rewards.shape[0])
    dl_dtype = dl_dtype or w.logits.dtype
    shards = []
    for r0, r1 in zip(row_cuts[:-1], row_cuts[1:]):
        row = []
        for k in range(len(col_starts) - 1):
            c0, c1 = col_starts[k], col_starts[k + 1]
            buf = api.alloc(r1 - r0, n_traj, w.n_groups, DEV, vocab=c1 - c0,
                            dlogits_dtype=dl_dtype, fill_nan=True)
            row.append(api.VocabShard(_view(w, r0, r1, c0, c1), k, col_starts, buf,
                                      row_offset=r0, n_rows_total=R, params=params))
        shards.append(row)
    if drive:
        api.vocab_sharded_fwd_bwd_local(shards)
        torch.cuda.synchronize()
    return shards


def assemble(w, shards, col_starts, row_cuts, expect_err=0):
    """The whole call's outputs from its shards, in run_gpu's format."""
    R = w.n_rows
    dl = torch.full((R, w.vocab), float("nan"), dtype=shards[0][0].buf.dlogits.dtype, device=DEV)
    logp = np.empty(R, np.float32)
    H = np.empty(R, np.float32)
    for (r0, r1), row in zip(zip(row_cuts[:-1], row_cuts[1:]), shards):
        lp0, h0 = P.np_(row[0].buf.token_logprobs), P.np_(row[0].buf.entropy)
        for k, s in enumerate(row):
            assert ml.rl_loss_check_device_error(s.buf.workspace) == expect_err
            dl[r0:r1, col_starts[k]:col_starts[k + 1]] = s.buf.dlogits
            # the merge runs in shard order: every column shard has the same bits
            np.testing.assert_array_equal(P.np_(s.buf.token_logprobs), lp0)
            np.testing.assert_array_equal(P.np_(s.buf.entropy), h0)
        logp[r0:r1], H[r0:r1] = lp0, h0
    first = shards[0][0].buf
    stats = first.read_stats()
    for row in shards:
        for s in row:
            assert s.buf.read_stats() == stats
            np.testing.assert_array_equal(P.np_(s.buf.advantages), P.np_(first.advantages))
            np.testing.assert_array_equal(P.np_(s.buf.group_sizes), P.np_(first.group_sizes))
    return dict(logp=logp, H=H, A=P.np_(first.advantages), group_sizes=P.np_(first.group_sizes),
                stats=stats, dlogits_t=dl)


V = 20480
LAYOUTS = {
    # (column starts, row cuts; None = the whole call's rows)
    "tp2": ([0, 10240, V], None),
    "tp3_unaligned": ([0, 7001, 13000, V], None),     # column starts off 16-byte boundaries
    "tp2_cp2": ([0, 10240, V], [0, 137]),
    "tp4_cp3": ([0, 5000, 10240, 15003, V], [0, 50, 50]),  # with an empty row shard
    "tp1": ([0, V], None),                               # one column shard: the whole vocabulary
    "tp8_uneven": ([0, 8, 1000, 1024, 9000, 9001, 15000, 20000, V], [0, 200]),
}
PARAMS = {
    "grpo": dict(),
    "rpp_kl": dict(estimator="reinforcepp", kl_coef=0.05),
    "opd_ent_tis": dict(opd_coef=0.3, entropy_coef=0.01, temperature=0.7, correction="tis",
                        corr_lo=0.0, corr_hi=2.0),
    "gspo_tis": dict(estimator="gspo", correction="tis", corr_lo=0.0, corr_hi=1.5),
    "topk_ent": dict(opd_coef=0.3, opd_topk=8, entropy_coef=0.01),
}


def _workload():
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=40, vocab=V,
                    rho_noise=0.3, ref_noise=0.2, teacher_noise=0.4, mask="prefix_u0_half",
                    topk=8, topk_noise=0.4)
    return wl.make(rec, DEV)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("layout", list(LAYOUTS))
@pytest.mark.parametrize("pname", list(PARAMS))
def test_vocab_sharded_call_matches_the_oracle(ov, kind, layout, pname):
    """Column shards (and row shards) of one call: log-probs, entropies,
    advantages, group sizes, N, clip counts, the metrics and the loss
    (1e-4 relative) against the oracle, every dLogit at 1e-2 relative /
    1e-5 absolute. The streaming kernel takes the slices whose rows start
    16-byte aligned; the others run in the cluster kernel."""
    ov(sweep_kernel=kind)
    w = _workload()
    params = dict(w.params, **PARAMS[pname])
    cols, cuts = LAYOUTS[layout]
    cuts = (cuts or [0]) + [w.n_rows]
    shards = run_sharded(w, cols, cuts, params)
    g = assemble(w, shards, cols, cuts)
    o = P.run_oracle(w, params=params)
    P.compare_forward(w, g, o, params=params)
    P.assert_dlogits_close(g["dlogits_t"].float().cpu().numpy(), o["dlogits"])


def test_vocab_sharded_fp32_logits_and_dlogits(ov):
    """fp32 logits and dLogits, three column shards with unaligned starts,
    two row shards (log-probs and entropy at 1e-5)."""
    rec = wl.shrink(wl.RECIPES["fp32"], n_prompts=4, traj_len=40, vocab=12288, rho_noise=0.4)
    w = wl.make(rec, DEV)
    cols, cuts = [0, 4097, 8190, 12288], [0, 301, w.n_rows]
    params = dict(w.params)
    g = assemble(w, run_sharded(w, cols, cuts, params), cols, cuts)
    o = P.run_oracle(w, params=params)
    P.compare_forward(w, g, o, params=params)
    P.assert_dlogits_close(g["dlogits_t"].float().cpu().numpy(), o["dlogits"])


def test_vocab_sharded_forward_only_leaves_dlogits_alone():
    """SWEEP without dLogits: the same log-probs and loss, dLogits untouched."""
    w = _workload()
    cols, cuts = [0, 10240, V], [0, w.n_rows]
    shards = run_sharded(w, cols, cuts, dict(w.params), drive=False)
    flat = [s for row in shards for s in row]
    for s in flat:
        s.count()
    for s in flat:
        s.partial()
    gathered = torch.stack([s.row_partials for s in flat])
    for s in flat:
        s.row_partials_all.copy_(gathered)
        s.sweep(forward_only=True)
        s.finish()
    torch.cuda.synchronize()
    for s in flat:
        assert torch.isnan(s.buf.dlogits.float()).all()
    whole = run_sharded(w, cols, cuts, dict(w.params))
    for a, b in zip(flat, [s for row in whole for s in row]):
        np.testing.assert_array_equal(P.np_(a.buf.token_logprobs), P.np_(b.buf.token_logprobs))
        assert a.buf.read_stats() == b.buf.read_stats()


def test_vocab_sharded_bad_target_is_reported():
    """A target outside the vocabulary: SWEEP on every column shard reports
    RL_ERR_TARGET_OUT_OF_RANGE and writes zeros for that row; the other rows
    match the oracle."""
    w = _workload()
    bad = 17
    y_ok = int(w.targets[bad])
    w.targets[bad] = V  # one past the end (no shard owns it)
    cols, cuts = [0, 10240, V], [0, w.n_rows]
    shards = run_sharded(w, cols, cuts, dict(w.params))
    g = assemble(w, shards, cols, cuts, expect_err=5)  # RL_ERR_TARGET_OUT_OF_RANGE
    assert g["logp"][bad] == 0 and g["H"][bad] == 0
    assert (g["dlogits_t"][bad].float() == 0).all()
    w.targets[bad] = y_ok
    o = P.run_oracle(w)
    good = np.setdiff1d(np.arange(w.n_rows), [bad])
    tol = P.logp_tol(w)
    np.testing.assert_allclose(g["logp"][good], o["logp"][good], atol=tol, rtol=0)
    np.testing.assert_allclose(g["H"][good], o["H"][good], atol=tol, rtol=0)
    P.assert_dlogits_close(g["dlogits_t"][good].float().cpu().numpy(), o["dlogits"][good])


@pytest.mark.parametrize("kind", ["cluster", "stream"])
def test_vocab_sharded_topk_ids_out_of_range_are_reported(ov, kind):
    """A top-K candidate id outside the vocabulary: SWEEP on every column
    shard reports RL_ERR_TOPK_ID_OUT_OF_RANGE and writes zeros for that row;
    the other rows match the oracle (with a valid id in its place)."""
    ov(sweep_kernel=kind)
    w = _workload()
    params = dict(w.params, opd_coef=0.3, opd_topk=8)
    bad = [5, 33]
    ids_ok = w.topk_ids.clone()
    w.topk_ids[5, 3] = V        # one past the end
    w.topk_ids[33, 0] = -1
    cols, cuts = [0, 10240, V], [0, w.n_rows]
    g = assemble(w, run_sharded(w, cols, cuts, params), cols, cuts, expect_err=9)
    for r in bad:
        assert g["logp"][r] == 0 and g["H"][r] == 0
        assert (g["dlogits_t"][r].float() == 0).all()
    w.topk_ids.copy_(ids_ok)
    o = P.run_oracle(w, params=params)
    good = np.setdiff1d(np.arange(w.n_rows), bad)
    tol = P.logp_tol(w)
    np.testing.assert_allclose(g["logp"][good], o["logp"][good], atol=tol, rtol=0)
    np.testing.assert_allclose(g["H"][good], o["H"][good], atol=tol, rtol=0)
    P.assert_dlogits_close(g["dlogits_t"][good].float().cpu().numpy(), o["dlogits"][good])


@pytest.mark.parametrize("kind", ["cluster", "stream"])
def test_vocab_shard_that_gives_up_zeroes_its_rows_everywhere(ov, kind):
    """Failure detection across shards, without a fault: the test hook makes
    every CTA of shard 0's partial sweep give up on its first wait (bounded
    by 1 ms). Shard 0 reports RL_ERR_DEVICE_TIMEOUT; its records carry the
    give-up mark, so the merge on EVERY shard writes zeros for those rows
    (finite outputs, zero dLogits) and shard 1's own error word stays clean.
    The next call without the hook matches the oracle."""
    ov(sweep_kernel=kind)
    w = _workload()
    cols, cuts = [0, 10240, V], [0, w.n_rows]
    shards = run_sharded(w, cols, cuts, dict(w.params), drive=False)
    s0, s1 = shards[0]
    for s in (s0, s1):
        s.count()
    ov(stall_first_wait_ns=1_000_000)
    s0.partial()
    ov(stall_first_wait_ns=-1)
    s1.partial()
    gathered = torch.stack([s0.row_partials, s1.row_partials])
    for s in (s0, s1):
        s.row_partials_all.copy_(gathered)
        s.sweep()
        s.finish()
    torch.cuda.synchronize()
    assert ml.rl_loss_check_device_error(s0.buf.workspace) == 8  # RL_ERR_DEVICE_TIMEOUT
    assert ml.rl_loss_check_device_error(s1.buf.workspace) == 0
    for s in (s0, s1):
        assert (s.buf.token_logprobs == 0).all() and (s.buf.entropy == 0).all()
        assert torch.equal(s.buf.dlogits, torch.zeros_like(s.buf.dlogits))
        assert s.buf.read_stats()["loss"] == 0.0
    g = assemble(w, run_sharded(w, cols, cuts, dict(w.params)), cols, cuts)
    o = P.run_oracle(w)
    P.compare_forward(w, g, o)
    P.assert_dlogits_close(g["dlogits_t"].float().cpu().numpy(), o["dlogits"])


@pytest.mark.slow
def test_full_size_two_column_shards_equal_the_whole_call():
    """The headline batch (65,536 x 154,880 bf16) split into two column
    shards of 77,440 (TP 2): log-probs and entropies within 1e-5 of the
    unsharded call (the same fp32 sums in another grouping), every dLogit
    within 1e-2 relative / 1e-5 absolute of it, N and the group sizes equal,
    the loss within 1e-4 relative. (The unsharded call itself is compared
    with the float64 oracle on every row in test_full_size_every_row.)"""
    w = wl.make(wl.RECIPES["glm"], DEV)
    whole = P.run_gpu(w)
    assert whole["err"] == 0
    half = w.vocab // 2
    cols, cuts = [0, half, w.vocab], [0, w.n_rows]
    g = assemble(w, run_sharded(w, cols, cuts, dict(w.params)), cols, cuts)
    np.testing.assert_allclose(g["logp"], whole["logp"], atol=1e-5, rtol=0)
    np.testing.assert_allclose(g["H"], whole["H"], atol=1e-5, rtol=0)
    np.testing.assert_array_equal(g["group_sizes"], whole["group_sizes"])
    assert g["stats"]["n_tokens"] == whole["stats"]["n_tokens"]
    P.assert_loss_close(g["stats"]["loss"], whole["stats"]["loss"], what="TP 2 loss")
    for r0 in range(0, w.n_rows, 4096):  # in blocks of rows: fp32 copies of 4,096 rows
        a = g["dlogits_t"][r0:r0 + 4096].float()
        b = whole["dlogits_t"][r0:r0 + 4096].float()
        excess = (a - b).abs() - torch.clamp(1e-2 * b.abs(), min=1e-5)
        assert bool((excess <= 0).all()), (r0, float(excess.max()))
