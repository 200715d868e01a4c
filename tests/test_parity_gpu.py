"""GPU parity: the CUDA library against the float64 oracle, element by
element, on seeded workloads at sizes the oracle finishes in seconds (many
rows, every cluster size, ragged tails), plus edge cases, error paths,
determinism and batch invariance. All calls go through the C ABI."""

import os

import numpy as np
import pytest
import torch

import _parity as P
import oracle
from paper_2609_08368_gb300 import api, workloads as wl
from paper_2609_08368_gb300 import milesloss as ml

pytestmark = pytest.mark.gpu

DEV = "cuda"

SHRUNK = {
    "tiny": wl.RECIPES["tiny"],
    "qwen": wl.shrink(wl.RECIPES["qwen"], n_prompts=2, traj_len=16),
    "glm": wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=48),
    "agentic": wl.shrink(wl.RECIPES["agentic"], traj_len=2048, vocab=8192),
    "fp32": wl.shrink(wl.RECIPES["fp32"], n_prompts=8, traj_len=32),
    # wide rollout noise: many tokens past every clip threshold
    "glm_noisy": wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=64,
                           vocab=20480, rho_noise=0.35, ref_noise=0.3),
    "fp32_noisy": wl.shrink(wl.RECIPES["fp32"], n_prompts=4, traj_len=64, vocab=12288,
                            rho_noise=0.4),
}


@pytest.fixture(autouse=True)
def ov():
    """Launch-plan overrides for one test: ``ov(field=value, ...)`` adds to
    the test's overrides; none are left installed afterwards."""
    fields = {}

    def set_(**kw):
        fields.update(kw)
        ml.set_launch_overrides(**fields)
    ml.set_launch_overrides()
    yield set_
    ml.set_launch_overrides()


def _full_check(w, mode="fused", dl_dtype=None, params=None, fp32_floor=False):
    g = P.run_gpu(w, mode=mode, dl_dtype=dl_dtype, params=params)
    assert g["err"] == 0, ml.status_string(g["err"])
    o = P.run_oracle(w, params=params)
    floor = P.fp32_logp_loss_floor(w, o, params) if fp32_floor else 0.0
    P.compare_forward(w, g, o, params=params, loss_floor=floor)
    if mode != "fwd":
        P.assert_dlogits_close(g["dlogits_t"][:, :w.vocab].float().cpu().numpy(), o["dlogits"])
    return g, o


@pytest.mark.parametrize("name", list(SHRUNK))
def test_parity_fused(name):
    _full_check(wl.make(SHRUNK[name], DEV))


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("name", list(SHRUNK))
def test_parity_each_sweep_kernel(ov, kind, name):
    """Both vocabulary-sweep kernels (cluster exchange, and one CTA per row
    with an L2-served second read) on every workload."""
    ov(sweep_kernel=kind)
    _full_check(wl.make(SHRUNK[name], DEV))
    _full_check(wl.make(SHRUNK[name], DEV), mode="split")


@pytest.mark.parametrize("chunk,slots,hold,split", [
    (16384, 14, 1, 0), (16384, 14, 5, 1), (4096, 2, 0, 0), (4096, 2, 2, 1), (12288, 3, 2, 1),
    (12288, 3, 3, 0), (1024, 1, 1, 1), (1024, 1, 0, 0), (65536, 3, 2, 1), (75776, 3, 2, 1),
    (8192, 4, 4, 1)])
def test_stream_ring_shapes(ov, chunk, slots, hold, split):
    """The streaming kernel's ring: chunk sizes, slot counts, chunks kept in
    shared memory for pass B (0 to every slot) and the ragged chunk first or
    last, on rows of 2 to 88 chunks."""
    ov(sweep_kernel="stream")
    ov(stream_chunk_bytes=chunk)
    ov(stream_slots=slots)
    ov(stream_hold=hold)
    ov(stream_split_first=split)
    # ragged rows: 45,003 bf16 columns = 5,625 vectors and a 3-element tail
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=24, vocab=45003,
                    rho_noise=0.3)
    _full_check(wl.make(rec, DEV))
    rec = wl.shrink(wl.RECIPES["fp32"], n_prompts=1, group_size=4, traj_len=16, vocab=20001,
                    rho_noise=0.3)
    _full_check(wl.make(rec, DEV))


@pytest.mark.parametrize("per_sm,chunk,slots,hold,split", [
    (2, -1, -1, -1, -1), (2, 36864, 3, 2, 1), (2, 36864, 3, 3, 0), (2, 16384, 6, 2, 1),
    (2, 4096, 2, 0, 0), (2, 1024, 1, 1, 1), (4, -1, -1, -1, -1), (4, 12288, 4, 2, 1),
    (4, 9216, 5, 5, 0), (4, 2048, 3, 0, 1)])
def test_stream_several_ctas_per_sm(ov, per_sm, chunk, slots, hold, split):
    """The streaming kernel with two or four CTAs per SM (eight or four
    consumer warps each, a half or a quarter of the SM's shared memory for
    each ring), with its default ring and forced ones, on ragged bf16 and
    fp32 rows, fused and split, and with top-K OPD and the entropy bonus."""
    ov(sweep_kernel="stream")
    ov(stream_ctas_per_sm=per_sm)
    for f, v in (("stream_chunk_bytes", chunk), ("stream_slots", slots), ("stream_hold", hold),
                 ("stream_split_first", split)):
        if v >= 0:
            ov(**{f: v})
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=24, vocab=45003,
                    rho_noise=0.3)
    _full_check(wl.make(rec, DEV))
    _full_check(wl.make(rec, DEV), mode="split")
    rec = wl.shrink(wl.RECIPES["fp32"], n_prompts=1, group_size=4, traj_len=16, vocab=20001,
                    rho_noise=0.3)
    _full_check(wl.make(rec, DEV))
    w = wl.make(wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=24,
                          vocab=40960, topk=16), DEV)
    _full_check(w, params=dict(w.params, entropy_coef=0.01, opd_topk=16, opd_coef=0.5))


@pytest.mark.parametrize("vocab", [34816, 36864, 45000])
def test_fp32_rows_in_two_equal_chunks(vocab):
    """The launch plan of fused fp32 rows of 136-192 KB: one streaming CTA
    per SM, the row in two (nearly) equal chunks, neither kept for pass B:
    three 68 / 72 KB slots, or two of 88 KB for 45,000 columns (chunks of
    5,624 and 5,626 vectors)."""
    rec = wl.shrink(wl.RECIPES["fp32"], n_prompts=1, group_size=4, traj_len=16, vocab=vocab,
                    rho_noise=0.3)
    _full_check(wl.make(rec, DEV))
    _full_check(wl.make(rec, DEV), mode="split")


@pytest.mark.parametrize("name", ["tiny", "fp32", "glm_noisy"])
def test_parity_split_fwd_then_bwd(name):
    _full_check(wl.make(SHRUNK[name], DEV), mode="split")


def test_clip_decisions_are_exercised():
    w = wl.make(SHRUNK["glm_noisy"], DEV)
    params = dict(w.params, dual_clip_c=1.5)  # r > 1.5 is common at this noise
    g, _ = _full_check(w, params=params)
    st = g["stats"]
    assert st["n_clip_hi"] > 0 and st["n_clip_lo"] > 0 and st["n_dual_clip"] > 0


def test_dlogits_relative_error_on_order_p_entries():
    """With grad_loss = N the entries are O(p), so the relative bound is
    checked on every entry of magnitude >= 1e-6."""
    for name in ("tiny", "fp32_noisy"):
        w = wl.make(SHRUNK[name], DEV)
        N = int(w.loss_mask.sum())
        g = P.run_gpu(w, grad_loss=float(N), dl_dtype=torch.float32)
        o = P.run_oracle(w, grad_loss=float(N))
        got = g["dlogits_t"].cpu().numpy()
        terms = P.summand_magnitude(w, o, float(N))
        P.assert_rel_on_large(got, o["dlogits"], terms, floor=1e-6, rel=1e-3, cancel=1e-4)
        P.assert_dlogits_close(got, o["dlogits"])


@pytest.mark.parametrize("cluster", [1, 2, 4, 8])
def test_every_cluster_size(ov, cluster):
    ov(sweep_kernel="cluster")
    ov(cluster_size=cluster)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=24, vocab=20000 + 24)
    _full_check(wl.make(rec, DEV))


@pytest.mark.parametrize("threads,per_sm", [(256, 4), (256, 5), (512, 2)])
def test_every_block_shape(ov, threads, per_sm):
    ov(sweep_kernel="cluster")
    ov(cluster_threads=threads)
    ov(cluster_ctas_per_sm=per_sm)
    _full_check(wl.make(SHRUNK["glm_noisy"], DEV))


@pytest.mark.parametrize("stages", [1, 2, 3, 4])
def test_every_ring_depth(ov, stages):
    ov(sweep_kernel="cluster")
    ov(cluster_size=2)
    ov(cluster_stages=stages)
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=1, group_size=4, traj_len=40, vocab=6144)
    _full_check(wl.make(rec, DEV))


@pytest.mark.parametrize("vocab", [1, 2, 7, 9, 4097, 12345])
def test_ragged_vocab(vocab):
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=1, group_size=3, traj_len=5, vocab=vocab,
                    mask="none")
    _full_check(wl.make(rec, DEV))


def test_padded_and_misaligned_rows():
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=1, group_size=2, traj_len=24, vocab=1000)
    # ld = 1003 bf16 elements: rows are not 16-byte aligned (scalar path)
    w = wl.make(rec, DEV, ld=1003)
    g, o = _full_check(w)
    # padded, aligned rows; the dLogits padding must stay untouched (NaN)
    w = wl.make(rec, DEV, ld=1024)
    g = P.run_gpu(w, ld_out=1032)
    assert torch.isnan(g["dlogits_t"][:, 1000:]).all()
    o = P.run_oracle(w)
    P.assert_dlogits_close(g["dlogits_t"][:, :1000].float().cpu().numpy(), o["dlogits"])


def _extreme_rows(w):
    """Rows that stress the running-maximum and -inf handling of the sweeps:
    -inf logits (scattered, nearly all, a whole leading block, all but the
    target), a spike far above the rest (at the row's end, in its first
    chunk, on the target), a constant row, a ramp whose maximum is last,
    and a row shifted to -1000."""
    V = w.vocab
    z = w.logits[:, :V]
    y = w.targets.long()
    g = torch.Generator(device="cpu").manual_seed(5)
    ninf = float("-inf")
    keep_y = lambda r, row: row.index_fill_(0, y[r:r + 1], float(z[r, y[r]]))  # noqa: E731
    sc = torch.rand(V, generator=g) < 0.1
    row = z[0].clone(); row[sc.to(z.device)] = ninf; z[0] = keep_y(0, row)
    row = torch.full((V,), ninf, dtype=z.dtype, device=z.device)
    live = torch.randperm(V, generator=g)[:100].to(z.device)
    row[live] = z[1, live]; z[1] = keep_y(1, row)
    z[2, V - 1] = 150.0
    if int(y[2]) == V - 1:
        w.targets[2] = 0
    z[3, V - 1] = 150.0
    w.targets[3] = V - 1
    z[4] = 5.0
    z[5] = torch.linspace(-60.0, 60.0, V, device=z.device).to(z.dtype)
    z[6] = (z[6].float() - 1000.0).to(z.dtype)
    row = z[7].clone(); row[:min(V, 8192)] = ninf; z[7] = keep_y(7, row)
    z[8, V // 4] = 100.0
    row = torch.full((V,), ninf, dtype=z.dtype, device=z.device); z[9] = keep_y(9, row)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("extra", [dict(), dict(entropy_coef=0.01, temperature=0.7),
                                   dict(temperature=0.05)])
def test_extreme_logits(ov, kind, extra):
    """Extreme rows (see _extreme_rows) on both sweep kernels, fused and
    split, with and without the entropy term and temperature; a row of 200 KB
    runs in the streaming kernel in two ring chunks."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=4, vocab=100000)
    w = wl.make(rec, DEV)
    _extreme_rows(w)
    params = dict(w.params, **extra)
    # rollout and reference log-probs near the new rows' own (a log-ratio
    # past ~88 would overflow the fp32 exponentials of the ratio and of k3)
    lp, _, _ = oracle.row_log_softmax(P.host_logits(w), P.np_(w.targets),
                                      params.get("temperature", 1.0))
    lp = torch.from_numpy(lp).float().to(DEV)
    w.rollout_logprobs.copy_(lp + 0.05 * torch.sin(torch.arange(w.n_rows, device=DEV)))
    if w.ref_logprobs is not None:
        w.ref_logprobs.copy_(lp - 0.03)
    if w.old_logprobs is not None:
        w.old_logprobs.copy_(lp + 0.01)
    # rows shifted to -1000 (and divided by T = 0.05) have |lse| up to ~2e4:
    # their fp32 log-probs carry errors of ~eps |lse|, which the loss bound
    # takes as its floor (fp32_logp_loss_floor)
    g, o = _full_check(w, params=params, fp32_floor=True)
    for k in ("logp", "H"):
        assert np.all(np.isfinite(g[k])), k
    assert abs(float(g["H"][9])) < 1e-6 and abs(float(g["logp"][9])) < 1e-6
    # the objective and the reduction alone, on the GPU's own log-probs: 1e-4
    own = P.stats_on_gpu_logp(w, g, o, P.oracle_params(params))
    P.assert_loss_close(g["stats"]["loss"], own["loss"], what="loss on the GPU's log-probs")
    _full_check(w, mode="split", params=params, fp32_floor=True)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("ld,ld_out", [(100008, 100000), (100003, 100003), (100000, 100011)])
def test_long_rows_padded_and_misaligned(ov, kind, ld, ld_out):
    """Rows of 200 KB on both sweep kernels with a padded row stride, rows
    whose starts are not 16-byte aligned (the cluster kernel's element-wise
    path takes them whatever the kind), and a dLogits stride that is not
    16-byte aligned (scalar stores); fused and split."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=6, vocab=100000)
    w = wl.make(rec, DEV, ld=ld)
    for mode in ("fused", "split"):
        g = P.run_gpu(w, mode=mode, ld_out=ld_out)
        assert g["err"] == 0, ml.status_string(g["err"])
        o = P.run_oracle(w)
        P.compare_forward(w, g, o)
        P.assert_dlogits_close(g["dlogits_t"][:, :w.vocab].float().cpu().numpy(), o["dlogits"])
        if ld_out > w.vocab:
            assert torch.isnan(g["dlogits_t"][:, w.vocab:]).all()


@pytest.mark.parametrize("logits,vocab,ld,dl_dtype,ld_out", [
    ("bf16", 140003, 140008, torch.bfloat16, 140008),
    ("bf16", 140003, 140008, torch.float32, 140011),
    ("bf16", 131075, 131080, torch.float32, 131076),
    ("f32", 65541, 65544, torch.bfloat16, 65544),
    ("f32", 65541, 65544, torch.float32, 65547)])
def test_long_row_plan_shapes(logits, vocab, ld, dl_dtype, ld_out):
    """The streaming kernel's plan for rows of 240 KB and more (three 74 KB
    slots, the ragged remainder first, two chunks kept for pass B), chosen by
    the library for 16-byte aligned rows: vector counts that are not a
    multiple of 8 (the last chunk a few vectors short of a slot), elements
    past the last whole vector, bf16 and fp32 logits and dLogits, and
    dLogits strides that are 16-byte aligned (vector stores) or not (scalar
    stores); fused and split."""
    base = wl.RECIPES["glm" if logits == "bf16" else "fp32"]
    rec = wl.shrink(base, n_prompts=1, group_size=4, traj_len=6, vocab=vocab, rho_noise=0.3)
    w = wl.make(rec, DEV, ld=ld)
    for mode in ("fused", "split"):
        g = P.run_gpu(w, mode=mode, dl_dtype=dl_dtype, ld_out=ld_out)
        assert g["err"] == 0, ml.status_string(g["err"])
        o = P.run_oracle(w)
        P.compare_forward(w, g, o)
        P.assert_dlogits_close(g["dlogits_t"][:, :vocab].float().cpu().numpy(), o["dlogits"])
        if ld_out > vocab:
            assert torch.isnan(g["dlogits_t"][:, vocab:]).all()


@pytest.mark.parametrize("logits,vocab,ld,topk", [
    ("bf16", 262144, 262144, 0),       # 512 KB rows (a 256K vocabulary)
    ("bf16", 256000, 256000, 16),      # with top-K OPD
    ("bf16", 1000003, 1000008, 0),     # ~2 MB rows, elements past the last whole vector
    ("f32", 200003, 200004, 0)])       # ~800 KB fp32 rows
def test_very_long_rows(logits, vocab, ld, topk):
    """Rows far longer than the headline's (up to ~2 MB, tens of ring chunks
    per row, most of pass B's second read from L2): fused and split calls
    against the oracle, the padding of each row left untouched."""
    base = wl.RECIPES["glm" if logits == "bf16" else "fp32"]
    rec = wl.shrink(base, n_prompts=1, group_size=4, traj_len=6, vocab=vocab, rho_noise=0.3,
                    topk=topk)
    w = wl.make(rec, DEV, ld=ld)
    params = dict(w.params, opd_coef=0.3, opd_topk=topk) if topk else None
    for mode in ("fused", "split"):
        g = P.run_gpu(w, mode=mode, ld_out=ld, params=params)
        assert g["err"] == 0, ml.status_string(g["err"])
        o = P.run_oracle(w, params=params)
        P.compare_forward(w, g, o, params=params)
        P.assert_dlogits_close(g["dlogits_t"][:, :vocab].float().cpu().numpy(), o["dlogits"])
        if ld > vocab:
            assert torch.isnan(g["dlogits_t"][:, vocab:]).all()


@pytest.mark.parametrize("C", [2, 4, 8])
@pytest.mark.parametrize("logits,vocab,ld,dl_dtype,traj", [
    ("bf16", 262144, 262144, None, 60),        # 512 KB rows, several rows per cluster
    ("bf16", 100003, 100008, torch.float32, 60),  # elements past the last whole vector
    ("f32", 200003, 200004, None, 30),         # ~800 KB fp32 rows
    ("bf16", 100, 104, None, 8)])              # CTAs whose slice holds no vector of the row
def test_stream_clusters(ov, C, logits, vocab, ld, dl_dtype, traj):
    """The streaming kernel with a cluster of C CTAs per row (each CTA
    streams one slice of the row, the CTAs exchange their row sums and merge
    them in rank order): every output against the oracle, every CTA's part of
    dLogits, the row padding untouched, and bit-identical reruns."""
    ov(sweep_kernel="stream", stream_cluster=C)
    base = wl.RECIPES["glm" if logits == "bf16" else "fp32"]
    rec = wl.shrink(base, n_prompts=1, group_size=4, traj_len=traj, vocab=vocab, rho_noise=0.3,
                    ref_noise=0.2)
    w = wl.make(rec, DEV, ld=ld)
    params = dict(w.params, entropy_coef=0.01, kl_coef=0.05)
    g = P.run_gpu(w, dl_dtype=dl_dtype, ld_out=ld, params=params)
    assert g["err"] == 0, ml.status_string(g["err"])
    o = P.run_oracle(w, params=params)
    P.compare_forward(w, g, o, params=params)
    P.assert_dlogits_close(g["dlogits_t"][:, :vocab].float().cpu().numpy(), o["dlogits"])
    if ld > vocab:
        assert torch.isnan(g["dlogits_t"][:, vocab:]).all()
    again = P.run_gpu(w, dl_dtype=dl_dtype, ld_out=ld, params=params)
    assert torch.equal(again["dlogits_t"].view(torch.uint8), g["dlogits_t"].view(torch.uint8))
    np.testing.assert_array_equal(again["logp"], g["logp"])


@pytest.mark.parametrize("estimator", ["grpo", "reinforcepp", "gspo"])
@pytest.mark.parametrize("n_prompts", [8, 1200])
def test_ragged_and_empty_trajectories(estimator, n_prompts):
    """Trajectories of random lengths, some empty, with their row offsets in
    shared memory (32 trajectories) or, past what fits there, in global memory
    (4,800 trajectories)."""
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=n_prompts, group_size=4, traj_len=3,
                    vocab=512)
    w = wl.make(rec, DEV)
    rng = np.random.default_rng(n_prompts)
    n_traj = int(w.rewards.shape[0])
    cuts = np.sort(rng.integers(0, w.n_rows + 1, size=n_traj - 1))
    cu = np.concatenate([[0], cuts, [w.n_rows]]).astype(np.int32)
    assert (np.diff(cu) == 0).any()
    w.cu_seqlens.copy_(torch.from_numpy(cu))
    w.loss_mask.copy_(torch.from_numpy((rng.random(w.n_rows) < 0.7).astype(np.uint8)))
    _full_check(w, params=dict(w.params, estimator=estimator))


@pytest.mark.parametrize("kind", ["cluster", "stream"])
def test_fused_call_replays_from_a_cuda_graph(ov, kind):
    """The fused call only enqueues kernels on the caller's stream (no
    allocation, no synchronisation), so it can be captured in a CUDA graph;
    replays give bit-identical results to a direct call, also after the inputs
    change in place."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=8, vocab=100000)
    w = wl.make(rec, DEV)
    buf = api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, DEV, vocab=w.vocab,
                    dlogits_dtype=w.logits.dtype)
    call = api.GraphedCall(w, buf)
    for step in range(2):
        if step:
            w.logits.mul_(0.5)  # new inputs, same buffers
        call()
        torch.cuda.synchronize()
        got = (buf.dlogits.clone(), buf.token_logprobs.clone(), buf.read_stats()["loss"])
        api.fwd_bwd(w, buf)
        torch.cuda.synchronize()
        assert torch.equal(got[0], buf.dlogits) and torch.equal(got[1], buf.token_logprobs)
        assert got[2] == buf.read_stats()["loss"]
        assert ml.rl_loss_check_device_error(buf.workspace) == 0


@pytest.mark.parametrize("logit_dtype,dl_dtype", [("bf16", torch.float32), ("f32", torch.bfloat16)])
def test_mixed_dtypes(logit_dtype, dl_dtype):
    rec = wl.shrink(wl.RECIPES["fp32" if logit_dtype == "f32" else "tiny"], n_prompts=2,
                    group_size=4, traj_len=16, vocab=5000)
    _full_check(wl.make(rec, DEV), dl_dtype=dl_dtype)


def test_temperature_entropy_kl_correction_opd():
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=32, vocab=9000,
                    rho_noise=0.25, ref_noise=0.2, old_noise=0.1, teacher_noise=0.3)
    for params in (dict(temperature=0.7, eps_lo=0.2, eps_hi=0.28, dual_clip_c=3.0, kl_coef=0.05,
                        entropy_coef=0.01),
                   dict(temperature=1.3, correction="tis", corr_lo=0.0, corr_hi=1.1, kl_coef=0.1),
                   dict(correction="clip_or_pop", corr_lo=0.9, corr_hi=1.1, dual_clip_c=2.0),
                   dict(opd_coef=0.5, entropy_coef=0.002),
                   dict(normalize_std=False, unbiased_std=False)):
        w = wl.make(rec, DEV)
        _full_check(w, params=params)
        _full_check(w, mode="split", params=params)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [
    dict(correction="tis", corr_lo=0.0, corr_hi=1.1),
    dict(correction="clip_or_pop", corr_lo=0.9, corr_hi=1.1, dual_clip_c=2.0, kl_coef=0.05),
    dict(estimator="gspo", correction="tis", corr_lo=0.0, corr_hi=1.05),
], ids=["tis", "pop", "gspo_tis"])
def test_corrections_without_old_logprobs(ov, kind, params):
    """The corrections of Sec. 3.4 in a single-pass step: no old log-probs,
    so the correction ratio is the trainer's own log-prob of this pass
    against the rollout's (held constant) and the PPO ratio is taken against
    the rollout log-probs; fused and split, both sweep kernels."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=32, vocab=9000,
                    rho_noise=0.25, ref_noise=0.2)
    w = wl.make(rec, DEV)
    assert w.old_logprobs is None
    p = dict(w.params, **params)
    g, _ = _full_check(w, params=p)
    assert g["stats"]["n_corr_clip"] > 0
    _full_check(w, mode="split", params=p)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [
    dict(estimator="reinforcepp"),
    dict(estimator="reinforcepp_baseline", dual_clip_c=2.0, kl_coef=0.05),
    dict(estimator="reinforcepp", normalize_std=False, unbiased_std=False),
    dict(estimator="gspo", dual_clip_c=1.5, kl_coef=0.05, entropy_coef=0.01),
    dict(estimator="gspo", correction="tis", corr_lo=0.0, corr_hi=1.1, eps_lo=0.1, eps_hi=0.1),
    dict(estimator="gspo", correction="clip_or_pop", corr_lo=0.9, corr_hi=1.1, temperature=0.8),
], ids=["rpp", "rpp_base", "rpp_center", "gspo", "gspo_tis", "gspo_pop"])
def test_advantage_estimators(ov, kind, params):
    """REINFORCE++ (plain, baseline-relative) and GSPO (Sec. 3.4), fused and
    split, on both sweep kernels; trajectories of unequal training length."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=3, group_size=4, traj_len=20, vocab=9000,
                    rho_noise=0.3, ref_noise=0.2, old_noise=0.1, mask="prefix_u0_half")
    w = wl.make(rec, DEV)
    _full_check(w, params=params)
    _full_check(w, mode="split", params=params)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("K", [1, 4, 16])
def test_opd_topk(ov, kind, K):
    """The top-K on-policy distillation signal (Sec. 5.2) from candidate sets
    and teacher log-probs, in the sweep epilogue."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=24, vocab=12000,
                    rho_noise=0.3, ref_noise=0.2, topk=K, topk_noise=0.4)
    w = wl.make(rec, DEV)
    for params in (dict(opd_coef=0.5, opd_topk=K, dual_clip_c=2.0),
                   dict(opd_coef=-0.3, opd_topk=K, estimator="reinforcepp_baseline")):
        _full_check(w, params=params)
        _full_check(w, mode="split", params=params)


@pytest.mark.parametrize("kind,cluster", [("cluster", 0), ("cluster", 8), ("stream", 0)])
@pytest.mark.parametrize("K", [4, 64])
def test_opd_topk_long_rows(ov, kind, cluster, K):
    """Top-K OPD on rows of 200 KB: candidates spread over the CTAs of a
    cluster (4 by the plan, 8 forced; their partial sums merge in the row
    exchange) or over the streaming kernel's two ring chunks."""
    ov(sweep_kernel=kind)
    if cluster:
        ov(cluster_size=cluster)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=12, vocab=100000,
                    rho_noise=0.3, ref_noise=0.2, topk=K, topk_noise=0.4)
    w = wl.make(rec, DEV)
    params = dict(w.params, opd_coef=0.5, opd_topk=K)
    _full_check(w, params=params)
    _full_check(w, mode="split", params=params)


@pytest.mark.parametrize("vocab,ring", [
    (45003, (4096, 2, 1, 0)), (45003, (4096, 3, 2, 1)), (45003, (1024, 1, 0, 0)),
    (45003, (16384, 4, 4, 1)), (45003, (75776, 3, 2, 1)), (131072, None)])
def test_opd_topk_stream_ring_shapes(ov, vocab, ring):
    """Top-K OPD in the streaming kernel, whose top-K warp waits on and
    releases every ring slot and hands each row's part to warp 0: chunk
    sizes, slot counts, kept chunks and both splits (rows of 1 to 88 chunks,
    a ragged tail past the last whole vector), and the default plan of
    256 KB rows (three 74 KB slots, two kept)."""
    ov(sweep_kernel="stream")
    if ring:
        ov(**dict(zip(("stream_chunk_bytes", "stream_slots", "stream_hold", "stream_split_first"),
                      ring)))
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=16, vocab=vocab,
                    rho_noise=0.3, ref_noise=0.2, topk=16, topk_noise=0.4)
    w = wl.make(rec, DEV)
    params = dict(w.params, opd_coef=0.5, opd_topk=16)
    _full_check(w, params=params)
    _full_check(w, mode="split", params=params)


@pytest.mark.parametrize("kind", ["cluster", "stream"])
def test_no_training_tokens_and_empty_call(ov, kind):
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=1, group_size=2, traj_len=8, vocab=300)
    w = wl.make(rec, DEV)
    w.loss_mask.zero_()
    g = P.run_gpu(w)
    assert g["err"] == 0
    assert g["stats"]["n_tokens"] == 0 and g["stats"]["loss"] == 0.0
    assert (g["dlogits_t"] == 0).all()
    o = P.run_oracle(w)
    np.testing.assert_allclose(g["logp"], o["logp"], atol=2e-3)
    # zero rows: advantages still computed, statistics all zero
    buf = api.alloc(0, 2, 1, DEV, vocab=300, dlogits_dtype=torch.bfloat16)
    empty = torch.empty(0, dtype=torch.bfloat16, device=DEV)
    ml.rl_loss_fwd_bwd(empty.view(0, 300), torch.empty(0, dtype=torch.int32, device=DEV),
                       torch.empty(0, device=DEV), None, None, None,
                       torch.tensor([0.0, 1.0], device=DEV),
                       torch.zeros(2, dtype=torch.int32, device=DEV),
                       torch.zeros(3, dtype=torch.int32, device=DEV), 1,
                       torch.empty(0, dtype=torch.uint8, device=DEV), {}, buf.token_logprobs,
                       buf.entropy, buf.advantages, buf.group_sizes, buf.stats, buf.dlogits,
                       buf.workspace, vocab=300)
    torch.cuda.synchronize()
    st = buf.read_stats()
    assert st["n_tokens"] == 0 and st["loss"] == 0.0
    assert buf.group_sizes.tolist() == [2]
    np.testing.assert_allclose(buf.advantages.cpu().numpy(), [-2 ** -0.5, 2 ** -0.5], rtol=1e-6)


@pytest.mark.parametrize("kind", ["cluster", "stream", "streamC4"])
def test_device_errors_are_reported_not_trapped(ov, kind):
    """Bad inputs that the kernels' own checks turn into error codes (no
    trap); "streamC4": the streaming kernel with a cluster of four CTAs per
    row, every CTA of which writes its part of a bad row as zeros."""
    if kind.startswith("streamC"):
        ov(sweep_kernel="stream", stream_cluster=int(kind[-1]))
    else:
        ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["tiny"], n_prompts=2, group_size=2, traj_len=8, vocab=256)
    w = wl.make(rec, DEV)
    w.targets[3] = 256                     # outside [0, vocab)
    g = P.run_gpu(w)
    assert g["err"] == 5                   # RL_ERR_TARGET_OUT_OF_RANGE
    assert g["logp"][3] == 0.0 and (g["dlogits_t"][3] == 0).all()
    assert np.isfinite(g["logp"]).all()
    good = [r for r in range(w.n_rows) if r != 3]  # the other rows as in a clean call
    g2 = P.run_gpu(wl.make(rec, DEV))
    np.testing.assert_array_equal(g["logp"][good], g2["logp"][good])
    w = wl.make(rec, DEV)
    w.group_id[1] = 9
    assert P.run_gpu(w)["err"] == 6        # RL_ERR_GROUP_OUT_OF_RANGE
    w = wl.make(rec, DEV)
    w.cu_seqlens[2] = 3                    # not non-decreasing
    assert P.run_gpu(w)["err"] == 7        # RL_ERR_BAD_SEQLENS
    w = wl.make(rec, DEV)
    assert P.run_gpu(w)["err"] == 0        # the error word resets on the next call


@pytest.mark.parametrize("kind,topk", [(k, t) for k in ("cluster", "stream", "stream2", "stream4")
                                       for t in (0, 4)] + [("streamC2", 0), ("streamC8", 0)])
def test_a_wait_that_runs_out_is_reported(ov, kind, topk):
    """Failure detection on the GPU without a fault. The test hook
    stall_first_wait_ns makes the first wait for logits of every CTA of the
    sweep wait on a barrier that nothing completes, bounded by 1 ms; each CTA
    then gives up as it would on a copy that never arrives (it stops issuing
    copies, waits for the ones in flight and writes zeros for its rows). The
    call reports RL_ERR_DEVICE_TIMEOUT with every output finite and zero, and
    the next call without the hook is RL_OK and matches the oracle. The
    streaming kernel runs with one CTA per SM, or two or four ("stream2",
    "stream4"), or with a cluster of two or eight CTAs per row ("streamC2",
    "streamC8": the CTAs still exchange their row sums, which carry the
    give-up mark)."""
    if kind.startswith("streamC"):
        ov(sweep_kernel="stream", stream_cluster=int(kind[-1]))
    else:
        ov(sweep_kernel=kind.rstrip("24"))
        if kind[-1] in "24":
            ov(stream_ctas_per_sm=int(kind[-1]))
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=64, vocab=100000,
                    rho_noise=0.3, ref_noise=0.2, topk=topk, topk_noise=0.4)
    w = wl.make(rec, DEV)
    params = dict(w.params, opd_coef=0.5, opd_topk=topk) if topk else None
    for mode in ("fused", "split"):
        ov(stall_first_wait_ns=1_000_000)
        g = P.run_gpu(w, mode=mode, params=params)
        assert g["err"] == 8, ml.status_string(g["err"])  # RL_ERR_DEVICE_TIMEOUT
        assert np.all(g["logp"] == 0) and np.all(g["H"] == 0)
        assert torch.equal(g["dlogits_t"], torch.zeros_like(g["dlogits_t"]))
        st = g["stats"]
        assert st["loss"] == 0.0 and st["n_tokens"] == int(w.loss_mask.sum())
        ov(stall_first_wait_ns=-1)
        _full_check(w, mode=mode, params=params)


@pytest.mark.parametrize("kind,cluster", [("cluster", 0), ("cluster", 4), ("stream", 0)])
def test_topk_ids_out_of_range_are_reported(ov, kind, cluster):
    """A top-K OPD candidate id outside [0, vocab) zeros its row (as a bad
    target does) and the call reports RL_ERR_TOPK_ID_OUT_OF_RANGE; the other
    rows match the oracle."""
    ov(sweep_kernel=kind)
    if cluster:
        ov(cluster_size=cluster)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=4, traj_len=8, vocab=60000,
                    rho_noise=0.3, topk=8, topk_noise=0.4)
    w = wl.make(rec, DEV)
    params = dict(w.params, opd_coef=0.5, opd_topk=8)
    bad = [3, 17]
    w.topk_ids[3, 5] = w.vocab   # one past the end
    w.topk_ids[17, 0] = -1
    for mode in ("fused", "split"):
        g = P.run_gpu(w, mode=mode, params=params)
        assert g["err"] == 9, ml.status_string(g["err"])  # RL_ERR_TOPK_ID_OUT_OF_RANGE
        assert all(g["logp"][r] == 0 and g["H"][r] == 0 for r in bad)
        dl = g["dlogits_t"].float()
        assert all((dl[r] == 0).all() for r in bad)
        # the other rows against the oracle on the same call with valid ids
        # in place of the bad ones (a row's outputs do not depend on another
        # row's candidates)
        ids = P.np_(w.topk_ids).copy()
        ids[3, 5], ids[17, 0] = 0, 1
        o = oracle.rl_loss(P.host_logits(w), P.np_(w.targets), P.np_(w.rollout_logprobs),
                           P.np_(w.ref_logprobs), P.np_(w.rewards), P.np_(w.group_id),
                           P.np_(w.cu_seqlens), w.n_groups, P.np_(w.loss_mask),
                           P.oracle_params(params), topk_ids=ids,
                           topk_teacher=P.np_(w.topk_teacher))
        good = np.setdiff1d(np.arange(w.n_rows), bad)
        tol = P.logp_tol(w)
        np.testing.assert_allclose(g["logp"][good], o["logp"][good], atol=tol, rtol=0)
        np.testing.assert_allclose(g["H"][good], o["H"][good], atol=tol, rtol=0)
        P.assert_dlogits_close(dl[good][:, :w.vocab].cpu().numpy(), o["dlogits"][good])


def test_bitwise_reproducible_and_fwd_matches_fused():
    w = wl.make(SHRUNK["glm_noisy"], DEV)
    a = P.run_gpu(w)
    b = P.run_gpu(w)
    c = P.run_gpu(w, mode="fwd")
    assert torch.equal(a["dlogits_t"], b["dlogits_t"])
    np.testing.assert_array_equal(a["logp"], b["logp"])
    assert a["stats"] == b["stats"]
    np.testing.assert_array_equal(a["logp"], c["logp"])
    np.testing.assert_array_equal(a["H"], c["H"])
    assert a["stats"] == c["stats"]


# forward-only plans: clusters (16 KB rows), streaming with four, two and one
# CTAs per SM (60, 137 and 215 KB rows)
@pytest.mark.parametrize("vocab", [8000, 30000, 70000, 110000])
def test_batch_invariance_of_row_outputs(vocab):
    """A row's log-prob and entropy do not depend on where it sits or on how
    many other rows share the call."""
    rec = wl.shrink(wl.RECIPES["qwen"], n_prompts=2, group_size=4, traj_len=32, vocab=vocab)
    w = wl.make(rec, DEV)
    full = P.run_gpu(w, mode="fwd")
    perm = torch.randperm(w.n_rows, generator=torch.Generator().manual_seed(0)).to(DEV)
    sub = perm[:37]
    w2 = wl.Workload(rec, w.logits[sub].contiguous(), w.targets[sub].contiguous(),
                     w.rollout_logprobs[sub].contiguous(), None, None, None,
                     torch.tensor([0.0], device=DEV), torch.zeros(1, dtype=torch.int32, device=DEV),
                     torch.tensor([0, 37], dtype=torch.int32, device=DEV),
                     w.loss_mask[sub].contiguous(), 1, dict(w.params))
    part = P.run_gpu(w2, mode="fwd")
    idx = sub.cpu().numpy()
    np.testing.assert_array_equal(part["logp"], full["logp"][idx])
    np.testing.assert_array_equal(part["H"], full["H"][idx])


def test_grad_loss_device_scalar():
    w = wl.make(SHRUNK["tiny"], DEV)
    a = P.run_gpu(w, grad_loss=3.0, dl_dtype=torch.float32)
    buf = api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, DEV, vocab=w.vocab,
                    dlogits_dtype=torch.float32)
    api.fwd_bwd(w, buf, grad_loss=1.5, grad_loss_device=torch.tensor([2.0], device=DEV))
    torch.cuda.synchronize()
    assert torch.equal(buf.dlogits, a["dlogits_t"])


# ------------------------------------------------- hand-worked calls on the GPU

def _golden_case(name):
    import json
    import math
    with open(os.path.join(os.path.dirname(os.path.abspath(__file__)), "golden",
                           "hand_cases.json")) as f:
        c = {c["name"]: c for c in json.load(f)["cases"]}[name]

    def ev(x):
        return float(eval(x, {"math": math})) if isinstance(x, str) else float(x)
    return c, ev


@pytest.mark.parametrize("name", ["full_call_kl_opd", "full_call_topk_opd",
                                  "full_call_gspo_two_row_trajectories"])
def test_hand_worked_calls(name):
    """The whole calls worked by hand from the definitions (tests/golden),
    through the C ABI with fp32 logits, against the hand-derived loss and
    dLogits (not against the oracle)."""
    c, ev = _golden_case(name)
    import dataclasses
    rec = dataclasses.replace(wl.RECIPES["tiny"], vocab=2, dtype="f32")
    f32 = dict(dtype=torch.float32, device=DEV)
    i32 = dict(dtype=torch.int32, device=DEV)
    z = torch.tensor([[ev(v) for v in row] for row in c["z"]], **f32)
    rho = torch.tensor([ev(v) for v in c["rho"]], **f32)
    q = rho + torch.tensor([ev(v) for v in c["delta"]], **f32) if "delta" in c else None
    teacher = torch.tensor([ev(v) for v in c["teacher"]], **f32) if "teacher" in c else None
    ids = torch.tensor(c["topk_ids"], **i32) if "topk_ids" in c else None
    tt = (torch.tensor([[ev(v) for v in row] for row in c["topk_teacher"]], **f32)
          if "topk_teacher" in c else None)
    w = wl.Workload(rec, z, torch.tensor(c["y"], **i32), rho, q, None, teacher,
                    torch.tensor([ev(v) for v in c["w"]], **f32), torch.tensor(c["gid"], **i32),
                    torch.tensor(c["cu"], **i32),
                    torch.tensor(c["mask"], dtype=torch.uint8, device=DEV), c["n_groups"],
                    dict(c["params"]), ids, tt)
    g = P.run_gpu(w)
    assert g["err"] == 0, ml.status_string(g["err"])
    assert abs(g["stats"]["loss"] - ev(c["expect"]["loss"])) <= 2e-6
    if "dlogits" in c["expect"]:
        want = np.array([[ev(v) for v in row] for row in c["expect"]["dlogits"]])
        np.testing.assert_allclose(g["dlogits_t"].cpu().numpy(), want, rtol=1e-4, atol=1e-6)


# ---------------------------------------------------------------- full sizes

FULL = ["glm", "qwen", "agentic", "fp32"]


@pytest.fixture(scope="module")
def oracle_pool():
    """The float64 oracle's worker processes (spawned), one per host core."""
    import bench
    pool = bench.OraclePool()
    yield pool
    pool.close()


@pytest.mark.slow
@pytest.mark.parametrize("name", FULL)
def test_full_size_every_row(name, oracle_pool):
    """Full-size workloads (the headline one first: 65,536 x 154,880 bf16) in
    the launch configuration the benchmark times, EVERY row against the
    float64 oracle: the log-prob and entropy of every row, every dLogit
    (compared entry by entry in the oracle's worker processes at 1e-2
    relative / 1e-5 absolute), advantages, group sizes and N, the clip counts
    (exactly, under the oracle's rule on the GPU's log-probs; within the
    guard band against the oracle's own), the metrics, and the scalar loss
    to 1e-4 relative of the oracle's."""
    import bench
    w = wl.make(wl.RECIPES[name], DEV)
    g = P.run_gpu(w)
    assert g["err"] == 0, ml.status_string(g["err"])
    o_rows = bench.oracle_rows(w, oracle_pool, dlogits=g["dlogits_t"])
    assert o_rows["n_bad"] == 0, (f"{o_rows['n_bad']} dLogits outside the bound; worst "
                                  f"(row, col, gpu, oracle) = {o_rows['worst_at']}")
    p = P.oracle_params(w.params)
    mask = P.np_(w.loss_mask).astype(bool)
    A_traj, A_row, n_g = oracle.estimator_advantages(P.np_(w.rewards), P.np_(w.group_id),
                                                     w.n_groups, P.np_(w.cu_seqlens), mask, p)
    obj = oracle.token_objective(o_rows["logp"], P.np_(w.rollout_logprobs), P.np_(w.ref_logprobs),
                                 A_row, o_rows["H"], p, old=P.np_(w.old_logprobs))
    stats = oracle.loss_stats(obj, o_rows["logp"], P.np_(w.rollout_logprobs), o_rows["H"], mask)
    o = dict(obj, logp=o_rows["logp"], H=o_rows["H"], lse=o_rows["lse"], A_traj=A_traj,
             A_row=A_row, group_sizes=n_g, N=int(mask.sum()), stats=stats)
    P.compare_forward(w, g, o)
    del g, w, o_rows
    torch.cuda.empty_cache()


@pytest.mark.parametrize("kind", ["cluster", "stream"])
def test_chunked_call_equals_whole_call(ov, kind):
    """BEGIN, ROWS over blocks of rows (ragged last block), END give the same
    bits as one rl_loss_fwd_bwd; a forward-only chunk leaves dLogits alone."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=40, vocab=20480,
                    rho_noise=0.3, ref_noise=0.2, topk=4)
    w = wl.make(rec, DEV)
    params = P.gpu_params(w, dict(w.params, opd_coef=0.3, opd_topk=4))
    whole = P.run_gpu(w, params=params)
    for chunk in (7, 100, w.n_rows):
        buf = api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, DEV, vocab=w.vocab,
                        dlogits_dtype=w.logits.dtype, fill_nan=True)
        api.fwd_bwd_chunked(w, buf, chunk, params=params)
        torch.cuda.synchronize()
        assert ml.rl_loss_check_device_error(buf.workspace) == 0
        assert torch.equal(buf.dlogits, whole["dlogits_t"])
        np.testing.assert_array_equal(buf.token_logprobs.cpu().numpy(), whole["logp"])
        np.testing.assert_array_equal(buf.entropy.cpu().numpy(), whole["H"])
        assert buf.read_stats() == whole["stats"]
    buf = api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, DEV, vocab=w.vocab,
                    dlogits_dtype=w.logits.dtype, fill_nan=True)
    api.fwd_bwd_chunked(w, buf, 64, params=params, forward_only=True)
    torch.cuda.synchronize()
    assert torch.isnan(buf.dlogits.float()).all()
    np.testing.assert_array_equal(buf.token_logprobs.cpu().numpy(), whole["logp"])
    assert buf.read_stats() == whole["stats"]


def test_pipelined_host_call_matches_device_call():
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=64, vocab=40000,
                    rho_noise=0.2, ref_noise=0.1)
    w = wl.make(rec, DEV)
    whole = P.run_gpu(w)
    host = w.to("cpu")
    for k in ("logits", "targets", "rollout_logprobs", "ref_logprobs", "rewards", "group_id",
              "cu_seqlens", "loss_mask"):
        setattr(host, k, getattr(host, k).pin_memory())
    for depth, on_device in ((2, False), (3, False), (2, True)):
        call = api.PipelinedHostCall(host, DEV, chunk_rows=100, depth=depth,
                                     dlogits_on_device=on_device)
        assert call.out["dlogits"].is_cuda == on_device
        for _ in range(2):
            out = call()
            torch.cuda.synchronize()
            assert torch.equal(out["dlogits"].cpu(), whole["dlogits_t"].cpu())
            np.testing.assert_array_equal(out["token_logprobs"].numpy(), whole["logp"])
            assert ml.parse_stats(out["stats"].numpy().tobytes()) == whole["stats"]


# ---------------------------------------------------------- row-sharded calls

def _shard_of(w, r0, r1):
    """Rows [r0, r1) of a workload as one shard's workload (the per-trajectory
    inputs stay those of the whole call)."""
    sl = slice(r0, r1)

    def rows(t):
        return None if t is None else t[sl].contiguous()
    return wl.Workload(w.recipe, rows(w.logits), rows(w.targets), rows(w.rollout_logprobs),
                       rows(w.ref_logprobs), rows(w.old_logprobs), rows(w.teacher_logprobs),
                       w.rewards, w.group_id, w.cu_seqlens, rows(w.loss_mask), w.n_groups,
                       dict(w.params), rows(w.topk_ids), rows(w.topk_teacher))


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [dict(), dict(estimator="reinforcepp", kl_coef=0.05),
                                    dict(opd_coef=0.3, opd_topk=4, entropy_coef=0.01)],
                         ids=["grpo", "rpp", "topk"])
def test_row_sharded_call_equals_whole_call(ov, kind, params):
    """One call's rows split over shards (2 and 3 shards, trajectories cut at
    the boundaries, and an empty shard), driven phase by phase with the
    exchanges done by sums and maxima over the shards' small arrays: every
    shard's log-probs, entropies and dLogits are those of the whole call bit
    for bit, the advantages, group sizes and counts equal, the loss within
    1e-4 relative (its partial sums are added in another order)."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=40, vocab=20480,
                    rho_noise=0.3, ref_noise=0.2, topk=4, mask="prefix_u0_half")
    w = wl.make(rec, DEV)
    p = P.gpu_params(w, dict(w.params, **params))
    whole = P.run_gpu(w, params=p)
    R, n_traj = w.n_rows, int(w.rewards.shape[0])
    for cuts in ([0, 137, R], [0, 50, 50, 221, R]):
        shards = []
        for r0, r1 in zip(cuts[:-1], cuts[1:]):
            ws = _shard_of(w, r0, r1)
            buf = api.alloc(r1 - r0, n_traj, w.n_groups, DEV, vocab=w.vocab,
                            dlogits_dtype=w.logits.dtype, fill_nan=True)
            # (the shard's own top-K candidates: params without the whole
            # call's arrays, so that api.Shard attaches the shard's rows)
            shards.append(api.Shard(ws, r0, R, buf, params=dict(w.params, **params)))
        api.sharded_fwd_bwd_local(shards)
        torch.cuda.synchronize()
        for sh, (r0, r1) in zip(shards, zip(cuts[:-1], cuts[1:])):
            b = sh.buf
            assert ml.rl_loss_check_device_error(b.workspace) == 0
            assert torch.equal(b.dlogits, whole["dlogits_t"][r0:r1])
            np.testing.assert_array_equal(b.token_logprobs.cpu().numpy(), whole["logp"][r0:r1])
            np.testing.assert_array_equal(b.entropy.cpu().numpy(), whole["H"][r0:r1])
            np.testing.assert_array_equal(b.advantages.cpu().numpy(), whole["A"])
            np.testing.assert_array_equal(b.group_sizes.cpu().numpy(), whole["group_sizes"])
            st, ref = b.read_stats(), whole["stats"]
            for k in ("n_tokens", "n_clip_hi", "n_clip_lo", "n_dual_clip", "n_corr_clip",
                      "ratio_min", "ratio_max"):
                assert st[k] == ref[k], k
            P.assert_loss_close(st["loss"], ref["loss"], what="sharded loss")
            for k in ("pg_loss_mean", "kl_mean", "entropy_mean", "ratio_mean"):
                assert abs(st[k] - ref[k]) <= 1e-4 * max(abs(ref[k]), 1e-3), k


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [dict(estimator="gspo"),
                                    dict(estimator="gspo", correction="tis", corr_lo=0.0,
                                         corr_hi=1.5, entropy_coef=0.01, kl_coef=0.05)],
                         ids=["gspo", "gspo_tis_ent_kl"])
def test_row_sharded_gspo_matches_the_oracle(ov, kind, params):
    """GSPO over row shards (trajectories cut at the boundaries, an empty
    shard): the forward sweep, the exchange of per-trajectory sums, then each
    shard's sequence terms and dLogits. The assembled outputs match the
    float64 oracle at the stated tolerances, and the shards' log-probs are
    the whole call's bit for bit (the sequence sums only change the
    gradient's scalars)."""
    ov(sweep_kernel=kind)
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=2, group_size=4, traj_len=40, vocab=20480,
                    rho_noise=0.3, ref_noise=0.2, mask="prefix_u0_half")
    w = wl.make(rec, DEV)
    p = dict(w.params, **params)
    whole = P.run_gpu(w, params=p)
    R, n_traj = w.n_rows, int(w.rewards.shape[0])
    for cuts in ([0, 137, R], [0, 50, 50, 221, R]):
        shards = []
        for r0, r1 in zip(cuts[:-1], cuts[1:]):
            buf = api.alloc(r1 - r0, n_traj, w.n_groups, DEV, vocab=w.vocab,
                            dlogits_dtype=w.logits.dtype, fill_nan=True)
            shards.append(api.Shard(_shard_of(w, r0, r1), r0, R, buf, params=p))
        api.sharded_fwd_bwd_local(shards)
        torch.cuda.synchronize()
        dl = torch.cat([sh.buf.dlogits for sh in shards])
        for sh in shards:
            assert ml.rl_loss_check_device_error(sh.buf.workspace) == 0
        g = dict(logp=np.concatenate([P.np_(sh.buf.token_logprobs) for sh in shards]),
                 H=np.concatenate([P.np_(sh.buf.entropy) for sh in shards]),
                 A=P.np_(shards[0].buf.advantages), group_sizes=P.np_(shards[0].buf.group_sizes),
                 stats=shards[0].buf.read_stats())
        np.testing.assert_array_equal(g["logp"], whole["logp"])
        o = P.run_oracle(w, params=p)
        P.compare_forward(w, g, o, params=p)
        P.assert_dlogits_close(dl.float().cpu().numpy(), o["dlogits"])
