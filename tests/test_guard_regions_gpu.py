"""Guard regions around every buffer a call touches: a stand-in for a memory
checker, which these tests do not run.

Each input and output of a call is placed inside a larger device allocation,
with GUARD bytes before and after it:
- input guards hold the bytes 00 00 c0 7f repeated: a quiet NaN read as fp32
  (and every second bf16 a NaN), 2,143,289,344 read as int32 (out of range
  as a target, group id, row offset or top-K id). A read outside an input
  that reaches the arithmetic therefore shows up in the outputs or as a
  device error, and the call is compared bit for bit with the same call on
  unguarded buffers (and the same launch plan);
- output guards hold a byte pattern that must be intact after the call;
- every input is compared with a copy taken before the call (the library
  writes none of them).

The cases cover every sweep kernel and launch plan the library picks (the
streaming kernel with one, two and four CTAs per SM and with a cluster of two
or four CTAs per row, the fp32 two-chunk plan, clusters of 1, 2, 4 and 8
CTAs), top-K OPD in both kernels, the split
forward / backward pair, GSPO, the chunked row call, ragged and padded rows,
and the row- and vocabulary-sharded calls with their exchange buffers."""

import dataclasses

import pytest
import torch

import _parity as P
from paper_2609_08368_gb300 import api, workloads as wl
from paper_2609_08368_gb300 import milesloss as ml

pytestmark = pytest.mark.gpu

DEV = "cuda"
GUARD = 8192
IN_FILL = torch.tensor([0x00, 0x00, 0xC0, 0x7F], dtype=torch.uint8)
OUT_FILL = torch.tensor([0xA5, 0x5A, 0xC3, 0x3C], dtype=torch.uint8)


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


class Arena:
    """Guarded copies of tensors and the checks of their guards."""

    def __init__(self):
        self.items = []

    def put(self, t, fill, name):
        if t is None:
            return None
        assert t.is_contiguous()
        n = t.numel() * t.element_size()
        raw = torch.empty(GUARD + n + GUARD, dtype=torch.uint8, device=t.device)
        pat = fill.to(t.device).repeat(GUARD // fill.numel())
        raw[:GUARD] = pat
        raw[GUARD + n:] = pat
        inner = raw[GUARD:GUARD + n].view(t.dtype).view(t.shape)
        inner.copy_(t)
        self.items.append((name, raw, n, pat))
        return inner

    def check(self):
        torch.cuda.synchronize()
        for name, raw, n, pat in self.items:
            assert torch.equal(raw[:GUARD], pat), f"{name}: a byte before the buffer changed"
            assert torch.equal(raw[GUARD + n:], pat), f"{name}: a byte after the buffer changed"


INPUTS = ("logits", "targets", "rollout_logprobs", "ref_logprobs", "old_logprobs",
          "teacher_logprobs", "rewards", "group_id", "cu_seqlens", "loss_mask", "topk_ids",
          "topk_teacher")
OUTPUTS = ("token_logprobs", "entropy", "advantages", "group_sizes", "stats", "workspace",
           "dlogits")


def guard_workload(w, arena):
    g = {k: arena.put(getattr(w, k), IN_FILL, k) for k in INPUTS}
    return dataclasses.replace(w, **g)


def guard_buffers(buf, arena, tag=""):
    return api.Buffers(*(arena.put(getattr(buf, k), OUT_FILL, tag + k) for k in OUTPUTS))


def snapshot(w):
    return {k: getattr(w, k).clone() for k in INPUTS if getattr(w, k) is not None}


def bits(t):
    """A tensor's bytes (NaN-safe bitwise comparison)."""
    return t.contiguous().view(torch.uint8)


def assert_inputs_unchanged(w, snap):
    for k, before in snap.items():
        assert torch.equal(bits(getattr(w, k)), bits(before)), f"input {k} was written"


def assert_same_outputs(a, b):
    for k in ("token_logprobs", "entropy", "advantages", "group_sizes", "stats", "dlogits"):
        x, y = getattr(a, k), getattr(b, k)
        if x is None:
            assert y is None
            continue
        assert torch.equal(bits(x), bits(y)), f"{k} differs from the unguarded call"


def _alloc(w, mode, dl_dtype=None, ld_out=None):
    return api.alloc(w.n_rows, int(w.rewards.shape[0]), w.n_groups, DEV, vocab=w.vocab,
                     dlogits_dtype=None if mode == "fwd" else (dl_dtype or w.logits.dtype),
                     ld_out=ld_out, fill_nan=True)


def _drive(mode, w, buf, params):
    if mode == "fused":
        api.fwd_bwd(w, buf, params=params)
    elif mode == "split":
        api.fwd(w, buf, params=params)
        api.bwd(w, buf, params=params)
    elif mode == "fwd":
        api.fwd(w, buf, params=params)
    elif mode == "chunked":
        api.fwd_bwd_chunked(w, buf, 100, params=params)
    else:
        raise ValueError(mode)


def _rec(name, **kw):
    return wl.shrink(wl.RECIPES[name], **kw)


LONG = dict(n_prompts=1, group_size=4, traj_len=80)  # 320 rows: more rows than SMs
TOPK = dict(opd_coef=0.3, opd_topk=4)
# id: (recipe, launch overrides, mode, extra params, make() ld, dLogits ld)
CASES = {
    "stream_one_cta": (_rec("glm", **LONG), {}, "fused", {}, None, None),
    "stream_one_cta_topk": (_rec("glm", topk=4, **LONG), {}, "fused", TOPK, None, None),
    "stream_one_cta_split": (_rec("glm", **LONG), {}, "split", {}, None, None),
    "stream_one_cta_fwd": (_rec("glm", **LONG), {}, "fwd", {}, None, None),
    "stream_one_cta_gspo": (_rec("glm", **LONG), {}, "fused", dict(estimator="gspo"), None,
                            None),
    "stream_one_cta_padded": (_rec("glm", vocab=100000, **LONG), {}, "fused", {}, 100008,
                              100016),
    "stream_two_ctas": (_rec("glm", n_prompts=2, group_size=4, traj_len=80, vocab=32768), {},
                        "fused", {}, None, None),
    "stream_two_ctas_topk": (_rec("glm", n_prompts=2, group_size=4, traj_len=80, vocab=32768,
                                  topk=4), {}, "fused", TOPK, None, None),
    "stream_four_ctas": (_rec("glm", n_prompts=4, group_size=4, traj_len=80, vocab=16384), {},
                         "fused", {}, None, None),
    "stream_four_ctas_fwd": (_rec("glm", n_prompts=4, group_size=4, traj_len=80, vocab=16384),
                             {}, "fwd", {}, None, None),
    "fp32_two_ctas": (_rec("fp32", n_prompts=10, traj_len=8), {}, "fused", {}, None, None),
    "fp32_equal_halves": (_rec("fp32", n_prompts=10, traj_len=8, vocab=40000), {}, "fused", {},
                          None, None),
    "clusters_by_plan": (_rec("glm", n_prompts=2, group_size=4, traj_len=80, vocab=49152), {},
                         "fused", {}, None, None),
    "clusters_topk": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480, topk=4),
                      dict(sweep_kernel=0), "fused", TOPK, None, None),
    "clusters_split": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480),
                       dict(sweep_kernel=0), "split", {}, None, None),
    "cluster_1": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480),
                  dict(sweep_kernel=0, cluster_size=1), "fused", {}, None, None),
    "cluster_2": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480),
                  dict(sweep_kernel=0, cluster_size=2), "fused", {}, None, None),
    "cluster_4": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480),
                  dict(sweep_kernel=0, cluster_size=4), "fused", {}, None, None),
    "cluster_8": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480),
                  dict(sweep_kernel=0, cluster_size=8), "fused", {}, None, None),
    "stream_cluster_of_two": (_rec("glm", vocab=262144, n_prompts=1, group_size=4, traj_len=40),
                              {}, "fused", {}, None, None),
    "stream_cluster_of_four_ragged": (_rec("glm", vocab=100003, n_prompts=1, group_size=4,
                                           traj_len=40),
                                      dict(sweep_kernel=1, stream_cluster=4), "fused", {},
                                      100008, 100016),
    "ragged_vocab": (_rec("tiny", n_prompts=1, group_size=3, traj_len=50, vocab=12345), {},
                     "fused", {}, None, None),
    "misaligned_rows": (_rec("tiny", n_prompts=1, group_size=2, traj_len=24, vocab=1000), {},
                        "fused", {}, 1003, None),
    "chunked_rows": (_rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480), {},
                     "chunked", {}, None, None),
}


@pytest.mark.parametrize("case", list(CASES))
def test_call_stays_inside_its_buffers(ov, case):
    rec, over, mode, extra, ld, ld_out = CASES[case]
    if over:
        ov(**over)
    w = wl.make(rec, DEV, ld=ld)
    params = P.gpu_params(w, dict(w.params, **extra))
    ref = _alloc(w, mode, ld_out=ld_out)
    _drive(mode, w, ref, params)
    torch.cuda.synchronize()
    assert ml.rl_loss_check_device_error(ref.workspace) == 0

    arena = Arena()
    gw = guard_workload(w, arena)
    gbuf = guard_buffers(_alloc(w, mode, ld_out=ld_out), arena)
    snap = snapshot(gw)
    _drive(mode, gw, gbuf, P.gpu_params(gw, dict(w.params, **extra)))
    arena.check()
    assert ml.rl_loss_check_device_error(gbuf.workspace) == 0
    assert_inputs_unchanged(gw, snap)
    assert_same_outputs(gbuf, ref)


def _row_shard_run(w, cuts, params, arena=None):
    n_traj = int(w.rewards.shape[0])
    shards = []
    for r0, r1 in zip(cuts[:-1], cuts[1:]):
        sw = dataclasses.replace(
            w, **{k: (getattr(w, k)[r0:r1].contiguous() if getattr(w, k) is not None else None)
                  for k in ("logits", "targets", "rollout_logprobs", "ref_logprobs",
                            "old_logprobs", "teacher_logprobs", "loss_mask", "topk_ids",
                            "topk_teacher")})
        buf = api.alloc(r1 - r0, n_traj, w.n_groups, DEV, vocab=w.vocab,
                        dlogits_dtype=w.logits.dtype, fill_nan=True)
        if arena is not None:
            sw = guard_workload(sw, arena)
            buf = guard_buffers(buf, arena, f"rows {r0}: ")
        s = api.Shard(sw, r0, w.n_rows, buf, params=P.gpu_params(sw, params))
        if arena is not None:
            for k in ("counts", "traj_sums", "partials"):
                setattr(s, k, arena.put(getattr(s, k), OUT_FILL, f"rows {r0}: {k}"))
        shards.append(s)
    api.sharded_fwd_bwd_local(shards)
    torch.cuda.synchronize()
    return shards


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [dict(), dict(estimator="gspo")], ids=["grpo", "gspo"])
def test_row_shards_stay_inside_their_buffers(ov, kind, params):
    ov(sweep_kernel=0 if kind == "cluster" else 1)
    rec = _rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480)
    w = wl.make(rec, DEV)
    p = dict(w.params, **params)
    cuts = [0, 137, w.n_rows]
    ref = _row_shard_run(w, cuts, p)
    arena = Arena()
    got = _row_shard_run(w, cuts, p, arena)
    arena.check()
    for a, b in zip(got, ref):
        assert ml.rl_loss_check_device_error(a.buf.workspace) == 0
        assert_same_outputs(a.buf, b.buf)
        assert torch.equal(bits(a.partials), bits(b.partials))


def _vocab_shard_run(w, col_starts, params, arena=None):
    """Two column shards of one call, both run here; with an arena, every
    output and exchange buffer of each shard is guarded (the workload's
    inputs are guarded by the caller)."""
    R, n_traj = w.n_rows, int(w.rewards.shape[0])
    row = []
    for k in range(len(col_starts) - 1):
        c0, c1 = col_starts[k], col_starts[k + 1]
        sw = dataclasses.replace(w, logits=w.logits[:, c0:c1])
        buf = api.alloc(R, n_traj, w.n_groups, DEV, vocab=c1 - c0,
                        dlogits_dtype=w.logits.dtype, fill_nan=True)
        if arena is not None:
            buf = guard_buffers(buf, arena, f"columns {c0}: ")
        s = api.VocabShard(sw, k, col_starts, buf, params=P.gpu_params(w, params))
        if arena is not None:
            for f in ("counts", "traj_sums", "row_partials", "row_partials_all", "partials"):
                setattr(s, f, arena.put(getattr(s, f), OUT_FILL, f"columns {c0}: {f}"))
        row.append(s)
    api.vocab_sharded_fwd_bwd_local([row])
    torch.cuda.synchronize()
    return row


@pytest.mark.parametrize("kind", ["cluster", "stream"])
@pytest.mark.parametrize("params", [dict(), dict(opd_coef=0.3, opd_topk=4)],
                         ids=["grpo", "topk"])
def test_vocab_shards_stay_inside_their_buffers(ov, kind, params):
    ov(sweep_kernel=0 if kind == "cluster" else 1)
    rec = _rec("glm", n_prompts=2, group_size=4, traj_len=40, vocab=20480, topk=4)
    w = wl.make(rec, DEV)
    p = dict(w.params, **params)
    col_starts = [0, 10240, 20480]
    ref = _vocab_shard_run(w, col_starts, p)
    arena = Arena()
    gw = guard_workload(w, arena)
    snap = snapshot(gw)
    got = _vocab_shard_run(gw, col_starts, p, arena)
    arena.check()
    for a, b in zip(got, ref):
        assert ml.rl_loss_check_device_error(a.buf.workspace) == 0
        assert_same_outputs(a.buf, b.buf)
        assert torch.equal(bits(a.row_partials_all), bits(b.row_partials_all))
    assert_inputs_unchanged(gw, snap)
