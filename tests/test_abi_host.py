"""Host-side checks of the C ABI that need no GPU: the library builds for
sm_103a and loads, exports every entry point include/milesloss.h declares,
sizes workspaces, names its status codes, and rejects every invalid
argument before enqueuing anything."""

import ctypes
import os
import re

import pytest

from paper_2609_08368_gb300 import milesloss as ml

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
HEADER = os.path.join(ROOT, "include", "milesloss.h")

RL_ERR_INVALID_ARG = 1
RL_ERR_WORKSPACE_TOO_SMALL = 3


@pytest.fixture(scope="module")
def lib():
    return ml.load()


def declared_functions():
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(rl_[a-z_0-9]+)\s*\(", text)))


def test_header_declares_the_boundary():
    names = declared_functions()
    for want in ("rl_loss_fwd", "rl_loss_bwd", "rl_loss_fwd_bwd", "rl_loss_workspace_size",
                 "rl_loss_check_device_error", "rl_status_string"):
        assert want in names


def test_every_declared_symbol_is_exported(lib):
    for name in declared_functions():
        assert hasattr(lib, name), name


def test_abi_version_and_status_strings(lib):
    assert lib.rl_loss_abi_version() == 131
    seen = set()
    for code in range(0, 10):
        s = ml.status_string(code)
        assert s and s != "unknown status"
        seen.add(s)
    assert len(seen) == 10
    assert ml.status_string(99) == "unknown status"


def test_workspace_size(lib):
    a = ml.rl_loss_workspace_size(0, 0, 0)
    b = ml.rl_loss_workspace_size(65536, 64, 4)
    c = ml.rl_loss_workspace_size(131072, 64, 4)
    assert 0 < a < b < c
    assert b % 256 == 0
    # roughly 41 bytes of per-row state
    assert 40 * 65536 < b - a < 48 * 65536
    out = ctypes.c_size_t()
    assert lib.rl_loss_workspace_size(-1, 0, 0, ctypes.byref(out)) == RL_ERR_INVALID_ARG
    assert lib.rl_loss_workspace_size(1, 0, 0, None) == RL_ERR_INVALID_ARG


FAKE = 1 << 20  # never dereferenced: every case below fails validation first


class _Ptr:
    """A fake device pointer with the tensor method make_params reads."""

    def __init__(self, addr):
        self.addr = addr

    def data_ptr(self):
        return self.addr


def _fwd_bwd_args(**over):
    p = ml.make_params(**over.pop("params", {}))
    a = dict(logits=FAKE, dt=ml.RL_BF16, R=16, V=64, ld=64, targets=FAKE, rho=FAKE, q=None,
             old=None, teacher=None, rewards=FAKE, gid=FAKE, cu=FAKE, n_traj=2, n_groups=1,
             mask=FAKE, params=p, logp=FAKE, H=FAKE, adv=FAKE, gs=FAKE, stats=FAKE, g=1.0,
             gdev=None, dl=FAKE, dl_dt=ml.RL_BF16, ld_out=64, ws=FAKE * 2, ws_bytes=1 << 30)
    a.update(over)
    return a


def _call_fwd_bwd(lib, a):
    v = ctypes.c_void_p
    return lib.rl_loss_fwd_bwd(
        v(a["logits"]), a["dt"], a["R"], a["V"], a["ld"], v(a["targets"]), v(a["rho"]),
        v(a["q"]), v(a["old"]), v(a["teacher"]), v(a["rewards"]), v(a["gid"]), v(a["cu"]),
        a["n_traj"], a["n_groups"], v(a["mask"]), ctypes.byref(a["params"]), v(a["logp"]),
        v(a["H"]), v(a["adv"]), v(a["gs"]), v(a["stats"]), a["g"], v(a["gdev"]), v(a["dl"]),
        a["dl_dt"], a["ld_out"], v(a["ws"]), a["ws_bytes"], None)


INVALID = [
    dict(logits=None),
    dict(targets=None),
    dict(rho=None),
    dict(mask=None),
    dict(cu=None),
    dict(rewards=None),
    dict(gid=None),
    dict(dl=None),
    dict(dt=7),
    dict(dl_dt=5),
    dict(V=0),
    dict(R=-1),
    dict(ld=63),
    dict(ld_out=10),
    dict(n_traj=-1),
    dict(n_groups=0),
    dict(g=float("inf")),
    dict(ws=FAKE * 2 + 8),
    dict(ws=None),
    dict(params=dict(temperature=0.0)),
    dict(params=dict(temperature=float("nan"))),
    dict(params=dict(eps_lo=-0.1)),
    dict(params=dict(eps_hi=float("inf"))),
    dict(params=dict(dual_clip_c=1.0)),
    dict(params=dict(dual_clip_c=-2.0)),
    dict(params=dict(kl_coef=0.1)),                    # no ref log-probs
    dict(params=dict(kl_coef=-0.1), q=FAKE),
    dict(params=dict(entropy_coef=-1.0)),
    dict(params=dict(std_floor=0.0)),
    dict(params=dict(correction="tis", corr_lo=3.0, corr_hi=2.0), old=FAKE),
    dict(params=dict(correction=5), old=FAKE),
    dict(params=dict(opd_coef=0.5)),                   # no teacher log-probs
    dict(params=dict(opd_coef=float("nan")), teacher=FAKE),
    dict(params=dict(estimator=4)),
    dict(params=dict(estimator=-1)),
    dict(params=dict(opd_coef=0.5, opd_topk=4)),        # no candidate ids / teacher log-probs
    dict(params=dict(opd_coef=0.5, opd_topk=65), teacher=FAKE),
    dict(params=dict(opd_topk=-1)),
    dict(params=dict(opd_coef=0.5, opd_topk=4, opd_topk_ids=_Ptr(FAKE + 2),  # not 4-byte aligned
                     opd_topk_teacher=_Ptr(FAKE))),
    dict(params=dict(opd_coef=0.5, opd_topk=4, opd_topk_ids=_Ptr(FAKE),
                     opd_topk_teacher=_Ptr(FAKE + 1))),
]


@pytest.mark.parametrize("over", INVALID, ids=[str(i) for i in range(len(INVALID))])
def test_invalid_arguments_are_rejected_on_the_host(lib, over):
    params = over.pop("params", None)
    a = _fwd_bwd_args(**({"params": params} if params else {}), **over)
    assert _call_fwd_bwd(lib, a) == RL_ERR_INVALID_ARG


def test_workspace_too_small_is_rejected(lib):
    need = ml.rl_loss_workspace_size(16, 2, 1)
    a = _fwd_bwd_args(ws_bytes=need - 1)
    assert _call_fwd_bwd(lib, a) == RL_ERR_WORKSPACE_TOO_SMALL


def test_bwd_and_fwd_validate_too(lib):
    v = ctypes.c_void_p
    p = ml.make_params()
    # ld < vocab
    assert lib.rl_loss_bwd(v(FAKE), 0, 4, 64, 32, v(FAKE), v(FAKE), ctypes.byref(p), 1.0, None,
                           v(FAKE * 2), 1 << 30, v(FAKE), 0, 64, None) == RL_ERR_INVALID_ARG
    # workspace too small for the rows
    assert lib.rl_loss_bwd(v(FAKE), 0, 4096, 64, 64, v(FAKE), v(FAKE), ctypes.byref(p), 1.0, None,
                           v(FAKE * 2), 1024, v(FAKE), 0, 64, None) == RL_ERR_WORKSPACE_TOO_SMALL
    # fwd without rollout log-probs
    assert lib.rl_loss_fwd(v(FAKE), 0, 4, 64, 64, v(FAKE), None, None, None, None, v(FAKE),
                           v(FAKE), v(FAKE), 1, 1, v(FAKE), ctypes.byref(p), None, None, None,
                           None, None, v(FAKE * 2), 1 << 30, None) == RL_ERR_INVALID_ARG


def test_params_struct_layout_matches_header():
    assert ctypes.sizeof(ml.RlLossParams) == 80
    text = open(HEADER).read()
    body = text[text.index("typedef struct {", text.index("} rl_estimator;")):
                text.index("} rl_loss_params;")]
    body = re.sub(r"/\*.*?\*/", "", body, flags=re.S)
    fields = re.findall(r"(?:float|int32_t|const int32_t\s*\*|const float\s*\*)\s*"
                        r"([a-z_0-9]+(?:\s*,\s*[a-z_0-9]+)*)\s*;", body)
    names = [n.strip() for group in fields for n in group.split(",")]
    assert names == [f[0] for f in ml.RlLossParams._fields_]


def test_chunked_entry_validates(lib):
    v = ctypes.c_void_p
    p = ml.make_params()
    gspo = ml.make_params(estimator="gspo")

    def call(phase, r0, r1, params=p, logits=FAKE, dl=FAKE):
        return lib.rl_loss_fwd_bwd_rows(
            phase, r0, r1, v(logits), 0, 16, 64, 64, v(FAKE), v(FAKE), None, None, None,
            v(FAKE), v(FAKE), v(FAKE), 2, 1, v(FAKE), ctypes.byref(params), v(FAKE), v(FAKE),
            v(FAKE), v(FAKE), v(FAKE), 1.0, None, v(dl), 0, 64, v(FAKE * 2), 1 << 30, None)
    assert call(0, 0, 16) == RL_ERR_INVALID_ARG            # no phase
    assert call(8, 0, 16) == RL_ERR_INVALID_ARG            # unknown phase bit
    assert call(ml.RL_PHASE_ROWS, 4, 2) == RL_ERR_INVALID_ARG
    assert call(ml.RL_PHASE_ROWS, 0, 17) == RL_ERR_INVALID_ARG
    assert call(ml.RL_PHASE_ROWS, -1, 3) == RL_ERR_INVALID_ARG
    assert call(ml.RL_PHASE_ROWS, 0, 8, logits=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_PHASE_ALL, 0, 8, params=gspo) == 2     # GSPO: whole calls only
    assert call(ml.RL_PHASE_ROWS, 0, 16, params=gspo) == 2


def test_launch_overrides_struct_layout_matches_header():
    text = open(HEADER).read()
    body = text[text.index("typedef struct {", text.index("Launch-plan overrides")):
                text.index("} rl_launch_overrides;")]
    names = re.findall(r"(?:int32_t|int64_t)\s+([a-z_0-9]+)\s*;", body)
    assert names == [f[0] for f in ml.RlLaunchOverrides._fields_]
    # eleven int32 fields, four bytes of padding, one int64, one int32 and
    # four bytes of tail padding
    assert ctypes.sizeof(ml.RlLaunchOverrides) == 64


def test_every_launch_override_is_documented_in_the_header():
    text = open(HEADER).read()
    doc = text[text.index("Launch-plan overrides"):text.index("typedef struct {",
                                                             text.index("Launch-plan overrides"))]
    for name, _ in ml.RlLaunchOverrides._fields_:
        assert re.search(r"\*\s+" + name + r"\s", doc), name


def test_launch_overrides_are_validated_and_cleared(lib):
    o = ml.RlLaunchOverrides()
    assert lib.rl_launch_overrides_init(ctypes.byref(o)) == 0
    assert all(getattr(o, f) == -1 for f, _ in ml.RlLaunchOverrides._fields_)
    assert lib.rl_launch_overrides_init(None) == RL_ERR_INVALID_ARG
    try:
        ml.set_launch_overrides(sweep_kernel="stream", stream_slots=3, stream_hold=2)
        ml.set_launch_overrides(cluster_size=8, cluster_stages=4, stall_first_wait_ns=1000)
        ml.set_launch_overrides(sweep_kernel="stream", stream_ctas_per_sm=2)
        ml.set_launch_overrides(sweep_kernel="stream", stream_cluster=4)
        for bad in (dict(sweep_kernel=2), dict(cluster_size=16), dict(cluster_stages=0),
                    dict(stream_chunk_bytes=512), dict(stream_slots=17), dict(stream_hold=-2),
                    dict(stream_split_first=2), dict(stream_prefetch_bytes=24),
                    dict(stream_prefetch_bytes=1 << 21), dict(stall_first_wait_ns=-5),
                    dict(stall_first_wait_ns=10 ** 11), dict(stream_ctas_per_sm=0),
                    dict(stream_ctas_per_sm=3), dict(stream_cluster=0), dict(stream_cluster=3),
                    dict(stream_cluster=16)):
            with pytest.raises(ml.MilesLossError) as e:
                ml.set_launch_overrides(**bad)
            assert e.value.status == RL_ERR_INVALID_ARG
        with pytest.raises(TypeError):
            ml.set_launch_overrides(no_such_field=1)
        with ml.launch_overrides(sweep_kernel="cluster"):
            pass
    finally:
        ml.set_launch_overrides()
    assert lib.rl_set_launch_overrides(None) == 0


def test_library_reads_no_environment_variables():
    """Launch plans come from the library's own rules or the explicit
    overrides, never from the caller's environment."""
    csrc = os.path.join(ROOT, "paper_2609_08368_gb300", "csrc")
    for name in os.listdir(csrc):
        text = open(os.path.join(csrc, name)).read()
        assert "getenv" not in text, name


def test_sharded_entry_validates(lib):
    v = ctypes.c_void_p
    p = ml.make_params()
    gspo = ml.make_params(estimator="gspo")

    def call(phase, r0=0, total=16, R=16, params=p, counts=FAKE, partials=FAKE, stats=FAKE,
             sums=FAKE):
        return lib.rl_loss_shard_fwd_bwd(
            phase, r0, total, v(FAKE), 0, R, 64, 64, v(FAKE), v(FAKE), None, None, None,
            v(FAKE), v(FAKE), v(FAKE), 2, 1, v(FAKE), ctypes.byref(params), v(FAKE), v(FAKE),
            v(FAKE), v(FAKE), v(counts), v(sums), v(partials), v(stats), 1.0, None, v(FAKE), 0,
            64, v(FAKE * 2), 1 << 30, None)
    assert call(0) == RL_ERR_INVALID_ARG                      # no phase
    assert call(3) == RL_ERR_INVALID_ARG                      # one phase per call
    assert call(ml.RL_SHARD_SEQ) == RL_ERR_INVALID_ARG        # SEQ is GSPO's only
    assert call(ml.RL_SHARD_SWEEP, params=gspo, sums=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_SEQ, params=gspo, sums=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_SEQ, params=gspo, partials=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_COUNT, r0=8, total=16, R=9) == RL_ERR_INVALID_ARG  # past the call
    assert call(ml.RL_SHARD_COUNT, r0=-1) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_COUNT, counts=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_SWEEP, partials=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_FINISH, partials=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_SHARD_FINISH, stats=None) == RL_ERR_INVALID_ARG


def test_vocab_sharded_entry_validates(lib):
    """Every argument error of rl_loss_vocab_shard_fwd_bwd is caught on the
    host, before anything is enqueued (no GPU is needed)."""
    v = ctypes.c_void_p
    p = ml.make_params()

    def call(phase, shard=0, starts=(0, 40, 64), r0=0, total=16, R=16, params=p, counts=FAKE,
             rp=FAKE, rp_all=FAKE, partials=FAKE, stats=FAKE, ld=40, starts_ptr=True, sums=FAKE):
        arr = (ctypes.c_int64 * len(starts))(*starts)
        return lib.rl_loss_vocab_shard_fwd_bwd(
            phase, shard, len(starts) - 1, ctypes.cast(arr, v) if starts_ptr else None, r0, total,
            v(FAKE), 0, R, ld, v(FAKE), v(FAKE), None, None, None, v(FAKE), v(FAKE), v(FAKE), 2, 1,
            v(FAKE), ctypes.byref(params), v(FAKE), v(FAKE), v(FAKE), v(FAKE), v(counts), v(sums),
            v(rp), v(rp_all), v(partials), v(stats), 1.0, None, v(FAKE), 0, 64, v(FAKE * 2),
            1 << 30, None)
    C, PA, SW, FI = (ml.RL_VSHARD_COUNT, ml.RL_VSHARD_PARTIAL, ml.RL_VSHARD_SWEEP,
                     ml.RL_VSHARD_FINISH)
    assert call(0) == RL_ERR_INVALID_ARG                               # no phase
    assert call(6) == RL_ERR_INVALID_ARG
    assert call(ml.RL_VSHARD_SEQ) == RL_ERR_INVALID_ARG                # SEQ is GSPO's only
    assert call(C, starts_ptr=False) == RL_ERR_INVALID_ARG             # no column partition
    assert call(C, starts=(1, 40, 64)) == RL_ERR_INVALID_ARG           # does not start at 0
    assert call(C, starts=(0, 40, 40)) == RL_ERR_INVALID_ARG           # an empty shard
    assert call(C, starts=(0, 50, 40)) == RL_ERR_INVALID_ARG           # decreasing
    assert call(C, starts=(0, 40, 1 << 31)) == RL_ERR_INVALID_ARG      # ids past int32
    assert call(C, starts=tuple(range(66))) == RL_ERR_INVALID_ARG      # 65 shards
    assert call(C, shard=2) == RL_ERR_INVALID_ARG                      # no such shard
    assert call(C, shard=-1) == RL_ERR_INVALID_ARG
    assert call(PA, ld=39) == RL_ERR_INVALID_ARG                       # ld below the shard's 40 columns
    assert call(C, r0=8, total=16, R=9) == RL_ERR_INVALID_ARG          # rows past the call
    assert call(C, counts=None) == RL_ERR_INVALID_ARG
    assert call(PA, rp=None) == RL_ERR_INVALID_ARG
    assert call(PA, rp=FAKE + 4) == RL_ERR_INVALID_ARG                 # records not 16-byte aligned
    assert call(SW, rp_all=None) == RL_ERR_INVALID_ARG
    assert call(SW, rp_all=FAKE + 8) == RL_ERR_INVALID_ARG
    assert call(SW, partials=None) == RL_ERR_INVALID_ARG
    assert call(FI, partials=None) == RL_ERR_INVALID_ARG
    assert call(FI, stats=None) == RL_ERR_INVALID_ARG
    gspo = ml.make_params(estimator="gspo")
    assert call(SW, params=gspo, sums=None) == RL_ERR_INVALID_ARG     # GSPO writes its sums
    assert call(ml.RL_VSHARD_SEQ, params=gspo, sums=None) == RL_ERR_INVALID_ARG
    assert call(ml.RL_VSHARD_SEQ, params=gspo, partials=None) == RL_ERR_INVALID_ARG
    tk = ml.make_params(opd_coef=0.5, opd_topk=4, opd_topk_ids=_Ptr(FAKE + 2),
                        opd_topk_teacher=_Ptr(FAKE))                   # ids not 4-byte aligned
    assert call(PA, params=tk) == RL_ERR_INVALID_ARG
    tk = ml.make_params(opd_coef=0.5, opd_topk=4)                      # no candidate arrays
    assert call(PA, params=tk) == RL_ERR_INVALID_ARG
    assert call(PA, params=ml.make_params(temperature=0.0)) == RL_ERR_INVALID_ARG
