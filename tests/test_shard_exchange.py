"""The host side of row-sharded calls with two gloo ranks on CPU: each rank
holds one contiguous block of a call's rows (the second block starts inside
a trajectory), forms what its shard would hand to the exchanges (training
tokens per trajectory; the partial sums, counts and extremes of the
statistics over its rows, here from the float64 oracle), and the exchanges
of paper_2609_08368_gb300.api (all-reduce sums, and maxima for the
extremes) must give every rank the whole call's counts and statistics."""

import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


def _call():
    """A small call: 6 trajectories of unequal length in 2 groups, mask
    prefixes, rollout / reference log-probs near the logits' own."""
    import oracle
    rng = np.random.default_rng(5)
    lens = np.array([7, 3, 9, 5, 6, 4])
    cu = np.concatenate([[0], np.cumsum(lens)]).astype(np.int32)
    R, V = int(cu[-1]), 11
    z = rng.normal(0, 2, size=(R, V))
    y = rng.integers(0, V, size=R)
    p = oracle.LossParams(eps_lo=0.2, eps_hi=0.25, dual_clip_c=2.0, kl_coef=0.1,
                          correction="tis", corr_lo=0.0, corr_hi=1.2)
    logp, H, _ = oracle.row_log_softmax(z, y, p.temperature)
    rho = logp + rng.normal(0, 0.4, size=R)
    q = logp + rng.normal(0, 0.3, size=R)
    mask = np.ones(R, bool)
    for i in range(len(lens)):
        mask[cu[i]:cu[i] + 1 + i % 2] = False
    w = rng.random(6)
    gid = np.array([0, 0, 0, 1, 1, 1])
    _, A_row, _ = oracle.estimator_advantages(w, gid, 2, cu, mask, p)
    obj = oracle.token_objective(logp, rho, q, A_row, H, p)
    return dict(cu=cu, R=R, mask=mask, logp=logp, rho=rho, H=H, obj=obj, p=p)


def _shard_values(c, r0, r1):
    """What a shard of rows [r0, r1) hands to the exchanges."""
    cu, m = c["cu"], c["mask"]
    counts = np.array([m[max(cu[i], r0):max(min(cu[i + 1], r1), max(cu[i], r0))].sum()
                       for i in range(len(cu) - 1)], dtype=np.int32)
    sel = np.zeros(c["R"], bool)
    sel[r0:r1] = True
    sel &= m
    o = c["obj"]
    r, rc = o["r"][sel], o["rc"][sel]
    sums = [o["ell"][sel].sum(), o["pg"][sel].sum(), o["k3"][sel].sum(), c["H"][sel].sum(),
            r.sum(), np.abs(r - 1).sum(), np.abs(c["logp"][sel] - c["rho"][sel]).sum(),
            rc.sum(), np.abs(rc - 1).sum()]
    cnt = [sel.sum(), o["clip_hi"][sel].sum(), o["clip_lo"][sel].sum(), o["dual"][sel].sum(),
           o["corr_clip"][sel].sum()]
    mx = [-r.min() if r.size else -np.inf, r.max() if r.size else -np.inf]
    return counts, np.array(sums + cnt + mx, dtype=np.float64)


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_08368_gb300 import api
    c = _call()
    cut = [0, 12, c["R"]][rank:rank + 2]  # row 12 lies inside trajectory 2
    counts, part = _shard_values(c, *cut)
    t_counts = torch.from_numpy(counts)
    t_part = torch.from_numpy(part)
    api.exchange_counts(t_counts)
    api.exchange_partials(t_part)
    out[rank] = (t_counts.numpy().tolist(), t_part.numpy().tolist())
    dist.destroy_process_group()


def test_two_gloo_ranks_exchange_a_sharded_call():
    import oracle
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    mp.start_processes(_worker, args=(2, _free_port(), out), nprocs=2, start_method="spawn")
    c = _call()
    want_counts = oracle.training_tokens_per_trajectory(c["cu"], c["mask"]).tolist()
    st = oracle.loss_stats(dict(c["obj"]), c["logp"], c["rho"], c["H"], c["mask"])
    for rank in (0, 1):
        counts, part = out[rank]
        assert counts == want_counts
        s, n, mx = np.array(part[:9]), np.array(part[9:14]), part[14:]
        assert n.tolist() == [st["n_tokens"], st["n_clip_hi"], st["n_clip_lo"],
                              st["n_dual_clip"], st["n_corr_clip"]]
        N = n[0]
        for k, i in (("loss", 0), ("pg_loss_mean", 1), ("kl_mean", 2), ("entropy_mean", 3),
                     ("ratio_mean", 4), ("ratio_absdev_mean", 5), ("logprob_absdiff_mean", 6),
                     ("corr_ratio_mean", 7), ("corr_absdev_mean", 8)):
            assert abs(s[i] / N - st[k]) <= 1e-13 * max(1.0, abs(st[k])), k
        assert -mx[0] == st["ratio_min"] and mx[1] == st["ratio_max"]
    assert out[0] == out[1]
