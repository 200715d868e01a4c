"""The host side of vocabulary-sharded calls with two gloo ranks on CPU: each
rank holds one block of the vocabulary's columns of a call's logits, forms
the per-row records its shard's forward sweep writes (the format
include/milesloss.h gives for rl_loss_vocab_shard_fwd_bwd: a reference m in
log2 units, s, u, the target's logit where the shard holds it, and the part
of the row's top-K OPD candidates in its columns), and
paper_2609_08368_gb300.api.exchange_row_partials gathers them in shard
order. Merged in that order as the library's merge step does, the records
must give every rank each row's log-sum-exp, log-prob, entropy and top-K
signal as the float64 oracle computes them over the whole row."""

import os
import socket

import numpy as np
import torch
import torch.distributed as dist
import torch.multiprocessing as mp

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
LOG2E = 1.4426950408889634
COLS = [0, 23, 41]  # rank k holds columns [COLS[k], COLS[k + 1])
T = 0.8


def _free_port():
    with socket.socket() as s:
        s.bind(("127.0.0.1", 0))
        return s.getsockname()[1]


K = 5


def _call():
    rng = np.random.default_rng(11)
    R, V = 9, COLS[-1]
    z = rng.normal(0, 3, size=(R, V))
    z[3, :COLS[1]] = -np.inf          # a row whose first block holds nothing
    y = rng.integers(0, V, size=R)
    y[0], y[1] = 0, V - 1             # the first and the last column
    ids = np.stack([rng.choice(V, size=K, replace=False) for _ in range(R)])
    ids[2] = [1, 2, 3, 4, 5]          # every candidate in the first block
    ids[3] = [24, 30, 35, 40, 23]     # every candidate in the second
    teacher = rng.normal(-3, 1, size=(R, K))
    return z, y, ids, teacher


def _records(z, y, ids, teacher, c0, c1):
    """One shard's records of its columns [c0, c1): per row (m, s, u, zy) with
    any finite reference m (here the block's largest scaled logit), then the
    part of the candidates in the block (mt, sw, acc, bad)."""
    t = z[:, c0:c1] * (LOG2E / T)
    rec = np.zeros((z.shape[0], 8))
    for r in range(z.shape[0]):
        fin = t[r][np.isfinite(t[r])]
        if fin.size == 0:
            rec[r, :4] = (-np.inf, 0.0, 0.0, 0.0)
        else:
            m = fin.max()
            x = np.exp2(fin - m)
            rec[r, :4] = (m, x.sum(), (x * (fin - m)).sum(),
                          z[r, y[r]] if c0 <= y[r] < c1 else 0.0)
        mine = (ids[r] >= c0) & (ids[r] < c1)
        if not mine.any():
            rec[r, 4:] = (-np.inf, 0.0, 0.0, 0.0)
            continue
        tc = z[r, ids[r][mine]] * (LOG2E / T)
        mt = tc.max()
        wc = np.exp2(tc - mt)
        rec[r, 4:] = (mt, wc.sum(), (wc * (z[r, ids[r][mine]] / T - teacher[r][mine])).sum(), 0.0)
    return rec


def _merge(all_rec, y):
    """Each row's records in shard order: lse, logp, H and the top-K signal."""
    R = all_rec.shape[1]
    lse, logp, H, opd = np.empty(R), np.empty(R), np.empty(R), np.empty(R)
    for r in range(R):
        c = all_rec[:, r, 4:].astype(np.float64)
        livec = c[:, 1] > 0
        Mt = c[livec, 0].max()
        ft = np.exp2(c[livec, 0] - Mt)
        sw, acc = (ft * c[livec, 1]).sum(), (ft * c[livec, 2]).sum()
        e = all_rec[:, r, :4].astype(np.float64)
        live = e[:, 1] > 0
        M = e[live, 0].max()
        f = np.exp2(e[live, 0] - M)
        S = (f * e[live, 1]).sum()
        U = (f * ((e[live, 0] - M) * e[live, 1] + e[live, 2])).sum()
        owner = int(np.searchsorted(COLS, y[r], side="right") - 1)
        lse[r] = M * np.log(2) + np.log(S)
        H[r] = np.log(S) - U * np.log(2) / S
        logp[r] = e[owner, 3] / T - lse[r]
        opd[r] = acc / sw - lse[r]
    return lse, logp, H, opd


def _worker(rank, world, port, out):
    import sys
    sys.path.insert(0, ROOT)
    os.environ.update(MASTER_ADDR="127.0.0.1", MASTER_PORT=str(port))
    dist.init_process_group("gloo", rank=rank, world_size=world)
    from paper_2609_08368_gb300 import api
    z, y, ids, teacher = _call()
    mine = torch.from_numpy(
        _records(z, y, ids, teacher, COLS[rank], COLS[rank + 1]).astype(np.float32))
    gathered = torch.full((world, z.shape[0], 8), float("nan"))
    api.exchange_row_partials(mine, gathered)
    out[rank] = gathered.numpy().tolist()
    dist.destroy_process_group()


def test_two_gloo_ranks_gather_and_merge_row_records():
    import oracle
    ctx = mp.get_context("spawn")
    out = ctx.Manager().dict()
    mp.start_processes(_worker, args=(2, _free_port(), out), nprocs=2, start_method="spawn")
    z, y, ids, teacher = _call()
    logp_o, H_o, lse_o = oracle.row_log_softmax(z, y, T)
    opd_o = oracle.opd_topk_estimate(z, T, lse_o, ids, teacher)
    assert out[0] == out[1]
    g = np.array(out[0])
    for k in range(2):  # shard k's records at index k
        want = _records(z, y, ids, teacher, COLS[k], COLS[k + 1]).astype(np.float32)
        np.testing.assert_array_equal(g[k], want)
    lse, logp, H, opd = _merge(g, y)
    np.testing.assert_allclose(opd, opd_o, rtol=0, atol=1e-5)
    # float32 records: agreement to a few ulp of float32
    np.testing.assert_allclose(lse, lse_o, rtol=1e-6, atol=1e-6)
    np.testing.assert_allclose(logp, logp_o, rtol=0, atol=1e-5)
    np.testing.assert_allclose(H, H_o, rtol=0, atol=1e-5)
