"""Tensor-level convenience layer over the C ABI: allocates the outputs and
the workspace with torch (device memory only) and calls the library. No
arithmetic of the loss happens here."""

from __future__ import annotations

from dataclasses import dataclass

import torch

from . import milesloss as ml


@dataclass
class Buffers:
    token_logprobs: torch.Tensor
    entropy: torch.Tensor
    advantages: torch.Tensor
    group_sizes: torch.Tensor
    stats: torch.Tensor          # 128 raw bytes of one rl_loss_stats
    workspace: torch.Tensor
    dlogits: torch.Tensor | None

    def read_stats(self) -> dict:
        return ml.parse_stats(self.stats.cpu().numpy().tobytes())


def alloc(n_rows: int, n_traj: int, n_groups: int, device, vocab: int | None = None,
          dlogits_dtype=None, ld_out: int | None = None, fill_nan: bool = False) -> Buffers:
    """Output buffers for one call. ``fill_nan`` pre-fills the float outputs
    with NaN so that an element the library fails to write cannot pass a
    comparison."""
    def f32(n):
        t = torch.empty(n, dtype=torch.float32, device=device)
        if fill_nan:
            t.fill_(float("nan"))
        return t
    ws = torch.empty(ml.rl_loss_workspace_size(n_rows, n_traj, n_groups), dtype=torch.uint8,
                     device=device)
    dl = None
    if dlogits_dtype is not None:
        ld = vocab if ld_out is None else ld_out
        dl = torch.empty((n_rows, ld), dtype=dlogits_dtype, device=device)
        if fill_nan:
            dl.fill_(float("nan"))
    gs = torch.full((n_groups,), -7, dtype=torch.int32, device=device)
    st = torch.full((ml.STATS_BYTES,), 0xAB, dtype=torch.uint8, device=device)
    return Buffers(f32(n_rows), f32(n_rows), f32(n_traj), gs, st, ws, dl)


def _params(w, params):
    """The call's parameters; with top-K OPD on, the workload's candidate ids
    and teacher log-probs are attached unless the caller gave them."""
    p = dict(w.params if params is None else params)
    if p.get("opd_topk", 0) > 0 and "opd_topk_ids" not in p and w.topk_ids is not None:
        p.update(opd_topk_ids=w.topk_ids, opd_topk_teacher=w.topk_teacher)
    return p


def fwd_bwd(w, buf: Buffers, params=None, grad_loss=1.0, grad_loss_device=None, stream=None):
    """One fused forward+backward call on a ``workloads.Workload``."""
    ml.rl_loss_fwd_bwd(w.logits, w.targets, w.rollout_logprobs, w.ref_logprobs, w.old_logprobs,
                       w.teacher_logprobs, w.rewards, w.group_id, w.cu_seqlens, w.n_groups,
                       w.loss_mask, _params(w, params),
                       buf.token_logprobs, buf.entropy, buf.advantages, buf.group_sizes,
                       buf.stats, buf.dlogits, buf.workspace, grad_loss=grad_loss,
                       grad_loss_device=grad_loss_device, vocab=w.vocab, stream=stream)


def fwd(w, buf: Buffers, params=None, stream=None):
    ml.rl_loss_fwd(w.logits, w.targets, w.rollout_logprobs, w.ref_logprobs, w.old_logprobs,
                   w.teacher_logprobs, w.rewards, w.group_id, w.cu_seqlens, w.n_groups,
                   w.loss_mask, _params(w, params), buf.token_logprobs,
                   buf.entropy, buf.advantages, buf.group_sizes, buf.stats, buf.workspace,
                   vocab=w.vocab, stream=stream)


def bwd(w, buf: Buffers, params=None, grad_loss=1.0, grad_loss_device=None, stream=None):
    ml.rl_loss_bwd(w.logits, w.targets, w.loss_mask,
                   _params(w, params), buf.workspace, buf.dlogits,
                   grad_loss=grad_loss, grad_loss_device=grad_loss_device, vocab=w.vocab,
                   stream=stream)


class GraphedCall:
    """The fused call on fixed tensors, captured once in a CUDA graph; each
    call replays it on the current stream. The library only enqueues kernels
    (no allocation, no synchronisation), so the capture holds the whole call;
    the inputs may change in place between replays. For small calls the host
    launch cost of the three to four kernels is then paid once."""

    def __init__(self, w, buf: Buffers, params=None, grad_loss=1.0):
        s = torch.cuda.Stream()
        s.wait_stream(torch.cuda.current_stream())
        with torch.cuda.stream(s):
            fwd_bwd(w, buf, params=params, grad_loss=grad_loss)  # kernel attributes set outside capture
        torch.cuda.current_stream().wait_stream(s)
        torch.cuda.synchronize()
        self.graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(self.graph):
            fwd_bwd(w, buf, params=params, grad_loss=grad_loss)

    def __call__(self):
        self.graph.replay()


def _rows_call(w, buf, phase, r0, r1, logits, dlogits, params=None, grad_loss=1.0, stream=None):
    ml.rl_loss_fwd_bwd_rows(phase, r0, r1, w.n_rows, logits, w.targets, w.rollout_logprobs,
                            w.ref_logprobs, w.old_logprobs, w.teacher_logprobs, w.rewards,
                            w.group_id, w.cu_seqlens, w.n_groups, w.loss_mask,
                            _params(w, params), buf.token_logprobs,
                            buf.entropy, buf.advantages, buf.group_sizes, buf.stats, dlogits,
                            buf.workspace, w.vocab,
                            logits_dtype=(w.logits.dtype if w.logits is not None
                                          else (logits.dtype if logits is not None
                                                else torch.bfloat16)),
                            grad_loss=grad_loss, stream=stream)


def fwd_bwd_chunked(w, buf: Buffers, chunk_rows: int, params=None, grad_loss=1.0,
                    forward_only=False):
    """The fused call as BEGIN, one ROWS call per block of ``chunk_rows`` rows
    (each reading a view of the logits and writing a view of dLogits), END."""
    R = w.n_rows
    _rows_call(w, buf, ml.RL_PHASE_BEGIN, 0, R, None, None, params, grad_loss)
    for r0 in range(0, R, chunk_rows):
        r1 = min(R, r0 + chunk_rows)
        dl = None if forward_only else buf.dlogits[r0:r1]
        _rows_call(w, buf, ml.RL_PHASE_ROWS, r0, r1, w.logits[r0:r1], dl, params, grad_loss)
    _rows_call(w, buf, ml.RL_PHASE_END, 0, R, None, None, params, grad_loss)


class PipelinedHostCall:
    """The fused call with logits in pinned HOST memory, streamed through
    ``depth`` device chunk buffers: per chunk of rows, the host-to-device
    copy (one stream), the vocabulary sweep (the caller's stream) and, when
    dLogits go back to pinned host memory too, their device-to-host copy (a
    third stream) overlap with the other chunks'. A chunk's input copy waits
    only for the sweep ``depth`` chunks back, so the two copy directions can
    drift apart by that many chunks when the host link's rate varies. With
    ``dlogits_on_device`` the dLogits stay in one device tensor (where a
    trainer's backward pass reads them) and only the per-row results and the
    statistics come back. The small per-row inputs go to the device whole
    before the sweep (BEGIN needs all of them)."""

    SMALL = ("targets", "rollout_logprobs", "ref_logprobs", "old_logprobs", "teacher_logprobs",
             "rewards", "group_id", "cu_seqlens", "loss_mask", "topk_ids", "topk_teacher")

    def __init__(self, host_w, device, chunk_rows=4096, dlogits_dtype=None, depth=2,
                 dlogits_on_device=False):
        from . import workloads as wl
        self.host = host_w
        self.chunk = chunk_rows
        self.depth = int(depth)
        if self.depth < 2:
            raise ValueError("depth must be at least 2")
        R, V = host_w.n_rows, host_w.vocab
        self.dl_dtype = dlogits_dtype or host_w.logits.dtype

        def dev(t):
            return None if t is None else torch.empty_like(t, device=device)
        self.dev = wl.Workload(host_w.recipe, None, dev(host_w.targets),
                               dev(host_w.rollout_logprobs), dev(host_w.ref_logprobs),
                               dev(host_w.old_logprobs), dev(host_w.teacher_logprobs),
                               dev(host_w.rewards), dev(host_w.group_id), dev(host_w.cu_seqlens),
                               dev(host_w.loss_mask), host_w.n_groups, dict(host_w.params),
                               dev(host_w.topk_ids), dev(host_w.topk_teacher))
        n = min(chunk_rows, R)
        self.lg = [torch.empty((n, V), dtype=host_w.logits.dtype, device=device)
                   for _ in range(self.depth)]
        self.dl = None if dlogits_on_device else [
            torch.empty((n, V), dtype=self.dl_dtype, device=device) for _ in range(self.depth)]
        self.buf = alloc(R, int(host_w.rewards.shape[0]), host_w.n_groups, device, vocab=V)
        pin = dict(pin_memory=True)
        self.out = dict(
            dlogits=torch.empty((R, V), dtype=self.dl_dtype,
                                **(dict(device=device) if dlogits_on_device else pin)),
            token_logprobs=torch.empty(R, dtype=torch.float32, **pin),
            entropy=torch.empty(R, dtype=torch.float32, **pin),
            stats=torch.empty(ml.STATS_BYTES, dtype=torch.uint8, **pin))
        self.s_in = torch.cuda.Stream(device=device)
        self.s_out = torch.cuda.Stream(device=device)
        self.params = dict(host_w.params)
        if self.params.get("opd_topk", 0) > 0:
            self.params.update(opd_topk_ids=self.dev.topk_ids,
                               opd_topk_teacher=self.dev.topk_teacher)

    def bytes_in(self) -> int:
        h = self.host
        return h.logits[:, :h.vocab].numel() * h.logits.element_size() + sum(
            getattr(h, k).numel() * getattr(h, k).element_size()
            for k in self.SMALL if getattr(h, k) is not None)

    def bytes_out(self) -> int:
        """Bytes copied back to the host per call."""
        return sum(t.numel() * t.element_size() for t in self.out.values() if not t.is_cuda)

    def __call__(self, grad_loss=1.0):
        comp = torch.cuda.current_stream()
        h, d = self.host, self.dev
        R, V = h.n_rows, h.vocab
        for k in self.SMALL:
            if getattr(h, k) is not None:
                getattr(d, k).copy_(getattr(h, k), non_blocking=True)
        _rows_call(d, self.buf, ml.RL_PHASE_BEGIN, 0, R, None, None, self.params, grad_loss)
        comp_done = [None] * self.depth
        out_done = [None] * self.depth
        for i, r0 in enumerate(range(0, R, self.chunk)):
            r1 = min(R, r0 + self.chunk)
            b, n = i % self.depth, r1 - r0
            if comp_done[b] is not None:   # the sweep `depth` chunks back read lg[b]
                self.s_in.wait_event(comp_done[b])
            with torch.cuda.stream(self.s_in):
                self.lg[b][:n].copy_(h.logits[r0:r1, :V], non_blocking=True)
                in_done = torch.cuda.Event()
                in_done.record(self.s_in)
            comp.wait_event(in_done)
            if out_done[b] is not None:    # dl[b] was copied out
                comp.wait_event(out_done[b])
            dl = self.out["dlogits"][r0:r1] if self.dl is None else self.dl[b][:n]
            _rows_call(d, self.buf, ml.RL_PHASE_ROWS, r0, r1, self.lg[b][:n], dl,
                       self.params, grad_loss)
            comp_done[b] = torch.cuda.Event()
            comp_done[b].record(comp)
            if self.dl is not None:
                self.s_out.wait_event(comp_done[b])
                with torch.cuda.stream(self.s_out):
                    self.out["dlogits"][r0:r1].copy_(self.dl[b][:n], non_blocking=True)
                    out_done[b] = torch.cuda.Event()
                    out_done[b].record(self.s_out)
        _rows_call(d, self.buf, ml.RL_PHASE_END, 0, R, None, None, self.params, grad_loss)
        self.out["token_logprobs"].copy_(self.buf.token_logprobs, non_blocking=True)
        self.out["entropy"].copy_(self.buf.entropy, non_blocking=True)
        self.out["stats"].copy_(self.buf.stats, non_blocking=True)
        for e in out_done:
            if e is not None:
                comp.wait_event(e)
        return self.out


# ------------------------------------------------------------ row-sharded calls

class Shard:
    """One shard of a row-sharded fused call (rl_loss_shard_fwd_bwd): the
    workload ``w`` holds this shard's rows [row_offset, row_offset + rows) of
    a call of ``n_rows_total`` rows, with the whole call's rewards, group ids
    and cu_seqlens; ``buf`` its output buffers. ``count``, ``sweep`` and
    ``finish`` run the three phases; between them the shards' ``counts`` are
    summed and their ``partials`` combined (exchange_counts /
    exchange_partials, or any equivalent)."""

    def __init__(self, w, row_offset: int, n_rows_total: int, buf: Buffers, params=None,
                 grad_loss=1.0):
        self.w, self.row_offset, self.n_rows_total, self.buf = w, row_offset, n_rows_total, buf
        self.params = _params(w, params)
        self.grad_loss = grad_loss
        dev = w.targets.device
        n_traj = int(w.rewards.shape[0])
        self.counts = torch.zeros(n_traj, dtype=torch.int32, device=dev)
        self.traj_sums = torch.zeros((n_traj, 2), dtype=torch.float64, device=dev)
        self.partials = torch.zeros(ml.PARTIALS_DOUBLES, dtype=torch.float64, device=dev)

    @property
    def gspo(self) -> bool:
        return self.params.get("estimator", "grpo") == "gspo"

    def _call(self, phase, forward_only=False):
        w, b = self.w, self.buf
        ml.rl_loss_shard_fwd_bwd(phase, self.row_offset, self.n_rows_total, w.logits, w.targets,
                                 w.rollout_logprobs, w.ref_logprobs, w.old_logprobs,
                                 w.teacher_logprobs, w.rewards, w.group_id, w.cu_seqlens,
                                 w.n_groups, w.loss_mask, self.params, b.token_logprobs,
                                 b.entropy, b.advantages, b.group_sizes, self.counts,
                                 self.partials, b.stats, None if forward_only else b.dlogits,
                                 b.workspace, w.vocab, grad_loss=self.grad_loss,
                                 traj_sums=self.traj_sums)

    def count(self):
        self._call(ml.RL_SHARD_COUNT)

    def sweep(self, forward_only=False):
        self._call(ml.RL_SHARD_SWEEP, forward_only)

    def seq(self, forward_only=False):
        """GSPO only: after the shards' traj_sums have been added."""
        self._call(ml.RL_SHARD_SEQ, forward_only)

    def finish(self):
        self._call(ml.RL_SHARD_FINISH)


def exchange_counts(counts: torch.Tensor, group=None):
    """Sum the shards' per-trajectory training-token counts over the ranks of
    ``group`` (in place)."""
    import torch.distributed as dist
    dist.all_reduce(counts, op=dist.ReduceOp.SUM, group=group)


def exchange_traj_sums(traj_sums: torch.Tensor, group=None):
    """GSPO: add the shards' per-trajectory sums over the ranks of ``group``
    (in place)."""
    import torch.distributed as dist
    dist.all_reduce(traj_sums, op=dist.ReduceOp.SUM, group=group)


def exchange_partials(partials: torch.Tensor, group=None):
    """Combine the shards' rl_loss_partials over the ranks of ``group`` (in
    place): sums and counts by addition, the two maxima by maximum."""
    import torch.distributed as dist
    dist.all_reduce(partials[:ml.PARTIALS_SUMS], op=dist.ReduceOp.SUM, group=group)
    dist.all_reduce(partials[ml.PARTIALS_SUMS:], op=dist.ReduceOp.MAX, group=group)


def sharded_fwd_bwd(shard: Shard, group=None):
    """This rank's shard of a row-sharded fused call, one shard per rank,
    with the two exchanges over torch.distributed."""
    shard.count()
    exchange_counts(shard.counts, group)
    shard.sweep()
    if shard.gspo:
        exchange_traj_sums(shard.traj_sums, group)
        shard.seq()
    exchange_partials(shard.partials, group)
    shard.finish()


def sharded_fwd_bwd_local(shards):
    """Several shards of one call driven from one process (for instance on
    one GPU): the exchanges are sums and maxima over the shards' tensors."""
    for s in shards:
        s.count()
    total = torch.stack([s.counts for s in shards]).sum(0)
    for s in shards:
        s.counts.copy_(total)
        s.sweep()
    if shards and shards[0].gspo:
        sums = torch.stack([s.traj_sums for s in shards]).sum(0)
        for s in shards:
            s.traj_sums.copy_(sums)
            s.seq()
    p = torch.stack([s.partials for s in shards])
    comb = torch.cat([p[:, :ml.PARTIALS_SUMS].sum(0), p[:, ml.PARTIALS_SUMS:].max(0).values])
    for s in shards:
        s.partials.copy_(comb)
        s.finish()


# ------------------------------------------------------ vocabulary-sharded calls

class VocabShard:
    """One shard of a vocabulary-sharded fused call
    (rl_loss_vocab_shard_fwd_bwd): ``w.logits`` holds this shard's columns
    [col_starts[col_shard], col_starts[col_shard + 1]) of its rows (a view of
    a wider tensor is fine: its row stride is the ld), ``w.targets`` the
    vocabulary ids; rows may be sharded as well (``row_offset``,
    ``n_rows_total``, as in Shard). ``buf.dlogits`` holds the same columns.
    The phases are ``count``, ``partial``, ``sweep`` and ``finish``; between
    them the ROW shards' ``counts`` are summed, the COLUMN shards'
    ``row_partials`` gathered into ``row_partials_all`` (exchange_row_partials)
    and the ROW shards' ``partials`` combined."""

    def __init__(self, w, col_shard: int, col_starts, buf: Buffers, row_offset: int = 0,
                 n_rows_total: int | None = None, params=None, grad_loss=1.0):
        self.w, self.buf = w, buf
        self.col_shard, self.col_starts = int(col_shard), [int(c) for c in col_starts]
        self.row_offset = int(row_offset)
        self.n_rows_total = w.n_rows if n_rows_total is None else int(n_rows_total)
        self.params = _params(w, params)
        self.grad_loss = grad_loss
        dev = w.targets.device
        R, n_shards = w.n_rows, len(self.col_starts) - 1
        self.counts = torch.zeros(int(w.rewards.shape[0]), dtype=torch.int32, device=dev)
        self.traj_sums = torch.zeros((int(w.rewards.shape[0]), 2), dtype=torch.float64,
                                     device=dev)
        self.row_partials = torch.zeros((R, 8), dtype=torch.float32, device=dev)
        self.row_partials_all = torch.zeros((n_shards, R, 8), dtype=torch.float32, device=dev)
        self.partials = torch.zeros(ml.PARTIALS_DOUBLES, dtype=torch.float64, device=dev)

    def _call(self, phase, forward_only=False):
        w, b = self.w, self.buf
        ml.rl_loss_vocab_shard_fwd_bwd(
            phase, self.col_shard, self.col_starts, self.row_offset, self.n_rows_total, w.logits,
            w.targets, w.rollout_logprobs, w.ref_logprobs, w.old_logprobs, w.teacher_logprobs,
            w.rewards, w.group_id, w.cu_seqlens, w.n_groups, w.loss_mask, self.params,
            b.token_logprobs, b.entropy, b.advantages, b.group_sizes, self.counts,
            self.row_partials, self.row_partials_all, self.partials, b.stats,
            None if forward_only else b.dlogits, b.workspace, grad_loss=self.grad_loss,
            traj_sums=self.traj_sums)

    @property
    def gspo(self) -> bool:
        return self.params.get("estimator", "grpo") == "gspo"

    def count(self):
        self._call(ml.RL_VSHARD_COUNT)

    def partial(self):
        self._call(ml.RL_VSHARD_PARTIAL)

    def sweep(self, forward_only=False):
        self._call(ml.RL_VSHARD_SWEEP, forward_only)

    def seq(self, forward_only=False):
        """GSPO only: after the row shards' traj_sums have been added."""
        self._call(ml.RL_VSHARD_SEQ, forward_only)

    def finish(self):
        self._call(ml.RL_VSHARD_FINISH)


def exchange_row_partials(row_partials: torch.Tensor, row_partials_all: torch.Tensor,
                          group=None):
    """Gather the column shards' per-row records over the ranks of ``group``
    (rank k of the group holds column shard k): row_partials_all[k] =
    rank k's row_partials."""
    import torch.distributed as dist
    # (rank k's rows land at rows [k R, (k + 1) R) of the flattened output)
    dist.all_gather_into_tensor(row_partials_all.view(-1, row_partials.shape[-1]),
                                row_partials.contiguous(), group=group)


def vocab_sharded_fwd_bwd(shard: VocabShard, col_group=None, row_group=None):
    """This rank's shard of a vocabulary-sharded fused call over
    torch.distributed: ``col_group`` holds the column shards of this rank's
    rows (in shard order), ``row_group`` the ranks of the same column shard
    that hold the other rows (None with a single row shard)."""
    shard.count()
    if row_group is not None:
        exchange_counts(shard.counts, row_group)
    shard.partial()
    exchange_row_partials(shard.row_partials, shard.row_partials_all, col_group)
    shard.sweep()
    if shard.gspo:
        if row_group is not None:
            exchange_traj_sums(shard.traj_sums, row_group)
        shard.seq()
    if row_group is not None:
        exchange_partials(shard.partials, row_group)
    shard.finish()


def vocab_sharded_fwd_bwd_local(shards):
    """Shards of one call driven from one process (for instance on one
    GPU), ``shards[i][k]`` the column shard k of row shard i: the exchanges
    are sums, stacks and maxima over the shards' tensors."""
    flat = [s for row in shards for s in row]
    for s in flat:
        s.count()
    total = torch.stack([row[0].counts for row in shards]).sum(0)
    for s in flat:
        s.counts.copy_(total)
        s.partial()
    for row in shards:
        gathered = torch.stack([s.row_partials for s in row])
        for s in row:
            s.row_partials_all.copy_(gathered)
            s.sweep()
    if flat and flat[0].gspo:
        sums = torch.stack([row[0].traj_sums for row in shards]).sum(0)
        for s in flat:
            s.traj_sums.copy_(sums)
            s.seq()
    p = torch.stack([row[0].partials for row in shards])
    comb = torch.cat([p[:, :ml.PARTIALS_SUMS].sum(0), p[:, ml.PARTIALS_SUMS:].max(0).values])
    for s in flat:
        s.partials.copy_(comb)
        s.finish()
