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


def fwd_bwd(w, buf: Buffers, params=None, grad_loss=1.0, grad_loss_device=None, stream=None):
    """One fused forward+backward call on a ``workloads.Workload``."""
    ml.rl_loss_fwd_bwd(w.logits, w.targets, w.rollout_logprobs, w.ref_logprobs, w.old_logprobs,
                       w.teacher_logprobs, w.rewards, w.group_id, w.cu_seqlens, w.n_groups,
                       w.loss_mask, params if params is not None else w.params,
                       buf.token_logprobs, buf.entropy, buf.advantages, buf.group_sizes,
                       buf.stats, buf.dlogits, buf.workspace, grad_loss=grad_loss,
                       grad_loss_device=grad_loss_device, vocab=w.vocab, stream=stream)


def fwd(w, buf: Buffers, params=None, stream=None):
    ml.rl_loss_fwd(w.logits, w.targets, w.rollout_logprobs, w.ref_logprobs, w.old_logprobs,
                   w.teacher_logprobs, w.rewards, w.group_id, w.cu_seqlens, w.n_groups,
                   w.loss_mask, params if params is not None else w.params, buf.token_logprobs,
                   buf.entropy, buf.advantages, buf.group_sizes, buf.stats, buf.workspace,
                   vocab=w.vocab, stream=stream)


def bwd(w, buf: Buffers, params=None, grad_loss=1.0, grad_loss_device=None, stream=None):
    ml.rl_loss_bwd(w.logits, w.targets, w.loss_mask,
                   params if params is not None else w.params, buf.workspace, buf.dlogits,
                   grad_loss=grad_loss, grad_loss_device=grad_loss_device, vocab=w.vocab,
                   stream=stream)


class HostCall:
    """Fused forward+backward with the inputs and results in pinned HOST
    memory: every call copies the inputs host -> device, runs the loss, and
    copies dLogits, the per-row outputs and the statistics back. Device
    buffers are allocated once at construction."""

    INPUTS = ("logits", "targets", "rollout_logprobs", "ref_logprobs", "old_logprobs",
              "teacher_logprobs", "rewards", "group_id", "cu_seqlens", "loss_mask")

    def __init__(self, host_w, device, dlogits_dtype=None, dev_w=None, buf=None):
        """``dev_w`` / ``buf``: existing device buffers of the same shapes to
        reuse (their contents are overwritten by every call)."""
        self.host = host_w
        self.dev = host_w.to(device) if dev_w is None else dev_w
        n_traj = int(host_w.rewards.shape[0])
        dl_dtype = dlogits_dtype or host_w.logits.dtype
        self.buf = buf if buf is not None else alloc(
            host_w.n_rows, n_traj, host_w.n_groups, device, vocab=host_w.vocab,
            dlogits_dtype=dl_dtype)
        pin = dict(pin_memory=True)
        self.out = dict(
            dlogits=torch.empty(self.buf.dlogits.shape, dtype=dl_dtype, **pin),
            token_logprobs=torch.empty(host_w.n_rows, dtype=torch.float32, **pin),
            entropy=torch.empty(host_w.n_rows, dtype=torch.float32, **pin),
            stats=torch.empty(ml.STATS_BYTES, dtype=torch.uint8, **pin))

    def bytes_in(self) -> int:
        return sum(getattr(self.host, k).numel() * getattr(self.host, k).element_size()
                   for k in self.INPUTS if getattr(self.host, k) is not None)

    def bytes_out(self) -> int:
        return sum(t.numel() * t.element_size() for t in self.out.values())

    def __call__(self, grad_loss=1.0):
        for k in self.INPUTS:
            h = getattr(self.host, k)
            if h is not None:
                getattr(self.dev, k).copy_(h, non_blocking=True)
        fwd_bwd(self.dev, self.buf, grad_loss=grad_loss)
        self.out["dlogits"].copy_(self.buf.dlogits, non_blocking=True)
        self.out["token_logprobs"].copy_(self.buf.token_logprobs, non_blocking=True)
        self.out["entropy"].copy_(self.buf.entropy, non_blocking=True)
        self.out["stats"].copy_(self.buf.stats, non_blocking=True)
        return self.out
