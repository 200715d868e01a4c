"""Seeded synthetic inputs shaped like the paper's RL training batches.

This module only draws inputs. It holds none of the loss arithmetic; both the
CUDA library's callers (tests, bench) and the float64 oracle consume what it
produces. The one derived input is the "exact" sampled-token log-prob that
the rollout and reference log-probs are perturbed from; it is taken with
torch's library ``logsumexp`` in float64 on the rounded logits, because the
recipes below define the rollout log-probs as "exact + noise".

Five named recipes stand in for the paper's workloads (Sec. 9.1: sessions up
to 65,536 tokens, groups of 8 attempts, vocabularies near 150K, masked tool
output in agentic turns, Sec. 2.4). The paper's own dataset is not used.

  tiny        2 prompts x 4 = 8 traj x 256 tok, V 4,096, bf16 N(0,2^2)
  qwen        16 x 8 = 128 traj x 128 tok, V 151,936, bf16 N(0,3^2), +8 boost
  glm         64 traj x 1,024 tok (groups of 16), V 154,880, bf16, dual clip 3,
              k3 KL 0.01, dLogits bf16 (the headline workload)
  agentic     4 traj x 32,768 tok (one group), V 151,936, T = 0.7, tool spans
  fp32        512 traj x 256 tok (groups of 8), V 32,768, fp32, entropy bonus,
              equal-reward groups

Each recipe can be shrunk (fewer trajectories / tokens / vocab) for parity
tests while keeping its distributions.
"""

from __future__ import annotations

from dataclasses import dataclass, field, replace

import numpy as np
import torch


@dataclass(frozen=True)
class Recipe:
    name: str
    n_prompts: int
    group_size: int
    traj_len: int
    vocab: int
    dtype: str                      # "bf16" | "f32"
    logit_std: float
    boost: float = 0.0              # added to the target logit ...
    boost_frac: float = 0.0         # ... on this fraction of rows
    rho_noise: float = 0.05
    ref_noise: float | None = None  # None: no reference log-probs
    reward: str = "bernoulli0.5"    # see _rewards
    mask: str = "prefix_u32_128"    # see _mask
    params: dict = field(default_factory=dict)
    seed: int = 1000
    old_noise: float | None = None  # optional old (pi_old) log-probs
    teacher_noise: float | None = None  # optional OPD teacher log-probs
    topk: int = 0                   # OPD top-K candidates per row (the student's K most likely)
    topk_noise: float = 0.3         # teacher log-prob of a candidate = student's + N(0, s^2)

    @property
    def n_traj(self) -> int:
        return self.n_prompts * self.group_size

    @property
    def n_rows(self) -> int:
        return self.n_traj * self.traj_len


RECIPES = {
    "tiny": Recipe("tiny", 2, 4, 256, 4096, "bf16", 2.0, rho_noise=0.05,
                   reward="bernoulli0.5", mask="prefix_u32_128",
                   params=dict(temperature=1.0, eps_lo=0.2, eps_hi=0.2), seed=1001),
    "qwen": Recipe("qwen", 16, 8, 128, 151936, "bf16", 3.0, boost=8.0, boost_frac=0.7,
                   rho_noise=0.02, reward="bernoulli0.3", mask="prefix_frac0.25",
                   params=dict(temperature=1.0, eps_lo=0.2, eps_hi=0.28), seed=1002),
    "glm": Recipe("glm", 4, 16, 1024, 154880, "bf16", 3.0, boost=8.0, boost_frac=0.7,
                  rho_noise=0.05, ref_noise=0.1, reward="uniform", mask="prefix_frac0.25",
                  params=dict(temperature=1.0, eps_lo=0.2, eps_hi=0.2, dual_clip_c=3.0,
                              kl_coef=0.01), seed=1003),
    "agentic": Recipe("agentic", 1, 4, 32768, 151936, "bf16", 2.5, rho_noise=0.1,
                      reward="normal", mask="tool_spans",
                      params=dict(temperature=0.7, eps_lo=0.2, eps_hi=0.2), seed=1004),
    "fp32": Recipe("fp32", 64, 8, 256, 32768, "f32", 4.0, rho_noise=0.05, ref_noise=0.2,
                   reward="uniform_eq8", mask="prefix_frac0.25",
                   params=dict(temperature=1.0, eps_lo=0.2, eps_hi=0.2, dual_clip_c=3.0,
                               kl_coef=0.05, entropy_coef=0.001, std_floor=1e-6),
                   seed=1005),
}


def shrink(rec: Recipe, n_prompts=None, group_size=None, traj_len=None, vocab=None,
           **kw) -> Recipe:
    """A smaller copy of a recipe with the same distributions."""
    return replace(rec,
                   n_prompts=n_prompts or rec.n_prompts,
                   group_size=group_size or rec.group_size,
                   traj_len=traj_len or rec.traj_len,
                   vocab=vocab or rec.vocab, **kw)


@dataclass
class Workload:
    recipe: Recipe
    logits: torch.Tensor        # [R, ld] bf16 / f32 (only [:, :V] is data)
    targets: torch.Tensor       # [R] int32
    rollout_logprobs: torch.Tensor  # [R] f32
    ref_logprobs: torch.Tensor | None
    old_logprobs: torch.Tensor | None
    teacher_logprobs: torch.Tensor | None
    rewards: torch.Tensor       # [n_traj] f32
    group_id: torch.Tensor      # [n_traj] int32
    cu_seqlens: torch.Tensor    # [n_traj + 1] int32
    loss_mask: torch.Tensor     # [R] uint8
    n_groups: int
    params: dict
    topk_ids: torch.Tensor | None = None      # [R, K] int32
    topk_teacher: torch.Tensor | None = None  # [R, K] f32

    @property
    def n_rows(self) -> int:
        return int(self.targets.shape[0])

    @property
    def vocab(self) -> int:
        return self.recipe.vocab

    def to(self, device) -> "Workload":
        def mv(t):
            return None if t is None else t.to(device)
        return Workload(self.recipe, mv(self.logits), mv(self.targets),
                        mv(self.rollout_logprobs), mv(self.ref_logprobs),
                        mv(self.old_logprobs), mv(self.teacher_logprobs),
                        mv(self.rewards), mv(self.group_id), mv(self.cu_seqlens),
                        mv(self.loss_mask), self.n_groups, dict(self.params),
                        mv(self.topk_ids), mv(self.topk_teacher))


def _rewards(kind: str, n_traj: int, group_size: int, rng: np.random.Generator):
    if kind == "bernoulli0.5":
        return (rng.random(n_traj) < 0.5).astype(np.float32)
    if kind == "bernoulli0.3":
        return (rng.random(n_traj) < 0.3).astype(np.float32)
    if kind == "uniform":
        return rng.random(n_traj).astype(np.float32)
    if kind == "normal":
        return rng.standard_normal(n_traj).astype(np.float32)
    if kind == "uniform_eq8":
        # U[0,1], and every 8th group gets the constant 0.5 for all members:
        # equal-reward groups with no advantage signal.
        w = rng.random(n_traj).astype(np.float32)
        n_groups = n_traj // group_size
        for g in range(0, n_groups, 8):
            w[g * group_size:(g + 1) * group_size] = 0.5
        return w
    raise ValueError(kind)


def _mask(kind: str, n_traj: int, traj_len: int, rng: np.random.Generator):
    m = np.ones((n_traj, traj_len), dtype=np.uint8)
    if kind == "prefix_u32_128":
        for i in range(n_traj):
            m[i, :min(traj_len, int(rng.integers(32, 129)))] = 0
    elif kind == "prefix_frac0.25":
        m[:, :traj_len // 4] = 0
    elif kind == "prefix_u0_half":
        # prompt prefixes of U[0, traj_len/2] tokens: unequal training lengths
        for i in range(n_traj):
            m[i, :int(rng.integers(0, traj_len // 2 + 1))] = 0
    elif kind == "tool_spans":
        # Model-token spans U[64,512] alternate with masked tool-output spans
        # U[128,2048], starting with a model span.
        for i in range(n_traj):
            pos, model = 0, True
            while pos < traj_len:
                n = int(rng.integers(64, 513)) if model else int(rng.integers(128, 2049))
                if not model:
                    m[i, pos:pos + n] = 0
                pos += n
                model = not model
    elif kind == "none":
        pass
    else:
        raise ValueError(kind)
    return m.reshape(-1)


def exact_target_logprobs(logits: torch.Tensor, targets: torch.Tensor, vocab: int,
                          temperature: float, chunk_rows: int = 512) -> torch.Tensor:
    """Sampled-token log-probs of the rounded logits, in float64, via torch's
    library logsumexp; used only to build the perturbed rollout/ref inputs."""
    R = logits.shape[0]
    out = torch.empty(R, dtype=torch.float64, device=logits.device)
    for lo in range(0, R, chunk_rows):
        hi = min(R, lo + chunk_rows)
        s = logits[lo:hi, :vocab].to(torch.float64) / temperature
        tgt = s.gather(1, targets[lo:hi].long().unsqueeze(1)).squeeze(1)
        out[lo:hi] = tgt - torch.logsumexp(s, dim=1)
    return out


def make(rec: Recipe, device="cpu", ld: int | None = None) -> Workload:
    """Draw one batch of a recipe on ``device`` (seeded by ``rec.seed``)."""
    R, V, n_traj = rec.n_rows, rec.vocab, rec.n_traj
    ld = V if ld is None else ld
    assert ld >= V
    rng = np.random.Generator(np.random.PCG64(rec.seed))
    gen = torch.Generator(device=device)
    gen.manual_seed(rec.seed)

    tdt = torch.bfloat16 if rec.dtype == "bf16" else torch.float32
    logits = torch.empty((R, ld), dtype=tdt, device=device)
    if ld > V:
        logits[:, V:] = float("nan")  # padding is never read
    chunk = max(1, (1 << 26) // max(V, 1))
    for lo in range(0, R, chunk):
        hi = min(R, lo + chunk)
        z = torch.randn((hi - lo, V), generator=gen, device=device, dtype=torch.float32)
        logits[lo:hi, :V] = (z * rec.logit_std).to(tdt)
    targets = torch.randint(0, V, (R,), generator=gen, device=device, dtype=torch.int64)
    if rec.boost_frac > 0.0:
        sel = torch.rand(R, generator=gen, device=device) < rec.boost_frac
        rows = torch.nonzero(sel).squeeze(1)
        cols = targets[rows]
        boosted = (logits[rows, cols].to(torch.float32) + rec.boost).to(tdt)
        logits[rows, cols] = boosted
    targets = targets.to(torch.int32)

    T = float(rec.params.get("temperature", 1.0))
    exact = exact_target_logprobs(logits, targets, V, T)

    def noisy(sd):
        e = torch.randn(R, generator=gen, device=device, dtype=torch.float64) * sd
        return (exact + e).to(torch.float32)

    rho = noisy(rec.rho_noise)
    ref = noisy(rec.ref_noise) if rec.ref_noise is not None else None
    old = noisy(rec.old_noise) if rec.old_noise is not None else None
    teacher = noisy(rec.teacher_noise) if rec.teacher_noise is not None else None

    topk_ids = topk_teacher = None
    if rec.topk > 0:
        # the student's K most likely tokens and the teacher's log-probs of them
        K = min(rec.topk, V)
        topk_ids = torch.empty((R, K), dtype=torch.int32, device=device)
        topk_teacher = torch.empty((R, K), dtype=torch.float32, device=device)
        for lo in range(0, R, 512):
            hi = min(R, lo + 512)
            s = logits[lo:hi, :V].to(torch.float64) / T
            vals, ids = torch.topk(s, K, dim=1)
            lps = vals - torch.logsumexp(s, dim=1, keepdim=True)
            e = torch.randn((hi - lo, K), generator=gen, device=device, dtype=torch.float64)
            topk_ids[lo:hi] = ids.to(torch.int32)
            topk_teacher[lo:hi] = (lps + rec.topk_noise * e).to(torch.float32)

    w = _rewards(rec.reward, n_traj, rec.group_size, rng)
    gid = (np.arange(n_traj) // rec.group_size).astype(np.int32)
    cu = (np.arange(n_traj + 1) * rec.traj_len).astype(np.int32)
    mask = _mask(rec.mask, n_traj, rec.traj_len, rng)

    def dev(a):
        return torch.from_numpy(a).to(device)

    return Workload(rec, logits, targets, rho, ref, old, teacher, dev(w), dev(gid),
                    dev(cu), dev(mask), rec.n_prompts, dict(rec.params), topk_ids, topk_teacher)
