#!/usr/bin/env python
"""Throughput of the fused RL-loss forward+backward on GB300.

One step = one rl_loss_fwd_bwd call (advantage kernel, fused vocabulary
sweep, statistics kernel) over one synthetic batch shaped like the paper's
long agentic sessions: 65,536 rows (64 trajectories x 1,024 tokens, groups
of 16) x vocabulary 154,880, bf16 logits -> bf16 dLogits, dual clip 3, k3
KL 0.01 (the "glm" recipe of paper_2609_08368_gb300.workloads).

Prints one JSON line (rank 0). Under torchrun every rank runs its own
independent batch (weak scaling; the loss has no exchange between
replicas). ``--impl reference`` times the float64 CPU oracle instead.
"""

from __future__ import annotations

import argparse
import dataclasses
import hashlib
import json
import os
import re
import shutil
import statistics
import subprocess
import sys
import tempfile
import time

import numpy as np
import torch

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "RL-loss fwd+bwd tokens/sec at vocab 154,880 bf16; achieved HBM GB/s vs 8 TB/s"
NOMINAL_HBM_GBS = 8000.0
FALLBACK_HBM_GBS = 6800.0
PROFILE_SUMMARY = os.path.join(ROOT, "profiles", "stream_kernel_glm.md")
SWEEP_SOURCES = ["k_stream.cu", "stream_plan.h", "common.cuh", "kernels.h"]  # the kernel and its launch plan


def parse_args():
    ap = argparse.ArgumentParser()
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=200)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="glm")
    ap.add_argument("--e2e-steps", type=int, default=10)
    ap.add_argument("--e2e-chunk-rows", type=int, default=4096)
    ap.add_argument("--e2e-depth", type=int, default=2,
                    help="device chunk buffers of the pipelined host-buffer call")
    ap.add_argument("--cpu-sample-rows", type=int, default=0,
                    help="time the CPU oracle on this many random rows (0: on every row)")
    ap.add_argument("--no-e2e", action="store_true")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--n-prompts", type=int, default=None,
                    help="fewer groups (a smaller case of the same workload, for profiling)")
    ap.add_argument("--traj-len", type=int, default=None,
                    help="shorter trajectories (a smaller case, for profiling)")
    ap.add_argument("--vocab", type=int, default=None,
                    help="another vocabulary size (other row lengths, for profiling the "
                         "launch plans)")
    ap.add_argument("--estimator", default=None,
                    choices=["grpo", "reinforcepp", "reinforcepp_baseline", "gspo"],
                    help="another advantage estimator than the workload's (for profiling "
                         "the kernels of that path)")
    ap.add_argument("--sweep-kernel", choices=["cluster", "stream"], default=None,
                    help="force the vocabulary-sweep kernel (a launch-plan override, for "
                         "profiling the kernel the library would not pick)")
    ap.add_argument("--stream-cluster", type=int, default=None,
                    help="measurement aid: CTAs per row of the streaming kernel (1, 2, 4, 8; "
                         "fused calls without top-K)")
    ap.add_argument("--opd-topk", type=int, default=0,
                    help="top-K on-policy distillation with K candidates per row, coefficient "
                         "0.5 (for profiling the sweeps' top-K instantiations)")
    return ap.parse_args()


# ---------------------------------------------------------------- plumbing

def dist_setup():
    world = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    if world > 1:
        import torch.distributed as dist
        backend = "nccl" if torch.cuda.is_available() else "gloo"
        if backend == "nccl":
            torch.cuda.set_device(local)
        dist.init_process_group(backend=backend)
    elif torch.cuda.is_available():
        torch.cuda.set_device(local)
    return rank, world, local


def barrier(world):
    if world > 1:
        import torch.distributed as dist
        dist.barrier()


def max_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def sum_over_ranks(x: float, world: int) -> float:
    if world == 1:
        return x
    import torch.distributed as dist
    dev = "cuda" if dist.get_backend() == "nccl" else "cpu"
    t = torch.tensor([x], dtype=torch.float64, device=dev)
    dist.all_reduce(t, op=dist.ReduceOp.SUM)
    return float(t.item())


class ClockSampler:
    """nvidia-smi samples of the SM clock and throttle reasons while the
    timed region runs."""

    FIELDS = ("clocks.sm,clocks.max.sm,power.draw,clocks_event_reasons.active,"
              "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
              "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")
    REASONS = ("hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap")

    def __init__(self, device_index: int, period_ms: int = 50):
        self.proc = None
        self.path = None
        exe = shutil.which("nvidia-smi")
        if exe is None:
            return
        fd, self.path = tempfile.mkstemp(suffix=".csv")
        os.close(fd)
        self.cmd = [exe, "-i", str(device_index), f"--query-gpu={self.FIELDS}",
                    "--format=csv,noheader,nounits", "-lms", str(period_ms)]

    def start(self):
        if self.path is None:
            return
        self.fh = open(self.path, "w")
        self.proc = subprocess.Popen(self.cmd, stdout=self.fh, stderr=subprocess.DEVNULL)
        time.sleep(0.3)

    def stop(self):
        if self.proc is None:
            return None
        time.sleep(0.1)
        self.proc.terminate()
        try:
            self.proc.wait(timeout=5)
        except subprocess.TimeoutExpired:
            self.proc.kill()
        self.fh.close()
        rows = []
        for line in open(self.path):
            parts = [p.strip() for p in line.split(",")]
            if len(parts) != 8:
                continue
            try:
                rows.append((float(parts[0]), float(parts[1]), parts[2], parts[4:]))
            except ValueError:
                continue
        os.unlink(self.path)
        if not rows:
            return None
        sm = [r[0] for r in rows]
        reasons = sorted({self.REASONS[i] for r in rows for i, v in enumerate(r[3])
                          if v.lower() == "active"})
        try:
            power = max(float(r[2]) for r in rows)
        except ValueError:
            power = None
        return {"sm_mhz": statistics.median(sm), "sm_max_mhz": max(r[1] for r in rows),
                "sm_mhz_min": min(sm), "samples": len(rows), "power_w_max": power,
                "reasons": reasons}


def measured_peaks():
    path = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(path):
        with open(path) as f:
            return json.load(f), "measured"
    return {"hbm_gbs": FALLBACK_HBM_GBS}, "fallback"


def sweep_source_hash() -> str:
    """Hash of the sweep kernel's code and launch plan, comments and
    whitespace left out (a comment edit does not change what was captured;
    none of these files has a comment marker inside a string literal)."""
    h = hashlib.sha256()
    for name in SWEEP_SOURCES:
        with open(os.path.join(ROOT, "paper_2609_08368_gb300", "csrc", name)) as f:
            text = f.read()
        text = re.sub(r"/\*.*?\*/", " ", text, flags=re.S)
        text = re.sub(r"//[^\n]*", " ", text)
        h.update(" ".join(text.split()).encode())
    return h.hexdigest()[:16]


def profiled_traffic(rows_now: int, workload: str, vocab: int):
    """DRAM bytes of one sweep launch from the committed ncu summary, if it
    was taken on the current kernel source and on this workload's recipe and
    vocabulary; scaled by rows if captured on a smaller case."""
    if not os.path.exists(PROFILE_SUMMARY):
        return None
    text = open(PROFILE_SUMMARY).read()
    src = re.search(r"source_sha256:\s*([0-9a-f]+)", text)
    tb = re.search(r"dram_bytes_per_launch:\s*([0-9.eE+]+)", text)
    rows = re.search(r"rows_per_launch:\s*([0-9]+)", text)
    wk = re.search(r"workload:\s*(\S+)", text)
    voc = re.search(r"vocab:\s*([0-9]+)", text)
    if not (src and tb and rows and wk and voc) or src.group(1) != sweep_source_hash():
        return None
    if wk.group(1) != workload or int(voc.group(1)) != vocab:
        return None
    return float(tb.group(1)) * rows_now / int(rows.group(1))


def stream_ctas(row_bytes: int, grad: bool, topk: bool = False, elem_size: int = 2) -> int:
    """Streaming CTAs per SM the library picks for 16-byte aligned rows of
    row_bytes (0: the cluster kernel): one from 192 KB (fused) or 200 KB
    (forward only), two or four on shorter rows, clusters in between and
    below 20 KB."""
    KB = 1024
    if grad:
        if row_bytes >= 192 * KB:
            return 1
        if elem_size == 4 and 136 * KB <= row_bytes:
            return 1  # fp32 rows in two equal chunks
        if elem_size == 4 and not topk and 120 * KB < row_bytes <= 136 * KB:
            return 2  # fp32 rows of 120-136 KB
        if 56 * KB < row_bytes <= 80 * KB:
            return 2
        if not topk and 20 * KB <= row_bytes <= 56 * KB:
            return 4
        return 0
    if row_bytes >= 200 * KB:
        return 1
    if row_bytes > 112 * KB:
        return 2
    if row_bytes > 56 * KB:
        return 2 if topk else 4
    return 4 if (not topk and row_bytes >= 20 * KB) else 0


def stream_cluster(row_bytes: int, grad: bool, topk: bool = False) -> int:
    """CTAs per row of the streaming kernel the library picks (a cluster of
    them on rows of 480 KB and more in fused calls without top-K)."""
    KB = 1024
    if not grad or topk:
        return 1
    if row_bytes >= 1280 * KB:
        return 4
    return 2 if row_bytes >= 480 * KB else 1


def sweep_kernel_name(vocab: int, elem_size: int, grad: bool = True, topk: bool = False,
                      forced: str | None = None, forced_cluster: int | None = None) -> str:
    """The sweep kernel the library picks for these (16-byte aligned) rows,
    or the one the sweep_kernel / stream_cluster overrides force."""
    kind = "fused fwd+bwd" if grad else "forward-only"
    per = stream_ctas(vocab * elem_size, grad, topk, elem_size)
    if forced == "cluster":
        per = 0
    elif forced == "stream":
        per = max(per, 1)
    clu = stream_cluster(vocab * elem_size, grad, topk)
    if forced_cluster and grad and not topk:
        clu = forced_cluster
    if per == 1 and clu > 1:
        return f"k_stream ({kind} vocabulary sweep, a cluster of {clu} CTAs per row)"
    if per == 1:
        return f"k_stream ({kind} vocabulary sweep, one CTA per row)"
    if per > 1:
        return f"k_stream ({kind} vocabulary sweep, one CTA per row, {per} CTAs per SM)"
    return f"k_sweep ({kind} vocabulary sweep, clusters sharing a row)"


def launches_per_call(params: dict, n_groups: int) -> int:
    """Kernels one fused call launches: group statistics (when there are
    groups), advantages, the sweep and the statistics; GSPO adds the
    per-trajectory pass and the gradient sweep."""
    n = 3 + (1 if n_groups > 8 else 0)  # up to 8 groups, k_advantages computes them itself
    return n + (2 if params.get("estimator", "grpo") == "gspo" else 0)


def algorithmic_bytes_per_row(w, dl_dtype) -> int:
    """Logits read once + dLogits written once + the per-row inputs and
    outputs (target, rollout log-prob, optional ref / old / teacher
    log-probs, mask byte, log-prob and entropy out, top-K OPD candidates)."""
    es_in = w.logits.element_size()
    es_out = torch.tensor([], dtype=dl_dtype).element_size()
    small = 4 + 4 + 1 + 4 + 4
    for t in (w.ref_logprobs, w.old_logprobs, w.teacher_logprobs):
        if t is not None:
            small += 4
    if w.topk_ids is not None:  # top-K OPD: candidate ids and teacher log-probs
        small += 8 * int(w.topk_ids.shape[1])
    return w.vocab * (es_in + es_out) + small


# ---------------------------------------------------------------- CPU oracle

def _widen_host(a: np.ndarray) -> np.ndarray:
    """bf16 bit patterns (uint16) or fp32 values as float64."""
    if a.dtype == np.uint16:
        return (a.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)
    return a.astype(np.float64)


def _oracle_rows_task(task):
    """One block of rows through the float64 oracle, in a worker process
    (spawned; it attaches to the parent's shared copy of the rows' logits,
    and of the GPU's dLogits of those rows when it is to compare them).
    Returns the rows' log-probs, entropies and lse, and for dLogits the count
    of entries outside 1e-2 relative / 1e-5 absolute and the largest
    error-to-bound ratio."""
    from multiprocessing import shared_memory

    import oracle

    (shm_z, shm_dl, shape, zdtype, dldtype, lo, hi, y, rho, q, old, A_row, mask, N, params,
     grad_loss) = task
    hz = shared_memory.SharedMemory(name=shm_z)
    hd = shared_memory.SharedMemory(name=shm_dl) if shm_dl else None
    try:
        z = np.ndarray(shape, dtype=zdtype, buffer=hz.buf)[lo:hi]
        o = oracle.rl_loss_rows(z, y, rho, q, A_row, mask, N, oracle.LossParams(**params),
                                grad_loss=grad_loss, old=old)
        out = dict(lo=lo, logp=o["logp"], H=o["H"], lse=o["lse"], n_bad=0, worst=0.0,
                   worst_at=None)
        if hd is not None:
            got = _widen_host(np.ndarray(shape, dtype=dldtype, buffer=hd.buf)[lo:hi])
            ref = o["dlogits"]
            ratio = np.abs(got - ref) / np.maximum(1e-2 * np.abs(ref), 1e-5)
            ratio[~np.isfinite(got)] = np.inf
            out["n_bad"] = int((ratio > 1.0).sum())
            i = np.unravel_index(int(np.argmax(ratio)), ratio.shape)
            out["worst"] = float(ratio[i])
            out["worst_at"] = (lo + int(i[0]), int(i[1]), float(got[i]), float(ref[i]))
    finally:
        hz.close()
        if hd is not None:
            hd.close()
    return out


def _oracle_worker_init():
    """Worker start-up: import the oracle and run it once on a tiny row so
    that first-call costs stay out of the timed samples."""
    import oracle

    oracle.rl_loss_rows(np.zeros((1, 8)), np.zeros(1, np.int64), np.zeros(1), None, np.zeros(1),
                        np.ones(1, bool), 1, oracle.LossParams())


class OraclePool:
    """A pool of spawned worker processes, one per host core this process
    may run on, that run the oracle on blocks of rows (spawned, so it may be
    started after CUDA initialisation)."""

    def __init__(self, workers: int | None = None):
        import multiprocessing as mp

        self.workers = workers or max(1, len(os.sched_getaffinity(0)))
        self.pool = (mp.get_context("spawn").Pool(self.workers, initializer=_oracle_worker_init)
                     if self.workers > 1 else None)
        if self.pool is not None:
            try:  # workers up and importing done; if they cannot start, run in this process
                self.pool.map_async(int, range(self.workers)).get(timeout=300)
            except Exception:  # noqa: BLE001
                self.pool.terminate()
                self.pool.join()
                self.pool, self.workers = None, 1

    def map(self, fn, tasks):
        if self.pool is None:
            return [fn(t) for t in tasks]
        return self.pool.map(fn, tasks, chunksize=1)

    def close(self):
        if self.pool is not None:
            self.pool.close()
            self.pool.join()


def _host_rows(t, rows):
    """Rows of a device tensor as a host numpy array (bf16 as uint16 bits)."""
    z = t[rows].cpu()
    if z.dtype == torch.bfloat16:
        return z.contiguous().view(torch.int16).numpy().view(np.uint16)
    return z.contiguous().numpy()


def oracle_rows(w, pool: OraclePool, rows=None, dlogits=None, grad_loss=1.0, block=2048,
                task_rows=32):
    """The float64 oracle over rows of a token-level workload (every row by
    default), with the call-wide advantages and N of the whole batch: the
    rows' log-probs, entropies and lse, and dLogits of every row computed
    (and, when the GPU's ``dlogits`` are given, compared entry by entry in
    the workers). The logits (and dLogits) go to the workers a block of rows
    at a time through shared memory. Returns a dict with the per-row arrays,
    the dLogits check, and ``seconds``: the wall time of the oracle's work
    (the blocks' host copies excluded)."""
    import oracle
    from multiprocessing import shared_memory

    p = oracle.LossParams(**w.params)

    def host(t):
        return None if t is None else t.cpu().numpy()

    R = w.n_rows
    rows = np.arange(R) if rows is None else np.asarray(rows)
    mask = host(w.loss_mask).astype(bool)
    _, A_row, _ = oracle.estimator_advantages(host(w.rewards), host(w.group_id), w.n_groups,
                                              host(w.cu_seqlens), mask, p)
    N = int(mask.sum())
    y, rho = host(w.targets), host(w.rollout_logprobs)
    q, old = host(w.ref_logprobs), host(w.old_logprobs)
    es = w.logits.element_size()
    blk = min(block, len(rows)) if len(rows) else 1
    hz = shared_memory.SharedMemory(create=True, size=max(1, blk * w.vocab * es))
    hd = None
    if dlogits is not None:
        hd = shared_memory.SharedMemory(create=True,
                                        size=max(1, blk * w.vocab * dlogits.element_size()))
    out = dict(logp=np.zeros(len(rows)), H=np.zeros(len(rows)), lse=np.zeros(len(rows)),
               n_bad=0, worst=0.0, worst_at=None, seconds=0.0, rows=rows, N=N, A_row=A_row)
    try:
        for b0 in range(0, len(rows), blk):
            sel = rows[b0:b0 + blk]
            n = len(sel)
            idx = torch.from_numpy(sel).to(w.logits.device)
            z = _host_rows(w.logits[:, :w.vocab], idx)
            zs = np.ndarray(z.shape, dtype=z.dtype, buffer=hz.buf)
            zs[:] = z
            dl_dtype = None
            if hd is not None:
                d = _host_rows(dlogits[:, :w.vocab], idx)
                ds = np.ndarray(d.shape, dtype=d.dtype, buffer=hd.buf)
                ds[:] = d
                dl_dtype = d.dtype
                del ds
            del zs
            tasks = []
            for lo in range(0, n, task_rows):
                hi = min(n, lo + task_rows)
                r = sel[lo:hi]
                tasks.append((hz.name, None if hd is None else hd.name, z.shape, z.dtype, dl_dtype,
                              lo, hi, y[r], rho[r], None if q is None else q[r],
                              None if old is None else old[r], A_row[r], mask[r], N,
                              dict(w.params), grad_loss))
            t0 = time.perf_counter()
            res = pool.map(_oracle_rows_task, tasks)
            out["seconds"] += time.perf_counter() - t0
            for o in res:
                lo = b0 + o["lo"]
                k = len(o["logp"])
                for key in ("logp", "H", "lse"):
                    out[key][lo:lo + k] = o[key]
                out["n_bad"] += o["n_bad"]
                if o["worst"] > out["worst"] or out["worst_at"] is None:
                    out["worst"] = o["worst"]
                    if o["worst_at"] is not None:
                        r0, col, g_, r_ = o["worst_at"]  # r0: the row within the block
                        out["worst_at"] = (int(sel[r0]), col, g_, r_)
    finally:
        hz.close()
        hz.unlink()
        if hd is not None:
            hd.close()
            hd.unlink()
    return out


def oracle_sample(w, n_rows: int, seed: int = 7, pool: "OraclePool | None" = None):
    """Times the float64 CPU oracle on ``n_rows`` random rows of the workload
    (every per-row output and dLogits of those rows, with the call-wide
    advantages and token count of the whole batch) on the pool's worker
    processes. Returns (rows/s, seconds, rows, cores)."""
    rng = np.random.default_rng(seed)
    rows = np.sort(rng.choice(w.n_rows, size=min(n_rows, w.n_rows), replace=False))
    own = pool is None
    pool = pool or OraclePool(workers=1)
    try:
        o = oracle_rows(w, pool, rows=rows)
    finally:
        if own:
            pool.close()
    return len(rows) / o["seconds"], o["seconds"], len(rows), pool.workers


def run_reference(args, rank, world):
    """The reference arm: the float64 CPU oracle as it stands, on the host
    cores, on bounded samples of the same workload."""
    if rank != 0:
        return
    from paper_2609_08368_gb300 import workloads as wl

    pool = OraclePool()  # spawned before any CUDA work
    rec = wl.RECIPES[args.workload]
    w = wl.make(rec, "cuda" if torch.cuda.is_available() else "cpu")
    rows_per_step = min(512, 32 * pool.workers)  # one 32-row block per worker
    try:
        for _ in range(args.warmup):
            oracle_sample(w, rows_per_step, seed=1, pool=pool)
        times = []
        for k in range(args.steps):
            _, dt, n, cores = oracle_sample(w, rows_per_step, seed=100 + k, pool=pool)
            times.append(dt)
    finally:
        pool.close()
    total = sum(times)
    value = rows_per_step * args.steps / total
    sample = (f"{rows_per_step} random rows of the {rec.n_rows} x {rec.vocab} batch per step "
              f"(all per-row outputs and dLogits; call-wide advantages and N), "
              f"{cores} worker processes")
    line = {"impl": "reference", "metric": METRIC, "value": value, "unit": "tokens/s",
            "n_gpus": world, "steps": args.steps, "warmup": args.warmup,
            "ms_per_step": 1e3 * total / args.steps,
            "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": "f64",
            "data": "synthetic",
            "config": {"workload": f"{args.workload}: {rec.n_rows} rows x vocab {rec.vocab}",
                       "rows": rec.n_rows, "vocab": rec.vocab},
            "cpu_baseline": {"value": value, "unit": "tokens/s", "cores": cores, "kind": "oracle",
                             "sample": sample},
            "e2e": {"value": value, "unit": "tokens/s", "h2d_bytes_per_step": 0,
                    "d2h_bytes_per_step": 0}}
    print(json.dumps(line), flush=True)


# ---------------------------------------------------------------- GPU arm

def _pinned_copy(w):
    """The workload's tensors copied into pinned host memory."""
    from paper_2609_08368_gb300 import workloads as wl

    def pin(t):
        if t is None:
            return None
        h = torch.empty(t.shape, dtype=t.dtype, pin_memory=True)
        h.copy_(t)
        return h
    return wl.Workload(w.recipe, pin(w.logits), pin(w.targets), pin(w.rollout_logprobs),
                       pin(w.ref_logprobs), pin(w.old_logprobs), pin(w.teacher_logprobs),
                       pin(w.rewards), pin(w.group_id), pin(w.cu_seqlens), pin(w.loss_mask),
                       w.n_groups, dict(w.params))


def e2e_host_memory_check(bytes_per_rank: int, ranks_on_host: int):
    """None if this host's available memory holds every local rank's pinned
    host buffers with a tenth to spare, else the reason to skip the e2e
    leg (pinning more than the host has would take the machine down)."""
    try:
        with open("/proc/meminfo") as f:
            avail = next(int(line.split()[1]) * 1024 for line in f
                         if line.startswith("MemAvailable:"))
    except (OSError, StopIteration, ValueError):
        return None
    need = bytes_per_rank * max(1, ranks_on_host)
    if need * 1.1 > avail:
        return (f"the e2e leg would pin {need / 1e9:.1f} GB of host memory for "
                f"{ranks_on_host} local rank(s), more than 0.9 x the {avail / 1e9:.1f} GB "
                f"available")
    return None


def copy_floor_ms(call, stream, steps: int, warm: bool = True) -> float:
    """Milliseconds per step of the pipelined call's logits and dLogits
    copies alone: per chunk of rows, the host-to-device copy of its logits on
    the input stream and, when the call copies dLogits back, the
    device-to-host copy of a dLogits buffer of the same rows on the output
    stream (after that chunk's input copy, as if the sweep took no time),
    through the call's own device buffers, so both directions run at once as
    in the call. What the call takes beyond this is what the sweep and the
    small copies add."""
    h = call.host
    R, V = h.n_rows, h.vocab

    def one():
        done = None
        for i, r0 in enumerate(range(0, R, call.chunk)):
            r1 = min(R, r0 + call.chunk)
            b, n = i % len(call.lg), r1 - r0
            with torch.cuda.stream(call.s_in):
                call.lg[b][:n].copy_(h.logits[r0:r1, :V], non_blocking=True)
                done = in_done = torch.cuda.Event()
                in_done.record(call.s_in)
            if call.dl is None:  # dLogits stay on the device: input copies only
                continue
            call.s_out.wait_event(in_done)
            with torch.cuda.stream(call.s_out):
                call.out["dlogits"][r0:r1].copy_(call.dl[b][:n], non_blocking=True)
                done = torch.cuda.Event()
                done.record(call.s_out)
        if done is not None:
            stream.wait_event(done)

    if warm:
        one()
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(steps):
        one()
    e1.record(stream)
    torch.cuda.synchronize()
    return e0.elapsed_time(e1) / steps


def vocab_tp2_timing(w, dev, dl_dtype, stream, reps: int = 10) -> dict:
    """The call as two column shards of its vocabulary (tensor parallelism 2,
    rl_loss_vocab_shard_fwd_bwd), both run one after the other on this GPU
    with the record exchange done on the device: each of two GPUs would
    spend about half of that (plus an all-gather of 16 B per row). Median of
    ``reps`` whole calls after 3 warm-ups."""
    from paper_2609_08368_gb300 import api, milesloss as ml, workloads as wl
    R, V, n_traj = w.n_rows, w.vocab, int(w.rewards.shape[0])
    half = (V // 2 + 7) // 8 * 8  # keeps the second shard's rows 16-byte aligned
    cols = [0, half, V]
    row = []
    for k in range(2):
        c0, c1 = cols[k], cols[k + 1]
        wk = wl.Workload(w.recipe, w.logits[:, c0:c1], w.targets, w.rollout_logprobs,
                         w.ref_logprobs, w.old_logprobs, w.teacher_logprobs, w.rewards,
                         w.group_id, w.cu_seqlens, w.loss_mask, w.n_groups, dict(w.params))
        b = api.alloc(R, n_traj, w.n_groups, dev, vocab=c1 - c0, dlogits_dtype=dl_dtype)
        row.append(api.VocabShard(wk, k, cols, b))
    shards = [row]
    for _ in range(3):
        api.vocab_sharded_fwd_bwd_local(shards)
    evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
           for _ in range(reps)]
    for b_, e_ in evs:
        b_.record(stream)
        api.vocab_sharded_fwd_bwd_local(shards)
        e_.record(stream)
    torch.cuda.synchronize()
    for s in row:
        err = ml.rl_loss_check_device_error(s.buf.workspace)
        if err:
            raise RuntimeError(f"device error (vocabulary shards): {ml.status_string(err)}")
    ms = statistics.median(b_.elapsed_time(e_) for b_, e_ in evs)
    del shards, row
    torch.cuda.empty_cache()
    return {"vocab_tp2_ms_per_shard": ms / 2,
            "vocab_tp2_how": "two column shards of the vocabulary, both on this GPU one after "
                             "the other; per shard: partial sweep, merge, gradient sweep, "
                             "statistics (the logits read twice, as in the split pair)"}


def e2e_leg(host_w, dev, args, stream, world, rows_all, dlogits_on_device: bool) -> dict:
    """The pipelined host-buffer call timed end to end, each timed step
    followed by one step of its copies alone (so that a change in the host
    link's rate during the measurement, from other processes on the host,
    falls on both)."""
    from paper_2609_08368_gb300 import api
    call = api.PipelinedHostCall(host_w, dev, chunk_rows=args.e2e_chunk_rows,
                                 depth=args.e2e_depth, dlogits_on_device=dlogits_on_device)
    call()
    copy_floor_ms(call, stream, 1)
    torch.cuda.synchronize()
    e0, e1 = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    call_ms, floor_steps = [], []
    barrier(world)
    for _ in range(args.e2e_steps):
        torch.cuda.synchronize()
        e0.record(stream)
        call()
        e1.record(stream)
        torch.cuda.synchronize()
        call_ms.append(e0.elapsed_time(e1))
        floor_steps.append(copy_floor_ms(call, stream, 1, warm=False))
    barrier(world)
    ms_e2e = max_over_ranks(statistics.fmean(call_ms), world)
    floor_ms = statistics.fmean(floor_steps)
    where = ("dLogits written to one device tensor; the per-row log-probs and entropies "
             "and the statistics copied back" if dlogits_on_device else
             "dLogits copied back to pinned host memory too, overlapped with the sweep")
    out = {"value": rows_all / (ms_e2e / 1e3), "unit": "tokens/s",
           "ms_per_step": ms_e2e, "steps": args.e2e_steps,
           "ms_per_step_each": call_ms, "copy_floor_ms_each": floor_steps,
           "how": f"logits from pinned host memory through rl_loss_fwd_bwd_rows in chunks of "
                  f"{args.e2e_chunk_rows} rows and {args.e2e_depth} device chunk buffers, "
                  f"the copies overlapped with the sweep; {where}",
           "h2d_bytes_per_step": call.bytes_in(), "d2h_bytes_per_step": call.bytes_out(),
           "copy_floor_ms": floor_ms, "frac_of_copy_floor": floor_ms / ms_e2e,
           # the host link's rate drops to a third or less for bursts of a few
           # hundred ms on some boxes, hitting the call and its copies alike:
           # the best step of each shows what the call adds on a steady link
           "best_ms_per_step": min(call_ms), "best_copy_floor_ms": min(floor_steps),
           "frac_of_copy_floor_best": min(floor_steps) / min(call_ms),
           "copy_floor_how": "the same logits (and, when they go back, dLogits) copied alone "
                             "on this box, in the same chunks, through the same device "
                             "buffers and copy streams (no sweep); one such step after each "
                             "timed step of the call"}
    del call
    return out


def run_ours(args, rank, world, local):
    from paper_2609_08368_gb300 import api, milesloss as ml, workloads as wl

    ml.load()
    ov = {}
    if args.sweep_kernel:
        ov["sweep_kernel"] = args.sweep_kernel
    if args.stream_cluster:
        ov["stream_cluster"] = args.stream_cluster
    if ov:
        ml.set_launch_overrides(**ov)
    dev = torch.device("cuda", local)
    rec = wl.RECIPES[args.workload]
    rec = wl.shrink(rec, n_prompts=args.n_prompts, traj_len=args.traj_len, vocab=args.vocab,
                    seed=rec.seed + 1000 * rank)  # each replica has its own batch
    if args.estimator:
        rec = dataclasses.replace(rec, params=dict(rec.params, estimator=args.estimator))
    if args.opd_topk:
        rec = dataclasses.replace(rec, topk=args.opd_topk,
                                  params=dict(rec.params, opd_topk=args.opd_topk, opd_coef=0.5))
    w = wl.make(rec, dev)
    R, V = w.n_rows, w.vocab
    dl_dtype = w.logits.dtype
    dt_name = "bf16" if w.logits.dtype == torch.bfloat16 else "f32"
    buf = api.alloc(R, int(w.rewards.shape[0]), w.n_groups, dev, vocab=V, dlogits_dtype=dl_dtype)
    stream = torch.cuda.current_stream()

    for _ in range(max(3, args.warmup)):
        api.fwd_bwd(w, buf)
    torch.cuda.synchronize()
    err = ml.rl_loss_check_device_error(buf.workspace)
    if err:
        raise RuntimeError(f"device error during warm-up: {ml.status_string(err)}")

    K = args.steps
    ev_sweep = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
                for _ in range(K)]
    for b, e in ev_sweep:  # torch creates the CUDA event handles on first record
        b.record(stream)
        e.record(stream)
    start, stop = torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True)
    clocks = ClockSampler(local)
    clocks.start()
    barrier(world)
    torch.cuda.synchronize()
    start.record(stream)
    for i in range(K):
        ml.rl_set_sweep_events(*ev_sweep[i])
        api.fwd_bwd(w, buf)
    stop.record(stream)
    torch.cuda.synchronize()
    barrier(world)
    ml.rl_set_sweep_events(None, None)
    clk = clocks.stop()
    ms_total = start.elapsed_time(stop)
    ms_total = max_over_ranks(ms_total, world)
    ms_step = ms_total / K
    sweep_ms = [b.elapsed_time(e) for b, e in ev_sweep]
    err = ml.rl_loss_check_device_error(buf.workspace)
    if err:
        raise RuntimeError(f"device error: {ml.status_string(err)}")
    stats = buf.read_stats()
    rows_all = sum_over_ranks(float(R), world)
    value = rows_all * K / (ms_total / 1e3)

    # the other two ways to call the loss, timed beside the fused call (median
    # of 20 after 3 warm-ups, whole call, CUDA events): the forward alone
    # (reads the logits once) and the split pair rl_loss_fwd + rl_loss_bwd
    # (reads them twice)
    also = {}
    for name, fn in (("fwd_only", lambda: api.fwd(w, buf)),
                     ("split_fwd_bwd", lambda: (api.fwd(w, buf), api.bwd(w, buf)))):
        for _ in range(3):
            fn()
        evs = [(torch.cuda.Event(enable_timing=True), torch.cuda.Event(enable_timing=True))
               for _ in range(20)]
        for b, e in evs:
            b.record(stream)
            fn()
            e.record(stream)
        torch.cuda.synchronize()
        also[name + "_ms"] = statistics.median(b.elapsed_time(e) for b, e in evs)
    err = ml.rl_loss_check_device_error(buf.workspace)
    if err:
        raise RuntimeError(f"device error: {ml.status_string(err)}")
    if w.params.get("estimator", "grpo") != "gspo" and not args.opd_topk:
        also.update(vocab_tp2_timing(w, dev, dl_dtype, stream))
    logit_bytes = R * V * w.logits.element_size()
    also["fwd_only_read_gbs"] = logit_bytes / (also["fwd_only_ms"] / 1e3) / 1e9
    also["split_fwd_bwd_tokens_per_s"] = R / (also["split_fwd_bwd_ms"] / 1e3)

    bpr = algorithmic_bytes_per_row(w, dl_dtype)  # before w is released for the e2e leg
    kernel_name = sweep_kernel_name(V, w.logits.element_size(), topk=bool(args.opd_topk),
                                    forced=args.sweep_kernel, forced_cluster=args.stream_cluster)
    w_params, n_groups = dict(w.params), w.n_groups
    step_bytes = bpr * R
    launch_bytes = step_bytes
    if w_params.get("estimator", "grpo") == "gspo":
        # GSPO's timed sweep is the forward-only one (k_seq and the gradient
        # sweep k_bwd follow it): it reads the logits and writes no dLogits
        launch_bytes = (bpr - V * torch.tensor([], dtype=dl_dtype).element_size()) * R
        kernel_name = sweep_kernel_name(V, w.logits.element_size(), grad=False,
                                        topk=bool(args.opd_topk), forced=args.sweep_kernel) + \
            ", GSPO's first pass (k_bwd reads the logits again for dLogits)"
    sweep_avg = statistics.fmean(sweep_ms)
    peaks, peak_kind = measured_peaks()
    peak = float(peaks["hbm_gbs"])
    achieved = launch_bytes / (sweep_avg / 1e3) / 1e9
    step_gbs = step_bytes / (ms_step / 1e3) / 1e9

    cpu = None
    # (the oracle's row pass covers the token-level estimators without
    # top-K OPD only)
    if rank == 0 and world == 1 and not args.no_cpu_baseline and \
            w.params.get("estimator", "grpo") != "gspo" and not args.opd_topk:
        pool = OraclePool()
        try:
            if args.cpu_sample_rows > 0:
                rps, secs, n, cores = oracle_sample(w, args.cpu_sample_rows, pool=pool)
                what = f"{n} random rows of the {R} x {V} batch"
            else:
                o = oracle_rows(w, pool)
                n, secs, cores = R, o["seconds"], pool.workers
                rps = R / secs
                what = f"all {R} rows of the {R} x {V} batch"
        finally:
            pool.close()
        cpu = {"value": rps, "unit": "tokens/s", "cores": cores, "kind": "oracle",
               "sample": f"{what} (every per-row output and dLogits of every row, with the "
                         f"call-wide advantages and N), {secs:.1f} s wall of oracle work on "
                         f"{cores} worker processes (the logits reach them through shared "
                         f"memory a block of rows at a time; those copies are not timed)"}

    # end to end through host buffers (pinned), one call per step
    e2e = None
    host_need = 2 * R * V * w.logits.element_size()  # pinned logits in, dLogits out
    host_skip = e2e_host_memory_check(host_need, int(os.environ.get("LOCAL_WORLD_SIZE", "1")))
    if host_skip and not args.no_e2e:
        e2e = {"skipped": host_skip}
    elif not args.no_e2e and args.e2e_steps > 0:
        host_w = _pinned_copy(w)
        del w, buf  # the pipelined call keeps its own chunk buffers
        torch.cuda.empty_cache()
        # the step's inputs from pinned host memory, its results (per-row
        # log-prob and entropy, the statistics) back; dLogits stay on the
        # device, where the trainer's backward pass reads them
        e2e = e2e_leg(host_w, dev, args, stream, world, rows_all, dlogits_on_device=True)
        torch.cuda.empty_cache()
        # the same with dLogits copied back to pinned host memory as well
        e2e["host_dlogits"] = e2e_leg(host_w, dev, args, stream, world, rows_all,
                                      dlogits_on_device=False)
        del host_w

    # the committed capture is of the default path (GRPO-style fused sweep,
    # no top-K): it does not describe the others
    traffic = None if (args.estimator or args.opd_topk or args.sweep_kernel or args.stream_cluster) \
        else profiled_traffic(R, args.workload, V)
    line = {
        "metric": METRIC, "value": value, "unit": "tokens/s", "n_gpus": world, "steps": K,
        "warmup": max(3, args.warmup), "ms_per_step": ms_step, "higher_is_better": True,
        "scaling": "weak", "vs_baseline": None, "dtype": dt_name, "data": "synthetic",
        "config": {"workload": f"{args.workload}: {R} rows ({rec.n_traj} traj x {rec.traj_len} "
                               f"tokens, groups of {rec.group_size}) x vocab {V}, "
                               f"{dt_name} logits "
                               f"-> dLogits",
                   "rows": R, "vocab": V, "parallelism": f"replicas x{world}",
                   **({"estimator": args.estimator} if args.estimator else {}),
                   **({"opd_topk": args.opd_topk} if args.opd_topk else {}),
                   **({"sweep_kernel": args.sweep_kernel} if args.sweep_kernel else {}),
                   **({"stream_cluster": args.stream_cluster} if args.stream_cluster else {}),
                   "l2": f"inputs larger than L2 ({step_bytes / 1e9:.1f} GB per step), "
                         "no flush"},
        "roofline": {"bound": "hbm", "achieved": achieved, "peak": peak, "unit": "GB/s",
                     "frac": achieved / peak, "traffic": traffic,
                     "kernel": kernel_name,
                     "bytes_per_launch": launch_bytes, "sweep_ms": sweep_avg,
                     "peak_kind": f"{peak_kind} copy bandwidth (MEASURED_PEAKS.json hbm_gbs)"
                     if peak_kind == "measured" else "fallback 6.8 TB/s",
                     "frac_of_8tbs": achieved / NOMINAL_HBM_GBS,
                     "traffic_gbs": None if traffic is None else traffic / (sweep_avg / 1e3) / 1e9},
        "step_hbm_gbs": step_gbs,
        "also": also,
        "cpu_baseline": cpu,
        "e2e": e2e,
        "gpu_launches": launches_per_call(w_params, n_groups) * K,
        "clocks": clk,
        "loss": stats["loss"],
    }
    if rank == 0:
        print(json.dumps(line), flush=True)


def main():
    args = parse_args()
    rank, world, local = dist_setup()
    try:
        if args.impl == "reference":
            run_reference(args, rank, world)
        else:
            run_ours(args, rank, world, local)
    finally:
        if world > 1:
            import torch.distributed as dist
            dist.destroy_process_group()


if __name__ == "__main__":
    main()
