"""Host-side helpers of bench.py and the tensor API, on CPU: the launch count
per call, the sweep-kernel naming rule, the profiled traffic's validity checks,
the algorithmic bytes per row, and the top-K parameter attachment."""

import dataclasses
import os
import sys

import torch

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
if ROOT not in sys.path:
    sys.path.insert(0, ROOT)

import bench  # noqa: E402
from paper_2609_08368_gb300 import api, workloads as wl  # noqa: E402


def test_launches_per_call():
    assert bench.launches_per_call({}, 4) == 3                     # glm: groups inline
    assert bench.launches_per_call({}, 64) == 4                    # fp32: k_groups too
    assert bench.launches_per_call({"estimator": "gspo"}, 4) == 5  # + k_seq, k_bwd
    assert bench.launches_per_call({"estimator": "reinforcepp"}, 1) == 3


def test_sweep_kernel_name_follows_the_plan_tiers():
    one, clusters = "one CTA per row)", "clusters sharing a row)"
    assert bench.sweep_kernel_name(154880, 2).endswith(one)
    assert bench.sweep_kernel_name(98304, 2).endswith(one)
    assert bench.sweep_kernel_name(98303, 2).endswith(clusters)      # bf16 80-192 KB
    assert bench.sweep_kernel_name(69632, 2).endswith(clusters)
    assert bench.sweep_kernel_name(34816, 4).endswith(one)           # fp32 136 KB: halves
    assert bench.sweep_kernel_name(38912, 4).endswith(one)           # fp32 152 KB
    assert bench.sweep_kernel_name(49151, 4).endswith(one)
    assert bench.sweep_kernel_name(40964, 2).endswith(clusters)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(32768, 4)      # fp32, 128 KB
    assert bench.sweep_kernel_name(65536, 2).endswith(clusters)      # bf16, 128 KB
    assert bench.sweep_kernel_name(32768, 4, topk=True).endswith(clusters)
    assert bench.sweep_kernel_name(36864, 4).endswith(one)           # fp32, 144 KB
    assert bench.sweep_kernel_name(57344, 2).endswith(clusters)      # bf16, 112 KB
    assert bench.sweep_kernel_name(49152, 4).endswith(one)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(32768, 2)      # 64 KB
    assert "2 CTAs per SM" in bench.sweep_kernel_name(40960, 2)      # 80 KB
    assert "4 CTAs per SM" in bench.sweep_kernel_name(28672, 2)      # 56 KB
    assert "4 CTAs per SM" in bench.sweep_kernel_name(16384, 2)      # 32 KB
    assert "4 CTAs per SM" in bench.sweep_kernel_name(10240, 2)      # 20 KB
    assert bench.sweep_kernel_name(10232, 2).endswith(clusters)      # below 20 KB
    assert bench.sweep_kernel_name(4096, 2).endswith(clusters)       # the tiny workload
    # with top-K OPD, no four-CTA plans
    assert bench.sweep_kernel_name(16384, 2, topk=True).endswith(clusters)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(32768, 2, topk=True)
    # forward-only calls: one CTA from 200 KB, two from 112 KB, four from 20 KB
    assert bench.sweep_kernel_name(154880, 2, grad=False).endswith(one)
    assert bench.sweep_kernel_name(102400, 2, grad=False).endswith(one)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(102392, 2, grad=False)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(77440, 2, grad=False)  # glm TP 2 shards
    assert "2 CTAs per SM" in bench.sweep_kernel_name(57348, 2, grad=False)
    assert "4 CTAs per SM" in bench.sweep_kernel_name(57344, 2, grad=False)
    assert "2 CTAs per SM" in bench.sweep_kernel_name(32768, 2, grad=False, topk=True)
    assert bench.sweep_kernel_name(8192, 2, grad=False).endswith(clusters)
    # the sweep_kernel override
    assert bench.sweep_kernel_name(32768, 4, forced="cluster").endswith(clusters)
    assert bench.sweep_kernel_name(65536, 2, forced="stream").endswith(one)
    # rows of 480 KB and more (fused, no top-K): a cluster of two, from 1.25 MB four
    assert bench.sweep_kernel_name(245759, 2).endswith(one)
    assert "a cluster of 2 CTAs per row" in bench.sweep_kernel_name(245760, 2)
    assert "a cluster of 2 CTAs per row" in bench.sweep_kernel_name(154880, 4)  # fp32, 620 KB
    assert "a cluster of 4 CTAs per row" in bench.sweep_kernel_name(655360, 2)
    assert bench.sweep_kernel_name(262144, 2, topk=True).endswith(one)
    assert bench.sweep_kernel_name(262144, 2, grad=False).endswith(one)
    # the stream_cluster override (fused calls without top-K only)
    assert "a cluster of 4 CTAs per row" in bench.sweep_kernel_name(154880, 2, forced_cluster=4)
    assert bench.sweep_kernel_name(154880, 2, topk=True, forced_cluster=4).endswith(one)


def test_profiled_traffic_only_for_its_workload_and_sources():
    t = bench.profiled_traffic(65536, "glm", 154880)
    # valid only while the sources hash to the capture's; scaled from the
    # captured rows to a full 65,536-row launch (40.6 GB algorithmic)
    assert t is None or 3.6e10 < t < 4.5e10
    assert bench.profiled_traffic(65536, "glm", 100000) is None
    assert bench.profiled_traffic(131072, "fp32", 32768) is None


def test_algorithmic_bytes_per_row():
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=2, traj_len=2, vocab=1000)
    w = wl.make(rec, "cpu")
    # bf16 in and out, plus target, rollout, ref log-prob, mask, logp and H out
    assert bench.algorithmic_bytes_per_row(w, torch.bfloat16) == 1000 * 4 + 4 + 4 + 4 + 1 + 4 + 4
    assert bench.algorithmic_bytes_per_row(w, torch.float32) == 1000 * 6 + 21
    # top-K OPD adds each row's K candidate ids and teacher log-probs
    rec = dataclasses.replace(rec, topk=4, params=dict(rec.params, opd_topk=4, opd_coef=0.5))
    w = wl.make(rec, "cpu")
    assert bench.algorithmic_bytes_per_row(w, torch.bfloat16) == 1000 * 4 + 21 + 4 * 8


def test_api_attaches_top_k_inputs():
    rec = wl.shrink(wl.RECIPES["glm"], n_prompts=1, group_size=2, traj_len=2, vocab=64, topk=4)
    w = wl.make(rec, "cpu")
    p = api._params(w, dict(w.params, opd_topk=4, opd_coef=0.5))
    assert p["opd_topk_ids"] is w.topk_ids and p["opd_topk_teacher"] is w.topk_teacher
    assert "opd_topk_ids" not in api._params(w, None)


def test_e2e_leg_is_skipped_when_the_host_cannot_pin_its_buffers():
    avail = next(int(line.split()[1]) * 1024 for line in open("/proc/meminfo")
                 if line.startswith("MemAvailable:"))
    assert bench.e2e_host_memory_check(avail // 4, 1) is None
    reason = bench.e2e_host_memory_check(avail, 1)
    assert reason and "host memory" in reason
    assert bench.e2e_host_memory_check(avail // 4, 8) is not None  # eight local ranks
