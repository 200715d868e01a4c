"""The streaming kernel's launch plan, checked on the host: stream_plan.h is
plain C++, so a small program built with the host compiler prints the plan
for every row length from 1 to 320 KB (and 16 bytes either side of each KB)
and on to 4 MB in steps of 32 KB, both element sizes, fused and forward-only
calls, top-K OPD on and off, at one GB300 SM's shared-memory limits. The plan
must fit the SM, keep no more chunks than it has slots, split long rows over a
cluster in whole 128-byte slices, and match the tiers bench.py names its
kernel by."""

import os
import shutil
import subprocess

import pytest

import bench

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))
OPTIN, PER_SM, RESERVED = 232448, 233472, 1024


@pytest.fixture(scope="module")
def table(tmp_path_factory):
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path_factory.mktemp("plan") / "stream_plan_table")
    subprocess.run([cxx, "-std=c++17", "-O1", "-Wall", "-Werror",
                    "-I", os.path.join(ROOT, "paper_2609_08368_gb300", "csrc"),
                    "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "stream_plan_table.cpp"), "-o", exe], check=True)
    out = subprocess.run([exe], check=True, capture_output=True, text=True).stdout
    keys = ("es", "grad", "topk", "row", "ctas", "ok", "chunk", "slots", "hold", "split",
            "smem", "cw", "cluster", "slice_vec")
    return [dict(zip(keys, map(int, line.split()))) for line in out.splitlines()]


def test_every_default_plan_fits_one_sm(table):
    assert len(table) == 2 * 2 * 2 * (320 + 118) * 3
    for p in table:
        assert p["ok"] == 1, p
        per = max(1, p["ctas"])
        assert p["cw"] * per == 16, p
        assert p["chunk"] % 128 == 0 and 1024 <= p["chunk"] <= 131072, p
        assert 1 <= p["slots"] <= 16 and 0 <= p["hold"] <= p["slots"], p
        extra = 1024 if p["topk"] else 0
        assert p["smem"] == p["slots"] * p["chunk"] + 1024 + extra, p
        assert p["smem"] <= OPTIN, p
        if per > 1:  # `per` CTAs fit one SM's shared memory
            assert per * (p["smem"] + RESERVED) <= PER_SM, p


def test_tiers_match_the_bench_names(table):
    for p in table:
        want = bench.stream_ctas(p["row"], bool(p["grad"]), bool(p["topk"]), p["es"])
        assert p["ctas"] == want, p
        assert p["cluster"] == bench.stream_cluster(p["row"], bool(p["grad"]), bool(p["topk"])), p


def test_long_rows_split_over_clusters_in_whole_slices(table):
    """Rows of 480 KB and more in fused calls without top-K run on a cluster
    of two (four from 1.25 MB) CTAs, one per SM, each with a slice of the row
    that starts on a 128-byte boundary; the slices cover the row's whole
    vectors and each CTA's ring is the one-CTA ring of its slice's length."""
    seen = set()
    for p in table:
        C = p["cluster"]
        if not p["grad"] or p["topk"] or p["row"] < 480 * 1024:
            assert C == 1, p
            continue
        assert C == (4 if p["row"] >= 1280 * 1024 else 2), p
        seen.add(C)
        vec = p["row"] // 16
        sv = p["slice_vec"]
        assert sv % 8 == 0 and sv * C >= vec and sv * (C - 1) < vec, p
        assert p["cw"] == 16, p
        assert p["chunk"] == (75776 if sv * 16 >= 240 * 1024 else 114688), p
    assert seen == {2, 4}


def _plan(table, es, grad, topk, row):
    return next(p for p in table if (p["es"], p["grad"], p["topk"], p["row"]) ==
                (es, grad, topk, row))


def test_plans_of_the_workloads(table):
    # rows like glm's (154,880 bf16 columns = 302.5 KB): one CTA, three 74 KB
    # slots, the last two chunks kept, the ragged chunk first
    p = _plan(table, 2, 1, 0, 303 * 1024 - 16)
    assert (p["ctas"], p["chunk"], p["slots"], p["hold"], p["split"]) == (1, 75776, 3, 2, 1)
    # fp32 workload rows (32,768 columns = 128 KB): two CTAs, six 18 KB slots, three kept
    p = _plan(table, 4, 1, 0, 128 * 1024)
    assert (p["ctas"], p["chunk"], p["slots"], p["hold"]) == (2, 18432, 6, 3)
    # fp32 rows of 144 KB: one CTA, the row in two equal chunks, none kept
    p = _plan(table, 4, 1, 0, 144 * 1024)
    assert (p["ctas"], p["chunk"], p["slots"], p["hold"]) == (1, 73728, 3, 0)
    # bf16 rows of 64 KB: two CTAs, three 36 KB slots; of 32 KB: four CTAs, 16 KB slots
    p = _plan(table, 2, 1, 0, 64 * 1024)
    assert (p["ctas"], p["chunk"], p["slots"]) == (2, 36864, 3)
    p = _plan(table, 2, 1, 0, 32 * 1024)
    assert (p["ctas"], p["chunk"], p["slots"], p["hold"]) == (4, 16384, 3, 1)
    # a 24 KB row is one chunk
    p = _plan(table, 2, 1, 0, 24 * 1024)
    assert (p["ctas"], p["chunk"]) == (4, 24576)
    # glm rows split over two vocabulary shards (77,440 columns = 151.25 KB),
    # forward only: two CTAs
    p = _plan(table, 2, 0, 0, 151 * 1024 + 16)
    assert p["ctas"] == 2


def test_fused_and_forward_rows_up_to_56kb_take_the_same_chunks(table):
    """So that a forward-only call sums a row in the same order as the fused
    call, and both give the same bits."""
    for p in table:
        if p["grad"] == 1 and p["topk"] == 0 and p["ctas"] == 4:
            q = _plan(table, p["es"], 0, 0, p["row"])
            assert q["ctas"] == 4 and q["chunk"] == p["chunk"] and q["split"] == p["split"], (p, q)


def test_forced_plans_of_a_long_row(tmp_path):
    """A 512 KB fused bf16 row (a cluster of two by default) under the
    overrides: forced CTAs per SM above one give one CTA per row (not an
    error), a forced cluster size is taken, forcing both is refused, and a
    top-K call stays on one CTA per row whatever the cluster override."""
    cxx = shutil.which("g++") or shutil.which("c++")
    if cxx is None:
        pytest.skip("no host C++ compiler")
    exe = str(tmp_path / "stream_plan_table")
    subprocess.run([cxx, "-std=c++17", "-O1", "-Wall", "-Werror",
                    "-I", os.path.join(ROOT, "paper_2609_08368_gb300", "csrc"),
                    "-I", os.path.join(ROOT, "include"),
                    os.path.join(ROOT, "tests", "stream_plan_table.cpp"), "-o", exe], check=True)
    out = subprocess.run([exe, "forced"], check=True, capture_output=True, text=True).stdout
    got = {tuple(map(int, line.split()[:3])): tuple(map(int, line.split()[3:]))
           for line in out.splitlines()}
    assert got[(-1, -1, 0)] == (1, 2, 16)    # the library's plan: two CTAs per row
    assert got[(2, -1, 0)] == (1, 1, 8)      # two CTAs per SM forced: one CTA per row
    assert got[(4, -1, 0)] == (1, 1, 4)
    assert got[(1, -1, 0)] == (1, 2, 16)     # one CTA per SM forced: the cluster stays
    assert got[(-1, 4, 0)] == (1, 4, 16)     # a cluster of four forced
    assert got[(1, 8, 0)] == (1, 8, 16)
    assert got[(2, 2, 0)][0] == 0            # both forced: no plan
    assert got[(-1, 4, 1)] == (1, 1, 16)     # top-K: one CTA per row
    assert got[(-1, 1, 0)] == (1, 1, 16)     # clusters forced off
