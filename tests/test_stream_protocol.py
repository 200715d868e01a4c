"""A host model of the streaming sweep kernel's shared-memory ring protocol
(csrc/k_stream.cu), checked without a GPU.

Four parties share the ring: the producer issues one bulk copy per task into
slot task % n_slots once every reader has released the task n_slots before;
the consumers wait for each task, release it, and meet the top-K warp once
per row (hand-off of the row's top-K part); the top-K warp (top-K OPD only)
waits for and releases every task too. Per row of n chunks, a row that
trains has tasks for pass A (chunks 0 .. n-1) and then for pass B's second
copies (chunks n-h-1 .. 0); pass B takes the last h chunks from the slots
pass A left them in, so the consumers release those only after pass B. The
model checks that every task a party waits for carries the chunk it expects,
that every task is released exactly once by every reader, that the hand-off
buffers are never overwritten before they are read, and that no wait can
block forever, over chunk counts, slot counts, kept chunks and masks."""

import random

import pytest


def producer_tasks(masks, n, grad, hold):
    for row, m in enumerate(masks):
        again = grad and m and n > 0
        h = min(hold, n) if again else 0
        for t in range(2 * n - h if again else n):
            yield row, (t if t < n else 2 * n - h - 1 - t)


def consumer_ops(masks, n, grad, hold):
    q0 = 0
    for row, m in enumerate(masks):
        trains = grad and m and n > 0
        h = min(hold, n) if trains else 0
        for c in range(n):
            yield "wait", q0 + c, (row, c)
            if c < n - h:
                yield "release", q0 + c
        yield "take_part", row
        if grad:
            order = []
            for j in range(n):
                c = n - h + j if j < h else n - 1 - j
                qq = q0 + n - h + j if j < h else q0 + n + (j - h)
                order.append(c)
                if m:
                    yield "wait", qq, (row, c)
                    yield "release", qq
            assert sorted(order) == list(range(n))
        q0 += 2 * n - h if (grad and m) else n


def topk_ops(masks, n, grad, hold):
    q0 = 0
    for row, m in enumerate(masks):
        trains = grad and m and n > 0
        h = min(hold, n) if trains else 0
        for c in range(n):
            yield "wait", q0 + c, (row, c)
            yield "release", q0 + c
        yield "give_part", row
        if grad and m:
            for j in range(h, n):
                qq = q0 + n + (j - h)
                yield "wait", qq, None
                yield "release", qq
        q0 += 2 * n - h if (grad and m) else n


def simulate(masks, n, grad, n_slots, hold, topk, consumer=consumer_ops):
    tasks = list(producer_tasks(masks, n, grad, hold))
    readers = [list(consumer(masks, n, grad, hold))]
    if topk:
        readers.append(list(topk_ops(masks, n, grad, hold)))
    pos = [0] * len(readers)
    released = [set() for _ in readers]
    issued = 0
    given, taken = set(), set()
    while True:
        progress = False
        while issued < len(tasks) and (issued < n_slots or
                                       all(issued - n_slots in r for r in released)):
            issued += 1
            progress = True
        for a, ops in enumerate(readers):
            while pos[a] < len(ops):
                op = ops[pos[a]]
                if op[0] == "wait":
                    if op[1] >= issued:
                        break
                    if op[2] is not None:
                        assert tasks[op[1]] == op[2], (op, tasks[op[1]])
                elif op[0] == "release":
                    assert op[1] < issued and op[1] not in released[a]
                    released[a].add(op[1])
                elif op[0] == "give_part":
                    # the part of row r goes to buffer r % 2 once row r - 2's
                    # part has been taken
                    if op[1] >= 2 and op[1] - 2 not in taken:
                        break
                    given.add(op[1])
                elif op[0] == "take_part" and topk:
                    if op[1] not in given:
                        break
                    taken.add(op[1])
                pos[a] += 1
                progress = True
        if issued == len(tasks) and all(p == len(o) for p, o in zip(pos, readers)):
            break
        assert progress, "a wait that never ends"
    for r in released:
        assert r == set(range(len(tasks)))


@pytest.mark.parametrize("topk", [False, True])
@pytest.mark.parametrize("grad", [False, True])
def test_ring_protocol(grad, topk):
    rng = random.Random(7)
    for n in range(0, 7):
        for n_slots in range(1, 6):
            for hold in range(0, n_slots + 1):
                for _ in range(12):
                    masks = [rng.random() < 0.6 for _ in range(rng.randint(0, 7))]
                    simulate(masks, n, grad, n_slots, hold, topk)


def test_model_catches_a_wrong_pass_b_order():
    """The model fails when pass B asks for a chunk the producer did not
    bring (here: the consumers walk the second copies first to last)."""
    def bad_consumer(masks, n, grad, hold):
        h = min(hold, n)
        for op in consumer_ops(masks, n, grad, hold):
            if op[0] == "wait" and op[1] >= n:
                row, c = op[2]
                yield "wait", op[1], (row, n - h - 1 - c)
            else:
                yield op
    simulate([True], 4, True, 3, 1, False)
    with pytest.raises(AssertionError):
        simulate([True], 4, True, 3, 1, False, consumer=bad_consumer)


@pytest.mark.parametrize("split_first", [0, 1])
def test_chunk_split(split_first):
    """Chunk boundaries: every vector in exactly one chunk, no chunk empty or
    larger than a slot; with the ragged chunk first, every later chunk starts
    on a 128-byte (8-vector) boundary."""
    for row_vec in list(range(1, 300)) + [19360, 18992, 16384, 12500]:
        for cv in (64, 72, 3584, 4736, 7168):
            n = (row_vec + cv - 1) // cv
            rem = row_vec - (n - 1) * cv
            f0 = min(cv, (rem + 7) & ~7) if split_first else cv

            def cs(c):
                return 0 if c == 0 else min(row_vec, f0 + (c - 1) * cv)

            sizes = [cs(c + 1) - cs(c) for c in range(n)]
            assert sum(sizes) == row_vec and all(1 <= x <= cv for x in sizes)
            if split_first and n > 1:
                assert all(cs(c) % 8 == 0 for c in range(n))


# --------------------------------------------------------------------------
# The give-up path: every party's waits, with one of them running out.
#
# A finer model than the one above: the ring's "full" and "empty" barriers
# count completed phases and are waited on by parity, as the kernel's
# mbarriers are; copies land at arbitrary later times; two consumer warps
# (the first one also takes the top-K hand-off) and the top-K warp arrive
# separately on "empty"; the consumers meet at a barrier twice per row. One
# chosen wait (or the test hook's stall of the consumers' first wait) gives
# up, which sets the CTA's flag; every later wait of every party that may
# end early (all but the producer's waits for its own copies) then returns
# at once. Checked over random schedules: no copy is issued into a slot while
# the copy issued there before is still in flight or a reader still holds
# the slot, a reader reads only the chunk of the task it waited for, every
# wait either completes, ends because of the flag or is the one chosen to
# run out (no wait needs a timeout of its own), no parity wait is fooled by
# a barrier two phases ahead, and when the producer returns no copy is in
# flight. A reader that gave up still releases its tasks (unread: what it
# computes from them is discarded, the rows are written as zeros), so the
# producer checks the flag after every completed wait before it re-arms a
# slot.
# --------------------------------------------------------------------------


class _Barrier:
    def __init__(self, count):
        self.count = count
        self.pending = count
        self.phase = 0  # completed phases

    def arrive(self):
        self.pending -= 1
        if self.pending == 0:
            self.phase += 1
            self.pending = self.count

    def test(self, k):
        """try_wait.parity for phase k: (parity answer, true answer)."""
        return (self.phase & 1) != (k & 1), self.phase > k


class _GiveUpSim:
    def __init__(self, masks, n, grad, NS, hold, topk, fail_site=None, stall=False, seed=0,
                 n_cons=2):
        self.masks, self.n, self.grad, self.NS, self.hold, self.topk = masks, n, grad, NS, hold, topk
        self.rng = random.Random(seed)
        self.tasks = list(producer_tasks(masks, n, grad, hold))
        self.fail_site = fail_site
        self.stall = stall
        self.abort = False
        self.failed = False
        self.readers = [f"C{i}" for i in range(n_cons)] + (["T"] if topk else [])
        self.full = [_Barrier(1) for _ in range(NS)]
        self.full_issued = [0] * NS  # copies issued into each slot
        self.empty = [_Barrier(len(self.readers)) for _ in range(NS)]
        self.tk_full = [_Barrier(1), _Barrier(1)]
        self.tk_empty = [_Barrier(1), _Barrier(1)]
        self.inflight = {}      # slot -> task of the copy not yet landed
        self.content = {}       # slot -> task whose chunk the slot holds
        self.holding = {r: set() for r in self.readers}
        self.wait_count = {}
        self.sync_arrived = {}  # barrier generation -> consumer warps arrived
        self.sync_gen = {}      # consumer warp -> generations it has arrived at
        self.producer_done = False

    # ---- parties (generators yielding requests, as the kernel's code runs)
    def producer(self):
        NS, n = self.NS, self.n
        q, stop = 0, False
        for m in self.masks:
            if stop:
                break
            again = self.grad and m and n > 0
            h = min(self.hold, n) if again else 0
            for _ in range(2 * n - h if again else n):
                s = q % NS
                if q >= NS:
                    ok = yield ("wait", self.empty[s], q // NS - 1, True, ("P", "empty"))
                    if not ok or self.abort:  # a reader may have released unread
                        stop = True
                        break
                yield ("issue", q)
                q += 1
        for s in range(NS):
            if q > s:
                last = q - 1 - ((q - 1 - s) % NS)
                yield ("wait", self.full[s], last // NS, False, ("P", "drain"))
        yield ("producer_done",)

    def consumer(self, me, warp0):
        NS, n = self.NS, self.n
        q0 = 0
        for i, m in enumerate(self.masks):
            trains = self.grad and m and n > 0
            h = min(self.hold, n) if trains else 0
            for c in range(n):
                q = q0 + c
                if i == 0 and c == 0 and self.stall:
                    yield ("wait", None, 0, True, (me, "stall"))
                    ok = False
                else:
                    ok = yield ("wait", self.full[q % NS], q // NS, True, (me, "full"))
                if ok:
                    yield ("read", me, q, self.tasks[q])
                if c < n - h:
                    yield ("release", me, q)
            gen = yield ("sync_arrive", me)
            yield ("sync_wait", gen)
            if self.topk and warp0:
                ok = yield ("wait", self.tk_full[i & 1], i >> 1, True, (me, "tk_full"))
                yield ("arrive", self.tk_empty[i & 1])
            gen = yield ("sync_arrive", me)
            yield ("sync_wait", gen)
            if self.grad:
                for j in range(n):
                    c = n - h + j if j < h else n - 1 - j
                    qq = q0 + n - h + j if j < h else q0 + n + (j - h)
                    if m and n > 0:
                        ok = yield ("wait", self.full[qq % NS], qq // NS, True, (me, "full"))
                        if ok:
                            yield ("read", me, qq, self.tasks[qq])
                        yield ("release", me, qq)
            q0 += 2 * n - h if (self.grad and m and n > 0) else n
        yield ("done", me)

    def topk_warp(self):
        NS, n = self.NS, self.n
        q0 = 0
        for i, m in enumerate(self.masks):
            trains = self.grad and m and n > 0
            h = min(self.hold, n) if trains else 0
            for c in range(n):
                q = q0 + c
                ok = yield ("wait", self.full[q % NS], q // NS, True, ("T", "full"))
                if ok:
                    yield ("read", "T", q, self.tasks[q])
                yield ("release", "T", q)
            if i >= 2:
                yield ("wait", self.tk_empty[i & 1], (i >> 1) - 1, True, ("T", "tk_empty"))
            yield ("arrive", self.tk_full[i & 1])
            if trains:
                for j in range(h, n):
                    qq = q0 + n + (j - h)
                    ok = yield ("wait", self.full[qq % NS], qq // NS, True, ("T", "full"))
                    if ok:
                        yield ("read", "T", qq, self.tasks[qq])
                    yield ("release", "T", qq)
            q0 += 2 * n - h if trains else n
        yield ("done", "T")

    # ---- scheduler
    def run(self):
        gens = {"P": self.producer()}
        for k, r in enumerate(r for r in self.readers if r != "T"):
            gens[r] = self.consumer(r, warp0=(k == 0))
        if self.topk:
            gens["T"] = self.topk_warp()
        req = {name: next(g) for name, g in gens.items()}
        # the flag as each party's current wait first read it: the kernel
        # reads it before its first test of the phase, so a wait may find
        # the phase complete although the flag went up in between
        self.flag_seen = {name: self.abort for name in gens}
        done = set()
        while len(done) < len(gens):
            actions = []
            for name, r in req.items():
                if name in done:
                    continue
                res = self._enabled(name, r)
                if res is not None:
                    actions.append((name, res))
            actions += [("land", s) for s in self.inflight]
            assert actions, f"a wait that never ends: {[(k, v[:2] + v[3:]) for k, v in req.items() if k not in done]}"
            name, res = self.rng.choice(actions)
            if name == "land":
                s = res
                self.content[s] = self.inflight.pop(s)
                self.full[s].arrive()
                continue
            r = req[name]
            kind = r[0]
            if kind == "wait":
                site = r[4]
                self.wait_count[site] = self.wait_count.get(site, 0) + 1
                if res == "fail":  # this wait runs out: the CTA's flag goes up
                    self.failed = self.abort = True
                    res = False
            if kind == "issue":
                q = r[1]
                s = q % self.NS
                assert s not in self.inflight, f"slot {s} re-armed over pending task {self.inflight[s]}"
                for rd, held in self.holding.items():
                    assert all(t % self.NS != s for t in held), f"slot {s} re-armed while {rd} holds it"
                assert self.full[s].phase == q // self.NS, "copy order"
                self.inflight[s] = q
                self.content.pop(s, None)
            elif kind == "read":
                _, me, q, expect = r
                s = q % self.NS
                assert q in self.holding[me], f"{me} reads task {q} it did not wait for"
                assert self.content.get(s) == q and s not in self.inflight, \
                    f"{me} reads task {q} from slot {s} holding {self.content.get(s)}"
                assert self.tasks[q] == expect
            elif kind == "release":
                _, me, q = r
                self.holding[me].discard(q)
                self.empty[q % self.NS].arrive()
            elif kind == "arrive":
                r[1].arrive()
            elif kind == "sync_arrive":
                g = self.sync_gen.get(r[1], 0)
                self.sync_gen[r[1]] = g + 1
                self.sync_arrived[g] = self.sync_arrived.get(g, 0) + 1
                res = g
            elif kind == "wait" and res:
                bar, k = r[1], r[2]
                if bar is not None and bar in self.full and name != "P":
                    self.holding[name].add(self.full.index(bar) + k * self.NS)
            elif kind == "producer_done":
                assert not self.inflight, f"the producer returns with copies in flight {self.inflight}"
                self.producer_done = True
            try:
                if kind in ("done", "producer_done"):
                    done.add(name)
                    continue
                req[name] = gens[name].send(res if kind in ("wait", "sync_arrive") else None)
                self.flag_seen[name] = self.abort
            except StopIteration:
                done.add(name)
        assert not self.inflight
        return self

    def _enabled(self, name, r):
        kind = r[0]
        if kind == "sync_wait":
            n_cons = sum(1 for x in self.readers if x != "T")
            return True if self.sync_arrived.get(r[1], 0) == n_cons else None
        if kind != "wait":
            return True
        _, bar, k, abortable, site = r
        ordinal = self.wait_count.get(site, 0)
        if abortable and self.flag_seen[name]:
            return False
        if bar is None:  # the stall: nothing completes it; it runs out
            if self.abort:
                return False
            return "fail" if not self.failed else None
        if self.fail_site == (site, ordinal) and abortable and not self.failed:
            return "fail"
        par, truth = bar.test(k)
        if par:
            assert truth, f"parity wait fooled at {site}"
            return True
        if abortable and self.abort:  # the flag, seen while polling
            return False
        return None


def _sites(masks, n, grad, NS, hold, topk):
    """Every wait site an uninterrupted run passes, with its ordinal."""
    sim = _GiveUpSim(masks, n, grad, NS, hold, topk, seed=1).run()
    return [(site, k) for site, cnt in sim.wait_count.items() if site[0] != "P" or
            site[1] == "empty" for k in range(cnt)]


@pytest.mark.parametrize("topk", [False, True])
@pytest.mark.parametrize("grad", [False, True])
def test_give_up_at_every_wait(grad, topk):
    rng = random.Random(11)
    cases = 0
    for n in (1, 2, 3, 5):
        for NS in (1, 2, 3):
            for hold in sorted({0, min(1, NS), NS}):
                masks = [rng.random() < 0.7 for _ in range(rng.randint(1, 4))]
                # uninterrupted runs complete with no flag raised
                for seed in range(3):
                    sim = _GiveUpSim(masks, n, grad, NS, hold, topk, seed=seed).run()
                    assert not sim.abort
                for site in _sites(masks, n, grad, NS, hold, topk):
                    for seed in range(4):
                        sim = _GiveUpSim(masks, n, grad, NS, hold, topk, fail_site=site,
                                         seed=seed).run()
                        assert sim.failed and sim.abort and sim.producer_done
                        cases += 1
                for seed in range(4):
                    sim = _GiveUpSim(masks, n, grad, NS, hold, topk, stall=True, seed=seed).run()
                    assert sim.failed and sim.producer_done
    assert cases > 100


def _producer_without(sim, skip):
    """The kernel's producer with the waits at the sites in ``skip`` removed
    (a removed wait returns at once, as if its phase had completed)."""
    g = _GiveUpSim.producer(sim)
    r = next(g)
    while True:
        if r[0] == "wait" and r[4][1] in skip:
            r = g.send(True)
            continue
        res = yield r
        r = g.send(res)


@pytest.mark.parametrize("variant", ["no_drain", "drain_only_after_own_timeout",
                                     "no_flag_check"])
def test_give_up_model_catches_a_faulty_producer(variant):
    """The earlier producer waited for its copies in flight only when its own
    wait had run out; when a consumer gives up instead, the producer then
    returns with copies still landing. The model finds that, a producer with
    no final wait at all, and one that re-arms a slot after a completed wait
    without checking the flag (a reader that gave up released the slot while
    its copy was in flight or another reader still held it)."""
    class Early(_GiveUpSim):
        def producer(self):
            if variant == "no_flag_check":
                NS, n, q = self.NS, self.n, 0
                for m in self.masks:
                    again = self.grad and m and n > 0
                    h = min(self.hold, n) if again else 0
                    for _ in range(2 * n - h if again else n):
                        if q >= NS:
                            ok = yield ("wait", self.empty[q % NS], q // NS - 1, True,
                                        ("P", "empty"))
                            if not ok:
                                break
                        yield ("issue", q)
                        q += 1
                    else:
                        continue
                    break
                for s in range(NS):
                    if q > s:
                        last = q - 1 - ((q - 1 - s) % NS)
                        yield ("wait", self.full[s], last // NS, False, ("P", "drain"))
                yield ("producer_done",)
                return
            if variant == "no_drain":
                yield from _producer_without(self, {"drain"})
                return
            g = _GiveUpSim.producer(self)
            r = next(g)
            own_timeout = False
            while True:
                if r[0] == "wait" and r[4][1] == "drain" and not own_timeout:
                    r = g.send(True)
                    continue
                res = yield r
                if r[0] == "wait" and r[4] == ("P", "empty") and res is False:
                    own_timeout = self.fail_site is not None and self.fail_site[0] == ("P", "empty")
                r = g.send(res)
    caught = 0
    for seed in range(100):
        for site in [(("C0", "full"), k) for k in range(4)] + [(("C1", "full"), 1),
                                                               (("T", "full"), 1)]:
            try:
                Early([True, True, False, True], 3, True, 2, 1, True, fail_site=site,
                      seed=seed).run()
            except AssertionError as e:
                assert ("copies in flight" in str(e)) == (variant != "no_flag_check"), str(e)
                caught += 1
    assert caught > 0


# ------------------------------------------- the row exchange of a cluster

class XBar:
    """An mbarrier as the exchange uses it: one pending arrival per phase
    (the CTA's own arrive.expect_tx) and a transaction count that the peers'
    st.async stores decrement, possibly before the arrival raised it."""

    def __init__(self):
        self.phase, self.pending, self.tx = 0, 1, 0

    def _maybe_complete(self):
        if self.pending == 0 and self.tx == 0:
            self.phase += 1
            self.pending = 1

    def complete_tx(self, n):
        self.tx -= n
        self._maybe_complete()

    def arrive_expect_tx(self, n):
        self.tx += n
        self.pending -= 1
        assert self.pending == 0, "more arrivals than the barrier expects in one phase"
        self._maybe_complete()


def run_exchange(C, rows, seed, give_up=None):
    """C CTAs of one cluster exchange their row sums for `rows` rows (k_stream's
    kClu path): per row, write the own entry, push it to every peer (data and
    a 16-byte complete_tx on the peer's barrier for the row's parity), arrive
    with expect_tx (C - 1) x 16 unless the CTA gave up, wait for the phase,
    read the C entries. give_up = (cta, row): that CTA's wait on that row runs
    out (it stops waiting from then on). Random interleavings; returns what
    each CTA read per row."""
    rng = random.Random(seed)
    xs = [[[None] * C for _ in range(2)] for _ in range(C)]
    bars = [[XBar(), XBar()] for _ in range(C)]
    state = [dict(row=0, step="push", dead=False, read={}) for _ in range(C)]
    in_flight = []  # st.async stores not yet landed: (dst, slot, src, value)

    def runnable(c):
        s = state[c]
        if s["row"] >= rows:
            return False
        if s["step"] == "wait":
            slot = s["row"] & 1
            return s["dead"] or bars[c][slot].phase > (s["row"] >> 1)
        return True

    for _ in range(10 ** 6):
        choices = [("cta", c) for c in range(C) if runnable(c)]
        choices += [("land", k) for k in range(len(in_flight))]
        if not choices:
            break
        kind, k = rng.choice(choices)
        if kind == "land":
            dst, slot, src, value = in_flight.pop(k)
            xs[dst][slot][src] = value
            bars[dst][slot].complete_tx(16)
            continue
        s = state[k]
        i, slot = s["row"], s["row"] & 1
        if s["step"] == "push":
            value = (k, i)
            xs[k][slot][k] = value
            for r in range(C):
                if r != k:
                    in_flight.append((r, slot, k, value))
            if s["dead"]:
                s["step"] = "read"
            else:
                bars[k][slot].arrive_expect_tx(16 * (C - 1))
                s["step"] = "wait"
        elif s["step"] == "wait":
            if give_up == (k, i) and bars[k][slot].phase <= (i >> 1):
                s["dead"] = True
            s["step"] = "read"
        else:  # read the C entries of the row, then the next row
            s["read"][i] = list(xs[k][slot])
            s["row"] += 1
            s["step"] = "push"
    assert all(s["row"] == rows for s in state), "a CTA never finished its rows"
    return state


@pytest.mark.parametrize("C", [2, 4, 8])
@pytest.mark.parametrize("seed", range(40))
def test_cluster_exchange_reads_every_peers_entry_of_the_same_row(C, seed):
    rows = 7
    state = run_exchange(C, rows, seed)
    for c in range(C):
        for i in range(rows):
            assert state[c]["read"][i] == [(r, i) for r in range(C)], (c, i)


@pytest.mark.parametrize("C", [2, 8])
@pytest.mark.parametrize("seed", range(20))
def test_cluster_exchange_with_a_cta_that_gave_up_still_ends(C, seed):
    """A CTA whose exchange wait ran out keeps pushing but waits no more:
    every CTA still finishes its rows (what a CTA that gave up reads is not
    used; its rows are written as zeros), and the others read correct
    entries up to the row where the peer gave up."""
    rows = 6
    gave_up = (seed % C, seed % rows)
    state = run_exchange(C, rows, seed, give_up=gave_up)
    for c in range(C):
        if c == gave_up[0]:
            continue
        for i in range(rows):
            assert state[c]["read"][i] == [(r, i) for r in range(C)], (c, i)


def test_cluster_exchange_model_catches_a_single_buffer():
    """The same model with one exchange slot per CTA (no row-parity double
    buffer) lets a fast peer's next row overwrite an entry before it is read:
    some interleaving reads a wrong row."""
    def run_single(C, rows, seed):
        rng = random.Random(seed)
        xs = [[None] * C for _ in range(C)]
        bars = [XBar() for _ in range(C)]
        st = [dict(row=0, step="push", read={}) for _ in range(C)]
        fl = []
        for _ in range(10 ** 5):
            ch = [("cta", c) for c in range(C) if st[c]["row"] < rows and
                  (st[c]["step"] != "wait" or bars[c].phase > st[c]["row"])]
            ch += [("land", k) for k in range(len(fl))]
            if not ch:
                break
            kind, k = rng.choice(ch)
            if kind == "land":
                d, s_, v = fl.pop(k)
                xs[d][s_] = v
                bars[d].complete_tx(16)
                continue
            s = st[k]
            if s["step"] == "push":
                xs[k][k] = (k, s["row"])
                fl += [(r, k, (k, s["row"])) for r in range(C) if r != k]
                bars[k].arrive_expect_tx(16 * (C - 1))
                s["step"] = "wait"
            elif s["step"] == "wait":
                s["step"] = "read"
            else:
                s["read"][s["row"]] = list(xs[k])
                s["row"] += 1
                s["step"] = "push"
        return st
    wrong = 0
    for seed in range(200):
        try:
            st = run_single(2, 5, seed)
        except AssertionError:
            wrong += 1
            continue
        wrong += any(st[c]["read"].get(i) != [(r, i) for r in range(2)]
                     for c in range(2) for i in range(5))
    assert wrong > 0
