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
