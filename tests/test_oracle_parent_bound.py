"""Pins of the oracle's parent-bound reservation (Section 4.3: a
reservation takes up to B siblings of the first ready parent and keeps the
relative order of every other queued entry).

Pinned by a hand-worked example (tests/golden/parent_bound_reserve.json),
by an independent closed form (below), by the cases that reduce to elastic
reservation, and by its interplay with recovery groups, GroupFailure queue
drops and a refused (capacity) call.

Closed form.  Rank each queued entry among the queued entries of its parent
(queue order) and cut every parent's entries into chunks of B.  Repeated
reservations take exactly these chunks, in increasing queue position of
each chunk's first entry: a reservation takes the head parent's next chunk
(its first up-to-B remaining entries), so the remaining entries of every
parent always start at a chunk boundary, and the queue's first remaining
entry is the first entry of the remaining chunk that starts earliest.
Without flush the sequence stops at the first chunk shorter than B.
"""
import json
import os

import numpy as np
import pytest

from oracle import ACCEPT, E_CAPACITY as CAPACITY, GROUP_FAILURE, OracleCtx


def _names(parents):
    ids, base = {}, 0
    for name, m in parents.items():
        for j in range(m):
            ids[f"{name}{j}"] = base + j
        base += m
    return ids


def _split(r):
    b, off = r["batched"], r["batch_off"]
    return [list(map(int, b[off[k]:off[k + 1]])) for k in range(r["n_batches"])]


def _queue(o, x, call=0):
    """The queue's entries in order, read by an elastic flush of batches of 1."""
    none = np.zeros(1, np.uint32)[:0]   # no candidates (NULL would mean all children)
    return list(map(int, o.batch_ready(x, call, none, 1, flush=True)["batched"]))


def chunk_schedule(window, parent_of, B, flush):
    """Batches and leftover of repeated parent-bound reservations, by the
    closed form in the module docstring."""
    seen, rank = {}, []
    for c in window:
        p = parent_of[c]
        rank.append(seen.get(p, 0))
        seen[p] = rank[-1] + 1
    batches, taken = [], set()
    for i, c in enumerate(window):
        p, r = parent_of[c], rank[i]
        if r % B:
            continue   # not the first entry of a chunk
        size = min(B, seen[p] - r)
        if size < B and not flush:
            break
        chunk = [d for j, d in enumerate(window) if parent_of[d] == p and r <= rank[j] < r + size]
        batches.append(chunk)
        taken.update(chunk)
    return batches, [c for c in window if c not in taken]


def test_worked_example(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "parent_bound_reserve.json")))
    ids = _names(g["parents"])
    inv = {v: k for k, v in ids.items()}
    queue = [ids[n] for n in g["queue"]]
    for case in g["cases"]:
        o = OracleCtx()
        x = o.expand(list(g["parents"].values()))["xid"]
        r = o.batch_ready_parent(x, 0, queue, case["B"], flush=case["flush"])
        assert [[inv[c] for c in b] for b in _split(r)] == case["batches"]
        assert [inv[c] for c in _queue(o, x)] == case["left"]
        o.close()
    o = OracleCtx()
    x = o.expand(list(g["parents"].values()))["xid"]
    b = o.batch_ready(x, 0, queue, 2)["batched"]
    assert [[inv[int(c)] for c in b[k:k + 2]] for k in range(0, b.size, 2)] == g["elastic_B2"]
    o.close()


def test_blocked_head_waits_then_flushes():
    """A head parent short of B blocks the queue until more of its
    siblings arrive or a flush."""
    o = OracleCtx()
    x = o.expand([3, 4])["xid"]                      # a0..a2 = 0..2, b0..b3 = 3..6
    r = o.batch_ready_parent(x, 0, [0, 3, 4, 5, 6], 2)
    assert r["n_batched"] == 0 and _split(r) == []   # a has 1 < 2 queued: nothing
    r = o.batch_ready_parent(x, 0, [1], 2)           # a's second sibling arrives
    assert _split(r) == [[0, 1], [3, 4], [5, 6]]
    r = o.batch_ready_parent(x, 0, [2], 2)
    assert r["n_batched"] == 0
    r = o.batch_ready_parent(x, 0, None, 2, flush=True)
    assert _split(r) == [[2]] and list(r["batch_off"]) == [0, 1]
    o.close()


@pytest.mark.parametrize("seed", range(40))
def test_closed_form_random(seed):
    rng = np.random.default_rng(900 + seed)
    P = int(rng.integers(1, 40))
    counts = rng.integers(0, 9, P).astype(np.uint32)
    N = int(counts.sum())
    parent_of = np.repeat(np.arange(P), counts)
    o = OracleCtx()
    x = o.expand(counts)["xid"]
    window, admitted = [], set()
    for step in range(int(rng.integers(1, 6))):
        cand = rng.integers(0, max(N, 1) + 2, int(rng.integers(0, N + 3))).astype(np.uint32)
        for c in map(int, cand):
            if c < N and c not in admitted:
                admitted.add(c)
                window.append(c)
        B = int(rng.choice([1, 2, 3, 5, 8]))
        flush = bool(rng.integers(0, 2))
        r = o.batch_ready_parent(x, 0, cand, B, flush=flush)
        want, window = chunk_schedule(window, parent_of, B, flush)
        assert _split(r) == want, (step, B, flush)
        assert r["batch_off"][-1] == r["n_batched"] == sum(map(len, want))
    assert _queue(o, x) == window
    o.close()


@pytest.mark.parametrize("seed", range(6))
def test_reduces_to_elastic(seed):
    """B = 1 or a single parent: parent-bound and elastic reservation take
    the same batches.  A queue of distinct parents with flush: the same
    entries in the same order, one per batch."""
    rng = np.random.default_rng(50 + seed)
    for counts, B in (([5, 3, 7, 2], 1), ([23], 4), ([1] * 17, 3)):
        N = sum(counts)
        cand = rng.permutation(N).astype(np.uint32)
        for flush in (False, True):
            if len(counts) > 1 and B > 1 and not flush:
                continue   # distinct parents without flush: the head is always short
            oa, ob = OracleCtx(), OracleCtx()
            xa, xb = oa.expand(counts)["xid"], ob.expand(counts)["xid"]
            ra = oa.batch_ready_parent(xa, 0, cand, B, flush=flush)
            rb = ob.batch_ready(xb, 0, cand, B, flush=flush)
            assert list(ra["batched"]) == list(rb["batched"])
            distinct = len(counts) > 1 and B > 1
            assert ra["n_batches"] == (N if distinct else rb["n_batches"])
            assert _queue(oa, xa) == _queue(ob, xb)
            oa.close()
            ob.close()


def test_recovery_group_and_group_failure_drop():
    o = OracleCtx()
    x = o.expand([4, 2, 3])["xid"]                   # a 0..3, b 4..5, c 6..8
    r = o.batch_ready_parent(x, 0, [0, 4, 1, 6, 5, 7], 2)
    assert _split(r) == [[0, 1], [4, 5], [6, 7]]
    # the attempt of batch [4, 5] fails and is retried: it goes ahead
    assert o.retry(x, 0, [5, 4])["n_retried"] == 2
    o.batch_ready_parent(x, 0, [2, 8, 3], 4)         # a: 2 < 4 queued, nothing yet
    # window now: recovery 5 4, then 2 8 3; a GroupFailure on parent c seals 8
    cm = o.gather_commit(x, np.array([6], np.uint32), np.array([GROUP_FAILURE], np.uint8),
                         np.zeros(1, np.uint32), np.zeros(1, np.uint64))
    assert list(cm["code"]) == [ACCEPT]
    r = o.batch_ready_parent(x, 0, None, 2, flush=True)
    assert _split(r) == [[5, 4], [2, 3]]
    assert o.stats()["queue_dropped"] == 1
    o.close()


def test_capacity_refusal_changes_nothing():
    counts = [3, 1, 4, 1, 5]
    cand = np.array([10, 0, 4, 3, 11, 1, 5, 9, 2, 6, 12, 7, 8, 13], np.uint32)
    ref = OracleCtx()
    xr = ref.expand(counts)["xid"]
    want = ref.batch_ready_parent(xr, 0, cand, 2, flush=True)
    o = OracleCtx()
    x = o.expand(counts)["xid"]
    r = o.batch_ready_parent(x, 0, cand, 2, flush=True, cap=want["n_batched"] - 1, check=False)
    assert r["status"] == CAPACITY
    r = o.batch_ready_parent(x, 0, cand, 2, flush=True, off_cap=want["n_batches"], check=False)
    assert r["status"] == CAPACITY
    r = o.batch_ready_parent(x, 0, cand, 2, flush=True)
    assert _split(r) == _split(want)
    assert o.stats() == ref.stats()
    o.close()
    ref.close()
