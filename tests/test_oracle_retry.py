"""Pins of the oracle's retry path (Section 4.4: a failed physical attempt is
retried at a higher generation; Eq. 2's IN-FLIGHT -> READY edge; Section
4.3: recovery queues reinsert the exact Grain group ahead of normal
entries).  Checked by hand-built sequences against Eq. (2)/(3), and by
Eq. (4) (schedule invariance): runs in which random batches fail, are
retried and deliver late stale reports assemble exactly the same results
as a run without failures."""
import numpy as np
import pytest

from oracle import (ACCEPT, GROUP_FAILURE, PRESENT, REJ_NOT_INFLIGHT, REJ_STALE_GEN, OracleCtx)
from tests.pipeline import host_arena
from workload import tiny


def _rep(children, states=None, ln=8):
    children = np.asarray(children, np.uint32)
    st = np.full(children.size, PRESENT, np.uint8) if states is None else np.asarray(states, np.uint8)
    return children, st, np.full(children.size, ln, np.uint32), children.astype(np.uint64) * ln


def test_retry_edge_generation_and_recovery_first():
    o = OracleCtx()
    x = o.expand([4, 4])["xid"]
    b1 = o.batch_ready(x, 0, [0, 1, 4, 5], 4)["batched"]          # first attempt
    assert list(b1) == [0, 1, 4, 5]
    o.batch_ready(x, 0, [2, 3, 6, 7], 8)                          # queued, not reserved
    # the attempt fails: its Grains go back to READY at generation 1
    assert o.retry(x, 0, b1)["n_retried"] == 4
    # a late report of the failed attempt: the Grain is READY, not in flight
    cm = o.gather_commit(x, *_rep([0]))
    assert list(cm["code"]) == [REJ_NOT_INFLIGHT]
    # the next reservation takes the recovery group first, then the queue
    b2 = o.batch_ready(x, 0, None, 4, flush=True)["batched"]
    assert list(b2) == [0, 1, 4, 5, 2, 3, 6, 7]
    # now in flight at generation 1: generation 0 is stale, 1 is accepted
    cm = o.gather_commit(x, *_rep([0, 0, 1]), gen=np.array([0, 1, 1], np.uint32))
    assert list(cm["code"]) == [REJ_STALE_GEN, ACCEPT, ACCEPT]
    st = o.stats()
    assert st["retried"] == 4 and st["retry_skipped"] == 0
    o.close()


def test_retry_skips_and_first_occurrence():
    o = OracleCtx(2)
    x = o.expand([3, 3], parent_call=np.array([0, 1], np.uint8))["xid"]
    o.batch_ready(x, 0, [0, 1], 1)
    o.batch_ready(x, 1, [3, 4], 1)
    # duplicates, another Call's Grain, a WAITING Grain, an out-of-range id
    r = o.retry(x, 0, [1, 0, 1, 3, 2, 99])
    assert r["n_retried"] == 2 and o.stats()["retry_skipped"] == 4
    b = o.batch_ready(x, 0, None, 8, flush=True)["batched"]
    assert list(b) == [1, 0, 2]                                  # group order = list order
    cm = o.gather_commit(x, *_rep([1, 0, 2]), gen=np.array([1, 1, 0], np.uint32))
    assert list(cm["code"]) == [ACCEPT] * 3
    o.close()


def test_groups_keep_their_order_and_barrier_drops_retried():
    o = OracleCtx()
    x = o.expand([2, 2, 2, 3])["xid"]          # parents 0..3: children 0-1, 2-3, 4-5, 6-8
    g1 = o.batch_ready(x, 0, [0, 2], 2)["batched"]
    g2 = o.batch_ready(x, 0, [4, 6], 2)["batched"]
    o.retry(x, 0, g2)
    o.retry(x, 0, g1)
    # recovery groups in the order they failed, then the newly admitted ones
    assert list(o.batch_ready(x, 0, [1, 3], 2)["batched"]) == [4, 6, 0, 2, 1, 3]
    # 7 runs, fails and waits in the recovery queue; then a GroupFailure of
    # its sibling 6 (in flight at generation 1) seals it and the WAITING 8
    o.batch_ready(x, 0, [7], 1)
    o.retry(x, 0, [7])
    cm = o.gather_commit(x, *_rep([6], [GROUP_FAILURE]), gen=np.array([1], np.uint32))
    assert list(cm["code"]) == [ACCEPT]
    before = o.stats()["queue_dropped"]
    out = o.batch_ready(x, 0, None, 8, flush=True)["batched"]
    assert list(out) == [5] and o.stats()["queue_dropped"] == before + 1
    o.close()


def _pass(lv, arena, rng, fail_p):
    """Dispatch in waves of batches; each batch's attempt fails with
    probability fail_p (retried, its reports delivered later as stale)."""
    o = OracleCtx()
    x = o.expand(lv.counts)["xid"]
    results = {}
    late = []
    order = rng.permutation(lv.n_children).astype(np.uint32)
    waves = np.array_split(order, 6)
    gen = np.zeros(lv.n_children, np.uint32)
    for w in range(len(waves) + 20):
        cand = waves[w] if w < len(waves) else np.zeros(0, np.uint32)
        b = o.batch_ready(x, 0, cand, 32, flush=True)["batched"]
        if b.size == 0 and w >= len(waves):
            break
        reps = []
        for batch in np.array_split(b, max(1, b.size // 32)):
            if batch.size and rng.random() < fail_p:
                late.append(batch.copy())                       # reports of the failed attempt
                o.retry(x, 0, batch)
                gen[batch] += 1
            else:
                reps.append(batch)
        ch = np.concatenate(reps) if reps else np.zeros(0, np.uint32)
        if late and rng.random() < 0.5:                          # stale reports arrive late
            stale = late.pop(0)
            ch = np.concatenate([stale, ch])
            g = np.concatenate([gen[stale] - 1, gen[ch[stale.size:]]])
        else:
            g = gen[ch]
        ch = ch.astype(np.uint32)
        cm = o.gather_commit(x, ch, lv.state[ch], lv.length[ch], lv.arena_off[ch],
                             gen=g.astype(np.uint32), arena_bytes=lv.arena_bytes)
        a = o.assemble(x, arena, n_parents=max(cm["n_done"], 1))
        for i, p in enumerate(cm["done"]):
            s, e = int(a["out_off"][i]), int(a["out_off"][i + 1])
            results[int(p)] = (int(a["parent_status"][i]), bytes(a["out"][s:e]))
    st = o.stats()
    o.close()
    return results, st


@pytest.mark.parametrize("seed", [0, 1, 2])
def test_schedule_invariance_under_retries(seed):
    lv = tiny().top
    arena = host_arena(lv)
    clean, _ = _pass(lv, arena, np.random.default_rng(seed), 0.0)
    retried, st = _pass(lv, arena, np.random.default_rng(seed), 0.3)
    assert st["retried"] > 0 and st["rej_stale_gen"] > 0
    assert retried == clean and len(clean) == lv.n_parents
