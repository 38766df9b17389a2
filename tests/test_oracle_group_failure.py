"""Pins of the oracle's GroupFailure containment (Section 4.4, Figure 5):
a GroupFailure report fails its own Grain and installs a barrier for its
(Call, parent) — queued siblings are suppressed before dispatch, reports of
in-flight siblings are rejected, siblings sealed earlier keep their facts,
and other parents are unaffected.  Checked against the figure's worked
example, hand-built orderings, and a closed-form count over a seeded
readiness schedule whose unaffected parents must assemble exactly as in a
run without the failure."""
import json
import os

import numpy as np
import pytest

from oracle import (ACCEPT, GROUP_FAILURE, PRESENT, REJ_BARRIER, REJ_NOT_INFLIGHT, REJ_STALE_GEN,
                    SUPPRESSED, OracleCtx)
from tests.pipeline import host_arena
from workload import tiny


def _names(parents):
    ids, base = {}, 0
    for name, m in parents.items():
        for j in range(m):
            ids[f"{name}{j}"] = base + j
        base += m
    return ids


def _reports(children, states, seed_len=8):
    children = np.asarray(children, dtype=np.uint32)
    return (children, np.asarray(states, np.uint8), np.full(children.size, seed_len, np.uint32),
            children.astype(np.uint64) * seed_len)


def test_fig5_group_failure(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "fig5_reserve.json")))
    ids = _names(g["parents"])
    pnames = list(g["parents"])
    gf = g["group_failure"]
    o = OracleCtx()
    x = o.expand(list(g["parents"].values()))["xid"]
    earlier = [ids[n] for n in g["earlier"]]
    o.batch_ready(x, 0, earlier, len(earlier))
    cm = o.gather_commit(x, *_reports(earlier, [PRESENT] * len(earlier)))
    assert all(cm["code"] == ACCEPT) and cm["n_done"] == 0
    br = o.batch_ready(x, 0, [ids[n] for n in g["queue"]], g["reserve"], flush=False)
    assert sorted(int(c) for c in br["batched"]) == sorted(ids[n] for n in g["reserved"])
    # B1 reports the GroupFailure first; then the in-flight B2, then A1 and C1
    order = [gf["failing_report"]] + gf["rejected_in_flight"] + gf["commit"]
    states = [GROUP_FAILURE] + [PRESENT] * (len(order) - 1)
    cm = o.gather_commit(x, *_reports([ids[n] for n in order], states))
    assert list(cm["code"]) == [ACCEPT] + [REJ_BARRIER] * len(gf["rejected_in_flight"]) \
        + [ACCEPT] * len(gf["commit"])
    # every parent resolves: A and C by their commits, B by the barrier
    assert [pnames[p] for p in cm["done"]] == ["A", "B", "C"]
    st = o.stats()
    assert st["barrier_in_flight"] == len(gf["rejected_in_flight"])
    assert st["barrier_not_dispatched"] == len(gf["suppressed_before_dispatch"])
    assert st["rej_barrier"] == len(gf["rejected_in_flight"])
    a = o.assemble(x, None, n_parents=3)
    assert list(a["parent_status"]) == [PRESENT, SUPPRESSED, PRESENT]
    # B3 never enters a batch: the next reservation drops it
    fl = o.batch_ready(x, 0, None, g["reserve"], flush=True)
    assert fl["n_batched"] == 0
    assert o.stats()["queue_dropped"] == len(gf["suppressed_before_dispatch"])
    o.close()


def test_reports_before_the_failure_in_one_commit_stand():
    # one parent of 4, all in flight; reports: B2 (before), B1 GroupFailure, B3 (after)
    o = OracleCtx()
    x = o.expand([4, 2])["xid"]
    o.batch_ready(x, 0, None, 6, flush=True)
    cm = o.gather_commit(x, *_reports([2, 1, 3], [PRESENT, GROUP_FAILURE, PRESENT]))
    assert list(cm["code"]) == [ACCEPT, ACCEPT, REJ_BARRIER]
    st = o.stats()
    # B0 (never reported, in flight) and B3 are suppressed while in flight
    assert st["barrier_in_flight"] == 2 and st["barrier_not_dispatched"] == 0
    assert list(cm["done"]) == [0]
    # a report for the barrier-sealed B0 later: rejected as such; a stale one as stale
    cm2 = o.gather_commit(x, *_reports([0, 0], [PRESENT, PRESENT]), gen=np.array([0, 7], np.uint32))
    assert list(cm2["code"]) == [REJ_BARRIER, REJ_STALE_GEN]
    # a second GroupFailure for the same parent cannot install anything
    cm3 = o.gather_commit(x, *_reports([3, 4, 5], [GROUP_FAILURE, PRESENT, PRESENT]))
    assert list(cm3["code"]) == [REJ_BARRIER, ACCEPT, ACCEPT] and list(cm3["done"]) == [1]
    o.close()


def test_waiting_siblings_are_never_admitted():
    counts = [5, 3]
    o = OracleCtx()
    x = o.expand(counts)["xid"]
    o.batch_ready(x, 0, [0], 1, flush=True)           # only child 0 of parent 0 runs
    cm = o.gather_commit(x, *_reports([0], [GROUP_FAILURE]))
    assert list(cm["code"]) == [ACCEPT] and list(cm["done"]) == [0]
    assert o.stats()["barrier_not_dispatched"] == 4
    br = o.batch_ready(x, 0, None, 2, flush=True)     # the other parent's children only
    assert sorted(int(c) for c in br["batched"]) == [5, 6, 7]
    # a GroupFailure that is not in flight installs nothing
    cm = o.gather_commit(x, *_reports([1], [GROUP_FAILURE]))
    assert list(cm["code"]) == [REJ_BARRIER]
    o.close()


def _schedule(lv, W, rng):
    """Readiness wave per child and a report order per wave."""
    ready_wave = rng.integers(0, W, lv.n_children)
    order = [rng.permutation(np.flatnonzero(ready_wave == w)).astype(np.uint32) for w in range(W)]
    return ready_wave, order


def _run(lv, arena, W, order, poisoned_children):
    """Wave by wave: admit and dispatch the wave's ready children, then commit
    their reports in the wave's order; poisoned children report GroupFailure."""
    o = OracleCtx()
    x = o.expand(lv.counts)["xid"]
    outs = {}
    for w in range(W):
        br = o.batch_ready(x, 0, order[w], 64, flush=True)
        ch = order[w][np.isin(order[w], br["batched"])]   # suppressed Grains never run
        st = lv.state[ch].copy()
        st[np.isin(ch, poisoned_children)] = GROUP_FAILURE
        cm = o.gather_commit(x, ch, st, lv.length[ch], lv.arena_off[ch], arena_bytes=lv.arena_bytes)
        a = o.assemble(x, arena, n_parents=max(cm["n_done"], 1))
        for i, p in enumerate(cm["done"]):
            s, e = int(a["out_off"][i]), int(a["out_off"][i + 1])
            outs[int(p)] = (int(a["parent_status"][i]), bytes(a["out"][s:e]))
    stats = o.stats()
    o.close()
    return outs, stats


@pytest.mark.parametrize("seed", [0, 1])
def test_rq4_analog_closed_form_and_unaffected_parents(seed):
    # Section 6 RQ4: a failure at ordinal 0 of the largest parents
    lv = tiny().top
    arena = host_arena(lv)
    rng = np.random.default_rng(100 + seed)
    W = 8
    ready_wave, order = _schedule(lv, W, rng)
    big = np.argsort(-lv.counts.astype(np.int64), kind="stable")[:12]
    off = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
    poisoned = off[big].astype(np.uint32)                      # child (p, 0)
    clean, _ = _run(lv, arena, W, order, np.array([], np.uint32))
    pois, st = _run(lv, arena, W, order, poisoned)
    # closed form of the suppressed siblings
    not_disp = in_flight = 0
    for p, c0 in zip(big, poisoned):
        w0 = ready_wave[c0]
        pos = {int(c): i for i, c in enumerate(order[w0])}
        for c in range(off[p], off[p + 1]):
            if c == c0:
                continue
            if ready_wave[c] > w0:
                not_disp += 1
            elif ready_wave[c] == w0 and pos[c] > pos[int(c0)]:
                in_flight += 1
    assert st["barrier_not_dispatched"] == not_disp and st["barrier_in_flight"] == in_flight
    assert st["rej_barrier"] == in_flight
    # every parent resolves; poisoned ones are Suppressed, the rest are as in the clean run
    assert set(pois) == set(clean) == set(range(lv.n_parents))
    for p in range(lv.n_parents):
        if p in set(int(b) for b in big):
            assert pois[p] == (SUPPRESSED, b"")
        else:
            assert pois[p] == clean[p]
