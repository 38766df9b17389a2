"""GroupFailure containment on the GPU (Section 4.4, Figure 5) against the
oracle: every verdict, completed-parent list, reserved batch, assembled
byte and counter is compared exactly.

Covers the figure's worked example, a GroupFailure ordered among sibling
reports of the same call (before / after / duplicated), barriers over
WAITING, READY and IN-FLIGHT siblings, several Calls, multi-wave streaming
with the failure at ordinal 0 of the largest parents (the paper's RQ4
set-up), and a 100k-child parent whose barrier seals 99,999 siblings.
"""
import json
import os

import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


from tests.lockstep import Lockstep, dev  # noqa: E402
from tests.pipeline import host_arena  # noqa: E402
from workload import DROPPED, FAILED, PRESENT, SUPPRESSED, docpage, streaming  # noqa: E402

GF = 5   # report kind GroupFailure


def _arena_dev(a):
    return dev(a if a.size else np.zeros(1, np.uint8), np.uint8)


def _names(parents):
    ids, base = {}, 0
    for name, m in parents.items():
        for j in range(m):
            ids[f"{name}{j}"] = base + j
        base += m
    return ids


def _rep(children, states, ln=8):
    children = np.asarray(children, np.uint32)
    return (children, np.asarray(states, np.uint8), np.full(children.size, ln, np.uint32),
            children.astype(np.uint64) * ln)


def test_fig5_on_gpu(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "fig5_reserve.json")))
    ids = _names(g["parents"])
    gf = g["group_failure"]
    arena = np.arange(256, dtype=np.uint8)
    with Lockstep() as ls:
        x = ls.expand(np.array(list(g["parents"].values()), np.uint32))["xid"]
        ad = _arena_dev(arena)
        earlier = [ids[n] for n in g["earlier"]]
        ls.batch_ready(x, 0, earlier, len(earlier))
        ls.commit(x, *_rep(earlier, [PRESENT] * 3), arena_bytes=arena.size)
        ls.batch_ready(x, 0, [ids[n] for n in g["queue"]], g["reserve"])
        order = [gf["failing_report"]] + gf["rejected_in_flight"] + gf["commit"]
        r = ls.commit(x, *_rep([ids[n] for n in order], [GF] + [PRESENT] * (len(order) - 1)),
                      arena_bytes=arena.size)
        assert list(r["code"]) == [0, 5, 0, 0]
        ls.assemble(x, arena, ad, parents=None, n_parents=3)
        fl = ls.batch_ready(x, 0, None, g["reserve"], flush=True)
        assert fl["n_batched"] == 0
        ls.check_stats()


def test_group_failure_ordering_within_a_call():
    arena = np.arange(4096, dtype=np.uint8)
    with Lockstep() as ls:
        x = ls.expand(np.array([6, 3, 4], np.uint32))["xid"]
        ad = _arena_dev(arena)
        ls.batch_ready(x, 0, [0, 1, 2, 3, 6, 7, 9], 1, flush=True)   # 4, 5, 8, 10..12 stay WAITING
        ls.batch_ready(x, 0, [4, 10], 8, flush=False)                 # READY, queued
        # parent 0: sibling before the failure stands, the failure, a sibling
        # after it, a duplicate of that sibling, the failure's own duplicate,
        # a report for a queued sibling; parent 1 untouched; parent 2 a stale one
        ch = [1, 2, 0, 3, 3, 2, 4, 6, 7, 9, 9]
        st = [PRESENT, GF, PRESENT, PRESENT, FAILED, GF, PRESENT, PRESENT, PRESENT, PRESENT, GF]
        gen = np.array([0, 0, 0, 0, 0, 0, 0, 0, 0, 0, 3], np.uint32)
        r = ls.commit(x, *_rep(ch, st), gen=gen, arena_bytes=arena.size)
        ls.assemble(x, arena, ad, parents=None, n_parents=3)
        # the queued sibling 4 leaves the queue undispatched; 10 stays
        ls.batch_ready(x, 0, None, 8, flush=True)
        # later reports for barrier-sealed Grains
        r2 = ls.commit(x, *_rep([4, 5, 5, 8, 10, 11, 12], [PRESENT] * 4 + [GF, PRESENT, PRESENT]),
                       gen=np.array([0, 0, 9, 0, 0, 0, 0], np.uint32), arena_bytes=arena.size)
        ls.assemble(x, arena, ad, parents=[0, 1, 2, 2], n_parents=4)
        ls.check_stats()
        assert 5 in set(int(v) for v in r["code"]) and 5 in set(int(v) for v in r2["code"])


@pytest.mark.parametrize("seed", range(3))
def test_random_group_failures_many_calls(seed):
    rng = np.random.default_rng(4000 + seed)
    P = 3000
    counts = rng.integers(0, 12, P).astype(np.uint32)
    calls = rng.integers(0, 3, P).astype(np.uint8)
    N = int(counts.sum())
    arena = rng.integers(0, 256, N * 16 + 64).astype(np.uint8)
    with Lockstep(n_calls=3) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        ad = _arena_dev(arena)
        perm = rng.permutation(N).astype(np.uint32)
        chunks = np.array_split(perm, 6)
        for w, cand in enumerate(chunks):
            reserved = []
            for c in range(3):
                reserved.append(ls.batch_ready(x, c, cand, int(rng.choice([1, 7, 64])),
                                               flush=(w % 2 == 1))["batched"])
            got = np.concatenate(reserved)
            got = got[rng.permutation(got.size)]
            # some reports twice, some for children never reserved, some GroupFailures
            extra = rng.choice(N, size=max(1, got.size // 20)).astype(np.uint32)
            ch = np.concatenate([got, got[: got.size // 10], extra])
            ch = ch[rng.permutation(ch.size)]
            st = rng.choice([PRESENT] * 12 + [2, FAILED, 4, GF], ch.size).astype(np.uint8)
            ln = rng.integers(0, 16, ch.size).astype(np.uint32)
            of = (ch.astype(np.uint64) * 16)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=arena.size)
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        for c in range(3):
            ls.batch_ready(x, c, None, 5, flush=True)
        ls.check_stats()


@pytest.mark.parametrize("seed", range(3))
def test_random_group_failures_without_repeats(seed):
    """Calls with GroupFailures but no repeated report of a Grain take the
    barrier pass spread over the grid: every reserved child reports once, in
    random order, some as GroupFailure, some with a stale generation; plus
    reports for children that were never dispatched."""
    rng = np.random.default_rng(6000 + seed)
    P = 20000
    counts = rng.integers(0, 40, P).astype(np.uint32)
    calls = rng.integers(0, 2, P).astype(np.uint8)
    N = int(counts.sum())
    arena = rng.integers(0, 256, N * 16 + 64).astype(np.uint8)
    with Lockstep(n_calls=2) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        ad = _arena_dev(arena)
        perm = rng.permutation(N).astype(np.uint32)
        for w, cand in enumerate(np.array_split(perm, 5)):
            got = np.concatenate([ls.batch_ready(x, c, cand, 64, flush=True)["batched"] for c in range(2)])
            spare = np.setdiff1d(perm[: (w + 1) * N // 5], got)[: got.size // 8]   # not dispatched now
            ch = np.concatenate([got, spare]).astype(np.uint32)
            ch = ch[rng.permutation(ch.size)]
            st = rng.choice([PRESENT] * 30 + [FAILED, GF], ch.size).astype(np.uint8)
            gen = (rng.random(ch.size) < 0.02).astype(np.uint32) * 5   # a few stale
            ln = rng.integers(0, 16, ch.size).astype(np.uint32)
            cm = ls.commit(x, ch, st, ln, ch.astype(np.uint64) * 16, gen=gen, arena_bytes=arena.size)
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        for c in range(2):
            ls.batch_ready(x, c, None, 7, flush=True)
        ls.check_stats()
        assert ls.o.stats()["barrier_in_flight"] > 0


def test_rq4_analog_streaming_docpage():
    """Section 6 RQ4 on a document->page level: readiness in waves, reports
    per wave in a seeded order, GroupFailure at ordinal 0 of the 99 largest
    parents; only dispatched children report."""
    lv = docpage(parents=4000, waves=1).top
    a = host_arena(lv)
    rng = np.random.default_rng(77)
    W = 12
    ready_wave = rng.integers(0, W, lv.n_children)
    order = [rng.permutation(np.flatnonzero(ready_wave == w)).astype(np.uint32) for w in range(W)]
    off = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
    big = np.argsort(-lv.counts.astype(np.int64), kind="stable")[:99]
    poisoned = off[big].astype(np.uint32)
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        ad = _arena_dev(a)
        for w in range(W):
            br = ls.batch_ready(x, 0, order[w], 256, flush=True)
            ch = order[w][np.isin(order[w], br["batched"])]
            st = lv.state[ch].copy()
            st[np.isin(ch, poisoned)] = GF
            cm = ls.commit(x, ch, st, lv.length[ch], lv.arena_off[ch], arena_bytes=lv.arena_bytes)
            ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()
        st = ls.o.stats()
        assert st["barrier_not_dispatched"] > 0 and st["barrier_in_flight"] > 0


def test_barrier_on_a_100k_child_parent():
    counts = np.array([3, 100_000, 2], np.uint32)
    arena = np.arange(1024, dtype=np.uint8)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        ad = _arena_dev(arena)
        ls.batch_ready(x, 0, np.arange(0, 60_000, dtype=np.uint32), 1000)   # part dispatched
        ls.commit(x, *_rep([3, 4, 0, 5], [PRESENT, PRESENT, PRESENT, GF]), arena_bytes=arena.size)
        ls.assemble(x, arena, ad, parents=None, n_parents=3)
        ls.batch_ready(x, 0, None, 1000, flush=True)
        ls.check_stats()


@pytest.mark.parametrize("seed", range(2))
def test_heavy_parents_with_repeats_failures_and_barriers(seed):
    """Parents of 4,096 children or more (their members are counted down per
    CTA in shared memory, then once per parent) mixed with light ones, over
    several commits carrying repeated reports, failures, Dropped results and
    GroupFailures: every verdict, completion and assembled byte equals the
    oracle's (a report's order inside a call still decides)."""
    rng = np.random.default_rng(7100 + seed)
    counts = rng.integers(0, 6, 4000).astype(np.uint32)
    heavy = rng.choice(counts.size, 6, replace=False)
    counts[heavy] = [4096, 5000, 9000, 4095, 12000, 20000]   # one just below the threshold
    N = int(counts.sum())
    arena = rng.integers(0, 256, N * 8 + 64).astype(np.uint8)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        ad = _arena_dev(arena)
        ls.batch_ready(x, 0, None, 256, flush=True)
        perm = rng.permutation(N).astype(np.uint32)
        for w, chunk in enumerate(np.array_split(perm, 5)):
            rep = rng.choice(chunk, size=chunk.size // 8)
            ch = np.concatenate([chunk, rep])
            ch = ch[rng.permutation(ch.size)].astype(np.uint32)
            st = rng.choice([PRESENT] * 40 + [DROPPED, FAILED, SUPPRESSED] + ([GF] if w >= 2 else []),
                            ch.size).astype(np.uint8)
            ln = rng.integers(0, 9, ch.size).astype(np.uint32)
            of = ch.astype(np.uint64) * 8
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=arena.size)
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()
