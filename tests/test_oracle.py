"""Pins of the CPU oracle against what the paper and the mathematics fix:
the worked examples of Figures 1(c) and 5, closed forms of the expansion
(prefix sum, repeat), first-occurrence order of the FIFO, completion waves,
the Reduce rule enumerated over member outcomes, the generation fence, and
schedule invariance (Eq. 4) by brute force over arrival orders."""
import itertools
import json
import os

import numpy as np
import pytest

from oracle import (ACCEPT, DROPPED, E_CAPACITY, E_INVAL, FAILED, OK, PENDING, PRESENT,
                    REJ_DUPLICATE, REJ_INVALID, REJ_NOT_INFLIGHT, REJ_STALE_GEN, SUPPRESSED,
                    OracleCtx)
from tests.pipeline import (closed_form_done_wave, closed_form_lineage, closed_form_parent,
                            host_arena, run_level_oracle)
from workload import record_bytes, tiny, video


def _names(parents):
    """Map grain names like 'B2' to parent-major child ids."""
    ids, base = {}, 0
    for name, m in parents.items():
        for j in range(m):
            ids[f"{name}{j}"] = base + j
        base += m
    return ids


def _present_reports(children, seed_len=8):
    children = np.asarray(children, dtype=np.uint32)
    return (children, np.full(children.size, PRESENT, np.uint8),
            np.full(children.size, seed_len, np.uint32),
            (children.astype(np.uint64) * seed_len))


# --------------------------------------------------------------------- golden
def test_fig1c_fifo_batches_and_counters(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "fig1c_fifo.json")))
    ids = _names(g["parents"])
    names = {v: k for k, v in ids.items()}
    pnames = list(g["parents"])
    o = OracleCtx()
    ex = o.expand([g["parents"][p] for p in pnames])
    cand = [ids[x] for x in g["fifo"]]
    br = o.batch_ready(ex["xid"], 0, cand, g["batch_size"], flush=False)
    B = g["batch_size"]
    got = [[names[int(c)] for c in br["batched"][i:i + B]]
           for i in range(0, br["n_batched"], B)]
    assert got == g["batches"]
    # both dense batches report back; counters as drawn in the figure
    cm = o.gather_commit(ex["xid"], *_present_reports(br["batched"]))
    assert all(cm["code"] == ACCEPT)
    done = [pnames[p] for p in cm["done"]]
    assert done == g["complete_after_both_batches"]
    for p, (k, m) in g["counters_after_both_batches"].items():
        pi = pnames.index(p)
        committed = sum(1 for c in br["batched"] if ex["child_parent"][c] == pi)
        assert (committed, g["parents"][p]) == (k, m)


def test_fig5_elastic_reservation(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "fig5_reserve.json")))
    ids = _names(g["parents"])
    names = {v: k for k, v in ids.items()}
    o = OracleCtx()
    ex = o.expand(list(g["parents"].values()))
    first = o.batch_ready(ex["xid"], 0, [ids[x] for x in g["earlier"]], len(g["earlier"]))
    assert [names[int(c)] for c in first["batched"]] == g["earlier"]
    br = o.batch_ready(ex["xid"], 0, [ids[x] for x in g["queue"]], g["reserve"], flush=False)
    assert [names[int(c)] for c in br["batched"]] == g["reserved"]
    # the left-over grain is READY, not in flight: its report is refused ...
    left = [ids[x] for x in g["left_queued"]]
    cm = o.gather_commit(ex["xid"], *_present_reports(left))
    assert list(cm["code"]) == [REJ_NOT_INFLIGHT]
    # ... and it comes out first on the next reservation
    fl = o.batch_ready(ex["xid"], 0, None, g["reserve"], flush=True)
    assert [names[int(c)] for c in fl["batched"]] == g["left_queued"]


# -------------------------------------------------------------- closed forms
@pytest.mark.parametrize("seed", [0, 1, 2, 3])
def test_expand_closed_form(seed):
    rng = np.random.default_rng(seed)
    P = int(rng.integers(1, 400))
    counts = rng.integers(0, 9, size=P).astype(np.uint32)
    counts[rng.random(P) < 0.2] = 0
    if seed == 3:
        counts[:] = 0
    o = OracleCtx()
    ex = o.expand(counts)
    offsets, cp, co, empties = closed_form_lineage(counts)
    assert np.array_equal(ex["offsets"], offsets)
    assert ex["n_children"] == int(offsets[-1])
    assert np.array_equal(ex["child_parent"], cp)
    assert np.array_equal(ex["child_ordinal"], co)
    assert np.array_equal(ex["empty_parents"], empties)
    # each child has exactly one parent and ordinals are 0..m-1 per parent
    for p in range(P):
        sel = co[cp == p]
        assert np.array_equal(np.sort(sel), np.arange(counts[p]))


def test_expand_errors():
    o = OracleCtx(n_calls=2)
    r = o.expand([3, 4], child_cap=6, check=False)
    assert r["status"] == E_CAPACITY and r["n_children"] == 7
    ok = o.expand([3, 4])
    assert ok["status"] == OK
    assert o.expand([1, 1, 1], parent_xid=ok["xid"], check=False)["status"] == E_INVAL
    assert o.expand([1] * 7, parent_xid=ok["xid"])["status"] == OK
    assert o.expand([1, 2], parent_call=[0, 2], check=False)["status"] == E_INVAL


@pytest.mark.parametrize("B", [1, 3, 64])
def test_batch_ready_all_children_in_id_order(B):
    counts = np.random.default_rng(B).integers(0, 7, size=50).astype(np.uint32)
    o = OracleCtx()
    ex = o.expand(counts)
    N = ex["n_children"]
    a = o.batch_ready(ex["xid"], 0, None, B, flush=False)
    full = (N // B) * B
    assert np.array_equal(a["batched"], np.arange(full))
    assert a["n_batches"] == N // B
    b = o.batch_ready(ex["xid"], 0, None, B, flush=True)
    assert np.array_equal(b["batched"], np.arange(full, N))
    assert b["n_batches"] == (1 if N % B else 0)


def _first_occurrences(cand, N, seen):
    """Distinct valid candidates in order of first occurrence, minus ``seen``."""
    cand = np.asarray(cand, dtype=np.int64)
    valid = cand[cand < N]
    _, idx = np.unique(valid, return_index=True)
    firsts = valid[np.sort(idx)]
    return [int(c) for c in firsts if int(c) not in seen]


@pytest.mark.parametrize("seed", range(6))
def test_batch_ready_fifo_order_over_waves(seed):
    rng = np.random.default_rng(100 + seed)
    counts = rng.integers(1, 6, size=40).astype(np.uint32)
    o = OracleCtx()
    ex = o.expand(counts)
    N = ex["n_children"]
    B = int(rng.integers(1, 9))
    expected_stream, seen, got_stream, bad = [], set(), [], 0
    for w in range(5):
        cand = rng.integers(0, N + 5, size=int(rng.integers(0, 40)))
        bad += int(np.sum(cand >= N))
        new = _first_occurrences(cand, N, seen)
        seen.update(new)
        expected_stream += new
        last = w == 4
        r = o.batch_ready(ex["xid"], 0, cand, B, flush=last)
        if not last:
            assert r["n_batched"] % B == 0
        got_stream += [int(c) for c in r["batched"]]
    assert got_stream == expected_stream
    assert o.stats()["ready_bad_candidates"] == bad


def test_batch_ready_calls_partition():
    counts = np.array([3, 2, 4, 1, 2], np.uint32)
    calls = np.array([0, 1, 0, 1, 1], np.uint8)
    o = OracleCtx(n_calls=2)
    ex = o.expand(counts, parent_call=calls)
    cp = ex["child_parent"]
    for call in (0, 1):
        r = o.batch_ready(ex["xid"], call, None, 2, flush=True)
        assert np.array_equal(r["batched"], np.flatnonzero(calls[cp] == call))


def test_calls_admit_independently_of_their_order():
    """Each Call admits only its own children (Section 4.3: one Ready Queue
    per Call), so with one shared candidate list, duplicates included, the
    Calls' reservations do not depend on the order the Calls run in, and each
    Call's batches over all waves (the last one flushing) are the candidate-
    order sequence of first occurrences of that Call's children."""
    rng = np.random.default_rng(9)
    P, C, B = 400, 4, 5
    counts = rng.integers(0, 6, P).astype(np.uint32)
    calls = rng.integers(0, C, P).astype(np.uint8)
    N = int(counts.sum())
    cp = np.repeat(np.arange(P), counts.astype(np.int64))
    cand = rng.integers(0, N, 3 * N).astype(np.uint32)
    waves = np.array_split(cand, 3)
    runs = []
    for order in ((0, 1, 2, 3), (3, 1, 0, 2)):
        o = OracleCtx(n_calls=C)
        x = o.expand(counts, parent_call=calls)["xid"]
        got = {c: [] for c in range(C)}
        for k, wv in enumerate(waves):
            for c in order:
                r = o.batch_ready(x, c, wv, B, flush=(k == len(waves) - 1))
                assert k == len(waves) - 1 or r["n_batched"] % B == 0
                got[c].append(r["batched"])
        o.close()
        runs.append(got)
    for c in range(C):
        for u, v in zip(runs[0][c], runs[1][c]):
            assert np.array_equal(u, v)
        seen, seq = set(), []
        for v in cand.tolist():
            if calls[cp[v]] == c and v not in seen:
                seen.add(v)
                seq.append(v)
        assert np.array_equal(np.concatenate(runs[0][c]), np.array(seq, np.uint32))


def test_batch_ready_capacity_leaves_state():
    o = OracleCtx()
    ex = o.expand([4, 4])
    r = o.batch_ready(ex["xid"], 0, [5, 1, 2, 7], 2, flush=True, cap=3, check=False)
    assert r["status"] == E_CAPACITY and r["n_batched"] == 4
    again = o.batch_ready(ex["xid"], 0, [5, 1, 2, 7], 2, flush=True, cap=4)
    assert list(again["batched"]) == [5, 1, 2, 7]


# --------------------------------------------------------------- completion
@pytest.mark.parametrize("waves", [1, 3, 17])
def test_commit_completes_parent_in_wave_of_last_child(waves):
    w = tiny(parents=120, salt=waves)
    lv = w.top
    from workload.configs import _wave_bounds
    lv.wave_bounds = _wave_bounds(lv.n_children, waves)
    o = OracleCtx()
    ex, br, res = run_level_oracle(o, lv, host_arena(lv))
    expect = closed_form_done_wave(lv)
    seen = []
    for wv, (cm, _) in enumerate(res):
        assert np.all(cm["code"] == ACCEPT)
        assert np.array_equal(cm["done"], np.flatnonzero(expect == wv))
        seen += list(cm["done"])
    assert sorted(seen) == list(range(lv.n_parents))


def test_commit_generation_fence():
    o = OracleCtx()
    ex = o.expand([2, 3])          # A0 A1 | B0 B1 B2
    x = ex["xid"]
    o.batch_ready(x, 0, [0, 1, 2, 3], 3, flush=False)   # 0,1,2 in flight; 3 READY
    ch = np.array([4, 3, 0, 1, 0, 9, 2, 1, 2], np.uint32)
    st = np.array([1, 1, 1, 1, 1, 1, 7, 3, 1], np.uint8)
    ln = np.array([8, 8, 8, 8, 8, 8, 8, 8, 99], np.uint32)
    of = np.array([0, 0, 0, 8, 0, 0, 0, 0, 90], np.uint64)
    gen = np.array([0, 0, 0, 0, 0, 0, 0, 1, 0], np.uint32)
    cm = o.gather_commit(x, ch, st, ln, of, gen=gen, arena_bytes=100)
    assert list(cm["code"]) == [REJ_NOT_INFLIGHT,   # waiting child
                                REJ_NOT_INFLIGHT,   # queued (READY) child
                                ACCEPT,             # A0
                                ACCEPT,             # A1
                                REJ_DUPLICATE,      # A0 again in the same commit
                                REJ_INVALID,        # no such child
                                REJ_INVALID,        # unknown outcome
                                REJ_STALE_GEN,      # A1 at a generation never issued
                                REJ_INVALID]        # payload past the arena end
    assert list(cm["done"]) == [0]
    # a later duplicate of A1 is refused and changes nothing
    again = o.gather_commit(x, np.array([1], np.uint32), np.array([3], np.uint8),
                            np.array([0], np.uint32), np.array([0], np.uint64))
    assert list(again["code"]) == [REJ_DUPLICATE] and again["n_done"] == 0
    a = o.assemble(x, np.zeros(100, np.uint8), parents=[0, 1])
    assert list(a["parent_status"]) == [PRESENT, PENDING]
    s = o.stats()
    assert (s["accepted"], s["rej_invalid"], s["rej_not_inflight"], s["rej_stale_gen"],
            s["rej_duplicate"]) == (2, 3, 2, 1, 2)


# ------------------------------------------------------------ Reduce rule
@pytest.mark.parametrize("m", [0, 1, 2, 3])
def test_reduce_rule_all_member_outcomes(m):
    outcomes = [PRESENT, DROPPED, FAILED, SUPPRESSED]
    seed = 77
    for combo in itertools.product(outcomes, repeat=m):
        o = OracleCtx()
        ex = o.expand([m])
        x = ex["xid"]
        if m:
            o.batch_ready(x, 0, None, 1, flush=True)
            lens = np.array([5 + 3 * j for j in range(m)], np.uint32)
            offs = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.uint64)
            arena = np.frombuffer(b"".join(record_bytes(seed, j, int(lens[j]))
                                           for j in range(m)), np.uint8)
            # reports arrive in reverse ordinal order
            order = np.arange(m)[::-1]
            cm = o.gather_commit(x, order.astype(np.uint32), np.array(combo, np.uint8)[order],
                                 lens[order], offs[order], arena_bytes=arena.size)
            assert list(cm["done"]) == [0]
        else:
            arena = np.zeros(1, np.uint8)
        a = o.assemble(x, arena, parents=[0])
        bad = any(c in (FAILED, SUPPRESSED) for c in combo)
        if bad:
            assert list(a["parent_status"]) == [SUPPRESSED] and a["out_bytes"] == 0
        else:
            want = b"".join(record_bytes(seed, j, 5 + 3 * j)
                            for j in range(m) if combo[j] == PRESENT)
            assert list(a["parent_status"]) == [PRESENT]
            assert bytes(a["out"][:a["out_bytes"]]) == want
            assert list(a["out_len"]) == [len(want)]


# ------------------------------------------------------ schedule invariance
def test_schedule_invariance_all_arrival_orders():
    """Eq. (4): final Items do not depend on arrival order, wave cuts or batch size."""
    counts = [2, 0, 3, 1]
    states = np.array([1, 2, 1, 1, 1, 3], np.uint8)   # child 5 (parent 3) FAILED
    lens = np.array([4, 9, 7, 1, 12, 6], np.uint32)
    offs = np.concatenate([[0], np.cumsum(lens)[:-1]]).astype(np.uint64)
    arena = np.arange(int(lens.sum()), dtype=np.uint8) * 7
    final = None
    for perm in itertools.permutations(range(6)):
        perm = np.array(perm, np.uint32)
        cut = int(perm[0]) % 6          # vary the wave split with the order
        B = 1 + int(perm[1])
        o = OracleCtx()
        x = o.expand(counts)["xid"]
        o.batch_ready(x, 0, None, B, flush=True)
        items = {}
        for chunk in (perm[:cut], perm[cut:]):
            cm = o.gather_commit(x, chunk, states[chunk], lens[chunk], offs[chunk],
                                 arena_bytes=arena.size)
            a = o.assemble(x, arena, parents=None, n_parents=4)
            for i, p in enumerate(cm["done"]):
                s, e = a["out_off"][i], a["out_off"][i + 1]
                items[int(p)] = (int(a["parent_status"][i]), bytes(a["out"][s:e]))
        a0 = o.assemble(x, arena, parents=[1])      # the empty expansion
        items[1] = (int(a0["parent_status"][0]), bytes(a0["out"][:a0["out_bytes"]]))
        if final is None:
            final = items
        assert items == final
    assert final[1] == (PRESENT, b"")
    assert final[3][0] == SUPPRESSED
    assert final[0] == (PRESENT, bytes(arena[0:4]))        # child 1 DROPPED
    assert final[2] == (PRESENT, bytes(arena[13:13 + 7 + 1 + 12]))


# ------------------------------------------------------------ whole levels
def test_tiny_config_assembled_bytes_closed_form():
    w = tiny(parents=300)
    lv = w.top
    o = OracleCtx()
    ex, br, res = run_level_oracle(o, lv, host_arena(lv))
    assert np.array_equal(br["batched"], np.arange(lv.n_children))
    assert br["n_batches"] == -(-lv.n_children // lv.batch_size)
    seen = 0
    for cm, a in res:
        for i, p in enumerate(cm["done"]):
            s, e = int(a["out_off"][i]), int(a["out_off"][i + 1])
            status, want = closed_form_parent(lv, int(p))
            assert int(a["parent_status"][i]) == status
            assert bytes(a["out"][s:e]) == want
            seen += 1
    assert seen == lv.n_parents


def test_nested_video_levels_closed_form():
    w = video(videos=60)
    top, leaf = w.levels
    o = OracleCtx()
    arena = host_arena(leaf)
    ex0 = o.expand(top.counts)
    x0 = ex0["xid"]
    ex1 = o.expand(leaf.counts, parent_xid=x0)
    x1 = ex1["xid"]
    o.batch_ready(x0, 0, None, top.batch_size, flush=True)
    o.batch_ready(x1, 0, None, leaf.batch_size, flush=True)
    ch, st, ln, of = leaf.reports(leaf.wave(0))
    cm1 = o.gather_commit(x1, ch, st, ln, of, arena_bytes=leaf.arena_bytes)
    assert cm1["n_done"] == top.n_children
    a1 = o.assemble(x1, arena, parents=None, n_parents=cm1["n_done"])
    # each clip's result becomes the report of that clip in the video expansion
    cm0 = o.gather_commit(x0, cm1["done"], a1["parent_status"], a1["out_len"],
                          a1["out_off"][:-1], arena_bytes=a1["out_bytes"])
    assert cm0["n_done"] == top.n_parents
    a0 = o.assemble(x0, a1["out"], parents=None, n_parents=cm0["n_done"])
    frame_off = np.concatenate([[0], np.cumsum(leaf.counts.astype(np.uint64))])
    clip_off = np.concatenate([[0], np.cumsum(top.counts.astype(np.uint64))])
    for i, v in enumerate(cm0["done"]):
        want = b"".join(record_bytes(leaf.payload_seed, f, 512)
                        for clip in range(int(clip_off[v]), int(clip_off[v + 1]))
                        for f in range(int(frame_off[clip]), int(frame_off[clip + 1])))
        s, e = int(a0["out_off"][i]), int(a0["out_off"][i + 1])
        assert bytes(a0["out"][s:e]) == want


def test_assemble_cursor_and_capacity():
    o = OracleCtx()
    x = o.expand([1, 1])["xid"]
    o.batch_ready(x, 0, None, 2, flush=True)
    arena = np.arange(20, dtype=np.uint8)
    o.gather_commit(x, np.array([0, 1], np.uint32), np.array([1, 1], np.uint8),
                    np.array([3, 5], np.uint32), np.array([2, 10], np.uint64), arena_bytes=20)
    r = o.assemble(x, arena, parents=[1, 0], out_cap=9, cursor=2, check=False)
    assert r["status"] == E_CAPACITY and r["out_bytes"] == 8
    r = o.assemble(x, arena, parents=[1, 0], out_cap=10, cursor=2)
    assert list(r["out_off"]) == [2, 7, 10] and r["cursor"] == 10
    assert list(r["out"][2:10]) == [10, 11, 12, 13, 14, 2, 3, 4]
