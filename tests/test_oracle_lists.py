"""Pins of the oracle's list-structured Reduce output and F.filter
(Section 4.2: present values in immutable ordinal order, Dropped members
excluded, zero survivors give a present empty list; Table 3's F.filter:
pass on true, drop on false, with the propagation precedence of Section
4.2).  The list entries are checked against the records themselves
(regenerated from the payload definition), not against the oracle."""
import numpy as np
import pytest

from oracle import DROPPED, FAILED, PRESENT, SUPPRESSED, OracleCtx
from tests.pipeline import host_arena
from workload import record_bytes, tiny


def test_filter_rule_closed_form():
    rng = np.random.default_rng(5)
    st = rng.choice([PRESENT, DROPPED, FAILED, SUPPRESSED], 1000).astype(np.uint8)
    keep = rng.integers(0, 2, 1000).astype(np.uint8)
    got = OracleCtx.filter_reports(st, keep)
    want = np.where((st == PRESENT) & (keep == 0), DROPPED, st)
    assert np.array_equal(got, want)


@pytest.mark.parametrize("seed", [0, 1])
def test_list_entries_split_the_concatenation(seed):
    lv = tiny().top
    rng = np.random.default_rng(70 + seed)
    # a filter drops some Present results (and leaves one parent with no survivors)
    keep = (rng.random(lv.n_children) < 0.8).astype(np.uint8)
    off = np.concatenate([[0], np.cumsum(lv.counts.astype(np.int64))])
    p_all = int(np.flatnonzero((lv.counts >= 2) & np.array(
        [not np.any(lv.state[off[p]:off[p + 1]] == FAILED) for p in range(lv.n_parents)]))[0])
    keep[off[p_all]:off[p_all + 1]] = 0
    state = OracleCtx.filter_reports(lv.state, keep)
    arena = host_arena(lv)
    o = OracleCtx()
    x = o.expand(lv.counts)["xid"]
    o.batch_ready(x, 0, None, lv.batch_size, flush=True)
    ch = lv.arrival
    o.gather_commit(x, ch, state[ch], lv.length[ch], lv.arena_off[ch], arena_bytes=lv.arena_bytes)
    lst = rng.permutation(lv.n_parents).astype(np.uint32)
    r = o.assemble_list(x, arena, parents=lst, cursor=11)
    assert r["status"] == 0
    for i, p in enumerate(lst):
        p = int(p)
        e0, e1 = int(r["elem_base"][i]), int(r["elem_base"][i + 1])
        s0, s1 = int(r["out_off"][i]), int(r["out_off"][i + 1])
        states = state[off[p]:off[p + 1]]
        if np.any((states == FAILED) | (states == SUPPRESSED)):
            assert r["parent_status"][i] == SUPPRESSED and e1 == e0 and s1 == s0
            continue
        assert r["parent_status"][i] == PRESENT and e1 - e0 == lv.counts[p]
        pos = s0
        for j in range(int(lv.counts[p])):
            c = off[p] + j
            assert r["elem_state"][e0 + j] == states[j]
            assert r["elem_off"][e0 + j] == pos
            want = record_bytes(lv.payload_seed, c, int(lv.length[c])) if states[j] == PRESENT else b""
            ln = int(r["elem_len"][e0 + j])
            assert bytes(r["out"][pos:pos + ln]) == want
            pos += ln
        assert pos == s1
        if p == p_all:
            assert s1 == s0 and all(r["elem_state"][e0:e1] == DROPPED)   # a present empty list
    o.close()


def test_list_capacity_refuses_and_changes_nothing():
    o = OracleCtx()
    x = o.expand([3, 2])["xid"]
    o.batch_ready(x, 0, None, 8, flush=True)
    ch = np.arange(5, dtype=np.uint32)
    o.gather_commit(x, ch, np.full(5, PRESENT, np.uint8), np.full(5, 4, np.uint32),
                    ch.astype(np.uint64) * 4, arena_bytes=64)
    arena = np.arange(64, dtype=np.uint8)
    r = o.assemble_list(x, arena, parents=[0, 1], elem_cap=4, check=False)
    assert r["status"] == 2 and r["n_elems"] == 5
    r = o.assemble_list(x, arena, parents=[0, 1], elem_cap=5)
    assert list(r["elem_base"]) == [0, 3, 5] and list(r["elem_len"]) == [4] * 5
    o.close()
