"""Pipeline drivers shared by the tests: run a workload level through the
oracle (host) and compute the closed-form expectations that pin it.

Closed forms here use only the workload's own draws and numpy library
routines (cumsum, repeat, unique, max-reduce), never the oracle.
"""
from __future__ import annotations

import numpy as np

from workload import FAILED, PRESENT, SUPPRESSED, Level, level_arena, record_bytes

host_arena = level_arena   # the level's host result arena (input generation)


def closed_form_lineage(counts: np.ndarray):
    counts = np.asarray(counts, dtype=np.uint64)
    offsets = np.concatenate([[0], np.cumsum(counts)]).astype(np.uint64)
    P = counts.size
    child_parent = np.repeat(np.arange(P, dtype=np.int64), counts.astype(np.int64)).astype(np.uint32)
    ordinal = (np.arange(offsets[-1], dtype=np.uint64) - offsets[child_parent]).astype(np.uint32)
    empties = np.flatnonzero(counts == 0).astype(np.uint32)
    return offsets, child_parent, ordinal, empties


def closed_form_done_wave(lv: Level) -> np.ndarray:
    """Wave in which each parent completes: the wave of its last-arriving child
    (-1 for empty parents)."""
    wave_of = np.empty(lv.n_children, dtype=np.int64)
    for w in range(lv.n_waves):
        wave_of[lv.wave(w)] = w
    _, child_parent, _, _ = closed_form_lineage(lv.counts)
    done = np.full(lv.n_parents, -1, dtype=np.int64)
    np.maximum.at(done, child_parent.astype(np.int64), wave_of)
    return done


def closed_form_parent(lv: Level, p: int):
    """(status, bytes) the Reduce rule gives parent p, from the drawn results."""
    off = int(lv.counts[:p].sum(dtype=np.uint64))
    m = int(lv.counts[p])
    states = lv.state[off:off + m]
    if np.any((states == FAILED) | (states == SUPPRESSED)):
        return SUPPRESSED, b""
    parts = [record_bytes(lv.payload_seed, off + j, int(lv.length[off + j]))
             for j in range(m) if states[j] == PRESENT]
    return PRESENT, b"".join(parts)


def run_level_oracle(o, lv: Level, arena: np.ndarray, parent_xid: int = -1):
    """expand -> one readiness wave (all children, flush) -> per arrival wave:
    commit + assemble of the parents that wave completed."""
    ex = o.expand(lv.counts, parent_xid=parent_xid, parent_call=lv.parent_call)
    xid = ex["xid"]
    br = o.batch_ready(xid, 0, None, lv.batch_size, flush=True)
    waves = []
    for w in range(lv.n_waves):
        ch, st, ln, of = lv.reports(lv.wave(w))
        cm = o.gather_commit(xid, ch, st, ln, of, arena_bytes=lv.arena_bytes)
        asm = o.assemble(xid, arena, parents=None, n_parents=cm["n_done"])
        waves.append((cm, asm))
    return ex, br, waves
