"""Seeded synthetic lineage workloads (the five benchmark configurations).

The paper's corpora (MinerU PDFs, videos) are not available, so these
generators stand in for them with the shapes the benchmark names: long-tailed
per-parent child counts (document -> page, video -> clip -> frame), a skewed
fan-out case and a streaming multi-Call case.  They hold none of the lineage
method's arithmetic: they only draw counts, per-child result attributes,
arrival orders and readiness orders.  Children are numbered parent-major
(child ``c`` of parent ``p`` with ordinal ``j`` is ``sum(counts[:p]) + j``),
which is how per-child arrays here are indexed.

Readings of unspecified details (rounding, Pareto form, wave cuts, arena
layout) are the ones recorded in the design notes:

* lognormal draws are rounded half-to-even (``np.rint``) and then clamped;
* Pareto(alpha) is the classic form with x_m = 1: ``floor(U ** (-1/alpha))``;
* W arrival waves cut one seeded permutation into W contiguous chunks, the
  first ``n mod W`` chunks one longer;
* result records of PRESENT children are packed back to back (no padding, so
  arbitrary alignment) in arrival order; FAILED children carry no payload.
"""
from __future__ import annotations

from dataclasses import dataclass, field
from typing import List, Optional

import numpy as np

# Eq. (1) Item outcomes as carried by result reports (same numbering as the C ABI)
PRESENT, DROPPED, FAILED, SUPPRESSED = 1, 2, 3, 4

BASE_SEED = 0x52415930


@dataclass
class Level:
    """One expansion level: parents, child counts and per-child results."""
    counts: np.ndarray                     # uint32[P]
    n_children: int
    batch_size: int
    n_calls: int = 1
    parent_call: Optional[np.ndarray] = None   # uint8[P]; None -> every child goes to call 0
    state: Optional[np.ndarray] = None     # uint8[N] result state per child
    length: Optional[np.ndarray] = None    # uint32[N] payload bytes (0 unless PRESENT)
    arena_off: Optional[np.ndarray] = None  # uint64[N] record offset (0 unless PRESENT)
    arena_bytes: int = 0
    arrival: Optional[np.ndarray] = None   # uint32[N] children in result-arrival order
    wave_bounds: Optional[np.ndarray] = None  # int64[W+1]
    readiness: Optional[np.ndarray] = None  # uint32[N] children in readiness order (None: all at expand)
    ready_bounds: Optional[np.ndarray] = None  # int64[R+1]
    key: Optional[np.ndarray] = None       # uint64[N] arrival key inside a wave (streaming case)
    payload_seed: int = 0

    @property
    def n_parents(self) -> int:
        return int(self.counts.size)

    def wave(self, w: int) -> np.ndarray:
        return self.arrival[self.wave_bounds[w]:self.wave_bounds[w + 1]]

    @property
    def n_waves(self) -> int:
        return int(self.wave_bounds.size - 1) if self.wave_bounds is not None else 0

    def reports(self, children: np.ndarray):
        """Result reports (child, state, len, arena_off) for the given children."""
        children = np.asarray(children, dtype=np.uint32)
        return (children, self.state[children], self.length[children],
                self.arena_off[children])


@dataclass
class Workload:
    name: str
    levels: List[Level] = field(default_factory=list)
    description: str = ""

    @property
    def top(self) -> Level:
        return self.levels[0]

    @property
    def leaf(self) -> Level:
        return self.levels[-1]

    @property
    def total_children(self) -> int:
        return int(sum(lv.n_children for lv in self.levels))


def _streams(cfg: int, salt: int = 0):
    ss = np.random.SeedSequence([BASE_SEED + cfg, salt])
    return [np.random.Generator(np.random.PCG64(s)) for s in ss.spawn(8)]


def _wave_bounds(n: int, w: int) -> np.ndarray:
    w = max(1, int(w))
    sizes = np.full(w, n // w, dtype=np.int64)
    sizes[: n % w] += 1
    return np.concatenate([[0], np.cumsum(sizes)]).astype(np.int64)


def _lognormal_int(rng, mu, sigma, size, lo=None, hi=None, dtype=np.uint32):
    x = np.rint(rng.lognormal(mu, sigma, size))
    if lo is not None or hi is not None:
        x = np.clip(x, lo if lo is not None else -np.inf, hi if hi is not None else np.inf)
    return x.astype(dtype)


def _finish_results(lv: Level, rng_state, rng_arrival, fail_rate: float,
                    record_len, n_waves: int, payload_seed: int,
                    arena_in_arrival_order: bool = True) -> None:
    n = lv.n_children
    if fail_rate > 0:
        failed = rng_state.random(n) < fail_rate
    else:
        failed = np.zeros(n, dtype=bool)
    lv.state = np.where(failed, FAILED, PRESENT).astype(np.uint8)
    length = np.asarray(record_len, dtype=np.uint32)
    if length.ndim == 0:
        length = np.full(n, int(length), dtype=np.uint32)
    length = np.where(failed, 0, length).astype(np.uint32)
    lv.length = length
    lv.arrival = rng_arrival.permutation(n).astype(np.uint32)
    lv.wave_bounds = _wave_bounds(n, n_waves)
    order = lv.arrival if arena_in_arrival_order else np.arange(n, dtype=np.uint32)
    ordered_len = length[order].astype(np.uint64)
    starts = np.cumsum(ordered_len) - ordered_len
    off = np.zeros(n, dtype=np.uint64)
    off[order] = starts
    lv.arena_off = np.where(failed, 0, off).astype(np.uint64)
    lv.arena_bytes = int(ordered_len.sum())
    lv.payload_seed = int(payload_seed)


def tiny(parents: int = 1000, salt: int = 0) -> Workload:
    """1,000 parents, counts LN(2.0, 1.0) in [1, 500], 64 B records, 3 % FAILED,
    one random arrival permutation, batch size 64, one Call."""
    r = _streams(1, salt)
    counts = _lognormal_int(r[0], 2.0, 1.0, parents, 1, 500)
    n = int(counts.sum(dtype=np.uint64))
    lv = Level(counts=counts, n_children=n, batch_size=64)
    _finish_results(lv, r[2], r[4], 0.03, 64, 1, int(r[7].integers(1 << 63)))
    return Workload("tiny single-level lineage (1k parents, 64 B records)", [lv])


def docpage(parents: int = 1_000_000, waves: int = 256, salt: int = 0) -> Workload:
    """Document -> page: counts LN(2.3, 1.0) in [1, 2000], payload LN(7.5, 0.8)
    bytes in [256, 65536], 5 % FAILED, 256 random arrival waves, batch 256."""
    r = _streams(2, salt)
    counts = _lognormal_int(r[0], 2.3, 1.0, parents, 1, 2000)
    n = int(counts.sum(dtype=np.uint64))
    lens = _lognormal_int(r[3], 7.5, 0.8, n, 256, 65536)
    lv = Level(counts=counts, n_children=n, batch_size=256)
    _finish_results(lv, r[2], r[4], 0.05, lens, waves, int(r[7].integers(1 << 63)))
    return Workload(f"document->page ({parents} documents, {waves} waves)", [lv])


def video(videos: int = 100_000, salt: int = 0) -> Workload:
    """Video -> clip -> frame: clips Pareto(1.5) capped at 1000, frames U[8, 64],
    512 B frame records, no failures, one random arrival wave, batch 1024."""
    r = _streams(3, salt)
    u = 1.0 - r[0].random(videos)            # (0, 1]
    clips = np.minimum(1000, np.floor(u ** (-1.0 / 1.5))).astype(np.uint32)
    n_clips = int(clips.sum(dtype=np.uint64))
    frames = r[1].integers(8, 65, size=n_clips).astype(np.uint32)
    n_frames = int(frames.sum(dtype=np.uint64))
    top = Level(counts=clips, n_children=n_clips, batch_size=1024)
    leaf = Level(counts=frames, n_children=n_frames, batch_size=1024)
    _finish_results(leaf, r[2], r[4], 0.0, 512, 1, int(r[7].integers(1 << 63)))
    return Workload(f"video->clip->frame ({videos} videos)", [top, leaf])


def skew(parents: int = 10_000_000, heavy: int = 1000, heavy_children: int = 100_000,
         salt: int = 0) -> Workload:
    """Extreme skew: every parent has 1 child except ``heavy`` uniformly placed
    parents with ``heavy_children`` each; 32 B records; one random arrival wave."""
    r = _streams(4, salt)
    counts = np.ones(parents, dtype=np.uint32)
    hot = r[1].choice(parents, size=heavy, replace=False)
    counts[hot] = heavy_children
    n = int(counts.sum(dtype=np.uint64))
    lv = Level(counts=counts, n_children=n, batch_size=256)
    _finish_results(lv, r[2], r[4], 0.0, 32, 1, int(r[7].integers(1 << 63)))
    return Workload(f"extreme skew ({parents} parents, {heavy}x{heavy_children})", [lv])


def streaming(total_children: int = 50_000_000, batch_size: int = 256,
              ready_waves: int = 1000, n_calls: int = 4, salt: int = 0) -> Workload:
    """Streaming multi-Call: parent p feeds Call p mod 4; counts LN(2.5, 1.2)
    (rounded, not clamped, so a few expansions are empty) drawn until their sum
    reaches ``total_children``; children become ready in 1,000 waves of one
    seeded permutation; 1 KB records; 2 % FAILED.  Results of the children
    reserved in a wave arrive in that wave, ordered by a per-child key."""
    r = _streams(5, salt)
    est = int(total_children / np.exp(2.5 + 0.72) * 1.1) + 16
    counts = _lognormal_int(r[0], 2.5, 1.2, est, None, None)
    csum = np.cumsum(counts, dtype=np.uint64)
    while csum[-1] < total_children:
        more = _lognormal_int(r[0], 2.5, 1.2, est, None, None)
        counts = np.concatenate([counts, more])
        csum = np.cumsum(counts, dtype=np.uint64)
    cut = int(np.searchsorted(csum, total_children, side="left")) + 1
    counts = counts[:cut].copy()
    n = int(counts.sum(dtype=np.uint64))
    P = counts.size
    lv = Level(counts=counts, n_children=n, batch_size=batch_size, n_calls=n_calls,
               parent_call=(np.arange(P) % n_calls).astype(np.uint8))
    _finish_results(lv, r[2], r[4], 0.02, 1024, 1, int(r[7].integers(1 << 63)),
                    arena_in_arrival_order=False)
    lv.arrival = None
    lv.wave_bounds = None
    lv.readiness = r[5].permutation(n).astype(np.uint32)
    lv.ready_bounds = _wave_bounds(n, ready_waves)
    lv.key = r[6].integers(0, 1 << 63, size=n, dtype=np.uint64)
    return Workload(f"streaming {n_calls} Calls ({n} children, batch {batch_size})", [lv])


def _restrict_order(order: np.ndarray, bounds: np.ndarray, keep_below: int):
    """The entries of `order` below `keep_below`, in order, with the bounds of
    the waves they fell in."""
    n_w = bounds.size - 1
    wave = np.repeat(np.arange(n_w, dtype=np.int64), np.diff(bounds))
    keep = order < keep_below
    kept = order[keep]
    per = np.bincount(wave[keep], minlength=n_w)
    return kept.astype(np.uint32), np.concatenate([[0], np.cumsum(per)]).astype(np.int64)


def _repack(lv: Level, order: np.ndarray) -> None:
    """Lay the PRESENT records out back to back in `order` (no padding)."""
    ordered_len = lv.length[order].astype(np.uint64)
    starts = np.cumsum(ordered_len) - ordered_len
    off = np.zeros(lv.n_children, dtype=np.uint64)
    off[order] = starts
    lv.arena_off = np.where(lv.length > 0, off, 0).astype(np.uint64)
    lv.arena_bytes = int(ordered_len.sum())


def _head_level(lv: Level, parents: int) -> Level:
    counts = lv.counts[:parents].copy()
    n = int(counts.sum(dtype=np.uint64))
    out = Level(counts=counts, n_children=n, batch_size=lv.batch_size, n_calls=lv.n_calls,
                parent_call=None if lv.parent_call is None else lv.parent_call[:parents].copy(),
                payload_seed=lv.payload_seed)
    if lv.state is not None:
        out.state = lv.state[:n].copy()
        out.length = lv.length[:n].copy()
    if lv.key is not None:
        out.key = lv.key[:n].copy()
    if lv.arrival is not None:
        out.arrival, out.wave_bounds = _restrict_order(lv.arrival, lv.wave_bounds, n)
    if lv.readiness is not None:
        out.readiness, out.ready_bounds = _restrict_order(lv.readiness, lv.ready_bounds, n)
    if out.length is not None:
        # arrival order when there is one (configs 1-4), else child order
        _repack(out, out.arrival if out.arrival is not None else np.arange(n, dtype=np.uint32))
    return out


def subset(wl: Workload, parents: int) -> Workload:
    """The first `parents` top-level parents of a drawn workload with all
    their descendants: the same draws (counts, outcomes, lengths, payload
    seed, arrival and readiness orders restricted to the kept children, wave
    by wave), the records packed into a smaller arena in the same order."""
    levels = []
    keep = parents
    for lv in wl.levels:
        keep = min(keep, lv.n_parents)
        h = _head_level(lv, keep)
        levels.append(h)
        keep = h.n_children   # the next level's parents are these children
    return Workload(f"{wl.name}, first {parents} parents", levels, wl.description)


CONFIGS = {
    "tiny": tiny,
    "docpage": docpage,
    "video": video,
    "skew": skew,
    "streaming": streaming,
}
