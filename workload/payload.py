"""Counter-based payload bytes for synthetic child results (host side).

Every PRESENT child result is a record of ``len`` bytes whose byte ``j`` is
byte ``j & 7`` (little endian) of ``mix64(x)`` with

    x = seed ^ (child * 0x9E3779B97F4A7C15) + (j >> 3) * 0xD1B54A32D192ED03   (mod 2**64)

``mix64`` is the SplitMix64 output finaliser (Steele, Lea and Flood,
"Fast splittable pseudorandom number generators", OOPSLA 2014; the
variant with Stafford's "Mix13" constants).  The bytes of a record depend
only on (seed, child, j), never on where the record sits in the arena, so a
checker can regenerate any expected output without reading the arena.

The device-side fill in ``csrc/payload_fill.cu`` implements the same
published definition independently; ``tests/test_workload.py`` checks that
both agree.  Nothing here belongs to the lineage method: this module only
makes inputs.
"""
from __future__ import annotations

import os
from concurrent.futures import ThreadPoolExecutor

import numpy as np

GOLDEN = np.uint64(0x9E3779B97F4A7C15)
WORDSTEP = np.uint64(0xD1B54A32D192ED03)
_M1 = np.uint64(0xBF58476D1CE4E5B9)
_M2 = np.uint64(0x94D049BB133111EB)


def mix64(z: np.ndarray) -> np.ndarray:
    """SplitMix64 finaliser on a uint64 array (wrapping arithmetic)."""
    z = np.asarray(z, dtype=np.uint64)
    with np.errstate(over="ignore"):
        z = (z ^ (z >> np.uint64(30))) * _M1
        z = (z ^ (z >> np.uint64(27))) * _M2
        z = z ^ (z >> np.uint64(31))
    return z


def record_bytes(seed: int, child: int, length: int) -> bytes:
    """The ``length`` payload bytes of one child's result record."""
    if length == 0:
        return b""
    n_words = (length + 7) // 8
    with np.errstate(over="ignore"):
        base = np.uint64(seed) ^ (np.uint64(child) * GOLDEN)
        x = base + np.arange(n_words, dtype=np.uint64) * WORDSTEP
    words = mix64(x).astype("<u8")
    return words.tobytes()[:length]


def records_concat(seed: int, children, lengths) -> bytes:
    """Concatenation of several children's records, in the order given."""
    return b"".join(record_bytes(seed, int(c), int(n)) for c, n in zip(children, lengths))


def _host_lib():
    import ctypes as C
    import os
    from .build import HOST_LIB, build_host
    if not os.path.exists(HOST_LIB):
        build_host()
    L = C.CDLL(HOST_LIB)
    L.wl_fill_host.argtypes = [C.c_void_p, C.c_uint64, C.c_void_p, C.c_void_p, C.c_void_p,
                               C.c_uint64, C.c_uint64]
    L.wl_fill_host.restype = C.c_int
    return L


def fill_host_arena(seed: int, children: np.ndarray, offsets: np.ndarray,
                    lengths: np.ndarray, arena_bytes: int, use_c: bool = True,
                    chunk_bytes: int = 1 << 26) -> np.ndarray:
    """Build a host arena (uint8) holding each listed child's record at its offset.

    Uses the C filler (``csrc/payload_host.c``) when gcc is available, else a
    numpy version vectorised over children in chunks of ``chunk_bytes``.
    Children with length 0 are skipped.
    """
    arena = np.zeros(max(arena_bytes, 1), dtype=np.uint8)[:arena_bytes]
    if use_c:
        try:
            L = _host_lib()
        except Exception:
            L = None
        if L is not None:
            c = np.ascontiguousarray(children, dtype=np.uint64)
            o = np.ascontiguousarray(offsets, dtype=np.uint64)
            ln = np.ascontiguousarray(lengths, dtype=np.uint64)
            # records never overlap, so chunks of children fill in parallel
            n_threads = max(1, min(16, (os.cpu_count() or 1), c.size // 100000))
            bounds = np.linspace(0, c.size, n_threads + 1).astype(np.int64)

            def part(k):
                s0, s1 = int(bounds[k]), int(bounds[k + 1])
                return L.wl_fill_host(arena.ctypes.data, arena_bytes, c.ctypes.data + 8 * s0,
                                      o.ctypes.data + 8 * s0, ln.ctypes.data + 8 * s0, s1 - s0,
                                      seed & ((1 << 64) - 1))
            with ThreadPoolExecutor(n_threads) as ex:
                if any(ex.map(part, range(n_threads))):
                    raise ValueError("record outside the arena")
            return arena
    children = np.asarray(children, dtype=np.uint64)
    offsets = np.asarray(offsets, dtype=np.uint64)
    lengths = np.asarray(lengths, dtype=np.int64)
    keep = lengths > 0
    children, offsets, lengths = children[keep], offsets[keep], lengths[keep]
    if children.size == 0:
        return arena
    csum = np.cumsum(lengths)
    start = 0
    while start < children.size:
        done_before = int(csum[start - 1]) if start else 0
        end = int(np.searchsorted(csum, done_before + chunk_bytes, side="right"))
        end = max(end, start + 1)
        c = children[start:end]
        o = offsets[start:end]
        ln = lengths[start:end]
        nw = (ln + 7) // 8
        owner = np.repeat(np.arange(c.size), nw)
        first_word = np.cumsum(nw) - nw
        widx = np.arange(owner.size, dtype=np.int64) - np.repeat(first_word, nw)
        with np.errstate(over="ignore"):
            x = (np.uint64(seed) ^ (c[owner] * GOLDEN)) + widx.astype(np.uint64) * WORDSTEP
        by = mix64(x).astype("<u8").view(np.uint8)
        # byte b of word row -> (child owner, byte-in-record widx*8 + b)
        bowner = np.repeat(owner, 8)
        bpos = (np.repeat(widx, 8) * 8 + np.tile(np.arange(8), owner.size))
        valid = bpos < ln[bowner]
        dst = o[bowner[valid]].astype(np.int64) + bpos[valid]
        arena[dst] = by[valid]
        start = end
    return arena


def level_arena(lv) -> np.ndarray:
    """The host result arena of a workload level: every child's record at
    its arena offset (FAILED children have none)."""
    n = lv.n_children
    return fill_host_arena(lv.payload_seed, np.arange(n, dtype=np.uint64), lv.arena_off,
                           lv.length, lv.arena_bytes)
