"""ctypes wrapper around the plain-C oracle (``oracle.c``).

TEST INFRASTRUCTURE ONLY: the tests, ``__graft_entry__.smoke()`` and the
benchmark's CPU-baseline leg use it; the GPU library never does.

Each method mirrors one oracle entry point on numpy host arrays and returns
numpy results.  Non-zero statuses raise :class:`OracleError` unless
``check=False`` is given, in which case the status is returned alongside.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional

import numpy as np

from .build import LIB, build

OK, E_INVAL, E_CAPACITY, E_OVERFLOW, E_STATE, E_OOM = range(6)
PENDING, PRESENT, DROPPED, FAILED, SUPPRESSED = range(5)
GROUP_FAILURE = 5   # report kind (Section 4.4): the Grain failed and its open siblings are suppressed
ACCEPT, REJ_INVALID, REJ_NOT_INFLIGHT, REJ_STALE_GEN, REJ_DUPLICATE, REJ_BARRIER = range(6)

_u8p = C.POINTER(C.c_uint8)
_u32p = C.POINTER(C.c_uint32)
_u64p = C.POINTER(C.c_uint64)
_i32p = C.POINTER(C.c_int32)


class OracleError(RuntimeError):
    def __init__(self, fn: str, status: int):
        super().__init__(f"{fn} returned status {status}")
        self.status = status


class _Stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in (
        "accepted", "rej_invalid", "rej_not_inflight", "rej_stale_gen", "rej_duplicate",
        "ready_bad_candidates", "assemble_incomplete", "rej_barrier", "barrier_not_dispatched",
        "barrier_in_flight", "queue_dropped", "retried", "retry_skipped")]


_lib = None


def lib():
    """The oracle library (``ORACLE_LIB`` overrides the path, used by the
    planted-mistake tests to load a deliberately broken copy)."""
    global _lib
    if _lib is None:
        path = os.environ.get("ORACLE_LIB")
        if not path:
            if not os.path.exists(LIB):
                build()
            path = LIB
        L = C.CDLL(path)
        L.or_ctx_create.restype = C.c_void_p
        L.or_ctx_create.argtypes = [C.c_uint32]
        L.or_ctx_destroy.argtypes = [C.c_void_p]
        L.or_ctx_reset.argtypes = [C.c_void_p]
        L.or_ctx_stats.argtypes = [C.c_void_p, C.POINTER(_Stats)]
        L.or_expand.argtypes = [C.c_void_p, C.c_int32, _u32p, C.c_uint64, _u8p, _u64p, _u32p,
                                _u32p, C.c_uint64, _u32p, _u64p, _u64p, _i32p]
        L.or_batch_ready_parent.argtypes = [C.c_void_p, C.c_int32, C.c_uint32, _u32p, C.c_uint64,
                                            C.c_uint32, C.c_int32, _u32p, C.c_uint64, _u64p,
                                            C.c_uint64, _u64p, _u64p]
        L.or_batch_ready_parent.restype = C.c_int
        L.or_batch_ready.argtypes = [C.c_void_p, C.c_int32, C.c_uint32, _u32p, C.c_uint64,
                                     C.c_uint32, C.c_int32, _u32p, C.c_uint64, _u64p, _u64p]
        L.or_gather_commit.argtypes = [C.c_void_p, C.c_int32, C.c_uint64, _u32p, _u8p, _u32p,
                                       _u64p, _u32p, C.c_uint64, _u8p, _u32p, C.c_uint64, _u64p]
        L.or_assemble.argtypes = [C.c_void_p, C.c_int32, _u8p, C.c_uint64, _u32p, C.c_uint64,
                                  _u8p, _u64p, _u32p, _u8p, C.c_uint64, _u64p, _u64p, _u64p]
        L.or_retry.argtypes = [C.c_void_p, C.c_int32, C.c_uint32, _u32p, C.c_uint64, _u64p]
        L.or_assemble_list.argtypes = [C.c_void_p, C.c_int32, _u8p, C.c_uint64, _u32p, C.c_uint64,
                                       _u8p, _u64p, _u32p, _u8p, C.c_uint64, _u64p, _u64p, _u64p,
                                       _u64p, _u8p, _u64p, _u32p, C.c_uint64, _u64p]
        L.or_assemble_size.argtypes = [C.c_void_p, C.c_int32, _u32p, C.c_uint64, _u64p, _u64p]
        L.or_assemble_size.restype = C.c_int
        L.or_filter_reports.argtypes = [_u8p, _u8p, C.c_uint64]
        L.or_filter_reports.restype = None
        for f in ("or_expand", "or_batch_ready", "or_gather_commit", "or_assemble", "or_retry",
                  "or_assemble_list"):
            getattr(L, f).restype = C.c_int
        _lib = L
    return _lib


def _ptr(a: Optional[np.ndarray], ctype):
    if a is None:
        return None
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctype)


def _arr(a, dtype) -> Optional[np.ndarray]:
    if a is None:
        return None
    a = np.ascontiguousarray(np.asarray(a), dtype=dtype)
    # an empty list stays a list (a valid pointer), unlike NULL ("all")
    return a if a.size else np.zeros(1, dtype)[:0]


class OracleCtx:
    """One source microbatch of lineage state, held by the oracle."""

    def __init__(self, n_calls: int = 1):
        self._h = lib().or_ctx_create(n_calls)
        if not self._h:
            raise OracleError("or_ctx_create", E_INVAL)
        self.n_calls = n_calls
        self._n_children = {}

    def close(self):
        if self._h:
            lib().or_ctx_destroy(self._h)
            self._h = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass

    def reset(self):
        lib().or_ctx_reset(self._h)
        self._n_children = {}

    def stats(self) -> dict:
        s = _Stats()
        lib().or_ctx_stats(self._h, C.byref(s))
        return {n: int(getattr(s, n)) for n, _ in _Stats._fields_}

    def expand(self, counts, parent_xid: int = -1, parent_call=None,
               child_cap: Optional[int] = None, check: bool = True):
        counts = _arr(counts, np.uint32)
        P = counts.size
        offsets = np.zeros(P + 1, dtype=np.uint64)
        total = int(counts.sum(dtype=np.uint64))
        cap = total if child_cap is None else child_cap
        n_alloc = max(min(total, cap), 1)
        cp = np.zeros(n_alloc, dtype=np.uint32)
        co = np.zeros(n_alloc, dtype=np.uint32)
        empty = np.zeros(max(P, 1), dtype=np.uint32)
        n = C.c_uint64(0)
        ne = C.c_uint64(0)
        xid = C.c_int32(-1)
        pc = _arr(parent_call, np.uint8)
        st = lib().or_expand(self._h, parent_xid, _ptr(counts, _u32p), P, _ptr(pc, _u8p),
                             _ptr(offsets, _u64p), _ptr(cp, _u32p), _ptr(co, _u32p), cap,
                             _ptr(empty, _u32p), C.byref(n), C.byref(ne), C.byref(xid))
        res = dict(status=st, xid=xid.value, offsets=offsets, n_children=n.value,
                   child_parent=cp[:n.value] if st == OK else None,
                   child_ordinal=co[:n.value] if st == OK else None,
                   empty_parents=empty[:ne.value].copy())
        if st == OK:
            self._n_children[xid.value] = n.value
        if check and st != OK:
            raise OracleError("or_expand", st)
        return res

    def batch_ready(self, xid: int, call: int = 0, cand=None, batch_size: int = 1,
                    flush: bool = False, cap: Optional[int] = None, check: bool = True):
        cand = _arr(cand, np.uint32)
        n_cand = 0 if cand is None else cand.size
        if cap is None:
            # never more than the expansion's children (plus a batch of slack)
            cap = self._n_children[xid] + batch_size
        out = np.zeros(max(cap, 1), dtype=np.uint32)
        nb = C.c_uint64(0)
        nbt = C.c_uint64(0)
        st = lib().or_batch_ready(self._h, xid, call, _ptr(cand, _u32p), n_cand, batch_size,
                                  int(flush), _ptr(out, _u32p), cap, C.byref(nb), C.byref(nbt))
        if check and st != OK:
            raise OracleError("or_batch_ready", st)
        return dict(status=st, batched=out[:nb.value].copy() if st == OK else None,
                    n_batched=nb.value, n_batches=nbt.value)

    def batch_ready_parent(self, xid: int, call: int = 0, cand=None, batch_size: int = 1,
                           flush: bool = False, cap: Optional[int] = None,
                           off_cap: Optional[int] = None, check: bool = True):
        """Admission plus parent-bound reservation (Section 4.3); the batches
        are batched[batch_off[k]:batch_off[k+1]]."""
        cand = _arr(cand, np.uint32)
        n_cand = 0 if cand is None else cand.size
        if cap is None:
            cap = self._n_children[xid]
        if off_cap is None:
            off_cap = cap + 1
        out = np.zeros(max(cap, 1), dtype=np.uint32)
        offs = np.zeros(max(off_cap, 1), dtype=np.uint64)
        nb = C.c_uint64(0)
        nbt = C.c_uint64(0)
        st = lib().or_batch_ready_parent(self._h, xid, call, _ptr(cand, _u32p), n_cand, batch_size,
                                         int(flush), _ptr(out, _u32p), cap, _ptr(offs, _u64p),
                                         off_cap, C.byref(nb), C.byref(nbt))
        if check and st != OK:
            raise OracleError("or_batch_ready_parent", st)
        ok = st == OK
        return dict(status=st, batched=out[:nb.value].copy() if ok else None,
                    batch_off=offs[:nbt.value + 1].copy() if ok else None,
                    n_batched=nb.value, n_batches=nbt.value)

    def assemble_list(self, xid: int, arena: Optional[np.ndarray], parents=None,
                      n_parents: Optional[int] = None, out_cap: Optional[int] = None,
                      cursor: Optional[int] = None, elem_cap: Optional[int] = None,
                      check: bool = True):
        """Assemble plus the list structure: per listed parent its member
        entries (outcome, output offset, length) in ordinal order."""
        parents = _arr(parents, np.uint32)
        n = parents.size if parents is not None else (n_parents if n_parents is not None else (1 << 22))
        arena_u8 = _arr(arena, np.uint8)
        arena_bytes = arena_u8.size
        if out_cap is None:
            out_cap = (cursor or 0) + self.assemble_size(xid, parents, n)[0]
        if elem_cap is None:
            elem_cap = self._n_children[xid]
        status = np.zeros(max(n, 1), np.uint8)
        out_off = np.zeros(n + 1, np.uint64)
        out_len = np.zeros(max(n, 1), np.uint32)
        out = np.zeros(max(out_cap, 1), np.uint8)
        eb = np.zeros(n + 1, np.uint64)
        es = np.zeros(max(elem_cap, 1), np.uint8)
        eo = np.zeros(max(elem_cap, 1), np.uint64)
        el = np.zeros(max(elem_cap, 1), np.uint32)
        ob, na, ne = C.c_uint64(0), C.c_uint64(0), C.c_uint64(0)
        cur = C.c_uint64(cursor) if cursor is not None else None
        st = lib().or_assemble_list(self._h, xid, _ptr(arena_u8, _u8p), arena_bytes, _ptr(parents, _u32p),
                                    n, _ptr(status, _u8p), _ptr(out_off, _u64p), _ptr(out_len, _u32p),
                                    _ptr(out, _u8p), out_cap, C.byref(cur) if cur is not None else None,
                                    C.byref(ob), C.byref(na), _ptr(eb, _u64p), _ptr(es, _u8p),
                                    _ptr(eo, _u64p), _ptr(el, _u32p), elem_cap, C.byref(ne))
        if check and st != OK:
            raise OracleError("or_assemble_list", st)
        k, m = na.value, ne.value
        return dict(status=st, parent_status=status[:k].copy(), out_off=out_off[:k + 1].copy(),
                    out_len=out_len[:k].copy(), out=out[:out_cap], out_bytes=ob.value,
                    n_assembled=k, cursor=None if cur is None else cur.value,
                    elem_base=eb[:k + 1].copy(), elem_state=es[:m].copy(), elem_off=eo[:m].copy(),
                    elem_len=el[:m].copy(), n_elems=m)

    def assemble_size(self, xid: int, parents, n: int):
        """(bytes, list entries) of an assembly, without changing anything."""
        b, e = C.c_uint64(0), C.c_uint64(0)
        lib().or_assemble_size(self._h, xid, _ptr(parents, _u32p), n, C.byref(b), C.byref(e))
        return b.value, e.value

    @staticmethod
    def filter_reports(state, keep):
        """F.filter on a report batch (returns the new states)."""
        st = np.ascontiguousarray(np.asarray(state, np.uint8)).copy()
        kp = np.ascontiguousarray(np.asarray(keep, np.uint8))
        lib().or_filter_reports(_ptr(st, _u8p), _ptr(kp, _u8p), st.size)
        return st

    def retry(self, xid: int, call: int, children, check: bool = True):
        """Failed attempt: IN-FLIGHT Grains back to READY at generation + 1, as one
        recovery group taken before the Ready Queue at the next reservation."""
        children = _arr(children, np.uint32)
        n = 0 if children is None else children.size
        k = C.c_uint64(0)
        st = lib().or_retry(self._h, xid, call, _ptr(children, _u32p), n, C.byref(k))
        if check and st != OK:
            raise OracleError("or_retry", st)
        return dict(status=st, n_retried=k.value)

    def gather_commit(self, xid: int, child, state, length, off, gen=None,
                      arena_bytes: int = (1 << 48) - 1, n_parents_hint: Optional[int] = None,
                      check: bool = True):
        child = _arr(child, np.uint32)
        state = _arr(state, np.uint8)
        length = _arr(length, np.uint32)
        off = _arr(off, np.uint64)
        gen = _arr(gen, np.uint32)
        n = child.size
        code = np.zeros(max(n, 1), dtype=np.uint8)
        cap = n if n_parents_hint is None else min(n, n_parents_hint)
        done = np.zeros(max(n, 1), dtype=np.uint32)
        nd = C.c_uint64(0)
        st = lib().or_gather_commit(self._h, xid, n, _ptr(child, _u32p), _ptr(state, _u8p),
                                    _ptr(length, _u32p), _ptr(off, _u64p), _ptr(gen, _u32p),
                                    arena_bytes, _ptr(code, _u8p), _ptr(done, _u32p),
                                    max(cap, n), C.byref(nd))
        if check and st != OK:
            raise OracleError("or_gather_commit", st)
        return dict(status=st, code=code[:n].copy(), done=done[:nd.value].copy(),
                    n_done=nd.value)

    def assemble(self, xid: int, arena: Optional[np.ndarray], parents=None,
                 n_parents: Optional[int] = None, out_cap: Optional[int] = None,
                 cursor: Optional[int] = None, want_len: bool = True, check: bool = True):
        """Assemble ``parents`` (None: the latest commit's completed parents).
        With ``arena=None`` only outcomes and offsets are computed (no bytes)."""
        parents = _arr(parents, np.uint32)
        if parents is not None:
            n = parents.size
        else:
            n = n_parents if n_parents is not None else (1 << 22)
        status = np.zeros(max(n, 1), dtype=np.uint8)
        out_off = np.zeros(n + 1, dtype=np.uint64)
        out_len = np.zeros(max(n, 1), dtype=np.uint32) if want_len else None
        arena_u8 = None if arena is None else _arr(arena, np.uint8)
        arena_bytes = 0 if arena_u8 is None else arena_u8.size
        sizes_only = arena_u8 is None
        if out_cap is None:
            if sizes_only:
                out_cap = (1 << 62)
            else:
                out_cap = (cursor or 0) + self.assemble_size(xid, parents, n)[0]
        out = None if sizes_only else np.zeros(max(out_cap, 1), dtype=np.uint8)
        ob = C.c_uint64(0)
        na = C.c_uint64(0)
        cur = C.c_uint64(cursor) if cursor is not None else None
        st = lib().or_assemble(self._h, xid, _ptr(arena_u8, _u8p), arena_bytes,
                               _ptr(parents, _u32p), n, _ptr(status, _u8p),
                               _ptr(out_off, _u64p), _ptr(out_len, _u32p), _ptr(out, _u8p),
                               out_cap, C.byref(cur) if cur is not None else None,
                               C.byref(ob), C.byref(na))
        if check and st != OK:
            raise OracleError("or_assemble", st)
        k = na.value
        return dict(status=st, parent_status=status[:k].copy(), out_off=out_off[:k + 1].copy(),
                    out_len=None if out_len is None else out_len[:k].copy(),
                    out=None if out is None else out[:out_cap], out_bytes=ob.value,
                    n_assembled=k, cursor=None if cur is None else cur.value)
