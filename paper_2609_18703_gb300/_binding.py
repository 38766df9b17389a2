"""Thin ctypes binding of the C ABI in include/rayorch_gpu.h.

Function names and argument order follow the C entry points.  Pointer
arguments accept a torch tensor (its data_ptr), a raw integer address or
None; host outputs (the h_ pointers) are returned instead of passed.  A
``want_host=False`` keeps a call asynchronous (no h_ outputs, no sync).

Nothing here computes: every step runs in libro_gb300.so.  If the library
is missing the import of a function raises instead of falling back.
"""
from __future__ import annotations

import ctypes as C
import os
from typing import Optional

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libro_gb300.so")

# call status
RO_OK, RO_E_INVAL, RO_E_CAPACITY, RO_E_OVERFLOW, RO_E_STATE, RO_E_OOM, RO_E_CUDA, RO_E_TIMEOUT = range(8)
# Item outcomes (Eq. 1)
RO_PENDING, RO_PRESENT, RO_DROPPED, RO_FAILED, RO_SUPPRESSED = range(5)
# report kind (Section 4.4): the Grain failed and its open siblings are suppressed
RO_GROUP_FAILURE = 5
# report verdicts (Eq. 3)
RO_ACCEPT, RO_REJ_INVALID, RO_REJ_NOT_INFLIGHT, RO_REJ_STALE_GEN, RO_REJ_DUPLICATE, RO_REJ_BARRIER = range(6)

STATUS_NAMES = {0: "RO_OK", 1: "RO_E_INVAL", 2: "RO_E_CAPACITY", 3: "RO_E_OVERFLOW",
                4: "RO_E_STATE", 5: "RO_E_OOM", 6: "RO_E_CUDA", 7: "RO_E_TIMEOUT"}

EXPORTS = ("ro_ctx_create", "ro_ctx_destroy", "ro_ctx_reset", "ro_ctx_sync", "ro_ctx_stats",
           "ro_ctx_set_streams", "ro_ctx_set_call_streams", "ro_ctx_join", "ro_ctx_selftest_timeout", "ro_last_error", "ro_ctx_profile", "ro_ctx_profile_read", "ro_expand", "ro_batch_ready",
           "ro_batch_ready_calls", "ro_retry", "ro_batch_ready_parent", "ro_gather_commit", "ro_assemble", "ro_assemble_list", "ro_filter_reports",
           "ro_expand_noalloc")

# kernel ids (RO_K_*), in launch order of the path
KERNELS = ("expand_scan", "expand_fill", "ready_count", "ready_scatter", "commit_scatter",
           "commit_plan", "asm_parents", "asm_members", "asm_copy", "retry_claim", "retry_scatter",
           "pb_keys", "pb_hist", "pb_rowscan", "pb_sort", "pb_bounds", "pb_heads", "pb_mark",
           "pb_scan", "pb_emit", "commit_fix", "ready_fused")


class RoError(RuntimeError):
    def __init__(self, fn: str, status: int, msg: str = ""):
        super().__init__(f"{fn}: {STATUS_NAMES.get(status, status)} {msg}".rstrip())
        self.status = status


class _Stats(C.Structure):
    _fields_ = [(n, C.c_uint64) for n in (
        "accepted", "rej_invalid", "rej_not_inflight", "rej_stale_gen", "rej_duplicate",
        "ready_bad_candidates", "assemble_incomplete", "rej_barrier", "barrier_not_dispatched",
        "barrier_in_flight", "queue_dropped", "retried", "retry_skipped")]


_lib = None
_vp = C.c_void_p
_u64 = C.c_uint64
_u32 = C.c_uint32
_i32 = C.c_int32
_pu64 = C.POINTER(C.c_uint64)
_pi32 = C.POINTER(C.c_int32)


def load(path: Optional[str] = None):
    """Load libro_gb300.so (built in-tree by ``paper_2609_18703_gb300.build``)."""
    global _lib
    if _lib is not None:
        return _lib
    path = path or LIB_PATH
    if not os.path.exists(path):
        raise RuntimeError(f"{path} is missing: build it with "
                           "`python -m paper_2609_18703_gb300.build` (needs nvcc)")
    L = C.CDLL(path)
    L.ro_ctx_create.argtypes = [C.POINTER(_vp), _i32, _vp, _u32]
    L.ro_ctx_destroy.argtypes = [_vp]
    L.ro_ctx_reset.argtypes = [_vp]
    L.ro_ctx_sync.argtypes = [_vp]
    L.ro_ctx_stats.argtypes = [_vp, C.POINTER(_Stats)]
    L.ro_ctx_set_streams.argtypes = [_vp, _vp, _vp]
    L.ro_ctx_set_call_streams.argtypes = [_vp, C.POINTER(_vp), _u32]
    L.ro_ctx_join.argtypes = [_vp]
    L.ro_ctx_selftest_timeout.argtypes = [_vp, _u32]
    L.ro_last_error.argtypes = [_vp]
    L.ro_last_error.restype = C.c_char_p
    L.ro_ctx_profile.argtypes = [_vp, _u32]
    L.ro_ctx_profile_read.argtypes = [_vp, _pu64, _pu64, C.POINTER(C.c_double), _u32]
    L.ro_expand.argtypes = [_vp, _i32, _vp, _u64, _vp, _vp, _vp, _vp, _u64, _vp, _pu64, _pu64, _pi32]
    L.ro_batch_ready.argtypes = [_vp, _i32, _u32, _vp, _u64, _u32, _i32, _vp, _u64, _vp, _pu64, _pu64]
    L.ro_batch_ready_calls.argtypes = [_vp, _i32, _u32, C.POINTER(C.c_uint32), _vp, _u64, _u32, _i32,
                                       C.POINTER(_vp), _pu64, C.POINTER(_vp)]
    L.ro_retry.argtypes = [_vp, _i32, _u32, _vp, _u64, _pu64]
    L.ro_gather_commit.argtypes = [_vp, _i32, _u64, _vp, _vp, _vp, _vp, _vp, _vp, _u64, _vp, _vp, _u64,
                                   _vp, _pu64]
    L.ro_assemble.argtypes = [_vp, _i32, _vp, _u64, _vp, _u64, _vp, _vp, _vp, _vp, _vp, _u64, _vp, _vp,
                              _pu64]
    L.ro_assemble_list.argtypes = [_vp, _i32, _vp, _u64, _vp, _u64, _vp, _vp, _vp, _vp, _vp, _u64, _vp,
                                   _vp, _pu64, _vp, _vp, _vp, _vp, _u64, _vp, _pu64]
    L.ro_filter_reports.argtypes = [_vp, _vp, _vp, _u64]
    L.ro_batch_ready_parent.argtypes = [_vp, _i32, C.c_uint32, _vp, _u64, C.c_uint32, _i32, _vp,
                                        _u64, _vp, _u64, _vp, _vp, _pu64, _pu64]
    L.ro_expand_noalloc.argtypes = [_vp, _u64, _vp, _vp, _vp, _u64, _vp, _vp, _pu64, _pu64]
    for f in EXPORTS:
        if f != "ro_last_error":
            getattr(L, f).restype = C.c_int32
    _lib = L
    return L


def _ptr(x):
    if x is None:
        return None
    if isinstance(x, int):
        return x
    if hasattr(x, "data_ptr"):
        # pinned host tensors are reachable from the GPU (ro_assemble accepts
        # them for the arena and the output); pageable ones are not
        if hasattr(x, "is_cuda") and not x.is_cuda and not x.is_pinned():
            raise ValueError("argument is a pageable CPU tensor (pin it or move it to the GPU)")
        return x.data_ptr()
    raise TypeError(f"cannot pass {type(x)!r} as a pointer")


def _stream_handle(stream) -> Optional[int]:
    if stream is None:
        return None
    if isinstance(stream, int):
        return stream
    return stream.cuda_stream


def ro_last_error(ctx) -> str:
    s = load().ro_last_error(ctx)
    return s.decode() if s else ""


def _check(fn, st, ctx=None, allow=()):
    if st != RO_OK and st not in allow:
        raise RoError(fn, st, ro_last_error(ctx) if ctx else "")
    return st


def ro_ctx_create(device: int = 0, stream=None, n_calls: int = 1) -> int:
    h = _vp()
    st = load().ro_ctx_create(C.byref(h), device, _stream_handle(stream), n_calls)
    _check("ro_ctx_create", st)
    return h.value


def ro_ctx_destroy(ctx) -> int:
    return load().ro_ctx_destroy(ctx)


def ro_ctx_reset(ctx) -> int:
    return load().ro_ctx_reset(ctx)


def ro_ctx_sync(ctx) -> int:
    return load().ro_ctx_sync(ctx)


def ro_ctx_set_streams(ctx, plan_stream=None, copy_stream=None) -> int:
    """Assembly planning / copy streams (torch.cuda.Stream, raw handle or None)."""
    st = load().ro_ctx_set_streams(ctx, _stream_handle(plan_stream), _stream_handle(copy_stream))
    return _check("ro_ctx_set_streams", st, ctx)


def ro_ctx_set_call_streams(ctx, streams) -> int:
    """Streams for the Calls' admissions: streams[k] (torch.cuda.Stream, raw
    handle or None) runs ro_batch_ready for Call k."""
    handles = (_vp * max(len(streams), 1))(*[_stream_handle(s) for s in streams])
    st = load().ro_ctx_set_call_streams(ctx, handles, len(streams))
    return _check("ro_ctx_set_call_streams", st, ctx)


def ro_ctx_join(ctx) -> int:
    """The context's stream waits (on the GPU) for the plan, copy, completion
    scan and Call streams."""
    return _check("ro_ctx_join", load().ro_ctx_join(ctx), ctx)


def ro_ctx_stats(ctx) -> dict:
    s = _Stats()
    st = load().ro_ctx_stats(ctx, C.byref(s))
    out = {n: int(getattr(s, n)) for n, _ in _Stats._fields_}
    out["status"] = st
    return out


def ro_ctx_profile(ctx, kernel_mask: int) -> int:
    return load().ro_ctx_profile(ctx, kernel_mask)


def ro_ctx_profile_read(ctx) -> dict:
    """{kernel name: (launches, launches timed, summed device ms)} since the last read."""
    k = len(KERNELS)
    la = (C.c_uint64 * k)()
    ti = (C.c_uint64 * k)()
    ms = (C.c_double * k)()
    st = load().ro_ctx_profile_read(ctx, la, ti, ms, k)
    _check("ro_ctx_profile_read", st, ctx)
    return {name: (int(la[i]), int(ti[i]), float(ms[i])) for i, name in enumerate(KERNELS)}


def ro_expand(ctx, parent_xid, d_counts, n_parents, d_parent_call, d_offsets, d_child_parent,
              d_child_ordinal, child_cap, d_empty_parents=None):
    """Returns (status, n_children, n_empty, xid)."""
    n = _u64(0)
    ne = _u64(0)
    xid = _i32(-1)
    st = load().ro_expand(ctx, parent_xid, _ptr(d_counts), n_parents, _ptr(d_parent_call),
                          _ptr(d_offsets), _ptr(d_child_parent), _ptr(d_child_ordinal), child_cap,
                          _ptr(d_empty_parents), C.byref(n), C.byref(ne), C.byref(xid))
    return st, n.value, ne.value, xid.value


def ro_batch_ready(ctx, xid, call, d_cand, n_cand, batch_size, flush, d_batched, batched_cap,
                   d_n_batched=None, want_host: bool = True):
    """Returns (status, n_batched, n_batches); the counts are None without want_host."""
    nb = _u64(0)
    nbt = _u64(0)
    st = load().ro_batch_ready(ctx, xid, call, _ptr(d_cand), n_cand, batch_size, int(flush),
                               _ptr(d_batched), batched_cap, _ptr(d_n_batched),
                               C.byref(nb) if want_host else None,
                               C.byref(nbt) if want_host else None)
    return (st, nb.value, nbt.value) if want_host else (st, None, None)


def ro_ctx_selftest_timeout(ctx, kind: int) -> int:
    """Runs one bounded device-side wait that nothing releases; returns the
    status (RO_E_TIMEOUT expected)."""
    return load().ro_ctx_selftest_timeout(ctx, kind)


def ro_batch_ready_calls(ctx, xid, calls, d_cand, n_cand, batch_size, flush, d_batched, batched_cap,
                         d_n_batched=None):
    """Admissions of several Calls from one candidate list (one launch);
    d_batched, batched_cap and d_n_batched are per-Call sequences.  Returns
    the status."""
    n = len(calls)
    c_calls = (C.c_uint32 * n)(*calls)
    c_b = (_vp * n)(*[_ptr(d) for d in d_batched])
    c_cap = (C.c_uint64 * n)(*batched_cap)
    c_nb = (_vp * n)(*[_ptr(d) for d in d_n_batched]) if d_n_batched is not None else None
    return load().ro_batch_ready_calls(ctx, xid, n, c_calls, _ptr(d_cand), n_cand, batch_size,
                                       int(flush), c_b, c_cap, c_nb)


def ro_retry(ctx, xid, call, d_children, n, want_host: bool = True):
    """Returns (status, n_retried); n_retried is None without want_host."""
    k = _u64(0)
    st = load().ro_retry(ctx, xid, call, _ptr(d_children), n, C.byref(k) if want_host else None)
    return (st, k.value) if want_host else (st, None)


def ro_gather_commit(ctx, xid, n, d_n, d_child, d_state, d_len, d_arena_off, d_gen, arena_bytes,
                     d_code=None, d_done_parents=None, done_cap=0, d_n_done=None,
                     want_host: bool = True):
    """Returns (status, n_done); n_done is None without want_host."""
    nd = _u64(0)
    st = load().ro_gather_commit(ctx, xid, n, _ptr(d_n), _ptr(d_child), _ptr(d_state), _ptr(d_len),
                                 _ptr(d_arena_off), _ptr(d_gen), arena_bytes, _ptr(d_code),
                                 _ptr(d_done_parents), done_cap, _ptr(d_n_done),
                                 C.byref(nd) if want_host else None)
    return (st, nd.value) if want_host else (st, None)


def ro_assemble(ctx, xid, d_arena, arena_bytes, d_parents, n_parents, d_n_parents, d_status,
                d_out_off, d_out_len, d_out, out_cap, d_out_cursor=None, d_out_bytes=None,
                want_host: bool = True):
    """Returns (status, out_bytes); out_bytes is None without want_host."""
    ob = _u64(0)
    st = load().ro_assemble(ctx, xid, _ptr(d_arena), arena_bytes, _ptr(d_parents), n_parents,
                            _ptr(d_n_parents), _ptr(d_status), _ptr(d_out_off), _ptr(d_out_len),
                            _ptr(d_out), out_cap, _ptr(d_out_cursor), _ptr(d_out_bytes),
                            C.byref(ob) if want_host else None)
    return (st, ob.value) if want_host else (st, None)


def ro_assemble_list(ctx, xid, d_arena, arena_bytes, d_parents, n_parents, d_n_parents, d_status,
                     d_out_off, d_out_len, d_out, out_cap, d_out_cursor, d_out_bytes, d_elem_base,
                     d_elem_state, d_elem_off, d_elem_len, elem_cap, d_n_elems=None,
                     want_host: bool = True):
    """Returns (status, out_bytes, n_elems); the counts are None without want_host."""
    ob = _u64(0)
    ne = _u64(0)
    st = load().ro_assemble_list(ctx, xid, _ptr(d_arena), arena_bytes, _ptr(d_parents), n_parents,
                                 _ptr(d_n_parents), _ptr(d_status), _ptr(d_out_off), _ptr(d_out_len),
                                 _ptr(d_out), out_cap, _ptr(d_out_cursor), _ptr(d_out_bytes),
                                 C.byref(ob) if want_host else None, _ptr(d_elem_base),
                                 _ptr(d_elem_state), _ptr(d_elem_off), _ptr(d_elem_len), elem_cap,
                                 _ptr(d_n_elems), C.byref(ne) if want_host else None)
    return (st, ob.value, ne.value) if want_host else (st, None, None)


def ro_batch_ready_parent(ctx, xid, call, d_cand, n_cand, batch_size, flush, d_batched,
                          batched_cap, d_batch_off=None, batch_off_cap=0, d_n_batched=None,
                          d_n_batches=None, want_host: bool = True):
    """Admission plus parent-bound reservation.  Returns (status, n_batched,
    n_batches); the counts are None without want_host (no synchronisation)."""
    nb, nbt = _u64(0), _u64(0)
    st = load().ro_batch_ready_parent(ctx, xid, call, _ptr(d_cand), n_cand, batch_size, int(flush),
                                      _ptr(d_batched), batched_cap, _ptr(d_batch_off), batch_off_cap,
                                      _ptr(d_n_batched), _ptr(d_n_batches),
                                      C.byref(nb) if want_host else None,
                                      C.byref(nbt) if want_host else None)
    return (st, nb.value, nbt.value) if want_host else (st, None, None)


def ro_filter_reports(ctx, d_state, d_keep, n) -> int:
    """F.filter on a report batch (in place, on the context's stream)."""
    return load().ro_filter_reports(ctx, _ptr(d_state), _ptr(d_keep), n)


def ro_expand_noalloc(d_counts, n_parents, d_offsets, d_child_parent, d_child_ordinal, child_cap,
                      d_empty_parents=None, stream=None):
    """Context-free expansion that allocates nothing (static device scratch).
    Returns (status, n_children, n_empty)."""
    n = _u64(0)
    ne = _u64(0)
    st = load().ro_expand_noalloc(_ptr(d_counts), n_parents, _ptr(d_offsets), _ptr(d_child_parent),
                                  _ptr(d_child_ordinal), child_cap, _ptr(d_empty_parents),
                                  _stream_handle(stream), C.byref(n), C.byref(ne))
    return st, n.value, ne.value
