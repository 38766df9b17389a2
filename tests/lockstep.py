"""Run the same lineage operations through the GPU library (C ABI, device
buffers) and the CPU oracle, and compare every output element by element.

All outputs of this path are integers and bytes, so every comparison is
exact.  Used only by the GPU tests.
"""
from __future__ import annotations

from typing import Optional

import numpy as np
import torch

import paper_2609_18703_gb300 as ro
from oracle import OracleCtx

_VIEW = {np.uint8: torch.uint8, np.uint32: torch.int32, np.uint64: torch.int64,
         np.int32: torch.int32, np.int64: torch.int64}


def dev(a: np.ndarray, dtype) -> torch.Tensor:
    """Device copy of a host array with the same bytes (unsigned viewed as signed)."""
    a = np.ascontiguousarray(np.asarray(a), dtype=dtype)
    signed = {np.uint8: np.uint8, np.uint32: np.int32, np.uint64: np.int64}[dtype]
    t = torch.from_numpy(a.view(signed).copy() if a.size else np.zeros(1, signed))
    return t.cuda()


def empty(n: int, dtype) -> torch.Tensor:
    return torch.zeros(max(int(n), 1), dtype=_VIEW[dtype], device="cuda")


def host(t: torch.Tensor, dtype, n: Optional[int] = None) -> np.ndarray:
    a = t.cpu().numpy().view(dtype)
    return a if n is None else a[:n]


class Lockstep:
    def __init__(self, n_calls: int = 1, streams: bool = False, call_streams: bool = False):
        self.o = OracleCtx(n_calls)
        self.stream = torch.cuda.current_stream()
        self.ctx = ro.ro_ctx_create(0, self.stream, n_calls)
        if streams:   # assembly planning and copies on streams of their own
            self.side = (torch.cuda.Stream(), torch.cuda.Stream())
            ro.ro_ctx_set_streams(self.ctx, *self.side)
        if call_streams:   # each Call's admissions on a stream of its own
            self.call_side = [torch.cuda.Stream() for _ in range(n_calls)]
            ro.ro_ctx_set_call_streams(self.ctx, self.call_side)
        self.N = {}
        self.P = {}

    def close(self):
        if self.ctx:
            ro.ro_ctx_destroy(self.ctx)
            self.ctx = None
        self.o.close()

    def __enter__(self):
        return self

    def __exit__(self, *exc):
        self.close()

    # ---------------------------------------------------------------- expand
    def expand(self, counts, parent_xid: int = -1, parent_call=None,
               child_cap: Optional[int] = None, want_empty: bool = True) -> dict:
        counts = np.asarray(counts, dtype=np.uint32)
        P = counts.size
        total = int(counts.sum(dtype=np.uint64))
        cap = total if child_cap is None else child_cap
        r = self.o.expand(counts, parent_xid=parent_xid, parent_call=parent_call,
                          child_cap=cap, check=False)
        d_counts = dev(counts, np.uint32)
        d_pc = None if parent_call is None else dev(parent_call, np.uint8)
        d_off = empty(P + 1, np.uint64)
        n_alloc = min(total, cap)
        d_cp = empty(n_alloc, np.uint32)
        d_co = empty(n_alloc, np.uint32)
        d_empty = empty(P, np.uint32) if want_empty else None
        st, n, ne, xid = ro.ro_expand(self.ctx, parent_xid, d_counts, P, d_pc, d_off, d_cp, d_co,
                                      cap, d_empty)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert n == r["n_children"]
        if st != ro.RO_OK:
            return dict(status=st, n_children=n)
        assert ne == r["empty_parents"].size
        assert xid == r["xid"]
        assert np.array_equal(host(d_off, np.uint64, P + 1), r["offsets"])
        assert np.array_equal(host(d_cp, np.uint32, n), r["child_parent"])
        assert np.array_equal(host(d_co, np.uint32, n), r["child_ordinal"])
        if want_empty:
            assert np.array_equal(host(d_empty, np.uint32, ne), r["empty_parents"])
        self.N[xid] = n
        self.P[xid] = P
        return dict(status=st, xid=xid, n_children=n, n_empty=ne, offsets=r["offsets"])

    # ----------------------------------------------------------- batch_ready
    def batch_ready(self, xid: int, call: int = 0, cand=None, batch_size: int = 1,
                    flush: bool = False, cap: Optional[int] = None) -> dict:
        cand_np = None if cand is None else np.asarray(cand, dtype=np.uint32)
        n_cand = self.N[xid] if cand_np is None else cand_np.size
        if cap is None:
            cap = self.N[xid] + batch_size
        r = self.o.batch_ready(xid, call, cand_np, batch_size, flush, cap=cap, check=False)
        d_cand = None if cand_np is None else dev(cand_np, np.uint32)
        d_b = empty(cap, np.uint32)
        d_nb = empty(1, np.uint64)
        st, nb, nbt = ro.ro_batch_ready(self.ctx, xid, call, d_cand, 0 if cand_np is None else n_cand,
                                        batch_size, flush, d_b, cap, d_nb)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert nb == r["n_batched"]
        if st == ro.RO_OK:
            assert nbt == r["n_batches"]
            assert int(host(d_nb, np.uint64, 1)[0]) == nb
            got = host(d_b, np.uint32, nb)
            assert np.array_equal(got, r["batched"])
        return dict(status=st, batched=r["batched"], n_batched=nb)

    def batch_ready_calls(self, xid: int, calls, cand, batch_size: int = 1, flush: bool = False,
                          caps=None) -> list:
        """ro_batch_ready_calls (several Calls, one launch) against the
        oracle's admissions of the same Calls in turn.  Returns each Call's
        reserved children (None where its reservation was refused)."""
        cand = np.asarray(cand, dtype=np.uint32)
        if caps is None:
            caps = [self.N[xid] + batch_size] * len(calls)
        d_cand = dev(cand, np.uint32)
        d_b = [empty(max(int(c), 1), np.uint32) for c in caps]
        d_nb = [empty(1, np.uint64) for _ in calls]
        st = ro.ro_batch_ready_calls(self.ctx, xid, list(calls), d_cand, cand.size, batch_size, flush,
                                     d_b, [int(c) for c in caps], d_nb)
        assert st == ro.RO_OK, ro.ro_last_error(self.ctx)
        sync = ro.ro_ctx_sync(self.ctx)
        out, refused = [], False
        for k, c in enumerate(calls):
            r = self.o.batch_ready(xid, c, cand, batch_size, flush, cap=int(caps[k]), check=False)
            if r["status"] == ro.RO_E_CAPACITY:
                refused = True
                out.append(None)
                continue
            nb = int(host(d_nb[k], np.uint64, 1)[0])
            assert nb == r["n_batched"], (c, nb, r["n_batched"])
            assert np.array_equal(host(d_b[k], np.uint32, nb), r["batched"])
            out.append(r["batched"])
        assert sync == (ro.RO_E_CAPACITY if refused else ro.RO_OK), ro.ro_last_error(self.ctx)
        return out

    def batch_ready_parent(self, xid: int, call: int = 0, cand=None, batch_size: int = 1,
                           flush: bool = False, cap: Optional[int] = None,
                           off_cap: Optional[int] = None) -> dict:
        cand_np = None if cand is None else np.asarray(cand, dtype=np.uint32)
        n_cand = self.N[xid] if cand_np is None else cand_np.size
        if cap is None:
            cap = self.N[xid]
        if off_cap is None:
            off_cap = cap + 1
        r = self.o.batch_ready_parent(xid, call, cand_np, batch_size, flush, cap=cap,
                                      off_cap=off_cap, check=False)
        d_cand = None if cand_np is None else dev(cand_np, np.uint32)
        d_b = empty(cap, np.uint32)
        d_off = empty(off_cap, np.uint64)
        d_nb = empty(1, np.uint64)
        d_nbt = empty(1, np.uint64)
        st, nb, nbt = ro.ro_batch_ready_parent(self.ctx, xid, call, d_cand,
                                               0 if cand_np is None else n_cand, batch_size, flush,
                                               d_b, cap, d_off, off_cap, d_nb, d_nbt)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert nb == r["n_batched"] and nbt == r["n_batches"], (nb, nbt, r["n_batched"], r["n_batches"])
        if st == ro.RO_OK:
            assert int(host(d_nb, np.uint64, 1)[0]) == nb
            assert int(host(d_nbt, np.uint64, 1)[0]) == nbt
            assert np.array_equal(host(d_b, np.uint32, nb), r["batched"])
            assert np.array_equal(host(d_off, np.uint64, nbt + 1), r["batch_off"])
        return r

    # ------------------------------------------------------------- retry
    def retry(self, xid: int, call: int, children) -> dict:
        ch = np.asarray(children, np.uint32)
        r = self.o.retry(xid, call, ch, check=False)
        st, k = ro.ro_retry(self.ctx, xid, call, dev(ch, np.uint32), ch.size)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert k == r["n_retried"], (k, r["n_retried"])
        return r

    # ------------------------------------------------------------ commit
    def commit(self, xid: int, child, state, length, off, gen=None,
               arena_bytes: int = (1 << 48) - 1, device_count: bool = False,
               want_code: bool = True, want_done: bool = True) -> dict:
        child = np.asarray(child, np.uint32)
        n = child.size
        r = self.o.gather_commit(xid, child, state, length, off, gen=gen,
                                 arena_bytes=arena_bytes, check=False)
        d = [dev(child, np.uint32), dev(state, np.uint8), dev(length, np.uint32),
             dev(off, np.uint64)]
        d_gen = None if gen is None else dev(gen, np.uint32)
        d_code = empty(n, np.uint8) if want_code else None
        cap = max(min(n, self.P[xid]), 1)
        d_done = empty(cap, np.uint32) if want_done else None
        d_nd = empty(1, np.uint64)
        d_n = dev(np.array([n], np.uint64), np.uint64) if device_count else None
        st, nd = ro.ro_gather_commit(self.ctx, xid, n, d_n, *d, d_gen, arena_bytes, d_code, d_done,
                                     cap, d_nd)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert nd == r["n_done"]
        assert int(host(d_nd, np.uint64, 1)[0]) == nd
        if want_code:
            assert np.array_equal(host(d_code, np.uint8, n), r["code"])
        if want_done:
            assert np.array_equal(host(d_done, np.uint32, nd), r["done"])
        return r

    # ------------------------------------------------------------ assemble
    def assemble(self, xid: int, arena_np: Optional[np.ndarray], arena_dev: torch.Tensor,
                 parents=None, n_parents: Optional[int] = None, out_cap: Optional[int] = None,
                 out_dev: Optional[torch.Tensor] = None, cursor: Optional[int] = None,
                 want_len: bool = True, device_count: bool = False) -> dict:
        parents_np = None if parents is None else np.asarray(parents, np.uint32)
        r = self.o.assemble(xid, arena_np, parents=parents_np, n_parents=n_parents,
                            out_cap=out_cap, cursor=cursor, want_len=want_len, check=False)
        k = r["n_assembled"] if parents_np is None else parents_np.size
        n_host = parents_np.size if parents_np is not None else n_parents
        if out_cap is None:
            out_cap = (cursor or 0) + r["out_bytes"]
        if out_dev is None:
            out_dev = torch.zeros(max(out_cap, 1), dtype=torch.uint8, device="cuda")
        d_par = None if parents_np is None else dev(parents_np, np.uint32)
        d_np = dev(np.array([n_host], np.uint64), np.uint64) if (device_count and d_par is not None) else None
        d_status = empty(max(n_host, 1), np.uint8)
        d_off = empty(max(n_host, 1) + 1, np.uint64)
        d_len = empty(max(n_host, 1), np.uint32) if want_len else None
        d_cur = dev(np.array([cursor], np.uint64), np.uint64) if cursor is not None else None
        d_ob = empty(1, np.uint64)
        st, ob = ro.ro_assemble(self.ctx, xid, arena_dev, arena_dev.numel(), d_par, n_host, d_np,
                                d_status, d_off, d_len, out_dev, out_cap, d_cur, d_ob)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        assert ob == r["out_bytes"]
        if st != ro.RO_OK:
            return dict(status=st, out_bytes=ob)
        assert np.array_equal(host(d_status, np.uint8, k), r["parent_status"])
        assert np.array_equal(host(d_off, np.uint64, k + 1), r["out_off"])
        if want_len:
            assert np.array_equal(host(d_len, np.uint32, k), r["out_len"])
        base = cursor or 0
        if cursor is not None:
            assert int(host(d_cur, np.uint64, 1)[0]) == r["cursor"]
        if arena_np is not None and ob:
            got = out_dev[base:base + ob].cpu().numpy()
            want = r["out"][base:base + ob]
            if not np.array_equal(got, want):
                bad = np.flatnonzero(got != want)
                raise AssertionError(f"assembled bytes differ at {bad.size} positions, first {bad[:8]}")
        return dict(status=st, out_bytes=ob, out=out_dev, r=r)

    def assemble_list(self, xid: int, arena_np: np.ndarray, arena_dev: torch.Tensor, parents=None,
                      n_parents: Optional[int] = None, out_cap: Optional[int] = None,
                      cursor: Optional[int] = None, elem_cap: Optional[int] = None) -> dict:
        parents_np = None if parents is None else np.asarray(parents, np.uint32)
        if elem_cap is None:
            elem_cap = self.N[xid]
        r = self.o.assemble_list(xid, arena_np, parents=parents_np, n_parents=n_parents,
                                 out_cap=out_cap, cursor=cursor, elem_cap=elem_cap, check=False)
        n_host = parents_np.size if parents_np is not None else n_parents
        if out_cap is None:
            out_cap = (cursor or 0) + r["out_bytes"]
        out_dev = torch.zeros(max(out_cap, 1), dtype=torch.uint8, device="cuda")
        d_par = None if parents_np is None else dev(parents_np, np.uint32)
        d_status = empty(max(n_host, 1), np.uint8)
        d_off = empty(max(n_host, 1) + 1, np.uint64)
        d_len = empty(max(n_host, 1), np.uint32)
        d_cur = dev(np.array([cursor], np.uint64), np.uint64) if cursor is not None else None
        d_eb = empty(max(n_host, 1) + 1, np.uint64)
        d_es = empty(max(elem_cap, 1), np.uint8)
        d_eo = empty(max(elem_cap, 1), np.uint64)
        d_el = empty(max(elem_cap, 1), np.uint32)
        d_ne = empty(1, np.uint64)
        st, ob, ne = ro.ro_assemble_list(self.ctx, xid, arena_dev, arena_dev.numel(), d_par, n_host, None,
                                         d_status, d_off, d_len, out_dev, out_cap, d_cur, None, d_eb,
                                         d_es, d_eo, d_el, elem_cap, d_ne)
        assert st == r["status"], (st, r["status"], ro.ro_last_error(self.ctx))
        if st != ro.RO_OK:
            return r
        k, m = r["n_assembled"], r["n_elems"]
        assert ob == r["out_bytes"] and ne == m and int(host(d_ne, np.uint64, 1)[0]) == m
        assert np.array_equal(host(d_status, np.uint8, k), r["parent_status"])
        assert np.array_equal(host(d_off, np.uint64, k + 1), r["out_off"])
        assert np.array_equal(host(d_len, np.uint32, k), r["out_len"])
        assert np.array_equal(host(d_eb, np.uint64, k + 1), r["elem_base"])
        assert np.array_equal(host(d_es, np.uint8, m), r["elem_state"])
        assert np.array_equal(host(d_eo, np.uint64, m), r["elem_off"])
        assert np.array_equal(host(d_el, np.uint32, m), r["elem_len"])
        base = cursor or 0
        if ob:
            assert np.array_equal(out_dev[base:base + ob].cpu().numpy(), r["out"][base:base + ob])
        return r

    def filter(self, state, keep) -> np.ndarray:
        want = self.o.filter_reports(state, keep)
        d_s = dev(np.asarray(state, np.uint8), np.uint8)
        d_k = dev(np.asarray(keep, np.uint8), np.uint8)
        assert ro.ro_filter_reports(self.ctx, d_s, d_k, len(want)) == ro.RO_OK
        got = host(d_s, np.uint8, len(want))
        assert np.array_equal(got, want)
        return want

    def check_stats(self):
        g = ro.ro_ctx_stats(self.ctx)
        assert g.pop("status") == ro.RO_OK
        assert g == self.o.stats(), (g, self.o.stats())
