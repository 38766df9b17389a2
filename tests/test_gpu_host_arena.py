"""Assembly with the arena and/or the output in pinned host memory (the copy
reads the needed payload bytes and writes the assembled bytes in place over
the host link) against the oracle: every status, offset, length, byte and
counter equal.  Covers waves of the document->page level, many small
records per chunk (skew), list-structured output, cursors across waves with
separate streams, and the refusal of pageable host memory.
"""
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


import paper_2609_18703_gb300 as ro  # noqa: E402
from tests.lockstep import Lockstep, dev, empty  # noqa: E402
from tests.pipeline import host_arena  # noqa: E402
from workload import docpage, skew, tiny  # noqa: E402


def _pinned(a: np.ndarray) -> torch.Tensor:
    return torch.from_numpy(a if a.size else np.zeros(1, np.uint8)).pin_memory()


def _arena(a: np.ndarray, where: str) -> torch.Tensor:
    return _pinned(a) if where == "host" else dev(a if a.size else np.zeros(1, np.uint8), np.uint8)


def _run(ls, lv, a_np, arena_t, out_where, cursor=False):
    x = ls.expand(lv.counts, parent_call=lv.parent_call)["xid"]
    ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
    cur = 0 if cursor else None
    total = 0
    outs = []
    for w in range(lv.n_waves):
        ch, st, ln, of = lv.reports(lv.wave(w))
        cm = ls.commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1))
        n = max(cm["n_done"], 1)
        want = ls.o.assemble_size(x, None, cm["n_done"])[0]
        cap = (cur or 0) + want
        out = (torch.zeros(max(cap, 1), dtype=torch.uint8).pin_memory() if out_where == "host"
               else torch.zeros(max(cap, 1), dtype=torch.uint8, device="cuda"))
        r = ls.assemble(x, a_np, arena_t, parents=None, n_parents=n, out_cap=cap, out_dev=out,
                        cursor=cur)
        outs.append(out)
        total += r["out_bytes"]
        if cursor:
            cur += r["out_bytes"]
    return x, total


@pytest.mark.parametrize("arena_where,out_where", [("host", "device"), ("device", "host"),
                                                   ("host", "host")])
def test_docpage_waves(arena_where, out_where):
    lv = docpage(parents=3000, waves=12).top
    a = host_arena(lv)
    with Lockstep() as ls:
        _, total = _run(ls, lv, a, _arena(a, arena_where), out_where)
        assert total > 0
        ls.check_stats()


def test_host_buffers_with_streams_and_cursor():
    lv = docpage(parents=2000, waves=8).top
    a = host_arena(lv)
    with Lockstep(streams=True) as ls:
        _run(ls, lv, a, _arena(a, "host"), "host", cursor=True)
        ls.check_stats()


def test_many_small_records_per_chunk():
    """32-byte records: chunks hold hundreds of pieces (the general staging
    path for a device arena); a host arena takes the direct path for all."""
    lv = skew(parents=20000, heavy=4, heavy_children=6000).top
    a = host_arena(lv)
    for where in ("host", "device"):
        with Lockstep() as ls:
            _run(ls, lv, a, _arena(a, where), "host")
            ls.check_stats()


def test_list_output_from_host_arena():
    lv = tiny().top
    a = host_arena(lv)
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
        ch, st, ln, of = lv.reports(lv.wave(0))
        ls.commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1))
        ls.assemble_list(x, a, _pinned(a), parents=np.arange(lv.n_parents, dtype=np.uint32))
        ls.check_stats()


def test_pageable_host_memory_is_refused():
    lv = tiny().top
    a = host_arena(lv)
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
        ch, st, ln, of = lv.reports(lv.wave(0))
        ls.commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1))
        P = lv.n_parents
        d_status, d_off = empty(P, np.uint8), empty(P + 1, np.uint64)
        pageable = torch.from_numpy(a.copy())
        out_d = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
        # raw pointers reach the library, which refuses pageable memory
        st, _ = ro.ro_assemble(ls.ctx, x, pageable.data_ptr(), a.size, None, P, None, d_status,
                               d_off, None, out_d, out_d.numel(), None, None)
        assert st == ro.RO_E_INVAL
        host_out = torch.zeros(1 << 20, dtype=torch.uint8)
        st, _ = ro.ro_assemble(ls.ctx, x, dev(a, np.uint8), a.size, None, P, None, d_status, d_off,
                               None, host_out.data_ptr(), 1 << 20, None, None)
        assert st == ro.RO_E_INVAL
        # the binding itself refuses pageable tensors
        with pytest.raises(ValueError):
            ro.ro_assemble(ls.ctx, x, pageable, a.size, None, P, None, d_status, d_off, None,
                           out_d, out_d.numel(), None, None)
