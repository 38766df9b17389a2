"""List-structured Reduce output and F.filter on the GPU (Section 4.2,
Table 3) against the oracle: filtered report states, statuses, offsets,
assembled bytes, and every list entry (outcome, offset, length) compared
exactly, through the commit path and caller lists (repeats, incomplete and
out-of-range entries, cursors, capacity refusals)."""
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
from tests.lockstep import Lockstep, dev, empty, host  # noqa: E402
from tests.pipeline import host_arena  # noqa: E402
from workload import DROPPED, FAILED, PRESENT, SUPPRESSED, docpage, tiny  # noqa: E402


def _arena_dev(a):
    return dev(a if a.size else np.zeros(1, np.uint8), np.uint8)


@pytest.mark.parametrize("cfg", ["tiny", "docpage"])
def test_filtered_waves_with_lists(cfg):
    lv = tiny().top if cfg == "tiny" else docpage(parents=2500, waves=12).top
    a = host_arena(lv)
    ad = _arena_dev(a)
    rng = np.random.default_rng(31)
    keep = (rng.random(lv.n_children) < 0.85).astype(np.uint8)
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
        cursor = 0
        for w in range(lv.n_waves):
            ch, st, ln, of = lv.reports(lv.wave(w))
            st = ls.filter(st, keep[ch])
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            r = ls.assemble_list(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1),
                                 out_cap=cursor + int(lv.arena_bytes) + 64, cursor=cursor)
            cursor = r["cursor"]
        ls.check_stats()


def test_caller_lists_repeats_incomplete_and_capacity():
    rng = np.random.default_rng(12)
    P = 1500
    counts = rng.integers(0, 9, P).astype(np.uint32)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        N = ls.N[x]
        ls.batch_ready(x, 0, None, 64, flush=True)
        ln = rng.integers(0, 33, N).astype(np.uint32)
        st = rng.choice([PRESENT] * 7 + [DROPPED] * 2 + [FAILED], N).astype(np.uint8)
        of = (np.cumsum(ln.astype(np.uint64)) - ln).astype(np.uint64) + 3
        arena = rng.integers(0, 256, int(of[-1] + ln[-1]) + 16).astype(np.uint8)
        ad = _arena_dev(arena)
        half = rng.permutation(N)[: N // 2].astype(np.uint32)
        ls.commit(x, half, st[half], ln[half], of[half], arena_bytes=arena.size)
        lst = np.concatenate([rng.integers(0, P + 7, 2500), np.flatnonzero(counts == 0)[:20]])
        ls.assemble_list(x, arena, ad, parents=lst, cursor=5)
        # entries do not fit: refused, and the counters stay as the oracle's
        ls.assemble_list(x, arena, ad, parents=lst, cursor=5, elem_cap=3)
        rest = np.setdiff1d(np.arange(N, dtype=np.uint32), half)
        ls.commit(x, rest, st[rest], ln[rest], of[rest], arena_bytes=arena.size)
        ls.assemble_list(x, arena, ad, parents=rng.permutation(P).astype(np.uint32), cursor=0)
        ls.assemble_list(x, arena, ad, parents=np.zeros(0, np.uint32), cursor=9)
        ls.check_stats()


def test_present_empty_list():
    with Lockstep() as ls:
        x = ls.expand(np.array([3, 2, 4], np.uint32))["xid"]
        ls.batch_ready(x, 0, None, 16, flush=True)
        ch = np.arange(9, dtype=np.uint32)
        st = np.array([DROPPED, DROPPED, DROPPED, PRESENT, DROPPED, PRESENT, SUPPRESSED, PRESENT,
                       PRESENT], np.uint8)
        arena = np.arange(128, dtype=np.uint8)
        ls.commit(x, ch, st, np.full(9, 5, np.uint32), ch.astype(np.uint64) * 7,
                  arena_bytes=arena.size)
        r = ls.assemble_list(x, arena, _arena_dev(arena), parents=[0, 1, 2, 0])
        assert list(r["parent_status"]) == [PRESENT, PRESENT, SUPPRESSED, PRESENT]
        assert list(r["elem_base"]) == [0, 3, 5, 5, 8]
        ls.check_stats()


@pytest.mark.parametrize("second_list", [True, False])
def test_back_to_back_calls_reusing_outputs_on_streams(second_list):
    """Two list assemblies issued without waiting, on a context with
    planning and copy streams, into the same caller arrays: the second
    call's planning writes the list structure (and a caller list's
    outcomes) while the first call's copy may still be writing the same
    arrays.  The arrays end with the second call's values, as in stream
    order."""
    lv = docpage(parents=4000, waves=1).top
    a = host_arena(lv)
    ad = _arena_dev(a)
    rng = np.random.default_rng(77)
    with Lockstep(streams=True) as ls:
        x = ls.expand(lv.counts)["xid"]
        ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
        ch, st, ln, of = lv.reports(lv.wave(0))
        cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
        P, N = lv.n_parents, ls.N[x]
        cap = int(lv.arena_bytes) + 64
        first = np.arange(P, dtype=np.uint32)[::-1].copy()   # every parent: a long copy
        second = rng.choice(P, 300, replace=False).astype(np.uint32) if second_list else None
        n2 = second.size if second_list else max(cm["n_done"], 1)
        r2 = ls.o.assemble_list(x, a, parents=second, n_parents=n2, out_cap=cap, cursor=None,
                                elem_cap=N, check=False)
        assert r2["status"] == 0
        d_status, d_off, d_len = empty(P, np.uint8), empty(P + 1, np.uint64), empty(P, np.uint32)
        d_eb = empty(P + 1, np.uint64)
        d_es, d_eo, d_el = empty(N, np.uint8), empty(N, np.uint64), empty(N, np.uint32)
        out = torch.zeros(cap, dtype=torch.uint8, device="cuda")
        keep = []
        for par, n in ((first, P), (second, n2)):
            d_par = None if par is None else dev(par, np.uint32)
            keep.append(d_par)
            st, _, _ = ro.ro_assemble_list(ls.ctx, x, ad, ad.numel(), d_par, n, None, d_status, d_off,
                                           d_len, out, cap, None, None, d_eb, d_es, d_eo, d_el, N,
                                           None, want_host=False)
            assert st == ro.RO_OK, ro.ro_last_error(ls.ctx)
        assert ro.ro_ctx_join(ls.ctx) == ro.RO_OK
        torch.cuda.synchronize()
        k, m, ob = r2["n_assembled"], r2["n_elems"], r2["out_bytes"]
        assert np.array_equal(host(d_status, np.uint8, k), r2["parent_status"])
        assert np.array_equal(host(d_off, np.uint64, k + 1), r2["out_off"])
        assert np.array_equal(host(d_len, np.uint32, k), r2["out_len"])
        assert np.array_equal(host(d_eb, np.uint64, k + 1), r2["elem_base"])
        assert np.array_equal(host(d_es, np.uint8, m), r2["elem_state"])
        assert np.array_equal(host(d_eo, np.uint64, m), r2["elem_off"])
        assert np.array_equal(host(d_el, np.uint32, m), r2["elem_len"])
        assert np.array_equal(out[:ob].cpu().numpy(), r2["out"][:ob])
