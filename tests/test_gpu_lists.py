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


from tests.lockstep import Lockstep, dev  # noqa: E402
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
