"""GPU path (C ABI, sm_103a kernels) against the CPU oracle, element by element.

Sizes are chosen so the oracle finishes in seconds while the kernels still
run several tiles with ragged tails (expand tiles of 4096 parents and 4096
children, queue tiles of 2048 candidates, member tiles of 2048, copy chunks
of 16 KB).  Everything compared is integer or byte data: the bar is
bit-exact equality.
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


from tests.lockstep import Lockstep, dev  # noqa: E402
from tests.pipeline import host_arena  # noqa: E402
from workload import DROPPED, FAILED, PRESENT, SUPPRESSED, docpage, skew, streaming, tiny, video  # noqa: E402


def _arena_dev(a: np.ndarray):
    return dev(a if a.size else np.zeros(1, np.uint8), np.uint8)


def run_level(ls, lv, arena_np, arena_d, parent_xid=-1, device_count=False):
    ex = ls.expand(lv.counts, parent_xid=parent_xid, parent_call=lv.parent_call)
    x = ex["xid"]
    ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
    last = None
    for w in range(lv.n_waves):
        ch, st, ln, of = lv.reports(lv.wave(w))
        cm = ls.commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1),
                       device_count=device_count)
        last = ls.assemble(x, arena_np, arena_d, parents=None, n_parents=max(cm["n_done"], 1))
    return x, last


# --------------------------------------------------------------------- expand
@pytest.mark.parametrize("shape", ["one", "zeros", "wide", "heavy", "empties_run", "all_empty"])
def test_expand_parity(shape):
    rng = np.random.default_rng(hash(shape) % 2**32)
    if shape == "one":
        counts = np.array([3], np.uint32)
    elif shape == "zeros":
        counts = rng.integers(0, 10, 9001).astype(np.uint32)
        counts[rng.random(9001) < 0.25] = 0
    elif shape == "wide":
        counts = rng.integers(1, 700, 3001).astype(np.uint32)
    elif shape == "heavy":
        counts = np.ones(20000, np.uint32)
        counts[[5, 777, 19999]] = [40000, 12345, 9000]
    elif shape == "empties_run":
        counts = np.zeros(30000, np.uint32)
        counts[[0, 15000, 29999]] = [5000, 7, 6000]
    else:
        counts = np.zeros(5000, np.uint32)
    with Lockstep() as ls:
        ls.expand(counts)
        ls.check_stats()


def test_expand_capacity_and_overflow():
    with Lockstep() as ls:
        r = ls.expand(np.array([5, 6, 7], np.uint32), child_cap=10)
        assert r["status"] == 2 and r["n_children"] == 18
        r = ls.expand(np.array([2**31, 2**31], np.uint32), child_cap=16)
        assert r["status"] == 3
        ok = ls.expand(np.array([5, 6, 7], np.uint32))
        assert ok["status"] == 0 and ok["xid"] == 0


# ---------------------------------------------------------------- batch_ready
@pytest.mark.parametrize("seed", range(4))
def test_batch_ready_waves_with_duplicates(seed):
    rng = np.random.default_rng(1000 + seed)
    counts = rng.integers(1, 9, 2500).astype(np.uint32)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        N = ls.N[x]
        B = int(rng.choice([1, 7, 64, 256, 3000]))
        for w in range(6):
            m = int(rng.integers(0, 5000))
            cand = rng.integers(0, N + 50, m).astype(np.uint32)
            ls.batch_ready(x, 0, cand, B, flush=(w == 5))
        ls.batch_ready(x, 0, None, B, flush=True)
        ls.check_stats()


def test_batch_ready_calls_and_capacity():
    rng = np.random.default_rng(7)
    counts = rng.integers(0, 6, 4000).astype(np.uint32)
    calls = (np.arange(4000) % 3).astype(np.uint8)
    with Lockstep(n_calls=3) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        N = ls.N[x]
        perm = rng.permutation(N).astype(np.uint32)
        # too small an output: refused, nothing changes, then retried
        r = ls.batch_ready(x, 1, perm[:3000], 16, flush=True, cap=10)
        assert r["status"] == 2
        for call in range(3):
            ls.batch_ready(x, call, perm[:3000], 16, flush=False)
        for call in range(3):
            ls.batch_ready(x, call, None, 16, flush=True)
        ls.check_stats()


# ------------------------------------------------------------ whole pipelines
def test_pipeline_tiny_config():
    lv = tiny().top
    a = host_arena(lv)
    with Lockstep() as ls:
        run_level(ls, lv, a, _arena_dev(a))
        ls.check_stats()


@pytest.mark.parametrize("device_count,streams", [(False, False), (True, False), (False, True)])
def test_pipeline_docpage_small(device_count, streams):
    lv = docpage(parents=2500, waves=16).top
    a = host_arena(lv)
    with Lockstep(streams=streams) as ls:
        run_level(ls, lv, a, _arena_dev(a), device_count=device_count)
        ls.check_stats()


def test_pipeline_skew_small():
    lv = skew(parents=30000, heavy=6, heavy_children=9000).top
    a = host_arena(lv)
    with Lockstep() as ls:
        run_level(ls, lv, a, _arena_dev(a))
        ls.check_stats()


def test_pipeline_video_nested():
    top, leaf = video(videos=400).levels
    a = host_arena(leaf)
    with Lockstep() as ls:
        x0 = ls.expand(top.counts)["xid"]
        ls.batch_ready(x0, 0, None, top.batch_size, flush=True)
        x1 = ls.expand(leaf.counts, parent_xid=x0)["xid"]
        ls.batch_ready(x1, 0, None, leaf.batch_size, flush=True)
        ch, st, ln, of = leaf.reports(leaf.wave(0))
        cm1 = ls.commit(x1, ch, st, ln, of, arena_bytes=leaf.arena_bytes)
        a1 = ls.assemble(x1, a, _arena_dev(a), parents=None, n_parents=cm1["n_done"])
        r1 = a1["r"]
        level1 = a1["out"][:a1["out_bytes"]].cpu().numpy()
        cm0 = ls.commit(x0, cm1["done"], r1["parent_status"], r1["out_len"], r1["out_off"][:-1],
                        arena_bytes=a1["out_bytes"])
        assert cm0["n_done"] == top.n_parents
        ls.assemble(x0, level1, _arena_dev(level1), parents=None, n_parents=cm0["n_done"])
        ls.check_stats()


@pytest.mark.parametrize("B", [32, 256, 2048])
def test_pipeline_streaming_calls(B):
    lv = streaming(total_children=60000, batch_size=B, ready_waves=25).top
    a = host_arena(lv)
    ad = _arena_dev(a)
    with Lockstep(n_calls=4) as ls:
        x = ls.expand(lv.counts, parent_call=lv.parent_call)["xid"]
        n_ready = lv.ready_bounds.size - 1
        for w in range(n_ready):
            cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
            reserved = [ls.batch_ready(x, c, cand, B, flush=(w == n_ready - 1))["batched"]
                        for c in range(4)]
            got = np.concatenate(reserved) if reserved else np.zeros(0, np.uint32)
            got = got[np.argsort(lv.key[got], kind="stable")]
            ch, st, ln, of = lv.reports(got)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()


# ------------------------------------------------------------ fence, duplicates
def test_generation_fence_and_codes():
    with Lockstep() as ls:
        x = ls.expand(np.array([2, 3], np.uint32))["xid"]
        ls.batch_ready(x, 0, np.array([0, 1, 2, 3], np.uint32), 3, flush=False)
        ch = np.array([4, 3, 0, 1, 0, 9, 2, 1, 2], np.uint32)
        st = np.array([1, 1, 1, 1, 1, 1, 7, 3, 1], np.uint8)
        ln = np.array([8, 8, 8, 8, 8, 8, 8, 8, 99], np.uint32)
        of = np.array([0, 0, 0, 8, 0, 0, 0, 0, 90], np.uint64)
        gen = np.array([0, 0, 0, 0, 0, 0, 0, 1, 0], np.uint32)
        ls.commit(x, ch, st, ln, of, gen=gen, arena_bytes=100)
        ls.commit(x, np.array([1, 1], np.uint32), np.array([3, 1], np.uint8),
                  np.array([0, 4], np.uint32), np.array([0, 0], np.uint64), arena_bytes=100)
        ls.check_stats()


@pytest.mark.parametrize("seed", range(5))
def test_duplicate_reports_first_in_array_order_wins(seed):
    rng = np.random.default_rng(50 + seed)
    counts = rng.integers(1, 12, 3000).astype(np.uint32)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        N = ls.N[x]
        ls.batch_ready(x, 0, None, 64, flush=True)
        arena = rng.integers(0, 256, 200000).astype(np.uint8)
        ad = _arena_dev(arena)
        done_total = 0
        order = rng.permutation(N)
        for chunk in np.array_split(order, 4):
            dup = rng.choice(chunk, size=max(1, chunk.size // 3))
            ch = np.concatenate([chunk, dup, dup[: dup.size // 2]]).astype(np.uint32)
            rng.shuffle(ch)
            m = ch.size
            st = rng.choice([PRESENT, PRESENT, PRESENT, DROPPED, FAILED, SUPPRESSED], m).astype(np.uint8)
            ln = rng.integers(0, 300, m).astype(np.uint32)
            of = rng.integers(0, 199000, m).astype(np.uint64)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=arena.size)
            done_total += cm["n_done"]
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        assert done_total == counts.size
        ls.check_stats()


# ------------------------------------------------------------ assemble corners
@pytest.mark.parametrize("streams", [False, True])
def test_assemble_lists_cursor_capacity_and_alignment(streams):
    rng = np.random.default_rng(9)
    P = 3000
    counts = rng.integers(0, 8, P).astype(np.uint32)
    with Lockstep(streams=streams) as ls:
        ex = ls.expand(counts)
        x = ex["xid"]
        N = ls.N[x]
        ls.batch_ready(x, 0, None, 32, flush=True)
        # tiny, odd-sized records (0..40 bytes, some Present with 0 bytes) packed back to back
        ln = rng.integers(0, 41, N).astype(np.uint32)
        st = rng.choice([PRESENT] * 8 + [DROPPED, FAILED], N).astype(np.uint8)
        ln[st != PRESENT] = 0
        of = (np.cumsum(ln.astype(np.uint64)) - ln).astype(np.uint64) + 5
        arena = rng.integers(0, 256, int(of[-1] + ln[-1]) + 16 if N else 16).astype(np.uint8)
        ad = _arena_dev(arena)
        order = rng.permutation(N).astype(np.uint32)
        half = order[: N // 2]
        ls.commit(x, half, st[half], ln[half], of[half], arena_bytes=arena.size)
        out = torch.zeros(1 << 20, dtype=torch.uint8, device="cuda")
        # explicit list mixing complete, incomplete, out-of-range, repeated and empty parents
        lst = np.concatenate([rng.integers(0, P + 10, 4000), np.flatnonzero(counts == 0)[:50]])
        ls.assemble(x, arena, ad, parents=lst, out_cap=out.numel(), out_dev=out, cursor=3)
        rest = order[N // 2:]
        ls.commit(x, rest, st[rest], ln[rest], of[rest], arena_bytes=arena.size)
        lst = rng.permutation(P).astype(np.uint32)
        r = ls.assemble(x, arena, ad, parents=lst, out_cap=17 + 100, out_dev=out, cursor=17)
        assert r["status"] == 2   # does not fit: nothing copied
        for cur in (0, 1, 7, 15, 16, 1001):
            ls.assemble(x, arena, ad, parents=lst, out_cap=out.numel(), out_dev=out, cursor=cur)
        ls.assemble(x, arena, ad, parents=lst[:0], out_cap=out.numel(), out_dev=out, cursor=5)
        ls.check_stats()


def test_assemble_large_records_and_hot_parent():
    rng = np.random.default_rng(11)
    counts = np.array([1, 3000, 2, 0, 40, 1], np.uint32)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        N = ls.N[x]
        ls.batch_ready(x, 0, None, 256, flush=True)
        ln = rng.integers(1, 65537, N).astype(np.uint32)
        small = rng.random(N) < 0.3
        ln[small] = rng.integers(1, 64, int(small.sum()))
        of = (np.cumsum(ln.astype(np.uint64)) - ln).astype(np.uint64)
        arena = rng.integers(0, 256, int(of[-1] + ln[-1])).astype(np.uint8)
        ad = _arena_dev(arena)
        order = rng.permutation(N).astype(np.uint32)
        st = np.full(N, PRESENT, np.uint8)
        for chunk in np.array_split(order, 3):
            cm = ls.commit(x, chunk, st[chunk], ln[chunk], of[chunk], arena_bytes=arena.size)
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()
