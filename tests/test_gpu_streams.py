"""Assembly on separate plan and copy streams (ro_ctx_set_streams).

The wave loop is issued without host synchronisation, so the lists and
plans of several waves are in flight at once and the context's ring slots
are reused while earlier waves are still being planned or copied.  Every
wave writes its per-parent outputs to buffers of its own; after one join all
of them are compared with the oracle, wave by wave, bit for bit.  The same
loop is also captured in a CUDA graph and replayed, and explicit parent
lists are assembled between commits (their outcomes must reflect exactly
the commits issued before them).
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
from oracle import OracleCtx  # noqa: E402
from tests.lockstep import dev, empty, host  # noqa: E402
from tests.pipeline import host_arena  # noqa: E402
from workload import docpage, skew  # noqa: E402


def oracle_waves(lv, arena_np, lists=None):
    """Oracle results per wave: the commit's completed parents and the
    assembly of them appended at a running cursor; with ``lists`` also the
    assembly of lists[w] (into an output of its own) right after wave w's commit."""
    o = OracleCtx(1)
    x = o.expand(lv.counts, parent_call=lv.parent_call)["xid"]
    o.batch_ready(x, 0, None, lv.batch_size, True, cap=lv.n_children + lv.batch_size)
    cursor, waves = 0, []
    for w in range(lv.n_waves):
        ch, st, ln, of = lv.reports(lv.wave(w))
        cm = o.gather_commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1))
        ex = None
        if lists is not None:
            ex = o.assemble(x, arena_np, parents=lists[w], want_len=True)
        a = o.assemble(x, arena_np, n_parents=max(cm["n_done"], 1), cursor=cursor)
        waves.append(dict(done=cm["done"], status=a["parent_status"], off=a["out_off"],
                          len=a["out_len"], bytes=a["out_bytes"], base=cursor,
                          out=a["out"][cursor:cursor + a["out_bytes"]].copy(), explicit=ex))
        cursor = a["cursor"]
    o.close()
    return waves, cursor


class AsyncPass:
    """Device inputs and per-wave outputs of one level, issued asynchronously."""

    def __init__(self, lv, arena_np, lists=None):
        self.lv = lv
        P, N, W = lv.n_parents, lv.n_children, lv.n_waves
        self.P, self.N, self.W = P, N, W
        self.counts = dev(lv.counts, np.uint32)
        self.pc = None if lv.parent_call is None else dev(lv.parent_call, np.uint8)
        self.offsets = empty(P + 1, np.uint64)
        self.cp, self.co = empty(N, np.uint32), empty(N, np.uint32)
        self.batched, self.nb = empty(N + lv.batch_size, np.uint32), empty(1, np.uint64)
        self.arena = dev(arena_np if arena_np.size else np.zeros(1, np.uint8), np.uint8)
        self.arena_bytes = max(int(lv.arena_bytes), 1)
        self.rep = []
        for w in range(W):
            ch, st, ln, of = lv.reports(lv.wave(w))
            self.rep.append((ch.size, dev(ch, np.uint32), dev(st, np.uint8), dev(ln, np.uint32),
                             dev(of, np.uint64)))
        self.done = [empty(P, np.uint32) for _ in range(W)]
        self.nd = [empty(1, np.uint64) for _ in range(W)]
        self.status = [empty(P, np.uint8) for _ in range(W)]
        self.off = [empty(P + 1, np.uint64) for _ in range(W)]
        self.len = [empty(P, np.uint32) for _ in range(W)]
        self.ob = empty(W, np.uint64)
        self.cursor = empty(1, np.uint64)
        self.out_cap = int(lv.arena_bytes) + 64
        self.out = torch.zeros(max(self.out_cap, 1), dtype=torch.uint8, device="cuda")
        self.lists = None
        if lists is not None:
            self.lists = [dev(l, np.uint32) for l in lists]
            self.list_n = [int(l.size) for l in lists]
            self.xs = [empty(l.size, np.uint8) for l in lists]
            self.xo = [empty(l.size + 1, np.uint64) for l in lists]
            self.xl = [empty(l.size, np.uint32) for l in lists]
            # each list's bytes go to an output of their own (no cursor)
            self.xcap = int(lv.arena_bytes) * 2 + 64
            self.xout = [torch.zeros(self.xcap, dtype=torch.uint8, device="cuda") for _ in lists]

    def expand(self, ctx):
        st, n, _, x = ro.ro_expand(ctx, -1, self.counts, self.P, self.pc, self.offsets, self.cp,
                                   self.co, self.N, None)
        assert st == ro.RO_OK and n == self.N, ro.ro_last_error(ctx)
        return x

    def waves(self, ctx, x):
        st, _, _ = ro.ro_batch_ready(ctx, x, 0, None, 0, self.lv.batch_size, 1, self.batched,
                                     self.N + self.lv.batch_size, self.nb, want_host=False)
        assert st == ro.RO_OK
        self.cursor.zero_()
        for w in range(self.W):
            n, ch, stt, ln, of = self.rep[w]
            st, _ = ro.ro_gather_commit(ctx, x, n, None, ch, stt, ln, of, None, self.arena_bytes,
                                        None, self.done[w], self.P, self.nd[w], want_host=False)
            assert st == ro.RO_OK
            if self.lists is not None:
                st, _ = ro.ro_assemble(ctx, x, self.arena, self.arena_bytes, self.lists[w],
                                       self.list_n[w], None, self.xs[w], self.xo[w], self.xl[w],
                                       self.xout[w], self.xcap, None, None, want_host=False)
                assert st == ro.RO_OK
            st, _ = ro.ro_assemble(ctx, x, self.arena, self.arena_bytes, None, self.P, None,
                                   self.status[w], self.off[w], self.len[w], self.out, self.out_cap,
                                   self.cursor, self.ob[w:], want_host=False)
            assert st == ro.RO_OK
        assert ro.ro_ctx_join(ctx) == ro.RO_OK

    def check(self, ref, total):
        torch.cuda.synchronize()
        obs = host(self.ob, np.uint64)
        for w, r in enumerate(ref):
            k = r["done"].size
            assert int(host(self.nd[w], np.uint64, 1)[0]) == k, w
            assert np.array_equal(host(self.done[w], np.uint32, k), r["done"]), w
            assert np.array_equal(host(self.status[w], np.uint8, k), r["status"]), w
            assert np.array_equal(host(self.off[w], np.uint64, k + 1), r["off"]), w
            assert np.array_equal(host(self.len[w], np.uint32, k), r["len"]), w
            assert int(obs[w]) == r["bytes"], w
            got = self.out[r["base"]:r["base"] + r["bytes"]].cpu().numpy()
            assert np.array_equal(got, r["out"]), f"wave {w}: assembled bytes differ"
            if r["explicit"] is not None:
                e = r["explicit"]
                m = self.list_n[w]
                assert np.array_equal(host(self.xs[w], np.uint8, m), e["parent_status"]), w
                assert np.array_equal(host(self.xo[w], np.uint64, m + 1), e["out_off"]), w
                assert np.array_equal(host(self.xl[w], np.uint32, m), e["out_len"]), w
                nb = e["out_bytes"]
                assert np.array_equal(self.xout[w][:nb].cpu().numpy(), e["out"][:nb]), w
        assert int(host(self.cursor, np.uint64, 1)[0]) == total


def _ctx(streams=True):
    ctx = ro.ro_ctx_create(0, torch.cuda.current_stream(), 1)
    side = None
    if streams:
        side = (torch.cuda.Stream(), torch.cuda.Stream())
        ro.ro_ctx_set_streams(ctx, *side)
    return ctx, side


@pytest.mark.parametrize("cfg", ["docpage", "skew"])
def test_async_waves_on_three_streams(cfg):
    lv = (docpage(parents=3000, waves=24) if cfg == "docpage"
          else skew(parents=20000, heavy=4, heavy_children=8000)).top
    a = host_arena(lv)
    ref, total = oracle_waves(lv, a)
    ps = AsyncPass(lv, a)
    ctx, _side = _ctx()
    try:
        ps.waves(ctx, ps.expand(ctx))
        assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
        ps.check(ref, total)
        # again on the same context (reused buffers, events and ring slots)
        ps.out.zero_()
        ro.ro_ctx_reset(ctx)
        ps.waves(ctx, ps.expand(ctx))
        assert ro.ro_ctx_sync(ctx) == ro.RO_OK
        ps.check(ref, total)
    finally:
        ro.ro_ctx_destroy(ctx)


def test_async_waves_captured_in_a_graph():
    lv = docpage(parents=2000, waves=12).top
    a = host_arena(lv)
    ref, total = oracle_waves(lv, a)
    ps = AsyncPass(lv, a)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        ctx = ro.ro_ctx_create(0, stream, 1)
        side = (torch.cuda.Stream(), torch.cuda.Stream())
        ro.ro_ctx_set_streams(ctx, *side)
        try:
            ps.waves(ctx, ps.expand(ctx))   # sizes every buffer
            assert ro.ro_ctx_sync(ctx) == ro.RO_OK
            ro.ro_ctx_reset(ctx)
            x = ps.expand(ctx)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                ps.waves(ctx, x)
            for _ in range(2):
                ps.out.zero_()
                for t in ps.status + ps.off + ps.len + ps.done:
                    t.zero_()
                ro.ro_ctx_reset(ctx)
                ps.expand(ctx)
                g.replay()
                assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
                ps.check(ref, total)
        finally:
            ro.ro_ctx_destroy(ctx)


def test_one_wave_captured_after_one_eager_commit():
    """A one-wave pass run once eagerly (its commit takes one completion
    stream), then captured and replayed twice (the captured commits take the
    next streams in turn): every stream's scan slot was sized by the eager
    call, so the capture never needs to grow a buffer, and each replay
    equals the oracle."""
    lv = docpage(parents=3000, waves=1).top
    a = host_arena(lv)
    ref, total = oracle_waves(lv, a)
    ps = AsyncPass(lv, a)
    stream = torch.cuda.Stream()
    with torch.cuda.stream(stream):
        ctx = ro.ro_ctx_create(0, stream, 1)
        ro.ro_ctx_set_streams(ctx, torch.cuda.Stream(), torch.cuda.Stream())
        try:
            ps.waves(ctx, ps.expand(ctx))
            assert ro.ro_ctx_sync(ctx) == ro.RO_OK
            for _ in range(2):
                ro.ro_ctx_reset(ctx)
                x = ps.expand(ctx)
                g = torch.cuda.CUDAGraph()
                with torch.cuda.graph(g, stream=stream):
                    ps.waves(ctx, x)
                ps.out.zero_()
                for t in ps.status + ps.off + ps.len + ps.done:
                    t.zero_()
                ro.ro_ctx_reset(ctx)
                ps.expand(ctx)
                g.replay()
                assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
                ps.check(ref, total)
        finally:
            ro.ro_ctx_destroy(ctx)


def test_explicit_lists_between_commits_see_exactly_the_earlier_commits():
    lv = docpage(parents=2500, waves=10).top
    rng = np.random.default_rng(21)
    P = lv.n_parents
    lists = [np.concatenate([rng.integers(0, P + 5, 700), rng.integers(0, 40, 64)]).astype(np.uint32)
             for _ in range(lv.n_waves)]
    a = host_arena(lv)
    ref, total = oracle_waves(lv, a, lists=lists)
    ps = AsyncPass(lv, a, lists=lists)
    ctx, _side = _ctx()
    try:
        ps.waves(ctx, ps.expand(ctx))
        assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
        ps.check(ref, total)
        st = ro.ro_ctx_stats(ctx)
        assert st.pop("status") == ro.RO_OK
        assert st["assemble_incomplete"] == sum(
            int((r["explicit"]["parent_status"] == ro.RO_PENDING).sum()) for r in ref)
    finally:
        ro.ro_ctx_destroy(ctx)


def test_set_streams_back_to_one_stream():
    lv = docpage(parents=1500, waves=6).top
    a = host_arena(lv)
    ref, total = oracle_waves(lv, a)
    ps = AsyncPass(lv, a)
    ctx, _side = _ctx()
    try:
        ps.waves(ctx, ps.expand(ctx))
        assert ro.ro_ctx_set_streams(ctx, None, None) == ro.RO_OK
        ps.out.zero_()
        ro.ro_ctx_reset(ctx)
        ps.waves(ctx, ps.expand(ctx))
        assert ro.ro_ctx_sync(ctx) == ro.RO_OK
        ps.check(ref, total)
    finally:
        ro.ro_ctx_destroy(ctx)


@pytest.mark.parametrize("B", [32, 256])
def test_call_admissions_on_streams_of_their_own(B):
    """Four Calls, each admitting on a stream of its own
    (ro_ctx_set_call_streams).  Per readiness wave the four admissions are
    issued without waiting, from one candidate list (each Call keeps its
    own children), so they run at the same time; every Call's reserved
    batches, the commit of their results and the assembly equal the
    oracle's, wave by wave."""
    from tests.lockstep import Lockstep
    from workload import streaming
    lv = streaming(total_children=80000, batch_size=B, ready_waves=20).top
    a = host_arena(lv)
    ad = dev(a if a.size else np.zeros(1, np.uint8), np.uint8)
    with Lockstep(n_calls=4, call_streams=True) as ls:
        x = ls.expand(lv.counts, parent_call=lv.parent_call)["xid"]
        N = ls.N[x]
        d_b = [empty(N + B, np.uint32) for _ in range(4)]
        d_nb = [empty(1, np.uint64) for _ in range(4)]
        n_ready = lv.ready_bounds.size - 1
        for w in range(n_ready):
            cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
            last = w == n_ready - 1
            d_cand = dev(cand, np.uint32)
            for c in range(4):
                st, _, _ = ro.ro_batch_ready(ls.ctx, x, c, d_cand, cand.size, B, last, d_b[c], N + B,
                                             d_nb[c], want_host=False)
                assert st == ro.RO_OK, ro.ro_last_error(ls.ctx)
            assert ro.ro_ctx_sync(ls.ctx) == ro.RO_OK
            got = []
            for c in range(4):
                r = ls.o.batch_ready(x, c, cand, B, last, cap=N + B, check=False)
                nb = int(host(d_nb[c], np.uint64, 1)[0])
                assert nb == r["n_batched"]
                assert np.array_equal(host(d_b[c], np.uint32, nb), r["batched"])
                got.append(r["batched"])
            got = np.concatenate(got)
            got = got[np.argsort(lv.key[got], kind="stable")]
            ch, st, ln, of = lv.reports(got)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()


def test_call_streams_with_failures_retries_and_capacity():
    """Call streams with the rest of the path in between: a GroupFailure
    commit, a retry and a refused admission (capacity) of one Call while the
    others admit; all equal the oracle's."""
    from tests.lockstep import Lockstep
    rng = np.random.default_rng(41)
    P = 3000
    counts = rng.integers(1, 9, P).astype(np.uint32)
    calls = (np.arange(P) % 3).astype(np.uint8)
    with Lockstep(n_calls=3, call_streams=True) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        N = ls.N[x]
        cand = rng.permutation(N).astype(np.uint32)
        r = [ls.batch_ready(x, c, cand[: N // 2], 4) for c in range(3)]
        # a GroupFailure from the first reserved child of Call 0
        ch = np.array([r[0]["batched"][0]], np.uint32)
        ls.commit(x, ch, np.array([5], np.uint8), np.array([8], np.uint32), np.array([0], np.uint64),
                  arena_bytes=64)
        ls.retry(x, 1, r[1]["batched"][:8])
        ls.batch_ready(x, 2, cand[N // 2:], 4, cap=3)          # refused: nothing changes
        for c in range(3):
            ls.batch_ready(x, c, cand[N // 2:], 4, flush=True)
        ls.check_stats()


def test_call_streams_captured_in_a_graph():
    """The streaming configuration's wave loop (four Calls, each admitting on
    a stream of its own; commit of the reserved children's results in key
    order; assembly at a running cursor on plan and copy streams) captured
    in a CUDA graph and replayed: every Call's reservation of every wave and
    every assembled output equal the oracle's."""
    from workload import streaming
    B = 64
    lv = streaming(total_children=60000, batch_size=B, ready_waves=16).top
    a = host_arena(lv)
    P, N, W, C = lv.n_parents, lv.n_children, lv.ready_bounds.size - 1, lv.n_calls
    # the oracle's pass: reservations per (wave, Call), then reports, commit, assembly
    o = OracleCtx(C)
    x = o.expand(lv.counts, parent_call=lv.parent_call)["xid"]
    ref, reports, cursor = [], [], 0
    for w in range(W):
        cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
        res = [o.batch_ready(x, c, cand, B, w == W - 1, cap=N + B)["batched"] for c in range(C)]
        got = np.concatenate(res)
        got = got[np.argsort(lv.key[got], kind="stable")]
        ch, st, ln, of = lv.reports(got)
        reports.append((ch.size, dev(ch, np.uint32), dev(st, np.uint8), dev(ln, np.uint32),
                        dev(of, np.uint64)))
        cm = o.gather_commit(x, ch, st, ln, of, arena_bytes=max(lv.arena_bytes, 1))
        asm = o.assemble(x, a, n_parents=max(cm["n_done"], 1), cursor=cursor)
        ref.append(dict(res=res, status=asm["parent_status"], off=asm["out_off"],
                        bytes=asm["out_bytes"], base=cursor,
                        out=asm["out"][cursor:cursor + asm["out_bytes"]].copy()))
        cursor = asm["cursor"]
    o.close()
    counts, pc = dev(lv.counts, np.uint32), dev(lv.parent_call, np.uint8)
    offsets, cp, co = empty(P + 1, np.uint64), empty(N, np.uint32), empty(N, np.uint32)
    cands = [dev(lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]], np.uint32) for w in range(W)]
    batched = [[empty(N + B, np.uint32) for _ in range(C)] for _ in range(W)]
    nb = [[empty(1, np.uint64) for _ in range(C)] for _ in range(W)]
    status = [empty(P, np.uint8) for _ in range(W)]
    off = [empty(P + 1, np.uint64) for _ in range(W)]
    ad = dev(a if a.size else np.zeros(1, np.uint8), np.uint8)
    out_cap = int(lv.arena_bytes) + 64
    out = torch.zeros(out_cap, dtype=torch.uint8, device="cuda")
    cur = empty(1, np.uint64)
    stream = torch.cuda.Stream()

    def waves(ctx, xid):
        cur.zero_()
        for w in range(W):
            n_c = int(lv.ready_bounds[w + 1] - lv.ready_bounds[w])
            for c in range(C):
                st, _, _ = ro.ro_batch_ready(ctx, xid, c, cands[w], n_c, B, w == W - 1, batched[w][c],
                                             N + B, nb[w][c], want_host=False)
                assert st == ro.RO_OK
            n, ch, stt, ln, of = reports[w]
            st, _ = ro.ro_gather_commit(ctx, xid, n, None, ch, stt, ln, of, None,
                                        max(int(lv.arena_bytes), 1), None, None, 0, None,
                                        want_host=False)
            assert st == ro.RO_OK
            st, _ = ro.ro_assemble(ctx, xid, ad, ad.numel(), None, P, None, status[w], off[w], None,
                                   out, out_cap, cur, None, want_host=False)
            assert st == ro.RO_OK
        assert ro.ro_ctx_join(ctx) == ro.RO_OK

    def expand(ctx):
        st, n, _, xid = ro.ro_expand(ctx, -1, counts, P, pc, offsets, cp, co, N, None)
        assert st == ro.RO_OK and n == N
        return xid

    def check():
        torch.cuda.synchronize()
        for w, r in enumerate(ref):
            for c in range(C):
                k = int(host(nb[w][c], np.uint64, 1)[0])
                assert np.array_equal(host(batched[w][c], np.uint32, k), r["res"][c]), (w, c)
            k = r["status"].size
            assert np.array_equal(host(status[w], np.uint8, k), r["status"]), w
            assert np.array_equal(host(off[w], np.uint64, k + 1), r["off"]), w
            got = out[r["base"]:r["base"] + r["bytes"]].cpu().numpy()
            assert np.array_equal(got, r["out"]), w
        assert int(host(cur, np.uint64, 1)[0]) == cursor

    with torch.cuda.stream(stream):
        ctx = ro.ro_ctx_create(0, stream, C)
        side = (torch.cuda.Stream(), torch.cuda.Stream())
        call_side = [torch.cuda.Stream() for _ in range(C)]
        ro.ro_ctx_set_streams(ctx, *side)
        ro.ro_ctx_set_call_streams(ctx, call_side)
        try:
            waves(ctx, expand(ctx))   # sizes every buffer
            assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
            check()
            ro.ro_ctx_reset(ctx)
            xid = expand(ctx)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                waves(ctx, xid)
            for _ in range(2):
                out.zero_()
                for t in status + off + [b for row in batched for b in row]:
                    t.zero_()
                ro.ro_ctx_reset(ctx)
                expand(ctx)
                g.replay()
                assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
                check()
        finally:
            ro.ro_ctx_destroy(ctx)


def test_captured_commits_with_repeats_and_group_failures():
    """A wave loop with repeated reports in some waves and GroupFailure
    reports in others (the commit's fix-up then orders the repeats and
    applies the barriers), captured in a CUDA graph and replayed, gives every
    verdict, completed list, status, offset and byte the oracle gives."""
    lv = docpage(parents=1500, waves=10).top
    a = host_arena(lv)
    rng = np.random.default_rng(5)
    W, P, N = lv.n_waves, lv.n_parents, lv.n_children
    reps = []
    for w in range(W):
        ch, st, ln, of = lv.reports(lv.wave(w))
        if w in (2, 5):   # repeats of some reports of this wave, later in the array
            idx = rng.choice(ch.size, 25, replace=False)
            ch, st = np.concatenate([ch, ch[idx]]), np.concatenate([st, st[idx]])
            ln, of = np.concatenate([ln, ln[idx]]), np.concatenate([of, of[idx]])
        if w in (3, 7):   # GroupFailures
            st = st.copy()
            st[rng.choice(ch.size, 4, replace=False)] = 5
        reps.append((ch, st, ln, of))
    o = OracleCtx(1)
    x = o.expand(lv.counts)["xid"]
    o.batch_ready(x, 0, None, lv.batch_size, True, cap=N + lv.batch_size)
    ref, cursor = [], 0
    for w in range(W):
        cm = o.gather_commit(x, *reps[w], arena_bytes=max(lv.arena_bytes, 1))
        asm = o.assemble(x, a, n_parents=max(cm["n_done"], 1), cursor=cursor)
        ref.append(dict(code=cm["code"], done=cm["done"], status=asm["parent_status"],
                        off=asm["out_off"], bytes=asm["out_bytes"], base=cursor,
                        out=asm["out"][cursor:cursor + asm["out_bytes"]].copy()))
        cursor = asm["cursor"]
    o.close()
    counts = dev(lv.counts, np.uint32)
    offsets, cp, co = empty(P + 1, np.uint64), empty(N, np.uint32), empty(N, np.uint32)
    batched = empty(N + lv.batch_size, np.uint32)
    dr = [tuple(dev(v, t) for v, t in zip(r, (np.uint32, np.uint8, np.uint32, np.uint64))) for r in reps]
    code = [empty(r[0].size, np.uint8) for r in reps]
    done = [empty(P, np.uint32) for _ in range(W)]
    status = [empty(P, np.uint8) for _ in range(W)]
    off = [empty(P + 1, np.uint64) for _ in range(W)]
    ad = dev(a if a.size else np.zeros(1, np.uint8), np.uint8)
    out_cap = int(lv.arena_bytes) + 64
    out = torch.zeros(out_cap, dtype=torch.uint8, device="cuda")
    cur = empty(1, np.uint64)
    stream = torch.cuda.Stream()

    def expand(ctx):
        st, n, _, xid = ro.ro_expand(ctx, -1, counts, P, None, offsets, cp, co, N, None)
        assert st == ro.RO_OK and n == N
        return xid

    def waves(ctx, xid):
        st, _, _ = ro.ro_batch_ready(ctx, xid, 0, None, 0, lv.batch_size, 1, batched, N + lv.batch_size,
                                     None, want_host=False)
        assert st == ro.RO_OK
        cur.zero_()
        for w in range(W):
            ch, stt, ln, of = dr[w]
            st, _ = ro.ro_gather_commit(ctx, xid, reps[w][0].size, None, ch, stt, ln, of, None,
                                        max(int(lv.arena_bytes), 1), code[w], done[w], P, None,
                                        want_host=False)
            assert st == ro.RO_OK
            st, _ = ro.ro_assemble(ctx, xid, ad, ad.numel(), None, P, None, status[w], off[w], None,
                                   out, out_cap, cur, None, want_host=False)
            assert st == ro.RO_OK
        assert ro.ro_ctx_join(ctx) == ro.RO_OK

    def check():
        torch.cuda.synchronize()
        for w, r in enumerate(ref):
            assert np.array_equal(host(code[w], np.uint8, r["code"].size), r["code"]), w
            k = r["done"].size
            assert np.array_equal(host(done[w], np.uint32, k), r["done"]), w
            assert np.array_equal(host(status[w], np.uint8, k), r["status"]), w
            assert np.array_equal(host(off[w], np.uint64, k + 1), r["off"]), w
            got = out[r["base"]:r["base"] + r["bytes"]].cpu().numpy()
            assert np.array_equal(got, r["out"]), w
        assert int(host(cur, np.uint64, 1)[0]) == cursor

    with torch.cuda.stream(stream):
        ctx = ro.ro_ctx_create(0, stream, 1)
        side = (torch.cuda.Stream(), torch.cuda.Stream())
        ro.ro_ctx_set_streams(ctx, *side)
        try:
            waves(ctx, expand(ctx))
            assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
            check()
            ro.ro_ctx_reset(ctx)
            xid = expand(ctx)
            g = torch.cuda.CUDAGraph()
            with torch.cuda.graph(g, stream=stream):
                waves(ctx, xid)
            for _ in range(2):
                out.zero_()
                for t in code + done + status + off:
                    t.zero_()
                ro.ro_ctx_reset(ctx)
                expand(ctx)
                g.replay()
                assert ro.ro_ctx_sync(ctx) == ro.RO_OK, ro.ro_last_error(ctx)
                check()
        finally:
            ro.ro_ctx_destroy(ctx)
