"""Full-size configurations.  The 1,000,000-document configuration (16.4M children,
38.8 GB arena, 256 arrival waves, batch 256), in the launch configuration
bench.py times, against the oracle on every output: lineage arrays, the
reserved batches, every wave's verdicts, completed-parent list, statuses,
offsets, lengths and all ~12 GB of assembled bytes.  The CUDA-graph replay of
the wave loop (what the benchmark runs) is then checked byte for byte
against the eager run.  Needs ~70 GB of host memory and ~60 GB on the GPU.
The extreme-skew (110M children), video -> clip -> frame (100,000 videos,
nested) and streaming (four Calls, 50M children, 1,000 readiness waves)
configurations run at full size too, each compared with the oracle call by
call."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module")
def setup():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    from workload import docpage
    return docpage()   # 1M parents, 256 waves


def test_docpage_full_size(setup):
    import paper_2609_18703_gb300 as ro
    from oracle import OracleCtx
    from tests.lockstep import host
    from tests.pipeline import host_arena
    from workload import record_bytes
    from workload.device import fill_payload

    lv = setup.top
    P, N, W, B = lv.n_parents, lv.n_children, lv.n_waves, lv.batch_size
    stream = torch.cuda.current_stream()
    i32 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int32)).cuda()
    i64 = lambda a: torch.from_numpy(np.ascontiguousarray(a).view(np.int64)).cuda()
    arr = lv.arrival
    d_counts = i32(lv.counts)
    d_child, d_state = i32(arr), torch.from_numpy(lv.state[arr]).cuda()
    d_len, d_off = i32(lv.length[arr]), i64(lv.arena_off[arr])
    arena_d = torch.empty(lv.arena_bytes, dtype=torch.uint8, device="cuda")
    fill_payload(arena_d, i64(lv.arena_off), i32(lv.length), lv.payload_seed)
    # the device fill follows the host definition (sampled records)
    rng = np.random.default_rng(3)
    for c in rng.choice(np.flatnonzero(lv.length), 200, replace=False):
        o, n = int(lv.arena_off[c]), int(lv.length[c])
        assert arena_d[o:o + n].cpu().numpy().tobytes() == record_bytes(lv.payload_seed, int(c), n)

    o = OracleCtx()
    ctx = ro.ro_ctx_create(0, stream, 1)
    # expand
    ex = o.expand(lv.counts)
    d_offsets = torch.empty(P + 1, dtype=torch.int64, device="cuda")
    d_cp = torch.empty(N, dtype=torch.int32, device="cuda")
    d_co = torch.empty(N, dtype=torch.int32, device="cuda")
    st, n, ne, xid = ro.ro_expand(ctx, -1, d_counts, P, None, d_offsets, d_cp, d_co, N, None)
    assert (st, n, ne) == (0, N, 0)
    assert np.array_equal(host(d_offsets, np.uint64), ex["offsets"])
    assert np.array_equal(host(d_cp, np.uint32), ex["child_parent"])
    assert np.array_equal(host(d_co, np.uint32), ex["child_ordinal"])
    # one readiness wave, all children, flush
    br = o.batch_ready(ex["xid"], 0, None, B, flush=True)
    d_b = torch.empty(N + B, dtype=torch.int32, device="cuda")
    st, nb, nbt = ro.ro_batch_ready(ctx, xid, 0, None, 0, B, 1, d_b, N + B)
    assert (st, nb, nbt) == (0, br["n_batched"], br["n_batches"])
    assert np.array_equal(host(d_b, np.uint32, nb), br["batched"])

    # 256 arrival waves: commit + assemble of the parents each completes
    out_d = torch.empty(lv.arena_bytes + 64, dtype=torch.uint8, device="cuda")
    d_status = torch.empty(P, dtype=torch.uint8, device="cuda")
    d_oo = torch.empty(P + 1, dtype=torch.int64, device="cuda")
    d_ol = torch.empty(P, dtype=torch.int32, device="cuda")
    d_cur = torch.zeros(1, dtype=torch.int64, device="cuda")
    d_code = torch.empty(N, dtype=torch.uint8, device="cuda")
    d_done = torch.empty(P, dtype=torch.int32, device="cuda")
    ledger = []   # (done parents, out_off) per wave, for the byte check
    for w in range(W):
        s, e = int(lv.wave_bounds[w]), int(lv.wave_bounds[w + 1])
        ch, stt, ln, of = lv.reports(lv.wave(w))
        cm = o.gather_commit(ex["xid"], ch, stt, ln, of, arena_bytes=lv.arena_bytes)
        st, nd = ro.ro_gather_commit(ctx, xid, e - s, None, d_child[s:e], d_state[s:e], d_len[s:e],
                                     d_off[s:e], None, lv.arena_bytes, d_code, d_done, P, None)
        assert (st, nd) == (0, cm["n_done"])
        assert np.array_equal(host(d_code, np.uint8, e - s), cm["code"])
        assert np.array_equal(host(d_done, np.uint32, nd), cm["done"])
        cur0 = int(d_cur.item())
        a = o.assemble(ex["xid"], None, parents=None, n_parents=max(nd, 1), cursor=cur0)
        st, ob = ro.ro_assemble(ctx, xid, arena_d, lv.arena_bytes, None, max(nd, 1), None, d_status,
                                d_oo, d_ol, out_d, out_d.numel(), d_cur, None)
        assert (st, ob) == (0, a["out_bytes"])
        assert np.array_equal(host(d_status, np.uint8, nd), a["parent_status"])
        assert np.array_equal(host(d_oo, np.uint64, nd + 1), a["out_off"])
        assert np.array_equal(host(d_ol, np.uint32, nd), a["out_len"])
        ledger.append(cm["done"])
    total = int(d_cur.item())
    assert ro.ro_ctx_sync(ctx) == 0
    gs = ro.ro_ctx_stats(ctx)
    gs.pop("status")
    assert gs == o.stats()

    # every assembled byte: the oracle assembles the same parent sequence
    # from a host copy of the arena
    arena_h = host_arena(lv)
    o2 = OracleCtx()
    x2 = o2.expand(lv.counts)["xid"]
    o2.batch_ready(x2, 0, None, B, flush=True)
    o2.gather_commit(x2, lv.arrival, lv.state[arr], lv.length[arr], lv.arena_off[arr],
                     arena_bytes=lv.arena_bytes)
    order = np.concatenate(ledger).astype(np.uint32)
    assert order.size == P
    ref = o2.assemble(x2, arena_h, parents=order, out_cap=total, want_len=False)
    assert ref["out_bytes"] == total
    del arena_h
    got = out_d[:total].cpu().numpy()
    assert np.array_equal(got, ref["out"][:total]), "assembled bytes differ"
    del ref

    # the benchmark's launch configuration: the wave loop captured in a CUDA
    # graph and replayed after a fresh expand gives the same bytes
    eager = out_d[:total].clone()
    ro.ro_ctx_reset(ctx)
    xid = ro.ro_expand(ctx, -1, d_counts, P, None, d_offsets, d_cp, d_co, N, None)[3]
    L = ro.load()
    g_stream = torch.cuda.Stream()
    ro.ro_ctx_destroy(ctx)
    ctx = ro.ro_ctx_create(0, g_stream, 1)
    with torch.cuda.stream(g_stream):
        xid = ro.ro_expand(ctx, -1, d_counts, P, None, d_offsets, d_cp, d_co, N, None)[3]
        bounds = lv.wave_bounds

        def wave_loop():
            bad = L.ro_batch_ready(ctx, xid, 0, None, 0, B, 1, d_b.data_ptr(), N + B, None, None, None)
            d_cur.zero_()
            for w in range(W):
                s, e = int(bounds[w]), int(bounds[w + 1])
                bad |= L.ro_gather_commit(ctx, xid, e - s, None, d_child.data_ptr() + 4 * s,
                                          d_state.data_ptr() + s, d_len.data_ptr() + 4 * s,
                                          d_off.data_ptr() + 8 * s, None, lv.arena_bytes, None, None,
                                          0, None, None)
                bad |= L.ro_assemble(ctx, xid, arena_d.data_ptr(), lv.arena_bytes, None, P, None,
                                     d_status.data_ptr(), d_oo.data_ptr(), d_ol.data_ptr(),
                                     out_d.data_ptr(), out_d.numel(), d_cur.data_ptr(), None, None)
            assert bad == 0
        wave_loop()            # sizes every buffer
        torch.cuda.synchronize()
        ro.ro_ctx_reset(ctx)
        xid = ro.ro_expand(ctx, -1, d_counts, P, None, d_offsets, d_cp, d_co, N, None)[3]
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph, stream=g_stream):
            wave_loop()
        for _ in range(2):
            out_d[:total].zero_()
            ro.ro_ctx_reset(ctx)
            assert ro.ro_expand(ctx, -1, d_counts, P, None, d_offsets, d_cp, d_co, N, None)[0] == 0
            graph.replay()
            torch.cuda.synchronize()
            assert int(d_cur.item()) == total
            assert torch.equal(out_d[:total], eager)
    assert ro.ro_ctx_sync(ctx) == 0
    ro.ro_ctx_destroy(ctx)


def _arena_dev(a):
    from tests.lockstep import dev
    return dev(a if a.size else np.zeros(1, np.uint8), np.uint8)


def test_skew_full_size():
    """The extreme-skew configuration at full size: 10,000,000 parents, 1,000
    of them with 100,000 children (109,999,000 children of 32 bytes), one
    arrival wave, batch 256: lineage arrays, reserved batches, every
    verdict, the completed list, statuses, offsets, lengths and all 3.5 GB
    of assembled bytes equal the oracle's."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from tests.lockstep import Lockstep
    from tests.pipeline import host_arena
    from workload import skew
    lv = skew().top
    assert lv.n_children == 109_999_000
    a = host_arena(lv)
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        ls.batch_ready(x, 0, None, lv.batch_size, flush=True)
        ch, st, ln, of = lv.reports(lv.wave(0))
        cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
        assert cm["n_done"] == lv.n_parents
        r = ls.assemble(x, a, _arena_dev(a), parents=None, n_parents=cm["n_done"])
        assert r["out_bytes"] == lv.arena_bytes   # no failures: every byte is assembled
        ls.check_stats()


def test_video_nested_full_size():
    """The video -> clip -> frame configuration at full size: 100,000 videos,
    their clips and frames (512-byte records), frames gathered into clips,
    the clips' assembled results committed as the reports of the videos'
    expansion and gathered again; every output of both levels equal to the
    oracle's."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from tests.lockstep import Lockstep
    from tests.pipeline import host_arena
    from workload import video
    top, leaf = video().levels
    assert top.n_parents == 100_000
    a = host_arena(leaf)
    with Lockstep() as ls:
        x0 = ls.expand(top.counts)["xid"]
        ls.batch_ready(x0, 0, None, top.batch_size, flush=True)
        x1 = ls.expand(leaf.counts, parent_xid=x0)["xid"]
        ls.batch_ready(x1, 0, None, leaf.batch_size, flush=True)
        ch, st, ln, of = leaf.reports(leaf.wave(0))
        cm1 = ls.commit(x1, ch, st, ln, of, arena_bytes=leaf.arena_bytes)
        assert cm1["n_done"] == leaf.n_parents
        a1 = ls.assemble(x1, a, _arena_dev(a), parents=None, n_parents=cm1["n_done"])
        del a
        r1 = a1["r"]
        level1 = a1["out"][:a1["out_bytes"]].cpu().numpy()
        cm0 = ls.commit(x0, cm1["done"], r1["parent_status"], r1["out_len"], r1["out_off"][:-1],
                        arena_bytes=a1["out_bytes"])
        assert cm0["n_done"] == top.n_parents
        ls.assemble(x0, level1, _arena_dev(level1), parents=None, n_parents=cm0["n_done"])
        ls.check_stats()


@pytest.mark.parametrize("B,admissions", [(32, "calls"), (256, "calls"), (2048, "calls"),
                                          (256, "call-streams")])
def test_streaming_full_size(B, admissions):
    """The streaming configuration at full size, at each batch size the
    benchmark sweeps, with the bench's default streams (assembly planning and
    copies on streams of their own) and its default admission (every Call's
    in one ro_batch_ready_calls per wave), and at B = 256 also with each
    Call's admissions on a stream of its own: four Calls, 50,000,050
    children of 1 KB, 1,000 readiness waves; per
    wave every Call admits the wave's ready children and reserves whole
    batches (the last wave flushes), the reserved children's results are
    committed in their key order and the completed parents assembled.  Every
    Call's reservation, every verdict, completed list, status, offset, length
    and every wave's assembled bytes equal the oracle's (compared wave by
    wave, so host memory stays bounded)."""
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    from tests.lockstep import Lockstep
    from tests.pipeline import host_arena
    from workload import streaming
    lv = streaming(batch_size=B).top
    assert lv.n_children == 50_000_050
    a = host_arena(lv)
    ad = _arena_dev(a)
    total = 0
    with Lockstep(n_calls=4, streams=True, call_streams=admissions == "call-streams") as ls:
        x = ls.expand(lv.counts, parent_call=lv.parent_call)["xid"]
        n_ready = lv.ready_bounds.size - 1
        for w in range(n_ready):
            cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
            last = w == n_ready - 1
            if admissions == "calls":
                reserved = ls.batch_ready_calls(x, [0, 1, 2, 3], cand, B, flush=last)
            else:
                reserved = [ls.batch_ready(x, c, cand, B, flush=last)["batched"] for c in range(4)]
            got = np.concatenate(reserved)
            got = got[np.argsort(lv.key[got], kind="stable")]
            ch, st, ln, of = lv.reports(got)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            r = ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
            total += r["out_bytes"]
        ls.check_stats()
        assert ls.o.stats()["ready_bad_candidates"] == 0
    assert total > 0
