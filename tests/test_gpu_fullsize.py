"""The 1,000,000-document configuration at full size (16.4M children,
38.8 GB arena, 256 arrival waves, batch 256), in the launch configuration
bench.py times, against the oracle on every output: lineage arrays, the
reserved batches, every wave's verdicts, completed-parent list, statuses,
offsets, lengths and all ~12 GB of assembled bytes.  The CUDA-graph replay of
the wave loop (what the benchmark runs) is then checked byte for byte
against the eager run.  Needs ~70 GB of host memory and ~60 GB on the GPU."""
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
