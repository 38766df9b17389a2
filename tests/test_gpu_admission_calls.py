"""ro_batch_ready_calls (Section 4.3): the admissions of several Calls from
one candidate list in one launch equal, Call by Call, the oracle's
admissions taken one after another (each Call admits only its own children
into its own queue): every Call's reserved batches and count, then the
commit of the reserved children's results and the assembly, wave by wave.
Covered: the streaming configuration's waves (no repeated candidates: one
grid barrier), lists with repeats and ids past the expansion (the claims'
second barrier), a refused Call beside admitted ones, and a list too long
for one cooperative grid (one admission after another)."""
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
from workload import streaming  # noqa: E402


def _admit_all(ls, x, calls, cand, B, flush, caps):
    return ls.batch_ready_calls(x, calls, cand, B, flush, caps)


@pytest.mark.parametrize("B", [32, 2048])
def test_streaming_waves_admitted_in_one_launch(B):
    lv = streaming(total_children=80000, batch_size=B, ready_waves=20).top
    a = host_arena(lv)
    ad = dev(a if a.size else np.zeros(1, np.uint8), np.uint8)
    with Lockstep(n_calls=4) as ls:
        x = ls.expand(lv.counts, parent_call=lv.parent_call)["xid"]
        N = ls.N[x]
        n_ready = lv.ready_bounds.size - 1
        for w in range(n_ready):
            cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
            got = _admit_all(ls, x, [0, 1, 2, 3], cand, B, w == n_ready - 1, [N + B] * 4)
            got = np.concatenate(got)
            got = got[np.argsort(lv.key[got], kind="stable")]
            ch, st, ln, of = lv.reports(got)
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=lv.arena_bytes)
            ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()


@pytest.mark.parametrize("seed", range(3))
def test_repeats_foreign_ids_and_a_refused_call(seed):
    rng = np.random.default_rng(9100 + seed)
    P = 3000
    counts = rng.integers(0, 9, P).astype(np.uint32)
    calls = (np.arange(P) % 3).astype(np.uint8)
    with Lockstep(n_calls=3) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        N = ls.N[x]
        B = int(rng.choice([1, 16, 64]))
        for w in range(5):
            m = int(rng.integers(0, 9000))
            cand = rng.integers(0, N + 40, m).astype(np.uint32)   # repeats and ids past N
            caps = [N + B] * 3
            if w == 2:
                caps[1] = 3   # Call 1 cannot take its batches: refused alone
            order = [int(c) for c in rng.permutation(3)]
            _admit_all(ls, x, order, cand, B, w == 4, [caps[c] for c in order])
        for c in range(3):
            ls.batch_ready(x, c, None, B, flush=True)
        ls.check_stats()


def test_list_longer_than_one_grid():
    """~1.4M candidates for 4 Calls: more CTAs than the device holds at
    once, so the Calls are admitted one after another."""
    rng = np.random.default_rng(77)
    P = 40000
    counts = rng.integers(1, 12, P).astype(np.uint32)
    calls = (np.arange(P) % 4).astype(np.uint8)
    with Lockstep(n_calls=4) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        N = ls.N[x]
        cand = np.concatenate([rng.permutation(N), rng.integers(0, N, 1_200_000)]).astype(np.uint32)
        _admit_all(ls, x, [3, 1, 0, 2], cand, 256, False, [N + 256] * 4)
        _admit_all(ls, x, [0, 1, 2, 3], cand[:5000], 256, True, [N + 256] * 4)
        ls.check_stats()


def test_bad_arguments_change_nothing():
    with Lockstep(n_calls=2) as ls:
        x = ls.expand(np.array([3, 4], np.uint32), parent_call=np.array([0, 1], np.uint8))["xid"]
        d_cand = dev(np.arange(7, dtype=np.uint32), np.uint32)
        d_b = [empty(16, np.uint32), empty(16, np.uint32)]
        assert ro.ro_batch_ready_calls(ls.ctx, x, [0, 0], d_cand, 7, 4, 1, d_b, [16, 16]) == ro.RO_E_INVAL
        assert ro.ro_batch_ready_calls(ls.ctx, x, [0, 2], d_cand, 7, 4, 1, d_b, [16, 16]) == ro.RO_E_INVAL
        assert ro.ro_batch_ready_calls(ls.ctx, x, [], d_cand, 7, 4, 1, [], []) == ro.RO_E_INVAL
        assert ro.ro_batch_ready_calls(ls.ctx, x, [0, 1], d_cand, 7, 0, 1, d_b, [16, 16]) == ro.RO_E_INVAL
        for c in range(2):
            ls.batch_ready(x, c, np.arange(7, dtype=np.uint32), 4, flush=True)
        ls.check_stats()


def test_empty_lists_flush_exact_and_short_capacities():
    """Edge cases of one launch over several Calls: an empty candidate list
    (one id past the expansion: only the windows earlier calls left move,
    on flush), a capacity exactly
    equal to a Call's reservation (admitted) and one entry short of it
    (refused, that Call alone), and a single Call through the same entry
    point; each against the oracle's admissions in turn.  The exact sizes
    come from a second context with the same history."""
    rng = np.random.default_rng(515)
    P = 2500
    counts = rng.integers(1, 7, P).astype(np.uint32)
    calls = (np.arange(P) % 3).astype(np.uint8)
    B = 16

    def history(ls):
        x = ls.expand(counts, parent_call=calls)["xid"]
        N = ls.N[x]
        perm = np.random.default_rng(516).permutation(N).astype(np.uint32)
        _admit_all(ls, x, [0, 1, 2], perm[:3001], B, False, [N + B] * 3)   # partial batches stay
        none = np.array([N + 5], np.uint32)   # one id past the expansion: admits nothing
        _admit_all(ls, x, [2, 0, 1], none, B, False, [N + B] * 3)       # nothing moves
        return x, N, perm

    with Lockstep(n_calls=3) as probe:
        x, N, perm = history(probe)
        sizes = [b.size for b in _admit_all(probe, x, [0, 1, 2], perm[3001:6001], B, False, [N + B] * 3)]
    assert sizes[0] > 0 and sizes[2] > 0
    with Lockstep(n_calls=3) as ls:
        x, N, perm = history(ls)
        got = _admit_all(ls, x, [0, 1, 2], perm[3001:6001], B, False, [sizes[0], N + B, sizes[2] - 1])
        assert got[0] is not None and got[0].size == sizes[0]
        assert got[1] is not None and got[2] is None   # refused alone
        _admit_all(ls, x, [1, 2, 0], np.array([N + 5], np.uint32), B, True, [N + B] * 3)   # the windows flush
        _admit_all(ls, x, [1], perm[6001:], B, True, [N + B])           # one Call
        for c in range(3):
            ls.batch_ready(x, c, None, B, flush=True)
        ls.check_stats()
