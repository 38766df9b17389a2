"""Parent-bound reservation on the GPU (Section 4.3) against the oracle:
every batch, batch boundary, count, later queue state (through the calls
that follow) and counter is compared exactly.

Covers the hand-worked example, random sequences mixing both policies over
windows of several tiles with 1-, 2- and 3-pass sorts by parent, several
Calls, recovery groups and GroupFailure drops, refused calls (capacity of
either output), the degenerate cases (empty window, one parent, B = 1,
B larger than any parent) and the 1,000,000-parent document->page window
that the benchmark reserves.
"""
import json
import os

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


from tests.lockstep import Lockstep  # noqa: E402
from workload import PRESENT, docpage  # noqa: E402

GF = 5
NONE = np.zeros(1, np.uint32)[:0]


def _names(parents):
    ids, base = {}, 0
    for name, m in parents.items():
        for j in range(m):
            ids[f"{name}{j}"] = base + j
        base += m
    return ids


def _rep(children, states=None, ln=8):
    children = np.asarray(children, np.uint32)
    st = np.full(children.size, PRESENT, np.uint8) if states is None else np.asarray(states, np.uint8)
    return children, st, np.full(children.size, ln, np.uint32), children.astype(np.uint64) * ln


def test_worked_example_on_gpu(golden_dir):
    g = json.load(open(os.path.join(golden_dir, "parent_bound_reserve.json")))
    ids = _names(g["parents"])
    queue = np.array([ids[n] for n in g["queue"]], np.uint32)
    for case in g["cases"]:
        with Lockstep() as ls:
            x = ls.expand(np.array(list(g["parents"].values()), np.uint32))["xid"]
            r = ls.batch_ready_parent(x, 0, queue, case["B"], flush=case["flush"])
            assert r["n_batches"] == len(case["batches"])
            left = ls.batch_ready(x, 0, NONE, 1, flush=True)
            assert left["n_batched"] == len(case["left"])
            ls.check_stats()


@pytest.mark.parametrize("P,maxc,seed", [(40, 9, 0), (300, 30, 1), (3000, 12, 2),
                                         (70000, 6, 3), (70000, 6, 4)])
def test_random_sequences(P, maxc, seed):
    """Windows of several tiles; P > 256 and P > 65536 need 2 and 3 sort passes."""
    rng = np.random.default_rng(7000 + seed)
    counts = rng.integers(0, maxc + 1, P).astype(np.uint32)
    N = int(counts.sum())
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        perm = rng.permutation(N).astype(np.uint32)
        parts = np.array_split(perm, 5)
        for k, part in enumerate(parts):
            # duplicates and ids out of range among the candidates
            cand = np.concatenate([part, part[: part.size // 7], [N + 3, N]]).astype(np.uint32)
            cand = cand[rng.permutation(cand.size)]
            B = int(rng.choice([1, 2, 3, 7, 64, 256]))
            if k == 2:   # an elastic reservation in between shares the queue
                ls.batch_ready(x, 0, cand, B, flush=False)
            else:
                ls.batch_ready_parent(x, 0, cand, B, flush=bool(k % 2))
        ls.batch_ready_parent(x, 0, NONE, int(rng.choice([5, 100])), flush=False)
        ls.batch_ready_parent(x, 0, NONE, 3, flush=True)
        ls.check_stats()


def test_several_calls():
    rng = np.random.default_rng(11)
    P = 5000
    counts = rng.integers(0, 10, P).astype(np.uint32)
    calls = rng.integers(0, 3, P).astype(np.uint8)
    N = int(counts.sum())
    with Lockstep(n_calls=3) as ls:
        x = ls.expand(counts, parent_call=calls)["xid"]
        cand = rng.permutation(N).astype(np.uint32)
        for c in range(3):
            ls.batch_ready_parent(x, c, cand[: N // 2], 4)
        for c in range(3):
            ls.batch_ready_parent(x, c, cand[N // 2:], 4, flush=(c != 1))
        ls.batch_ready(x, 1, NONE, 1, flush=True)
        ls.check_stats()


def test_recovery_groups_and_group_failure():
    rng = np.random.default_rng(12)
    P = 4000
    counts = rng.integers(1, 12, P).astype(np.uint32)
    N = int(counts.sum())
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        cand = rng.permutation(N).astype(np.uint32)
        r = ls.batch_ready_parent(x, 0, cand[: N // 2], 4)
        b, off = r["batched"], r["batch_off"]
        # every third batch fails and is retried, in a scrambled batch order
        failed = [b[off[k]:off[k + 1]] for k in range(0, r["n_batches"], 3)]
        for grp in failed[::-1]:
            ls.retry(x, 0, grp)
        # GroupFailure from the first child of some committed batches' parents
        ok = [b[off[k]] for k in range(1, r["n_batches"], 3)][:200]
        ls.commit(x, *_rep(ok, [GF] * len(ok)))
        ls.batch_ready_parent(x, 0, cand[N // 2:], 4)
        ls.batch_ready_parent(x, 0, NONE, 4, flush=True)
        ls.check_stats()


def test_refused_calls_change_nothing_but_the_prelude():
    rng = np.random.default_rng(13)
    counts = rng.integers(0, 20, 2000).astype(np.uint32)
    N = int(counts.sum())
    cand = rng.permutation(N).astype(np.uint32)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        ls.batch_ready_parent(x, 0, cand[:1000], 8)
        ls.batch_ready_parent(x, 0, cand[1000:], 8, flush=True, cap=N // 3)     # batched too small
        ls.batch_ready_parent(x, 0, cand[1000:], 8, flush=True, off_cap=5)      # boundaries too small
        ls.batch_ready_parent(x, 0, cand[1000:], 8, flush=True, off_cap=0)
        ls.batch_ready_parent(x, 0, cand[1000:], 8, flush=True)                 # fits
        ls.check_stats()


def test_degenerate_cases():
    with Lockstep() as ls:
        x = ls.expand(np.array([0, 0, 0], np.uint32))["xid"]          # no children at all
        ls.batch_ready_parent(x, 0, NONE, 4, flush=True)
        y = ls.expand(np.array([5000], np.uint32))["xid"]             # one parent: 0 sort passes
        ls.batch_ready_parent(y, 0, np.arange(4999, -1, -1, dtype=np.uint32)[:3001], 256)
        ls.batch_ready_parent(y, 0, None, 256, flush=True)
        z = ls.expand(np.arange(1, 600, dtype=np.uint32) % 7)["xid"]
        ls.batch_ready_parent(z, 0, None, 1)                          # B = 1
        w = ls.expand(np.arange(1, 600, dtype=np.uint32) % 7)["xid"]
        ls.batch_ready_parent(w, 0, None, 1 << 31)                    # no chunk is whole
        ls.batch_ready_parent(w, 0, None, 1 << 31, flush=True)
        ls.check_stats()


def test_document_page_window_full_size():
    """The benchmark's reservation: 1,000,000 parents (about 16.4M pages)
    admitted in arrival order, batches of 256 siblings, flush; whole
    arrays compared."""
    lv = docpage(parents=1_000_000, waves=256).top
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        r = ls.batch_ready_parent(x, 0, lv.arrival.astype(np.uint32), 256, flush=True)
        assert r["n_batched"] == lv.n_children
        ls.check_stats()
