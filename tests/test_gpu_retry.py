"""Retry at a new generation and recovery queues on the GPU (Section 4.4;
Eq. 2's IN-FLIGHT -> READY edge; Section 4.3) against the oracle: retried
counts, every reserved batch (recovery groups first), every verdict
(stale reports of failed attempts), every completed list, assembled byte
and counter compared exactly."""
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
from workload import PRESENT, docpage, tiny  # noqa: E402

GF = 5


def _rep(children, states=None, ln=8):
    children = np.asarray(children, np.uint32)
    st = np.full(children.size, PRESENT, np.uint8) if states is None else np.asarray(states, np.uint8)
    return children, st, np.full(children.size, ln, np.uint32), children.astype(np.uint64) * ln


def test_retry_sequence_on_gpu():
    arena = np.arange(1024, dtype=np.uint8)
    ad = dev(arena, np.uint8)
    with Lockstep(n_calls=2) as ls:
        x = ls.expand(np.array([4, 4, 3, 3], np.uint32), parent_call=np.array([0, 0, 1, 1], np.uint8))["xid"]
        b1 = ls.batch_ready(x, 0, [0, 1, 4, 5], 4)["batched"]
        ls.batch_ready(x, 0, [2, 3, 6, 7], 8)
        ls.batch_ready(x, 1, [8, 11, 9], 2, flush=True)
        ls.retry(x, 0, list(b1) + [1, 9, 2, 500])          # duplicate, other Call, READY, bad id
        ls.commit(x, *_rep([0, 8]), arena_bytes=arena.size)  # 0: READY now; 8: Call 1, fine
        ls.batch_ready(x, 0, None, 4, flush=True)
        ls.retry(x, 1, [11])
        ls.commit(x, *_rep([0, 0, 1, 4, 5, 2, 3, 6, 7, 9, 11]),
                  gen=np.array([0, 1, 1, 1, 1, 0, 0, 0, 0, 0, 1], np.uint32), arena_bytes=arena.size)
        ls.batch_ready(x, 1, None, 2, flush=True)
        ls.commit(x, *_rep([11, 10]), gen=np.array([1, 0], np.uint32), arena_bytes=arena.size)
        ls.assemble(x, arena, ad, parents=[0, 1, 2, 3], n_parents=4)
        ls.check_stats()


@pytest.mark.parametrize("seed", range(3))
def test_random_failed_attempts_with_late_stale_reports(seed):
    lv = tiny().top if seed < 2 else docpage(parents=3000, waves=1).top
    a = host_arena(lv)
    ad = dev(a if a.size else np.zeros(1, np.uint8), np.uint8)
    rng = np.random.default_rng(900 + seed)
    gen = np.zeros(lv.n_children, np.uint32)
    order = rng.permutation(lv.n_children).astype(np.uint32)
    waves = np.array_split(order, 6)
    late = []
    poisoned = set()
    with Lockstep() as ls:
        x = ls.expand(lv.counts)["xid"]
        for w in range(len(waves) + 25):
            cand = waves[w] if w < len(waves) else np.zeros(0, np.uint32)
            b = ls.batch_ready(x, 0, cand, 32, flush=True)["batched"]
            if b.size == 0 and w >= len(waves) and not late:
                break
            reps = []
            for batch in np.array_split(b, max(1, b.size // 32)):
                if batch.size and rng.random() < 0.3:
                    late.append(batch.copy())
                    ls.retry(x, 0, batch[rng.permutation(batch.size)])
                    gen[batch] += 1
                else:
                    reps.append(batch)
            ch = np.concatenate(reps).astype(np.uint32) if reps else np.zeros(0, np.uint32)
            st = lv.state[ch].copy()
            if seed == 1 and ch.size and rng.random() < 0.3:   # now and then a GroupFailure
                st[0] = GF
            g = gen[ch]
            if late and rng.random() < 0.5:
                stale = late.pop(0)
                ch = np.concatenate([stale, ch]).astype(np.uint32)
                st = np.concatenate([lv.state[stale], st])
                g = np.concatenate([np.maximum(gen[stale], 1) - 1, g])
            cm = ls.commit(x, ch, st, lv.length[ch], lv.arena_off[ch], gen=g.astype(np.uint32),
                           arena_bytes=lv.arena_bytes)
            ls.assemble(x, a, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()
        assert ls.o.stats()["retried"] > 0
