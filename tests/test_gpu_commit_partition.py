"""ro_gather_commit groups the reports of a large call by child range before
the fence (k_partition.cu; calls of at least 2^24 reports by default, such
as the extreme-skew configuration's 110M).  With RO_COMMIT_PARTITION_MIN=1 at
context creation every call takes that path; here the commit scenarios run
again on it, each against the oracle: the generation fence and every verdict
code (written back in the caller's order), a Grain reported several times in
one call (the lowest index wins), a device-side report count, GroupFailures
ordered among their siblings' reports, heavy parents with repeats and
barriers, retried attempts with late stale reports, and calls of ~400,000
reports over 1.2M children whose 256 ranges each hold many parents, with
repeats, ids past the expansion and GroupFailures."""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(autouse=True)
def _grouped(monkeypatch):
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()
    monkeypatch.setenv("RO_COMMIT_PARTITION_MIN", "1")


def test_grouped_fence_and_codes():
    from tests import test_gpu_parity
    test_gpu_parity.test_generation_fence_and_codes()


@pytest.mark.parametrize("seed", range(2))
def test_grouped_duplicates_first_in_array_order(seed):
    from tests import test_gpu_parity
    test_gpu_parity.test_duplicate_reports_first_in_array_order_wins(seed)


@pytest.mark.parametrize("device_count,streams", [(True, False), (False, True)])
def test_grouped_pipeline_docpage_small(device_count, streams):
    from tests import test_gpu_parity
    test_gpu_parity.test_pipeline_docpage_small(device_count, streams)


def test_grouped_pipeline_skew_small():
    from tests import test_gpu_parity
    test_gpu_parity.test_pipeline_skew_small()


def test_grouped_group_failure_ordering():
    from tests import test_gpu_group_failure
    test_gpu_group_failure.test_group_failure_ordering_within_a_call()


def test_grouped_random_group_failures():
    from tests import test_gpu_group_failure
    test_gpu_group_failure.test_random_group_failures_many_calls(0)


def test_grouped_heavy_parents_with_barriers():
    from tests import test_gpu_group_failure
    test_gpu_group_failure.test_heavy_parents_with_repeats_failures_and_barriers(0)


def test_grouped_retried_attempts():
    from tests import test_gpu_retry
    test_gpu_retry.test_random_failed_attempts_with_late_stale_reports(0)


def test_grouped_calls_over_many_ranges():
    from tests.lockstep import Lockstep, dev
    from workload import DROPPED, FAILED, PRESENT, SUPPRESSED
    GF = 5
    rng = np.random.default_rng(9100)
    counts = rng.integers(0, 8, 300_000).astype(np.uint32)
    heavy = rng.choice(counts.size, 4, replace=False)
    counts[heavy] = [5000, 20000, 4096, 70000]
    N = int(counts.sum())
    assert N > 256 * 4096   # every range edge distinct
    arena = rng.integers(0, 256, N * 4 + 64).astype(np.uint8)
    with Lockstep() as ls:
        x = ls.expand(counts)["xid"]
        ad = dev(arena, np.uint8)
        ls.batch_ready(x, 0, None, 256, flush=True)
        perm = rng.permutation(N).astype(np.uint32)
        for w, chunk in enumerate(np.array_split(perm, 3)):
            rep = rng.choice(chunk, size=chunk.size // 16)
            past = rng.integers(N, N + 1000, 50)
            ch = np.concatenate([chunk, rep, past])
            ch = ch[rng.permutation(ch.size)].astype(np.uint32)
            st = rng.choice([PRESENT] * 60 + [DROPPED, FAILED, SUPPRESSED, GF], ch.size).astype(np.uint8)
            ln = rng.integers(0, 5, ch.size).astype(np.uint32)
            of = ch.astype(np.uint64) * 4
            cm = ls.commit(x, ch, st, ln, of, arena_bytes=arena.size, device_count=(w == 1))
            ls.assemble(x, arena, ad, parents=None, n_parents=max(cm["n_done"], 1))
        ls.check_stats()
