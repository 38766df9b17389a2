"""Bounded device-side waits end with RO_E_TIMEOUT instead of hanging.

ro_ctx_selftest_timeout runs one wait that nothing releases (a decoupled
look-back whose predecessor tile never publishes; a grid barrier missing an
arrival), on scratch state of its own.  The call must come back with
RO_E_TIMEOUT within seconds, and the same context must then run a whole
document->page pass exactly as the oracle does (the time-out left no state
behind)."""
import time

import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


@pytest.mark.parametrize("kind", [0, 1])
def test_wait_gives_up_and_the_context_stays_usable(kind):
    import paper_2609_18703_gb300 as ro
    from tests.lockstep import Lockstep
    from tests.pipeline import host_arena
    from tests.test_gpu_parity import _arena_dev, run_level
    from workload import docpage
    with Lockstep() as ls:
        t0 = time.perf_counter()
        st = ro.ro_ctx_selftest_timeout(ls.ctx, kind)
        dt = time.perf_counter() - t0
        assert st == ro.RO_E_TIMEOUT, (st, ro.ro_last_error(ls.ctx))
        assert dt < 30.0
        assert ro.ro_ctx_sync(ls.ctx) == ro.RO_OK   # reported once
        lv = docpage(parents=600, waves=4).top
        a = host_arena(lv)
        run_level(ls, lv, a, _arena_dev(a))
        ls.check_stats()


def test_bad_kind_is_refused():
    import paper_2609_18703_gb300 as ro
    ctx = ro.ro_ctx_create(0, torch.cuda.current_stream(), 1)
    try:
        assert ro.ro_ctx_selftest_timeout(ctx, 7) == ro.RO_E_INVAL
    finally:
        ro.ro_ctx_destroy(ctx)
