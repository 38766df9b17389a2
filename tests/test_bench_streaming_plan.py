"""The streaming benchmark derives each readiness wave's reports on the host
(bench.streaming_plan): every Call's FIFO queue is its children in readiness
order and a wave reserves the whole batches its queue then holds (all on the
last wave).  Checked wave by wave against the oracle's own reservations."""
import numpy as np
import pytest

from bench import streaming_plan
from oracle import OracleCtx
from workload import streaming


@pytest.mark.parametrize("B", [32, 256, 2048])
def test_plan_matches_oracle_reservations(B):
    lv = streaming(total_children=60000, batch_size=B, ready_waves=25).top
    plan = streaming_plan(lv, B)
    assert sum(p.size for p in plan) == lv.n_children
    o = OracleCtx(4)
    x = o.expand(lv.counts, parent_call=lv.parent_call)["xid"]
    W = lv.ready_bounds.size - 1
    for w in range(W):
        cand = lv.readiness[lv.ready_bounds[w]:lv.ready_bounds[w + 1]]
        got = np.concatenate([o.batch_ready(x, c, cand, B, flush=(w == W - 1))["batched"]
                              for c in range(4)])
        got = got[np.argsort(lv.key[got], kind="stable")]
        assert np.array_equal(got, plan[w]), w
        o.gather_commit(x, *lv.reports(got), arena_bytes=lv.arena_bytes)
    o.close()


def test_copy_traffic_only_for_the_captured_workload_and_run():
    """The bench's roofline `traffic` is an ncu figure for one workload at one
    size and the default run options; any other run reports it as null."""
    import bench
    full = "document->page: 1000000 parents, 16399843 children, 256 arrival waves, batch 256"
    t, src = bench.measured_traffic(full, "asm_copy")
    captured = bench.TRAFFIC[(full, "asm_copy")][1] == bench.source_sha16("asm_copy")
    assert (t is not None and bool(src)) == captured   # null once the kernel's source changed
    assert bench.measured_traffic(full, "asm_copy", default_run=False) == (None, None)
    assert bench.measured_traffic(full, "commit_scatter") == (None, None)
    small = "document->page: 60000 parents, 979486 children, 16 arrival waves, batch 256"
    assert bench.measured_traffic(small, "asm_copy") == (None, None)
