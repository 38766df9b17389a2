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
