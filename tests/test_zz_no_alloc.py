"""ro_expand_noalloc — the allocation-free expansion — gives exactly what
ro_expand gives, through the C ABI, on two calls in a row.

It exists for callers that cannot call cudaMalloc (a memory budget owned by
another allocator, paths that must not synchronise the device, embedders
that forbid allocation after start-up); its scratch is a fixed static device
array, so this file checks that consecutive calls sharing that array stay
exact.  Named to be collected last."""
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


def _ctx_expand(ro, counts_d, P, cap):
    ctx = ro.ro_ctx_create(0, torch.cuda.current_stream(), 1)
    off = torch.empty(P + 1, dtype=torch.int64, device="cuda")
    cp = torch.empty(max(cap, 1), dtype=torch.int32, device="cuda")
    co = torch.empty(max(cap, 1), dtype=torch.int32, device="cuda")
    emp = torch.empty(max(P, 1), dtype=torch.int32, device="cuda")
    st, n, ne, _ = ro.ro_expand(ctx, -1, counts_d, P, None, off, cp, co, cap, emp)
    ro.ro_ctx_destroy(ctx)
    assert st == 0
    return n, ne, off, cp[:n], co[:n], emp[:ne]


@pytest.mark.parametrize("case", ["docpage_like", "skewed_with_empties"])
def test_noalloc_matches_ro_expand_twice(case):
    import paper_2609_18703_gb300 as ro
    rng = np.random.default_rng(17)
    if case == "docpage_like":
        counts = np.clip(np.rint(rng.lognormal(2.3, 1.0, 300_000)), 1, 2000).astype(np.uint32)
    else:
        counts = rng.integers(0, 4, 70_000).astype(np.uint32)
        counts[rng.choice(70_000, 20, replace=False)] = 50_000
    P = counts.size
    N = int(counts.sum(dtype=np.uint64))
    counts_d = torch.from_numpy(counts.view(np.int32)).cuda()
    n_ref, ne_ref, off_ref, cp_ref, co_ref, emp_ref = _ctx_expand(ro, counts_d, P, N)
    for _ in range(2):   # two calls in a row share the static scratch
        off = torch.full((P + 1,), -1, dtype=torch.int64, device="cuda")
        cp = torch.full((N,), -1, dtype=torch.int32, device="cuda")
        co = torch.full((N,), -1, dtype=torch.int32, device="cuda")
        emp = torch.full((P,), -1, dtype=torch.int32, device="cuda")
        st, n, ne = ro.ro_expand_noalloc(counts_d, P, off, cp, co, N, emp,
                                         torch.cuda.current_stream())
        assert (st, n, ne) == (0, n_ref, ne_ref)
        assert torch.equal(off, off_ref)
        assert torch.equal(cp, cp_ref) and torch.equal(co, co_ref)
        assert torch.equal(emp[:ne], emp_ref)


def test_noalloc_rejects_sizes_beyond_its_scratch():
    import paper_2609_18703_gb300 as ro
    counts_d = torch.ones(4, dtype=torch.int32, device="cuda")
    off = torch.empty(5, dtype=torch.int64, device="cuda")
    st, _, _ = ro.ro_expand_noalloc(counts_d, (1 << 24) + 1, off, None, None, 0)
    assert st == ro.RO_E_CAPACITY
    cp = torch.empty(4, dtype=torch.int32, device="cuda")
    st, n, _ = ro.ro_expand_noalloc(counts_d, 4, off, cp, cp, 3)   # N = 4 > child_cap
    assert st == ro.RO_E_CAPACITY and n == 4
