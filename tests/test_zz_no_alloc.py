"""ro_expand_noalloc — the allocation-free expansion — through the C ABI.

The entry point is for callers that cannot call cudaMalloc: code that runs
inside a memory budget another allocator owns, code that must not
synchronise the device the way cudaMalloc/cudaFree can, and embedders that
forbid allocation after start-up.  Its scratch is one fixed static device
array that every call shares, so these tests check that calls in a row stay
exact, that each result equals both the oracle's expansion and the
context-based ro_expand, and that sizes past the scratch are refused without
disturbing the next call.  Named to be collected last.
"""
import numpy as np
import pytest

torch = pytest.importorskip("torch")

pytestmark = pytest.mark.gpu

NA_MAX_PARENTS = 1 << 24
NA_MAX_CHILDREN = 1 << 27


@pytest.fixture(scope="module", autouse=True)
def _built():
    if not torch.cuda.is_available():
        pytest.skip("no CUDA device")
    import __graft_entry__
    __graft_entry__.build()


def _oracle_expand(counts):
    from oracle import OracleCtx
    o = OracleCtx()
    try:
        r = o.expand(counts)
    finally:
        o.close()
    return r


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


def _noalloc(ro, counts_d, P, cap, with_empties=True, stream=None):
    off = torch.full((P + 1,), -1, dtype=torch.int64, device="cuda")
    cp = torch.full((max(cap, 1),), -1, dtype=torch.int32, device="cuda")
    co = torch.full((max(cap, 1),), -1, dtype=torch.int32, device="cuda")
    emp = torch.full((max(P, 1),), -1, dtype=torch.int32, device="cuda") if with_empties else None
    torch.cuda.synchronize()
    st, n, ne = ro.ro_expand_noalloc(counts_d, P, off, cp, co, cap, emp,
                                     stream if stream is not None else torch.cuda.current_stream())
    return st, n, ne, off, cp, co, emp


def _u(t, dtype):
    return t.cpu().numpy().view(dtype)


def _check_against_oracle(ref, res, with_empties=True):
    st, n, ne, off, cp, co, emp = res
    assert st == 0
    assert n == ref["n_children"]
    np.testing.assert_array_equal(_u(off, np.uint64), ref["offsets"])
    np.testing.assert_array_equal(_u(cp[:n], np.uint32), ref["child_parent"])
    np.testing.assert_array_equal(_u(co[:n], np.uint32), ref["child_ordinal"])
    assert ne == ref["empty_parents"].size
    if with_empties:
        np.testing.assert_array_equal(_u(emp[:ne], np.uint32), ref["empty_parents"])


def _counts(case):
    rng = np.random.default_rng(17)
    if case == "docpage_like":
        return np.clip(np.rint(rng.lognormal(2.3, 1.0, 300_000)), 1, 2000).astype(np.uint32)
    if case == "skewed_with_empties":
        c = rng.integers(0, 4, 70_000).astype(np.uint32)
        c[rng.choice(70_000, 20, replace=False)] = 50_000
        return c
    if case == "no_parents":
        return np.zeros(0, np.uint32)
    if case == "all_empty":
        return np.zeros(5_000, np.uint32)
    if case == "one_parent":
        return np.array([9_000], np.uint32)
    raise ValueError(case)


@pytest.mark.parametrize("case", ["docpage_like", "skewed_with_empties", "no_parents", "all_empty",
                                  "one_parent"])
def test_noalloc_matches_oracle_and_ro_expand_twice(case):
    import paper_2609_18703_gb300 as ro
    counts = _counts(case)
    P = counts.size
    N = int(counts.sum(dtype=np.uint64))
    ref = _oracle_expand(counts)
    counts_d = torch.from_numpy(counts.view(np.int32)).cuda()
    n_ref, ne_ref, off_ref, cp_ref, co_ref, emp_ref = _ctx_expand(ro, counts_d, P, N)
    for _ in range(2):   # two calls in a row share the static scratch
        res = _noalloc(ro, counts_d, P, N)   # N == child_cap exactly
        _check_against_oracle(ref, res)
        st, n, ne, off, cp, co, emp = res
        assert (n, ne) == (n_ref, ne_ref)
        assert torch.equal(off, off_ref)
        assert torch.equal(cp[:n], cp_ref) and torch.equal(co[:n], co_ref)
        assert torch.equal(emp[:ne], emp_ref)


def test_noalloc_without_empty_list_and_on_two_streams():
    """NULL d_empty_parents; a call on one stream, then one on another stream
    right after it returns: the first call is complete on return, so the
    second cannot disturb it through the shared scratch."""
    import paper_2609_18703_gb300 as ro
    rng = np.random.default_rng(5)
    a = rng.integers(0, 40, 200_000).astype(np.uint32)
    b = np.clip(np.rint(rng.lognormal(2.0, 1.2, 150_000)), 0, 3000).astype(np.uint32)
    ref_a, ref_b = _oracle_expand(a), _oracle_expand(b)
    s1, s2 = torch.cuda.Stream(), torch.cuda.Stream()
    da = torch.from_numpy(a.view(np.int32)).cuda()
    db = torch.from_numpy(b.view(np.int32)).cuda()
    Na, Nb = ref_a["n_children"], ref_b["n_children"]
    ra = _noalloc(ro, da, a.size, Na, with_empties=False, stream=s1)
    rb = _noalloc(ro, db, b.size, Nb, with_empties=True, stream=s2)
    torch.cuda.synchronize()
    _check_against_oracle(ref_a, ra, with_empties=False)
    _check_against_oracle(ref_b, rb)


def test_noalloc_rejects_sizes_beyond_its_scratch_and_recovers():
    import paper_2609_18703_gb300 as ro
    small = np.array([3, 0, 5, 1], np.uint32)
    ref_small = _oracle_expand(small)
    ds = torch.from_numpy(small.view(np.int32)).cuda()
    # too many parents: refused before anything is launched
    off = torch.empty(5, dtype=torch.int64, device="cuda")
    st, _, _ = ro.ro_expand_noalloc(ds, NA_MAX_PARENTS + 1, off, None, None, 0)
    assert st == ro.RO_E_CAPACITY
    _check_against_oracle(ref_small, _noalloc(ro, ds, 4, 9))
    # more children than child_cap: the count is reported, the next call is exact
    st, n, _, _, _, _, _ = _noalloc(ro, ds, 4, 8)
    assert st == ro.RO_E_CAPACITY and n == 9
    _check_against_oracle(ref_small, _noalloc(ro, ds, 4, 9))
    # more children than the scratch's fill table covers (few huge parents)
    big = np.array([NA_MAX_CHILDREN - 7, 0, 8], np.uint32)
    db = torch.from_numpy(big.view(np.int32)).cuda()
    off = torch.full((4,), -1, dtype=torch.int64, device="cuda")
    st, n, ne = ro.ro_expand_noalloc(db, 3, off, None, None, NA_MAX_CHILDREN + 1)
    assert st == ro.RO_E_CAPACITY and n == NA_MAX_CHILDREN + 1 and ne == 1
    np.testing.assert_array_equal(_u(off, np.uint64),
                                  np.array([0, NA_MAX_CHILDREN - 7, NA_MAX_CHILDREN - 7,
                                            NA_MAX_CHILDREN + 1], np.uint64))
    _check_against_oracle(ref_small, _noalloc(ro, ds, 4, 9))


def test_noalloc_at_its_child_limit():
    """Exactly 2^27 children (the largest the static scratch takes), spread
    over a few large parents and many small ones."""
    import paper_2609_18703_gb300 as ro
    rng = np.random.default_rng(11)
    small = rng.integers(0, 6, 100_000).astype(np.uint32)
    big = np.full(8, 0, np.uint32)
    rest = NA_MAX_CHILDREN - int(small.sum())
    big[:] = rest // 8
    big[0] += rest - int(big.sum())
    counts = np.concatenate([big[:4], small, big[4:]])
    assert int(counts.sum(dtype=np.uint64)) == NA_MAX_CHILDREN
    ref = _oracle_expand(counts)
    dc = torch.from_numpy(counts.view(np.int32)).cuda()
    _check_against_oracle(ref, _noalloc(ro, dc, counts.size, NA_MAX_CHILDREN))
