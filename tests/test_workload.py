"""The seeded input generators: determinism, the shapes the configurations
name, and the counter-hash payload definition."""
import numpy as np

from workload import FAILED, PRESENT, docpage, mix64, record_bytes, skew, streaming, tiny, video


def test_mix64_reference_values():
    # SplitMix64 (Steele, Lea, Flood 2014): the first outputs of the generator
    # seeded with 0 are mix64(k * 0x9E3779B97F4A7C15) for k = 1, 2, 3.
    g = np.uint64(0x9E3779B97F4A7C15)
    with np.errstate(over="ignore"):
        xs = np.array([g * np.uint64(k) for k in (1, 2, 3)], dtype=np.uint64)
    assert [hex(int(v)) for v in mix64(xs)] == [
        "0xe220a8397b1dcdaf", "0x6e789e6aa1b965f4", "0x6c45d188009454f"]


def test_record_bytes_prefix_property():
    a = record_bytes(5, 123, 100)
    assert len(a) == 100 and record_bytes(5, 123, 37) == a[:37]
    assert record_bytes(5, 124, 100) != a and record_bytes(6, 123, 100) != a


def test_generators_are_deterministic_and_shaped():
    a, b = tiny(), tiny()
    assert np.array_equal(a.top.counts, b.top.counts)
    assert np.array_equal(a.top.arrival, b.top.arrival)
    lv = a.top
    assert lv.n_parents == 1000 and 1 <= lv.counts.min() and lv.counts.max() <= 500
    assert set(np.unique(lv.state)) <= {PRESENT, FAILED}
    assert np.all(lv.length[lv.state == PRESENT] == 64) and np.all(lv.length[lv.state == FAILED] == 0)
    # arena: present records packed back to back in arrival order
    order = lv.arrival[lv.state[lv.arrival] == PRESENT]
    assert np.array_equal(lv.arena_off[order], np.arange(order.size, dtype=np.uint64) * 64)
    d = docpage(parents=2000, waves=16)
    assert d.top.n_waves == 16 and d.top.wave_bounds[-1] == d.top.n_children
    pres = d.top.state == PRESENT
    assert d.top.length[pres].min() >= 256 and d.top.length[pres].max() <= 65536
    v = video(videos=500)
    assert v.levels[1].n_parents == v.levels[0].n_children
    assert v.levels[0].counts.max() <= 1000 and v.levels[1].counts.min() >= 8
    s = skew(parents=5000, heavy=10, heavy_children=300)
    assert s.top.n_children == 4990 + 3000
    st = streaming(total_children=20000, ready_waves=10)
    assert st.top.n_children >= 20000 and st.top.ready_bounds.size == 11
    assert np.array_equal(st.top.parent_call, np.arange(st.top.n_parents) % 4)
