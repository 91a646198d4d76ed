"""The seeded input generators: exact sampling tables, workload sizes, determinism."""
import numpy as np

from paper_2609_27209_gb300 import synth


def test_alias_table_reproduces_the_distribution_exactly():
    for p in [synth.chung_lu_weights(5000, 2.1, 40.0), np.random.default_rng(1).random(777)]:
        p = p / p.sum()
        prob, alias = synth.alias_table(p)
        n = p.size
        implied = prob / n + np.bincount(alias, weights=(1.0 - prob) / n, minlength=n)
        np.testing.assert_allclose(implied, p, rtol=1e-9, atol=1e-15)


def test_chung_lu_weights_hit_the_mean_and_the_cap():
    w = synth.chung_lu_weights(100000, 2.1, 50.0)
    assert abs(w.mean() - 50.0) < 1e-6 * 50
    assert w.max() <= np.sqrt(w.sum()) * (1 + 1e-9)
    assert np.all(np.diff(w) <= 0)


def test_small_workloads_sizes_and_determinism():
    n, s, d, w = synth.make_graph("ring_chords_n2000")
    assert n == 2000 and s.size == 10000 and w is None
    keys = np.minimum(s, d).astype(np.int64) * n + np.maximum(s, d)
    assert np.unique(keys).size == 10000 and np.all(s != d)
    n2, s2, d2, w2 = synth.make_graph("ring_chords_n2000")
    np.testing.assert_array_equal(s, s2)
    np.testing.assert_array_equal(d, d2)
    n, s, d, w = synth.make_graph("sbm_n20000")
    assert n == 20000 and 95000 < s.size < 115000 and w.dtype == np.float32 and np.all(w > 0)


def test_chung_lu_small_instance_is_simple_and_connected_by_the_ring():
    n, s, d, w = synth.chung_lu(3000, 2.3, 20000, "uniform_0.5_2", seed=9)
    keys = np.minimum(s, d).astype(np.int64) * n + np.maximum(s, d)
    assert np.unique(keys).size == keys.size and np.all(s != d)
    ring = np.arange(n, dtype=np.int64)
    ring_keys = np.minimum(ring, (ring + 1) % n) * n + np.maximum(ring, (ring + 1) % n)
    assert np.all(np.isin(ring_keys, keys))
    assert np.all((w >= 0.5) & (w <= 2.0))
