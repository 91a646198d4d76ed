"""Seeded synthetic graph inputs for ERC-LG.

This module draws edge lists and nothing else: it holds none of the method's arithmetic (no
Laplacian, projection, solve, resistance or curvature). Both the CUDA path and the CPU oracle are
fed from it, so the two sides always see identical inputs.

The paper's datasets (§4.1) are not available; the five workloads below stand in for them with the
sizes and degree structure of the graphs the paper measures on:

* ``ring_chords_n2000``      -- tiny sanity graph: a 2,000-cycle plus 8,000 distinct uniform chords.
* ``sbm_n20000``             -- stochastic block model, 10 equal blocks (Table 3 uses an SBM).
* ``chung_lu_n169343_g2.5``  -- power-law graph with the shape of ogbn-arxiv.
* ``chung_lu_n232965_g2.1``  -- dense power-law graph with the shape of Reddit.
* ``chung_lu_n2449029_g2.3`` -- large power-law graph with the shape of ogbn-products.

Every generator returns ``(n, src, dst, w)``: int32 endpoint arrays in a shuffled order with random
orientation (so canonicalisation is exercised), and float32 weights or ``None`` for unit weights.
"""
from __future__ import annotations

from dataclasses import dataclass, field

import numpy as np

JL_SEED = 0xE2C1  # Philox key shared by every workload's projection


@dataclass(frozen=True)
class Workload:
    """One synthetic workload: the graph recipe plus the solver parameters it is run with."""

    name: str
    n: int
    kind: str                 # "ring_chords" | "sbm" | "chung_lu"
    K: tuple                  # projection dimensions (the first is the default)
    kc: int                   # columns per streamed chunk
    eps: float                # regularisation (Eq. 5)
    tol: float                # CG relative-residual tolerance
    graph_seed: int
    params: dict = field(default_factory=dict)


WORKLOADS = {
    w.name: w
    for w in [
        Workload("ring_chords_n2000", 2_000, "ring_chords", (64,), 64, 1e-3, 1e-6, 1,
                 {"chords": 8_000}),
        Workload("sbm_n20000", 20_000, "sbm", (128,), 128, 1e-3, 1e-6, 2,
                 {"blocks": 10, "deg_in": 8.0, "deg_out": 0.5, "lognormal_sigma": 0.5}),
        Workload("chung_lu_n169343_g2.5", 169_343, "chung_lu", (256,), 256, 1e-3, 1e-6, 3,
                 {"gamma": 2.5, "m_target": 1_170_000, "weights": "unit"}),
        Workload("chung_lu_n232965_g2.1", 232_965, "chung_lu", (128,), 32, 1e-3, 1e-5, 4,
                 {"gamma": 2.1, "m_target": 57_300_000, "weights": "unit"}),
        Workload("chung_lu_n2449029_g2.3", 2_449_029, "chung_lu", (64, 256, 1024), 128, 1e-3,
                 1e-5, 5, {"gamma": 2.3, "m_target": 61_900_000, "weights": "uniform_0.5_2"}),
    ]
}


# ----------------------------------------------------------------------------------------------
# helpers on canonical 64-bit pair keys  (key = min * n + max)
# ----------------------------------------------------------------------------------------------
def _keys(u, v, n):
    a = np.minimum(u, v).astype(np.int64)
    b = np.maximum(u, v).astype(np.int64)
    return a * n + b


def _unique_sorted(k):
    """Sorted distinct values (a sort and a neighbour compare: much faster than np.unique's
    hashing path on tens of millions of int64 keys, same result)."""
    k = np.sort(np.asarray(k, dtype=np.int64))
    if k.size == 0:
        return k
    keep = np.empty(k.size, dtype=bool)
    keep[0] = True
    np.not_equal(k[1:], k[:-1], out=keep[1:])
    return k[keep]


def _ring_keys(n):
    i = np.arange(n, dtype=np.int64)
    return _keys(i, (i + 1) % n, n)


def _finish(rng, n, keys, weights="unit", sigma=0.5):
    """Sorted unique canonical keys -> shuffled, randomly oriented (n, src, dst, w)."""
    keys = _unique_sorted(keys)
    m = keys.size
    if weights == "unit":
        w = None
    elif weights == "lognormal":
        w = rng.lognormal(0.0, sigma, size=m).astype(np.float32)
    elif weights == "uniform_0.5_2":
        w = rng.uniform(0.5, 2.0, size=m).astype(np.float32)
    else:
        raise ValueError(weights)
    a = (keys // n).astype(np.int32)
    b = (keys % n).astype(np.int32)
    perm = rng.permutation(m)
    flip = rng.random(m) < 0.5
    a, b = a[perm], b[perm]
    src = np.where(flip, b, a).astype(np.int32)
    dst = np.where(flip, a, b).astype(np.int32)
    if w is not None:
        w = w[perm]
    return n, src, dst, w


def _draw_distinct(rng, count, draw_batch, n, exclude=None):
    """Collect `count` distinct canonical non-self-loop keys from repeated batch draws."""
    have = np.empty(0, dtype=np.int64)
    while have.size < count:
        need = count - have.size
        u, v = draw_batch(max(int(need * 1.1) + 16, 64))
        ok = u != v
        k = _keys(u[ok], v[ok], n)
        if exclude is not None:
            k = k[~np.isin(k, exclude)]
        have = _unique_sorted(np.concatenate([have, k]))
    if have.size > count:
        have = np.sort(rng.choice(have, size=count, replace=False))
    return have


# ----------------------------------------------------------------------------------------------
# workload generators
# ----------------------------------------------------------------------------------------------
def ring_chords(n, chords, seed):
    """A cycle i-(i+1 mod n) plus `chords` distinct uniform non-ring chords; unit weights."""
    rng = np.random.default_rng(seed)
    ring = _ring_keys(n)
    chord = _draw_distinct(
        rng, chords, lambda k: (rng.integers(0, n, k), rng.integers(0, n, k)), n, exclude=ring)
    return _finish(rng, n, np.concatenate([ring, chord]), "unit")


def sbm(n, blocks, deg_in, deg_out, sigma, seed):
    """Stochastic block model on contiguous equal blocks, plus a ring; lognormal(0, sigma) weights.

    In-block pair probability deg_in / (B - 1) and cross-block pair probability
    deg_out / (n - B), so the expected in-block and cross-block degrees are deg_in and deg_out.
    """
    rng = np.random.default_rng(seed)
    B = n // blocks
    p_in = deg_in / (B - 1)
    p_out = deg_out / (n - B)
    parts = [_ring_keys(n)]
    for b in range(blocks):
        cnt = rng.binomial(B * (B - 1) // 2, p_in)
        lo = b * B
        parts.append(_draw_distinct(
            rng, cnt, lambda k: (lo + rng.integers(0, B, k), lo + rng.integers(0, B, k)), n))
    cross_pairs = n * (n - 1) // 2 - blocks * (B * (B - 1) // 2)
    cnt = rng.binomial(cross_pairs, p_out)

    def cross(k):
        u = rng.integers(0, n, k)
        v = rng.integers(0, n, k)
        keep = (u // B) != (v // B)
        return u[keep], v[keep]

    parts.append(_draw_distinct(rng, cnt, cross, n))
    return _finish(rng, n, np.concatenate(parts), "lognormal", sigma)


def chung_lu_weights(n, gamma, mean_deg):
    """Expected degrees proportional to (i+1)^(-1/(gamma-1)), mean `mean_deg`, capped at sqrt(sum)."""
    base = (np.arange(n, dtype=np.float64) + 1.0) ** (-1.0 / (gamma - 1.0))
    s = mean_deg / base.mean()
    w = s * base
    for _ in range(100):
        cap = np.sqrt(w.sum())
        w = np.minimum(s * base, cap)
        s *= mean_deg / w.mean()
    return np.minimum(s * base, np.sqrt(w.sum()))


def alias_table(p):
    """Walker / Vose alias table of a discrete distribution p (sums to 1): (prob, alias)."""
    n = p.size
    q = np.asarray(p, dtype=np.float64) * n
    prob = np.ones(n)
    alias = np.arange(n, dtype=np.int64)
    small = np.nonzero(q < 1.0)[0].tolist()
    large = np.nonzero(q >= 1.0)[0].tolist()
    while small and large:
        s = small.pop()
        l = large.pop()
        prob[s] = q[s]
        alias[s] = l
        q[l] = (q[l] + q[s]) - 1.0
        (small if q[l] < 1.0 else large).append(l)
    return prob, alias


def alias_draw(rng, prob, alias, k):
    """k independent draws from the table's distribution."""
    i = rng.integers(0, prob.size, k)
    return np.where(rng.random(k) < prob[i], i, alias[i])


def chung_lu(n, gamma, m_target, weights, seed):
    """Chung-Lu power-law graph with `m_target` distinct edges, then a ring added for connectivity."""
    rng = np.random.default_rng(seed)
    wexp = chung_lu_weights(n, gamma, 2.0 * m_target / n)
    prob, alias = alias_table(wexp / wexp.sum())

    def draw(k):
        return alias_draw(rng, prob, alias, k), alias_draw(rng, prob, alias, k)

    body = _draw_distinct(rng, m_target, draw, n)
    return _finish(rng, n, np.concatenate([body, _ring_keys(n)]), weights)


def make_graph(name):
    """Generate the named workload's graph: returns (n, src, dst, w)."""
    wl = WORKLOADS[name]
    p = wl.params
    if wl.kind == "ring_chords":
        return ring_chords(wl.n, p["chords"], wl.graph_seed)
    if wl.kind == "sbm":
        return sbm(wl.n, p["blocks"], p["deg_in"], p["deg_out"], p["lognormal_sigma"],
                   wl.graph_seed)
    if wl.kind == "chung_lu":
        return chung_lu(wl.n, p["gamma"], p["m_target"], p["weights"], wl.graph_seed)
    raise ValueError(wl.kind)


# ----------------------------------------------------------------------------------------------
# small graph families with closed-form resistances (used by the tests)
# ----------------------------------------------------------------------------------------------
def cycle(n, weight=1.0):
    i = np.arange(n, dtype=np.int32)
    return n, i, ((i + 1) % n).astype(np.int32), np.full(n, weight, np.float32)


def path(n, weight=1.0):
    i = np.arange(n - 1, dtype=np.int32)
    return n, i, i + 1, np.full(n - 1, weight, np.float32)


def complete(n):
    u, v = np.triu_indices(n, 1)
    return n, u.astype(np.int32), v.astype(np.int32), None


def random_tree(n, seed, weighted=True):
    """Uniform random recursive tree: node i>0 attaches to a uniform earlier node."""
    rng = np.random.default_rng(seed)
    child = np.arange(1, n, dtype=np.int32)
    parent = np.array([rng.integers(0, i) for i in range(1, n)], dtype=np.int32)
    w = rng.uniform(0.5, 2.0, n - 1).astype(np.float32) if weighted else None
    return n, parent, child, w


def random_multigraph(n, m, seed, self_loops=True, weighted=True):
    """Random edge list with duplicates, both orientations and (optionally) self-loops."""
    rng = np.random.default_rng(seed)
    src = rng.integers(0, n, m).astype(np.int32)
    dst = rng.integers(0, n, m).astype(np.int32)
    if m >= 4:  # force some exact duplicates and reversed duplicates
        k = m // 4
        src[-k:], dst[-k:] = dst[:k], src[:k]
    if not self_loops:
        bad = src == dst
        dst[bad] = (dst[bad] + 1) % n
    w = rng.uniform(0.25, 4.0, m).astype(np.float32) if weighted else None
    return n, src, dst, w


def random_connected(n, extra, seed, weighted=True):
    """A ring plus `extra` random chords (connected); weights uniform in [0.5, 2] if weighted."""
    rng = np.random.default_rng(seed)
    keys = np.concatenate([_ring_keys(n), _keys(rng.integers(0, n, extra),
                                                 rng.integers(0, n, extra), n)])
    keys = keys[(keys // n) != (keys % n)]
    return _finish(rng, n, keys, "uniform_0.5_2" if weighted else "unit")


# ----------------------------------------------------------------------------------------------
# seeded dense inputs for single-call parity tests
# ----------------------------------------------------------------------------------------------
def random_block(n, kc, ld, seed):
    """n x ld float32 block: standard normal in the first kc columns, zero padding after."""
    rng = np.random.default_rng(seed)
    X = np.zeros((n, ld), np.float32)
    X[:, :kc] = rng.standard_normal((n, kc)).astype(np.float32)
    return X


def random_positive(size, seed, lo=0.05, hi=2.0):
    """float32 values uniform in [lo, hi)."""
    return np.random.default_rng(seed).uniform(lo, hi, size).astype(np.float32)


def random_normal(size, seed, scale=1.0):
    return (np.random.default_rng(seed).standard_normal(size) * scale).astype(np.float32)
