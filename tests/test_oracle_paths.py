"""Pins for the oracle's exhaustive path search (Def. 1-2, Eq. 1-2).  CPU only.

Pinned to: hand-worked golden cases; a textbook chain dynamic program (Viterbi)
written here; the full routine product (no Eq. 1 reduction); an independent
exact block-wise search; and invariants of the cost definition.
"""
import itertools
import json
import os

import numpy as np
import pytest

import oracle
from oracle.paths import articulation_layers, blockwise_search, full_routine_product
from synth import random_dag

INF = oracle.INF
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _lc(rows):
    return np.array([[INF if v is None else v for v in r] for r in rows], dtype=np.int64)


def _adapt_const(n_edges, ns, a):
    ac = np.full((n_edges, ns, ns), a, dtype=np.int64)
    for e in range(n_edges):
        np.fill_diagonal(ac[e], 0)
    return ac


def test_golden_island_chain():
    g = json.load(open(os.path.join(GOLDEN, "path_chain_island.json")))
    lc = _lc(g["layer_cost"])
    for case in g["cases"]:
        ac = _adapt_const(len(g["edges"]), 2, case["adapt"])
        t, asg, nmin = oracle.brute_force(lc, g["edges"], ac)
        assert t == case["expect_cost"]
        assert list(asg) == case["expect_assign"]
        assert nmin == 1


def test_golden_net_c():
    g = json.load(open(os.path.join(GOLDEN, "path_net_c.json")))
    lc = _lc(g["layer_cost"])
    ac = _adapt_const(len(g["edges"]), 2, g["adapt_any_change"])
    t, asg, nmin = oracle.brute_force(lc, g["edges"], ac)
    assert (t, list(asg), nmin) == (g["expect_cost"], g["expect_assign"], 1)
    t2, asg2 = blockwise_search(lc, g["edges"], ac)
    assert t2 == t and list(asg2) == g["expect_assign"]


def test_fastest_per_schema_is_eq1():
    out = oracle.fastest_per_schema([0, 1, 0, 2, 1], [7, 9, 3, 4, 11], 4)
    assert list(out) == [3, 9, 4, INF]


def _viterbi_chain(lc, ac):
    """Textbook chain DP: D_i(y) = F_i(y) + min_x D_{i-1}(x) + a_i(x, y)."""
    n, ns = lc.shape
    D = [int(v) for v in lc[0]]
    for i in range(1, n):
        nd = []
        for y in range(ns):
            best = INF
            for x in range(ns):
                if D[x] == INF or lc[i, y] == INF:
                    continue
                a = 0 if x == y else int(ac[i - 1, x, y])
                if a == INF:
                    continue
                best = min(best, D[x] + a + int(lc[i, y]))
            nd.append(best)
        D = nd
    return min(D)


@pytest.mark.parametrize("seed", range(40))
def test_chain_matches_textbook_dp(seed):
    rng = np.random.default_rng(seed)
    n, ns = int(rng.integers(2, 9)), int(rng.integers(1, 4))
    lc = rng.integers(0, 100, size=(n, ns)).astype(np.int64)
    lc[rng.random((n, ns)) < 0.1] = INF
    edges = [(i, i + 1) for i in range(n - 1)]
    ac = rng.integers(0, 60, size=(len(edges), ns, ns)).astype(np.int64)
    t, asg, _ = oracle.brute_force(lc, edges, ac)
    assert t == _viterbi_chain(lc, ac)
    if t != INF:
        assert oracle.path_cost(lc, edges, ac, asg) == t


@pytest.mark.parametrize("seed", range(25))
def test_eq1_reduction_matches_full_routine_product(seed):
    rng = np.random.default_rng(100 + seed)
    n_inner = int(rng.integers(1, 5))
    edges = random_dag(rng, n_inner)
    n, ns = n_inner + 2, int(rng.integers(1, 4))
    cands = [[(0, 0)]] + [[(int(rng.integers(0, ns)), int(rng.integers(1, 50)))
                           for _ in range(int(rng.integers(1, 4)))] for _ in range(n_inner)] \
        + [[(0, 0)]]
    ac = rng.integers(0, 30, size=(len(edges), ns, ns)).astype(np.int64)
    lc = np.stack([oracle.fastest_per_schema([c[0] for c in cs], [c[1] for c in cs], ns)
                   for cs in cands])
    t, _, _ = oracle.brute_force(lc, edges, ac)
    assert t == full_routine_product(cands, edges, ac, ns)


def _series_parallel(rng, n_blocks):
    """Chain of residual-like blocks: every block is a small DAG between two articulations."""
    edges, n = [], 1
    for _ in range(n_blocks):
        a = n - 1
        kind = int(rng.integers(0, 3))
        if kind == 0:          # plain edge
            edges.append((a, n)); n += 1
        elif kind == 1:        # identity shortcut: a -> x -> y -> m, a -> m
            edges += [(a, n), (n, n + 1), (n + 1, n + 2), (a, n + 2)]; n += 3
        else:                  # projection shortcut: a -> x -> y -> z -> m, a -> p -> m
            edges += [(a, n), (n, n + 1), (n + 1, n + 2), (a, n + 3), (n + 2, n + 4),
                      (n + 3, n + 4)]; n += 5
    return n, edges


@pytest.mark.parametrize("seed", range(30))
def test_blockwise_matches_exhaustive(seed):
    rng = np.random.default_rng(200 + seed)
    n, edges = _series_parallel(rng, int(rng.integers(1, 4)))
    ns = int(rng.integers(2, 4))
    if ns ** n > 2_000_000:
        ns = 2
    lc = rng.integers(0, 100, size=(n, ns)).astype(np.int64)
    lc[0, 1:] = INF
    lc[-1, 1:] = INF
    ac = rng.integers(0, 40, size=(len(edges), ns, ns)).astype(np.int64)
    t, asg, nmin = oracle.brute_force(lc, edges, ac)
    t2, asg2 = blockwise_search(lc, edges, ac)
    assert t == t2
    assert oracle.path_cost(lc, edges, ac, asg2) == t
    if nmin == 1:
        assert list(asg) == list(asg2)


def test_articulation_layers_residual():
    # 0 -> 1 -> 2 -> 3, 0 -> 3, 3 -> 4
    assert articulation_layers(5, [(0, 1), (1, 2), (2, 3), (0, 3), (3, 4)]) == [0, 3, 4]


def test_invariants():
    rng = np.random.default_rng(7)
    edges = random_dag(rng, 6)
    n, ns = 8, 3
    lc = rng.integers(0, 100, size=(n, ns)).astype(np.int64)
    ac = rng.integers(0, 40, size=(len(edges), ns, ns)).astype(np.int64)
    t, asg, _ = oracle.brute_force(lc, edges, ac)
    # a constant added to every schema of one layer shifts the optimum by it
    lc2 = lc.copy()
    lc2[3] += 17
    assert oracle.brute_force(lc2, edges, ac)[0] == t + 17
    # free adapts: the optimum is the per-layer minimum
    t0, _, _ = oracle.brute_force(lc, edges, np.zeros_like(ac))
    assert t0 == int(lc.min(axis=1).sum())
    # identical schemas: every assignment is optimal
    lc3 = np.repeat(lc[:, :1], ns, axis=1)
    t3, asg3, nmin = oracle.brute_force(lc3, edges, np.zeros_like(ac))
    assert nmin == ns ** n and list(asg3) == [0] * n
    # no feasible schema for a layer: infeasible
    lc4 = lc.copy()
    lc4[2, :] = INF
    assert oracle.brute_force(lc4, edges, ac)[0] == INF


def test_tie_break_is_lexicographic():
    lc = np.array([[0, 0], [5, 5], [0, 0]], dtype=np.int64)
    ac = np.zeros((2, 2, 2), dtype=np.int64)
    t, asg, nmin = oracle.brute_force(lc, [(0, 1), (1, 2)], ac)
    assert t == 5 and nmin == 8 and list(asg) == [0, 0, 0]
