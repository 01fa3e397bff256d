"""Fused-boundary routines (routines that write a schema other than the one
they read: a qint8 routine with the dequantisation in its epilogue): the
candidates, and DPRS over (read, written) schema pairs against an exhaustive
search over one candidate per layer.  CPU only: costs are injected."""
import numpy as np
import pytest

import oracle
from oracle.paths import brute_force_candidates
from paper_2110_06037_gb300 import SN_SELECT_BRUTE, SN_SELECT_DPRS, SnError, build_graph
from paper_2110_06037_gb300 import _sn

from test_dprs import random_net

INF = oracle.INF
LAMBDA = [("f16", "nhwc"), ("qi8", "nhwc"), ("f16", "nchw")]


def _graph(layers, ns):
    return build_graph(layers, (1, 4, 3, 3), ("f16", "nhwc"), ("f16", "nhwc"), LAMBDA[:ns], torch_alloc=False)


def test_qint8_routines_offer_float_outputs_of_their_layout():
    rng = np.random.default_rng(1)
    g = _graph(random_net(rng, 3), 3)
    t = g.cost_table()
    uni = g.schema_universe()
    fused = [c for c in range(len(t["cost"])) if t["out_schema"][c] != t["schema"][c]]
    assert fused
    for c in fused:
        rd, wr = uni[t["schema"][c]], uni[t["out_schema"][c]]
        assert rd[0] == "qi8" and wr[0] != "qi8" and rd[1] == wr[1]
        # the same routine and parameter exists with its ordinary output
        assert any(t["routine"][k] == t["routine"][c] and t["variant"][k] == t["variant"][c]
                   and t["schema"][k] == t["schema"][c] and t["out_schema"][k] == t["schema"][c]
                   and t["layer"][k] == t["layer"][c] for k in range(len(t["cost"])))
    # float routines never change the schema they write
    assert all(uni[t["schema"][c]][0] == "qi8" for c in fused)


def _random_costs(g, rng):
    t = g.cost_table()
    c = rng.integers(1, 1000, size=len(t["cost"])).astype(np.int64)
    c[rng.random(len(c)) < 0.1] = INF
    c[t["routine"] == 0] = 0
    t["cost"] = c
    a = rng.integers(0, 400, size=t["adapt"].shape).astype(np.int64)
    a[rng.random(a.shape) < 0.05] = INF
    for e in range(a.shape[0]):
        np.fill_diagonal(a[e], 0)
    t["adapt"] = a
    g.set_cost_table(t)
    return t


def _cands_per_layer(t):
    out = []
    for i in range(t["n_layers"]):
        idx = np.flatnonzero(t["layer"] == i)
        out.append([(int(t["cost"][c]), int(t["schema"][c]), int(t["out_schema"][c])) for c in idx])
    return out


@pytest.mark.parametrize("seed", range(40))
def test_dprs_over_schema_pairs_equals_exhaustive_search(seed):
    rng = np.random.default_rng(9100 + seed)
    ns = 2 if seed % 2 else 3
    layers = random_net(rng, int(rng.integers(1, 4)))
    g = _graph(layers, ns)
    t = _random_costs(g, rng)
    per = _cands_per_layer(t)
    if np.prod([len(c) for c in per], dtype=float) > 3e5:
        pytest.skip("candidate product too large to enumerate")
    ref, pick = brute_force_candidates(per, t["edges"].tolist(), t["adapt"])
    try:
        tot, sch, cand = g.select_path(SN_SELECT_DPRS)
    except SnError as e:
        assert ref == INF and e.status == _sn.SN_EINFEASIBLE
        return
    assert tot == ref
    # the chosen candidates realise the total
    chosen = [(int(t["cost"][c]), int(t["schema"][c]), int(t["out_schema"][c])) for c in cand]
    realised = sum(c[0] for c in chosen)
    for e, (u, v) in enumerate(t["edges"].tolist()):
        if chosen[u][2] != chosen[v][1]:
            realised += int(t["adapt"][e][chosen[u][2]][chosen[v][1]])
    assert realised == ref
    if len(layers) <= 3:
        assert g.select_path(SN_SELECT_BRUTE)[0] == ref


@pytest.mark.parametrize("seed", range(20))
def test_pair_problem_without_fused_choices_is_the_plain_problem(seed):
    """With every fused candidate infeasible the pair problem keeps only the
    diagonal pairs, so its optimum is the plain DPRS optimum over schemas
    (checked against the oracle's exhaustive search of Def. 2)."""
    rng = np.random.default_rng(9300 + seed)
    layers = random_net(rng, int(rng.integers(1, 5)))
    g = _graph(layers, 2)
    t = _random_costs(g, rng)
    t["cost"][t["out_schema"] != t["schema"]] = INF
    g.set_cost_table(t)
    ns, n = t["n_schemas"], t["n_layers"]
    lc = np.array([oracle.fastest_per_schema(t["schema"][t["layer"] == i], t["cost"][t["layer"] == i], ns)
                   for i in range(n)])
    ref, _, _ = oracle.brute_force(lc, t["edges"], t["adapt"])
    try:
        tot, _, cand = g.select_path(SN_SELECT_DPRS)
    except SnError as e:
        assert ref == INF and e.status == _sn.SN_EINFEASIBLE
        return
    assert tot == ref
    assert all(t["out_schema"][c] == t["schema"][c] for c in cand)


# ---------------------------------------------------------------------------
# pins of the oracle's exhaustive search over candidates (fused boundaries)
# ---------------------------------------------------------------------------

def _golden_fused():
    import json
    import os
    here = os.path.dirname(os.path.abspath(__file__))
    with open(os.path.join(here, "golden", "path_fused_boundary.json")) as f:
        return json.load(f)


def test_candidate_search_reaches_the_hand_worked_fused_optimum():
    """Def. 1-2 read for fused boundaries: each edge is charged the adapt from
    the producer's WRITTEN schema to the consumer's READ schema.  The golden
    lists every choice with its cost by hand; the optimum uses the qint8
    routine that writes f16, and charging the edge from its read schema
    instead would move the optimum."""
    g = _golden_fused()
    ns = len(g["schemas"])
    a = np.zeros((len(g["edges"]), ns, ns), np.int64)
    a[:, 0, 1] = g["adapt"]["F->Q (quantise)"]
    a[:, 1, 0] = g["adapt"]["Q->F (dequantise)"]
    cands = [[tuple(c) for c in layer] for layer in g["candidates"]]
    cost, pick = brute_force_candidates(cands, g["edges"], a)
    assert cost == g["expect_cost"]
    assert pick == g["expect_pick"]


def test_candidate_search_equals_schema_search_without_fused_candidates():
    """When every candidate writes the schema it reads, the search over one
    candidate per layer is the plain problem of Def. 2: its optimum equals the
    exhaustive search over schema assignments of F_i(lambda) (Eq. 1)."""
    for seed in range(60):
        rng = np.random.default_rng(9500 + seed)
        n, ns = int(rng.integers(3, 7)), int(rng.integers(2, 4))
        edges = [(i, i + 1) for i in range(n - 1)]
        for _ in range(int(rng.integers(0, 3))):  # a few skip edges (still a DAG in index order)
            u = int(rng.integers(0, n - 2))
            v = int(rng.integers(u + 2, n))
            if (u, v) not in edges:
                edges.append((u, v))
        cands, lc = [], np.full((n, ns), INF, np.int64)
        for i in range(n):
            layer = []
            for _ in range(int(rng.integers(1, 4))):
                s = int(rng.integers(0, ns))
                c = 0 if i in (0, n - 1) else int(rng.integers(1, 100))
                layer.append((c, s, s))
                lc[i, s] = min(lc[i, s], c)
            cands.append(layer)
        a = rng.integers(0, 40, size=(len(edges), ns, ns)).astype(np.int64)
        for e in range(len(edges)):
            np.fill_diagonal(a[e], 0)
        got, pick = brute_force_candidates(cands, edges, a)
        ref, _, _ = oracle.brute_force(lc, edges, a)
        assert got == ref, seed
        if got < INF:
            # the chosen candidates, read as a schema assignment, cost the same
            assign = [cands[i][k][1] for i, k in enumerate(pick)]
            assert oracle.path_cost(lc, edges, a, assign) == ref


def test_pair_blockwise_search_equals_candidate_search():
    """The oracle's block-wise exact search over (read, written) pair states
    (used on nets too large to enumerate) equals the exhaustive search over
    one candidate per layer, on random nets with fused candidates."""
    from oracle.paths import blockwise_search
    from test_dprs import oracle_pair_cost
    for seed in range(40):
        rng = np.random.default_rng(9700 + seed)
        layers = random_net(rng, int(rng.integers(1, 4)))
        g = _graph(layers, 3 if seed % 2 else 2)
        t = _random_costs(g, rng)
        per = _cands_per_layer(t)
        if np.prod([len(c) for c in per], dtype=float) > 2e5:
            continue
        ref, _ = brute_force_candidates(per, t["edges"].tolist(), t["adapt"])
        lcp, pairs = oracle_pair_cost(t)
        got, _ = blockwise_search(lcp, t["edges"], t["adapt"], pairs=pairs)
        assert got == ref, seed


def test_pair_blockwise_search_without_fused_states_is_the_plain_search():
    from oracle.paths import blockwise_search
    rng = np.random.default_rng(4)
    for _ in range(20):
        n, ns = int(rng.integers(3, 8)), 2
        edges = [(i, i + 1) for i in range(n - 1)]
        lc = rng.integers(1, 50, size=(n, ns)).astype(np.int64)
        lc[0] = lc[-1] = 0
        ac = rng.integers(0, 30, size=(len(edges), ns, ns)).astype(np.int64)
        pairs = [(r, w) for r in range(ns) for w in range(ns)]
        lcp = np.full((n, len(pairs)), INF, np.int64)
        for r in range(ns):
            lcp[:, r * ns + r] = lc[:, r]
        assert blockwise_search(lcp, edges, ac, pairs=pairs)[0] == blockwise_search(lc, edges, ac)[0]
