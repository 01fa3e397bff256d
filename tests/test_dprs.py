"""DPRS (Alg. 1) through the C ABI against the oracle's exhaustive search
(Def. 2) on the same integer cost tables.  CPU only: cost tables are injected
with sn_set_cost_table, no kernel runs.

Spec bar: the selected path equals brute-force enumeration bit-exactly
wherever the minimum is unique; on ties the totals are equal and the DPRS
path is one of the minimisers.
"""
import json
import os

import numpy as np
import pytest

import oracle
import synth
from oracle.paths import blockwise_search
from paper_2110_06037_gb300 import SN_SELECT_BRUTE, SN_SELECT_DPRS, SnError, build_graph
from paper_2110_06037_gb300.api import Graph
from paper_2110_06037_gb300 import _sn

INF = oracle.INF
GOLDEN = os.path.join(os.path.dirname(__file__), "golden")
SCHEMAS3 = [("f32", "nchw"), ("f32", "nhwc"), ("f16", "nhwc")]


def _conv1x1(c):
    return {"type": "conv2", "params": dict(c_in=c, c_out=c, kh=1, kw=1, sh=1, sw=1, ph=0, pw=0,
                                             groups=1, act="relu"),
            "weight": np.zeros((c, c, 1, 1), np.float32), "bias": np.zeros(c, np.float32)}


def _add():
    return {"type": "add", "params": {"act": "none"}}


def random_net(rng, n_steps):
    """Random 1-in-1-out net of 1x1 convs (any fan-out) and adds (fan-in 2)."""
    layers, open_ = [], {-1}
    for _ in range(n_steps):
        cands = sorted(open_)
        if len(cands) >= 2 and rng.random() < 0.4:
            a, b = rng.choice(cands, 2, replace=False)
            l = _add()
            l["inputs"] = [int(a), int(b)]
            open_ -= {int(a), int(b)}
        else:
            src = int(rng.integers(-1, len(layers))) if rng.random() < 0.5 else int(rng.choice(cands))
            l = _conv1x1(4)
            l["inputs"] = [src]
            open_.discard(src)
        layers.append(l)
        open_.add(len(layers) - 1)
    while len(open_) > 1:
        a, b = sorted(open_)[:2]
        l = _add()
        l["inputs"] = [a, b]
        open_ -= {a, b}
        layers.append(l)
        open_.add(len(layers) - 1)
    return layers


def make_graph(layers, schemas, in_shape=(1, 4, 3, 3)):
    s0 = schemas[0]
    return build_graph(layers, in_shape, s0, s0, schemas, torch_alloc=False)


def random_costs(g, rng, p_inf=0.1, hi=1000, adapt_hi=400):
    t = g.cost_table()
    c = rng.integers(1, hi, size=len(t["cost"])).astype(np.int64)
    c[rng.random(len(c)) < p_inf] = INF
    io = t["routine"] == 0
    c[io] = 0
    t["cost"] = c
    ns = t["n_schemas"]
    a = rng.integers(0, adapt_hi, size=t["adapt"].shape).astype(np.int64)
    a[rng.random(a.shape) < p_inf / 2] = INF
    for e in range(a.shape[0]):
        np.fill_diagonal(a[e], 0)
    t["adapt"] = a
    g.set_cost_table(t)
    return t


def oracle_layer_cost(t):
    n, ns = t["n_layers"], t["n_schemas"]
    lc = np.zeros((n, ns), np.int64)
    for i in range(n):
        m = t["layer"] == i
        lc[i] = oracle.fastest_per_schema(t["schema"][m], t["cost"][m], ns)
    return lc


def oracle_pair_cost(t):
    """Per layer, the cheapest candidate of every (read, written) schema pair
    (INF where none): the states of the pair problem."""
    n, ns = t["n_layers"], t["n_schemas"]
    pairs = [(r, w) for r in range(ns) for w in range(ns)]
    lc = np.full((n, len(pairs)), INF, np.int64)
    for c in range(len(t["cost"])):
        k = int(t["schema"][c]) * ns + int(t["out_schema"][c])
        lc[t["layer"][c], k] = min(lc[t["layer"][c], k], int(t["cost"][c]))
    return lc, pairs


def has_fused(t):
    return bool((t["out_schema"] != t["schema"]).any())


def realised_cost(t, cand):
    """T of a choice of one candidate per layer: their times plus, on every
    edge, the adapt from the producer's written schema to the consumer's read
    schema (Def. 1, fused boundaries)."""
    tot = sum(int(t["cost"][c]) for c in cand)
    for e, (u, v) in enumerate(t["edges"].tolist()):
        w, r = int(t["out_schema"][cand[u]]), int(t["schema"][cand[v]])
        if w != r:
            tot += int(t["adapt"][e][w][r])
    return tot


def check_against_oracle(g, t, exhaustive=True):
    if has_fused(t):
        # some routine writes another schema: the exact pair-state search
        lcp, pairs = oracle_pair_cost(t)
        ref, _ = blockwise_search(lcp, t["edges"], t["adapt"], pairs=pairs)
        try:
            tot, sch, cand = g.select_path(SN_SELECT_DPRS)
        except SnError as e:
            assert e.status == _sn.SN_EINFEASIBLE and ref == INF
            return None
        assert tot == ref, (tot, ref)
        assert realised_cost(t, cand) == ref
        return None
    lc = oracle_layer_cost(t)
    if exhaustive:
        ref, asg, nmin = oracle.brute_force(lc, t["edges"], t["adapt"])
    else:
        ref, asg = blockwise_search(lc, t["edges"], t["adapt"])
        nmin = None
    try:
        tot, sch, cand = g.select_path(SN_SELECT_DPRS)
    except SnError as e:
        assert e.status == _sn.SN_EINFEASIBLE and ref == INF
        return None
    assert tot == ref, (tot, ref)
    assert oracle.path_cost(lc, t["edges"], t["adapt"], sch) == ref
    if nmin == 1:
        assert list(sch) == list(asg)
    # the chosen routine is F_i(lambda) of the chosen schema (Eq. 1)
    for i, c in enumerate(cand):
        assert t["layer"][c] == i and t["schema"][c] == sch[i]
        assert t["cost"][c] == lc[i, sch[i]]
    return nmin


@pytest.mark.parametrize("seed", range(150))
def test_dprs_equals_brute_force_random_dags(seed):
    rng = np.random.default_rng(seed)
    ns = 2 if seed % 3 else 3
    layers = random_net(rng, int(rng.integers(1, 8 if ns == 3 else 10)))
    g = make_graph(layers, SCHEMAS3[:ns])
    t = random_costs(g, rng)
    check_against_oracle(g, t)


@pytest.mark.parametrize("seed", range(30))
def test_library_brute_force_equals_oracle(seed):
    rng = np.random.default_rng(1000 + seed)
    layers = random_net(rng, int(rng.integers(1, 8)))
    g = make_graph(layers, SCHEMAS3[:2])
    t = random_costs(g, rng)
    lc = oracle_layer_cost(t)
    ref, asg, nmin = oracle.brute_force(lc, t["edges"], t["adapt"])
    try:
        tot, sch, _ = g.select_path(SN_SELECT_BRUTE)
    except SnError as e:
        assert ref == INF and e.status == _sn.SN_EINFEASIBLE
        return
    assert tot == ref
    if nmin == 1:
        assert list(sch) == list(asg)


def test_nested_branch_counterexample():
    """1->2, 1->3, 2->4, 2->5, {4,3}->6, {6,5}->7: C_4 = {1,2} but C_3 = {1},
    so the constraint sets of a merge's predecessors differ (Alg. 1 assumes
    they are equal).  DPRS with the union of the sets must still be exact."""
    L = []
    def conv(src):
        l = _conv1x1(4); l["inputs"] = [src]; L.append(l); return len(L) - 1
    def add(a, b):
        l = _add(); l["inputs"] = [a, b]; L.append(l); return len(L) - 1
    l1 = conv(-1)
    l2 = conv(l1)
    l3 = conv(l1)
    l4 = conv(l2)
    l5 = conv(l2)
    l6 = add(l4, l3)
    add(l6, l5)
    for seed in range(200):
        rng = np.random.default_rng(5000 + seed)
        g = make_graph(L, SCHEMAS3[: 2 + seed % 2])
        t = random_costs(g, rng, p_inf=0.05)
        check_against_oracle(g, t)


def test_unique_minimum_instances_match_exactly():
    """Bit-exact path equality on instances whose minimum is unique."""
    hits = 0
    for seed in range(300):
        rng = np.random.default_rng(9000 + seed)
        g = make_graph(random_net(rng, 6), SCHEMAS3[:2])
        t = random_costs(g, rng, p_inf=0.0, hi=10 ** 6, adapt_hi=10 ** 6)
        if check_against_oracle(g, t) == 1:
            hits += 1
    assert hits > 250


def test_ties_give_a_minimiser():
    for seed in range(60):
        rng = np.random.default_rng(7000 + seed)
        g = make_graph(random_net(rng, 6), SCHEMAS3[:2])
        t = random_costs(g, rng, p_inf=0.0, hi=3, adapt_hi=2)  # many ties
        check_against_oracle(g, t)


def test_golden_island_chain_through_abi():
    gold = json.load(open(os.path.join(GOLDEN, "path_chain_island.json")))
    L = []
    for src in (-1, 0, 1):
        l = _conv1x1(4)
        l["inputs"] = [src]
        L.append(l)
    g = make_graph(L, [("f32", "nchw"), ("f32", "nhwc")])
    t = g.cost_table()
    for case in gold["cases"]:
        cost = np.zeros_like(t["cost"])
        for c in range(len(cost)):
            i, s = t["layer"][c], t["schema"][c]
            v = gold["layer_cost"][i][s]
            cost[c] = INF if v is None else v
        t["cost"] = cost
        a = np.full_like(t["adapt"], case["adapt"])
        for e in range(a.shape[0]):
            np.fill_diagonal(a[e], 0)
        t["adapt"] = a
        g.set_cost_table(t)
        tot, sch, _ = g.select_path(SN_SELECT_DPRS)
        assert tot == case["expect_cost"] and list(sch) == case["expect_assign"]


def test_golden_net_c_through_abi():
    gold = json.load(open(os.path.join(GOLDEN, "path_net_c.json")))
    # internal layers 1..8 = user layers 0..7; layer 8 (user 7) merges 5 and 7
    L = []
    def conv(src):
        l = _conv1x1(4); l["inputs"] = [src]; L.append(l); return len(L) - 1
    def add(a, b):
        l = _add(); l["inputs"] = [a, b]; L.append(l); return len(L) - 1
    u1 = conv(-1)          # internal 1
    u2 = conv(u1)          # 2
    u3 = conv(u2)          # 3
    u4 = conv(u2)          # 4
    u5 = add(u3, u4)       # 5
    u6 = conv(u1)          # 6
    u7 = conv(u6)          # 7
    add(u5, u7)            # 8
    g = make_graph(L, [("f32", "nchw"), ("f32", "nhwc")])
    t = g.cost_table()
    assert sorted(map(tuple, t["edges"].tolist())) == sorted(map(tuple, gold["edges"]))
    cost = np.zeros_like(t["cost"])
    for c in range(len(cost)):
        v = gold["layer_cost"][t["layer"][c]][t["schema"][c]]
        cost[c] = INF if v is None else v
    t["cost"] = cost
    a = np.full_like(t["adapt"], gold["adapt_any_change"])
    for e in range(a.shape[0]):
        np.fill_diagonal(a[e], 0)
    t["adapt"] = a
    g.set_cost_table(t)
    tot, sch, _ = g.select_path(SN_SELECT_DPRS)
    assert tot == gold["expect_cost"] and list(sch) == gold["expect_assign"]


@pytest.mark.parametrize("net", ["resnet50", "mobilenet_v2", "vgg16", "mobilenet_v3"])
def test_dprs_equals_blockwise_search_on_real_nets(net):
    """Nets too large to enumerate: the oracle's block-wise exact search."""
    build = {"resnet50": synth.resnet50, "mobilenet_v2": synth.mobilenet_v2, "vgg16": synth.vgg16,
             "mobilenet_v3": synth.mobilenet_v3}[net]
    _, layers = build(1, res=32)
    sch = [("f16", "nchw"), ("f16", "nhwc")]
    g = build_graph(layers, (1, 3, 32, 32), ("f32", "nchw"), ("f32", "nchw"), sch, torch_alloc=False)
    for seed in range(3):
        rng = np.random.default_rng(seed)
        t = random_costs(g, rng, p_inf=0.05)
        check_against_oracle(g, t, exhaustive=False)
