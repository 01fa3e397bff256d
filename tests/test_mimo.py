"""Nets with several inputs and outputs (section IV-E): the auxiliary input
layer feeds every input layer, the auxiliary output layer merges every
output, and DPRS (Alg. 1) on the resulting 1-in-1-out net equals the
oracle's exhaustive search (Def. 2).  CPU only: costs are injected."""
import numpy as np
import pytest

import oracle
from paper_2110_06037_gb300 import SN_SELECT_BRUTE, SN_SELECT_DPRS, SnError, build_graph
from paper_2110_06037_gb300 import _sn
from paper_2110_06037_gb300.api import Graph

from test_dprs import _add, _conv1x1, check_against_oracle, random_costs

S2 = [("f32", "nchw"), ("f32", "nhwc")]
SCHEMAS3 = [("f32", "nchw"), ("f32", "nhwc"), ("f16", "nhwc")]
SHAPE = (1, 4, 3, 3)


def two_in_two_out():
    a = dict(_conv1x1(4), inputs=[-1])
    b = dict(_conv1x1(4), inputs=[-2])
    c = dict(_add(), inputs=[0, 1])
    d = dict(_conv1x1(4), inputs=[2])
    return [a, b, c, d]


def test_structure_of_a_two_input_two_output_net():
    layers = two_in_two_out()
    g = build_graph(layers, SHAPE, S2[0], S2[0], S2, torch_alloc=False, extra_inputs=[SHAPE], outputs=[0, 3])
    assert g.io_counts() == (2, 2)
    t = g.cost_table()
    n = t["n_layers"]
    assert n == 2 + len(layers) + 1
    # input layer 1: one zero-cost routine in the input schema, fed by layer 0
    m1 = t["layer"] == 1
    assert m1.sum() == 1 and t["routine"][m1][0] == 0 and t["schema"][m1][0] == 0
    assert [0, 1] in t["edges"].tolist()
    # user layer u is internal layer u + 2; the output layer merges outputs 0 and 3 in order
    into_out = [int(e[0]) for e in t["edges"] if e[1] == n - 1]
    assert into_out == [0 + 2, 3 + 2]
    assert [g.layer_shape(j) for j in into_out] == [SHAPE, SHAPE]


def test_input_and_output_declarations_are_validated():
    g = Graph(SHAPE, S2[0], S2[0], S2, torch_alloc=False)
    g.add_layer(_sn.SN_L_CONV2, _conv1x1(4)["params"], (-1,), np.zeros((4, 4, 1, 1), np.float32), None)
    with pytest.raises(SnError) as e:
        g.add_input(SHAPE)  # after a layer
    assert e.value.status == _sn.SN_ESTATE
    with pytest.raises(SnError):
        g.set_outputs([5])
    with pytest.raises(SnError):
        g.set_outputs([0, 0])
    with pytest.raises(SnError):
        g.add_layer(_sn.SN_L_CONV2, _conv1x1(4)["params"], (-2,), np.zeros((4, 4, 1, 1), np.float32), None)
    # a declared input that feeds nothing makes the net invalid
    g2 = Graph(SHAPE, S2[0], S2[0], S2, torch_alloc=False)
    assert g2.add_input(SHAPE) == -2
    g2.add_layer(_sn.SN_L_CONV2, _conv1x1(4)["params"], (-1,), np.zeros((4, 4, 1, 1), np.float32), None)
    with pytest.raises(SnError) as e:
        g2.cost_table()
    assert "feeds no layer" in str(e.value)


def random_mimo(rng, n_in, n_steps):
    """Random DAG of 1x1 convs and adds over n_in inputs; returns (layers,
    outputs) with 1-3 outputs covering every sink."""
    layers = []
    srcs = list(range(-1, -1 - n_in, -1))
    used = set()
    for _ in range(n_steps):
        pool = srcs + list(range(len(layers)))
        if len(pool) >= 2 and rng.random() < 0.35:
            a, b = rng.choice(pool, 2, replace=False)
            layers.append(dict(_add(), inputs=[int(a), int(b)]))
            used |= {int(a), int(b)}
        else:
            s = int(rng.choice(pool))
            layers.append(dict(_conv1x1(4), inputs=[s]))
            used.add(s)
    for s in srcs:  # every input feeds some layer
        if s not in used:
            layers.append(dict(_conv1x1(4), inputs=[s]))
            used.add(s)
    sinks = [i for i in range(len(layers)) if i not in used]
    extra = [int(i) for i in rng.choice(len(layers), size=min(len(layers), int(rng.integers(0, 2))), replace=False)
             if i not in sinks]
    return layers, sinks + extra


@pytest.mark.parametrize("seed", range(60))
def test_dprs_equals_brute_force_on_mimo_nets(seed):
    rng = np.random.default_rng(7000 + seed)
    n_in = int(rng.integers(1, 4))
    ns = 2 if seed % 3 else 3
    layers, outs = random_mimo(rng, n_in, int(rng.integers(1, 6)))
    if len(layers) + n_in + 1 > (11 if ns == 3 else 15):
        pytest.skip("too many assignments for the exhaustive search")
    g = build_graph(layers, SHAPE, SCHEMAS3[0], SCHEMAS3[0], SCHEMAS3[:ns], torch_alloc=False,
                    extra_inputs=[SHAPE] * (n_in - 1), outputs=outs)
    t = random_costs(g, rng)
    check_against_oracle(g, t)
    # the library's own exhaustive search agrees
    lc_ref, _, _ = oracle.brute_force(
        np.array([oracle.fastest_per_schema(t["schema"][t["layer"] == i], t["cost"][t["layer"] == i],
                                            t["n_schemas"]) for i in range(t["n_layers"])]),
        t["edges"], t["adapt"])
    try:
        tot, _, _ = g.select_path(SN_SELECT_BRUTE)
        assert tot == lc_ref
    except SnError as e:
        assert lc_ref == oracle.INF and e.status == _sn.SN_EINFEASIBLE


def test_oracle_net_with_two_inputs():
    """The oracle's multi-input forward: a side input of zeros added to a
    branch leaves the single-input result unchanged, and ids -1 / -2 pick
    the first / second array."""
    from oracle.net import run_net
    rng = np.random.default_rng(3)
    conv = dict(_conv1x1(4), inputs=[-1])
    conv["weight"] = rng.standard_normal((4, 4, 1, 1)).astype(np.float32)
    conv["params"] = dict(conv["params"], act="none")
    x = rng.standard_normal(SHAPE).astype(np.float32)
    side = rng.standard_normal(SHAPE).astype(np.float32)
    one = run_net([conv], x)
    two = run_net([conv, dict(_add(), inputs=[0, -2])], [x, np.zeros_like(side)])
    assert np.array_equal(one, two)
    swapped = run_net([dict(conv, inputs=[-2])], [side, x])
    assert np.array_equal(swapped, one)
