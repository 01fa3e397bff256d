"""Chained launches of consecutive tensor-core convolutions (SN_OPT_CHAIN).

The plan runs every run of two or more conv2/igemm_tc layers as one
persistent launch whose tiles wait on the tiles they read.  The routine and
its parameters per layer are those of the selected path, so:
  * with every conv on a tensor-core variant that has no K split, the chained
    run gives the same bits as one launch per layer;
  * with mixed variants (every output-channel tile width, one or two channel
    blocks per stage, CTA pairs and K splits in the per-layer run) both runs
    match the oracle within the fp16/bf16 tolerance;
  * a whole profiled ResNet-50 at batch 32 runs chained, sampled images
    against the oracle;
and the plan counts one launch per chain.
The nets are ResNet-50 (residual adds fused into their convs) at a small
input, so that the later stages have ragged tiles (pixel counts and channel
counts that are not multiples of the tile) and few tiles per layer.
"""
import numpy as np
import pytest

import synth
from oracle.net import run_net
from paper_2110_06037_gb300 import (SN_OPT_CHAIN, SN_OPT_CUDA_GRAPH, SN_SELECT_DPRS, build_graph, fuse_residual,
                                    routine_name)

from gpu_helpers import TOL, from_device, maxrel, raw_bits, to_device

pytestmark = pytest.mark.gpu


def _force_tc(g, layers, pick):
    """Every conv layer on conv2/igemm_tc (variant chosen by pick(layer, n_variants)) in
    the NHWC schema; every other layer on its first candidate."""
    t = g.cost_table()
    uni = g.schema_universe()
    path, tc_layers = [], 0
    for i in range(t["n_layers"]):
        idx = np.flatnonzero(t["layer"] == i)
        tc = [c for c in idx if routine_name(int(t["routine"][c])) == "conv2/igemm_tc"
              and uni[t["schema"][c]][1] == "nhwc" and t["out_schema"][c] == t["schema"][c]]
        if tc:
            tc_layers += 1
            path.append(int(tc[pick(i, len(tc)) % len(tc)]))
        else:
            nhwc = [c for c in idx if uni[t["schema"][c]][1] == "nhwc"]
            path.append(int(nhwc[0] if nhwc else idx[0]))
    g.set_path(path)
    return tc_layers


def _run(g, xd, chain, graph=False):
    import torch
    g.set_option(SN_OPT_CHAIN, 1 if chain else 0)
    g.set_option(SN_OPT_CUDA_GRAPH, 1 if graph else 0)
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        y = g.run(xd)
        y2 = g.run(xd)  # a second launch: the completion counters were reset by the first
    s.synchronize()
    assert torch.equal(y, y2)
    return y


@pytest.mark.parametrize("dt", ["bf16", "f16"])
def test_chained_run_equals_per_layer_launches_bit_for_bit(dt):
    import torch
    x, layers = synth.resnet50(2, res=64)
    fused = fuse_residual(layers, x.shape)
    sch = (dt, "nhwc")
    g = build_graph(fused, x.shape, (dt, "nchw"), (dt, "nchw"), [sch])
    n_tc = _force_tc(g, fused, lambda i, n: 0)  # variant 0: 64-channel tiles, one CTA, no K split
    assert n_tc >= 50
    xd = to_device(x, (dt, "nchw"))
    y_chain = _run(g, xd, chain=True)
    _, k_chain = g.plan_stats()
    y_layer = _run(g, xd, chain=False)
    _, k_layer = g.plan_stats()
    assert k_chain < k_layer - 40, (k_chain, k_layer)
    assert np.array_equal(raw_bits(y_chain), raw_bits(y_layer))
    ref = run_net(layers, x, dt)
    assert maxrel(from_device(y_chain, (dt, "nchw")), ref) <= TOL[dt]
    # replayed from a CUDA graph: the same bits again
    y_graph = _run(g, xd, chain=True, graph=True)
    assert torch.equal(y_graph, y_chain)


@pytest.mark.parametrize("seed", [1, 2, 3])
def test_chained_run_with_mixed_variants_matches_oracle(seed):
    x, layers = synth.resnet50(2, res=96, seed=seed)
    fused = fuse_residual(layers, x.shape)
    g = build_graph(fused, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), [("bf16", "nhwc")])
    rng = np.random.default_rng(seed)
    _force_tc(g, fused, lambda i, n: int(rng.integers(0, n)))
    xd = to_device(x, ("bf16", "nchw"))
    ref = run_net(layers, x, "bf16")
    y_chain = from_device(_run(g, xd, chain=True), ("bf16", "nchw"))
    y_layer = from_device(_run(g, xd, chain=False), ("bf16", "nchw"))
    assert maxrel(y_chain, ref) <= TOL["bf16"]
    assert maxrel(y_layer, ref) <= TOL["bf16"]


def test_profiled_resnet50_b32_runs_chained():
    import torch
    x, layers = synth.resnet50(32)
    fused = fuse_residual(layers, x.shape)
    g = build_graph(fused, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), [("bf16", "nchw"), ("bf16", "nhwc")])
    g.profile(warmup=1, iters=3, topk=1, passes=2)
    g.select_path(SN_SELECT_DPRS)
    g.set_option(SN_OPT_CHAIN, 1)
    y = g.run(to_device(x, ("bf16", "nchw")))
    torch.cuda.synchronize()
    n_ops, n_kern = g.plan_stats()
    assert n_kern < n_ops - 20, (n_ops, n_kern)  # the conv layers run as a chain
    got = from_device(y, ("bf16", "nchw"))
    for n in (0, 23):
        ref = run_net(layers, x[n:n + 1], "bf16")
        assert maxrel(got[n:n + 1], ref) <= TOL["bf16"]
