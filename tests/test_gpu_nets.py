"""End-to-end on the GPU: profile -> DPRS -> run, against the oracle.

  * tiny CNN, fp32 (routine paths small enough to enumerate): the DPRS path on
    the profiled cost table equals the oracle's exhaustive search, and the
    output matches the oracle within 1e-4; random forced paths (mixed
    schemas, adapts on edges) match as well.
  * MobileNetV2 b1 fp16, ResNet-50 b1 fp16: DPRS equals the oracle's exact
    block-wise search on the profiled table; output within 2e-2.
  * ResNet-50 b32 bf16: sampled images of the batch against the oracle.
  * VGG16 bf16 (64x64 input, batch 2) and MobileNetV3-Large b1 fp16: DPRS
    equals the block-wise search; output within 2e-2.
  * The same nets with every residual add fused into its conv2: DPRS equals
    the block-wise search, outputs within 2e-2 of the (unfused) oracle.
"""
import numpy as np
import pytest

import oracle
import synth
from oracle.net import run_net
from oracle.paths import blockwise_search
from paper_2110_06037_gb300 import SN_OPT_CUDA_GRAPH, SN_SELECT_BRUTE, SN_SELECT_DPRS, build_graph, fuse_residual

from gpu_helpers import TOL, from_device, maxrel, to_device
from test_dprs import has_fused, oracle_layer_cost, oracle_pair_cost, realised_cost

pytestmark = pytest.mark.gpu

F32 = [("f32", "nchw"), ("f32", "nhwc")]
F16 = [("f16", "nchw"), ("f16", "nhwc")]
BF16 = [("bf16", "nchw"), ("bf16", "nhwc")]


def _exact_pair_total(t):
    """The exact optimum of the pair problem (some routine writes another
    schema): the oracle's block-wise search over (read, written) states."""
    lcp, pairs = oracle_pair_cost(t)
    return blockwise_search(lcp, t["edges"], t["adapt"], pairs=pairs)[0]


def _profile_select_run(layers, x, in_schema, out_schema, schemas, exhaustive, warmup=1, iters=5):
    import torch
    g = build_graph(layers, x.shape, in_schema, out_schema, schemas)
    g.profile(warmup=warmup, iters=iters, topk=2, passes=3)
    t = g.cost_table()
    if has_fused(t):
        total, sch, cand = g.select_path(SN_SELECT_DPRS)
        assert total == _exact_pair_total(t)
        assert realised_cost(t, cand) == total
        y = g.run(to_device(x, in_schema))
        torch.cuda.synchronize()
        return g, from_device(y, out_schema)
    lc = oracle_layer_cost(t)
    if exhaustive:
        ref_total, ref_asg, nmin = oracle.brute_force(lc, t["edges"], t["adapt"])
    else:
        ref_total, ref_asg = blockwise_search(lc, t["edges"], t["adapt"])
        nmin = None
    total, sch, cand = g.select_path(SN_SELECT_DPRS)
    assert total == ref_total
    assert oracle.path_cost(lc, t["edges"], t["adapt"], sch) == ref_total
    if nmin == 1:
        assert list(sch) == list(ref_asg)
    y = g.run(to_device(x, in_schema))
    torch.cuda.synchronize()
    return g, from_device(y, out_schema)


def test_tiny_cnn_fp32_profile_dprs_run():
    x, layers = synth.tiny_cnn()
    g, got = _profile_select_run(layers, x, ("f32", "nchw"), ("f32", "nchw"), F32, exhaustive=True)
    total_b, _, _ = g.select_path(SN_SELECT_BRUTE)
    total_d, _, _ = g.select_path(SN_SELECT_DPRS)
    assert total_b == total_d
    ref = run_net(layers, x, "f32")
    assert maxrel(got, ref) <= TOL["f32"]


def test_tiny_cnn_random_forced_paths():
    import torch
    x, layers = synth.tiny_cnn()
    ref = run_net(layers, x, "f32")
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nhwc"), F32)
    t = g.cost_table()
    rng = np.random.default_rng(0)
    xd = to_device(x, ("f32", "nchw"))
    for _ in range(12):
        pc = [int(rng.choice(np.flatnonzero(t["layer"] == i))) for i in range(t["n_layers"])]
        g.set_path(pc)
        y = g.run(xd)
        torch.cuda.synchronize()
        assert maxrel(from_device(y, ("f32", "nhwc")), ref) <= TOL["f32"]


def test_mixed_precision_schemas_tiny():
    """fp16 and fp32 schemas in one net: adapts cast between them."""
    import torch
    x, layers = synth.tiny_cnn()
    sch = [("f32", "nchw"), ("f16", "nhwc")]
    g = build_graph(layers, x.shape, ("f32", "nchw"), ("f32", "nchw"), sch)
    t = g.cost_table()
    rng = np.random.default_rng(1)
    xd = to_device(x, ("f32", "nchw"))
    ref = run_net(layers, x, "f32")
    for _ in range(6):
        pc = [int(rng.choice(np.flatnonzero(t["layer"] == i))) for i in range(t["n_layers"])]
        g.set_path(pc)
        y = g.run(xd)
        torch.cuda.synchronize()
        assert maxrel(from_device(y, ("f32", "nchw")), ref) <= TOL["f16"]


def test_mobilenet_v2_b1_fp16():
    x, layers = synth.mobilenet_v2(1)
    g, got = _profile_select_run(layers, x, ("f16", "nchw"), ("f16", "nchw"), F16, exhaustive=False)
    ref = run_net(layers, x, "f16")
    assert maxrel(got, ref) <= TOL["f16"]


def test_mobilenet_v3_b1_fp16():
    """MobileNetV3-Large: hard swish / hard sigmoid, squeeze-excite scales."""
    x, layers = synth.mobilenet_v3(1)
    g, got = _profile_select_run(layers, x, ("f16", "nchw"), ("f16", "nchw"), F16, exhaustive=False)
    ref = run_net(layers, x, "f16")
    assert maxrel(got, ref) <= TOL["f16"]


def test_vgg16_bf16():
    """VGG16 (fc6 as a whole-map convolution) at a 64x64 input, batch 2."""
    x, layers = synth.vgg16(2, res=64)
    g, got = _profile_select_run(layers, x, ("bf16", "nchw"), ("bf16", "nchw"), BF16, exhaustive=False)
    ref = run_net(layers, x, "bf16")
    assert maxrel(got, ref) <= TOL["bf16"]


def test_resnet50_b1_fp16_and_graph_replay():
    import torch
    x, layers = synth.resnet50(1)
    g, got = _profile_select_run(layers, x, ("f16", "nchw"), ("f16", "nchw"), F16, exhaustive=False)
    ref = run_net(layers, x, "f16")
    assert maxrel(got, ref) <= TOL["f16"]
    # CUDA-graph replay gives the same bits as eager launches
    xd = to_device(x, ("f16", "nchw"))
    s = torch.cuda.Stream()
    with torch.cuda.stream(s):
        y1 = g.run(xd)
        g.set_option(SN_OPT_CUDA_GRAPH, 1)
        y2 = g.run(xd)
        y3 = g.run(xd)
    s.synchronize()
    assert torch.equal(y1, y2) and torch.equal(y2, y3)


def test_resnet50_b32_bf16_sampled():
    import torch
    x, layers = synth.resnet50(32)
    g = build_graph(layers, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), BF16)
    g.profile(warmup=1, iters=3, topk=1, passes=2)
    t = g.cost_table()
    if has_fused(t):
        ref_total = _exact_pair_total(t)
    else:
        ref_total, _ = blockwise_search(oracle_layer_cost(t), t["edges"], t["adapt"])
    total, sch, _ = g.select_path(SN_SELECT_DPRS)
    assert total == ref_total
    y = g.run(to_device(x, ("bf16", "nchw")))
    torch.cuda.synchronize()
    got = from_device(y, ("bf16", "nchw"))
    for n in (0, 31):
        ref = run_net(layers, x[n:n + 1], "bf16")
        assert maxrel(got[n:n + 1], ref) <= TOL["bf16"]


def test_fused_mobilenet_v2_b1_fp16():
    x, layers = synth.mobilenet_v2(1)
    fused = fuse_residual(layers, x.shape)
    g, got = _profile_select_run(fused, x, ("f16", "nchw"), ("f16", "nchw"), F16, exhaustive=False)
    assert maxrel(got, run_net(layers, x, "f16")) <= TOL["f16"]


def test_fused_resnet50_b1_fp16():
    x, layers = synth.resnet50(1)
    fused = fuse_residual(layers, x.shape)
    g, got = _profile_select_run(fused, x, ("f16", "nchw"), ("f16", "nchw"), F16, exhaustive=False)
    assert maxrel(got, run_net(layers, x, "f16")) <= TOL["f16"]


def test_fused_resnet50_b32_bf16_sampled():
    import torch
    x, layers = synth.resnet50(32)
    fused = fuse_residual(layers, x.shape)
    g = build_graph(fused, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), BF16)
    g.profile(warmup=1, iters=3, topk=1, passes=2)
    t = g.cost_table()
    if has_fused(t):
        ref_total = _exact_pair_total(t)
    else:
        ref_total, _ = blockwise_search(oracle_layer_cost(t), t["edges"], t["adapt"])
    total, sch, _ = g.select_path(SN_SELECT_DPRS)
    assert total == ref_total
    y = g.run(to_device(x, ("bf16", "nchw")))
    torch.cuda.synchronize()
    got = from_device(y, ("bf16", "nchw"))
    for n in (0, 17):
        ref = run_net(layers, x[n:n + 1], "bf16")
        assert maxrel(got[n:n + 1], ref) <= TOL["bf16"]


def test_run_host_copies_inside_the_call():
    """sn_run_host: input from host memory, output to host memory, the copies
    queued by the library on the caller's stream; same bits as sn_run on
    device buffers, pinned or pageable host memory, eager or graph replay."""
    import torch
    x, layers = synth.resnet50(2, res=64)
    fused = fuse_residual(layers, x.shape)
    g = build_graph(fused, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), BF16)
    g.profile(warmup=1, iters=2, topk=1, passes=1)
    g.select_path(SN_SELECT_DPRS)
    xd = to_device(x, ("bf16", "nchw"))
    ref = g.run(xd)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    for graph in (0, 1):
        g.set_option(SN_OPT_CUDA_GRAPH, graph)
        for pinned in (True, False):
            xh = xd.cpu().pin_memory() if pinned else xd.cpu()
            oh = torch.empty(ref.shape, dtype=ref.dtype).pin_memory() if pinned else torch.empty(ref.shape, dtype=ref.dtype)
            for _ in range(2):
                g.run_host(xh, oh, stream=s)
            s.synchronize()
            assert torch.equal(oh, ref.cpu()), (graph, pinned)


def test_run_host_back_to_back_calls_keep_their_inputs():
    """Consecutive sn_run_host calls without a synchronisation in between,
    each on its own pinned input and output: the uploads go through two
    landing buffers used in turn on the graph's copy stream, so a call's
    upload overlaps the previous call's net; every output must still be the
    one of its own input (same bits as sn_run on that input)."""
    import torch
    x, layers = synth.resnet50(2, res=64)
    g = build_graph(layers, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), BF16, fuse=True)
    g.profile(warmup=1, iters=2, topk=1, passes=1)
    g.select_path(SN_SELECT_DPRS)
    rng = np.random.default_rng(3)
    xs = [to_device((x * rng.uniform(0.5, 1.5)).astype(np.float32), ("bf16", "nchw")) for _ in range(5)]
    refs = [g.run(xd).clone() for xd in xs]
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    for graph in (0, 1):
        g.set_option(SN_OPT_CUDA_GRAPH, graph)
        xh = [xd.cpu().pin_memory() for xd in xs]
        oh = [torch.empty(refs[0].shape, dtype=refs[0].dtype).pin_memory() for _ in xs]
        for _ in range(2):
            for i in range(len(xs)):
                g.run_host(xh[i], oh[i], stream=s)
        s.synchronize()
        for i in range(len(xs)):
            assert torch.equal(oh[i], refs[i].cpu()), (graph, i)


@pytest.mark.parametrize("chain", [0, 1])
def test_liveness_arena_same_bits_less_memory(chain):
    """Activations placed by liveness in one arena give the same bits as one
    place per blob, with and without chained launches, and take less memory
    without them (ResNet-50, profiled path, batch 2)."""
    import torch
    from paper_2110_06037_gb300 import SN_OPT_CHAIN, SN_OPT_SHARE_BUFFERS
    x, layers = synth.resnet50(2, res=96)
    g = build_graph(layers, x.shape, ("bf16", "nchw"), ("bf16", "nchw"), BF16, fuse=True)
    g.profile(warmup=1, iters=2, topk=1, passes=1)
    g.select_path(SN_SELECT_DPRS)
    g.set_option(SN_OPT_CHAIN, chain)
    xd = to_device(x, ("bf16", "nchw"))
    g.set_option(SN_OPT_SHARE_BUFFERS, 0)
    y0 = g.run(xd).clone()
    a0, u0 = g.plan_memory()
    g.set_option(SN_OPT_SHARE_BUFFERS, 1)
    y1 = g.run(xd)
    y2 = g.run(xd)
    torch.cuda.synchronize()
    a1, u1 = g.plan_memory()
    assert u0 == u1 and a0 == u0
    # a chained launch keeps everything it touches live across the chain, so
    # sharing then only happens outside it
    assert a1 <= u1 if chain else a1 < 0.5 * u1, (a1, u1)
    assert torch.equal(y0, y1) and torch.equal(y1, y2)
    ref = run_net(layers, x, "bf16")
    assert maxrel(from_device(y1, ("bf16", "nchw")), ref) <= TOL["bf16"]
