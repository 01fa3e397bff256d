"""The tensor-core convolution that writes the next layer's layout: reading
NHWC, its epilogue stores the result in NCHW of the same dtype (a fused
boundary, offered to DPRS as a (read, written) candidate).  Its output must be
bit for bit the plain routine's NHWC output permuted by the adapt routine,
for every routine-parameter combination that offers it (no K split), with
and without the fused residual input, at ragged sizes."""
import numpy as np
import pytest

from paper_2110_06037_gb300 import SN_OPT_CUDA_GRAPH, build_graph, routine_name

from gpu_helpers import raw_bits, to_device

pytestmark = pytest.mark.gpu

LAM = [("bf16", "nhwc"), ("bf16", "nchw")]


def _net(rng, C, K, k, s, res):
    w = (rng.standard_normal((K, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    b = (rng.standard_normal(K) * 0.1).astype(np.float32)
    return [{"type": "conv2", "inputs": [-1, -2] if res else [-1],
             "params": dict(c_in=C, c_out=K, kh=k, kw=k, sh=s, sw=s, ph=k // 2, pw=k // 2, act="relu"),
             "weight": w, "bias": b}]


@pytest.mark.parametrize("shape", [(4, 64, 128, 14, 3, 1, False), (4, 64, 64, 7, 1, 1, True),
                                   (2, 128, 256, 10, 3, 2, False), (3, 64, 192, 9, 1, 1, True)])
def test_nchw_writer_equals_conv_then_adapt(shape):
    import torch
    N, C, K, H, k, s, res = shape
    rng = np.random.default_rng(N + C + K + H)
    P = (H + 2 * (k // 2) - k) // s + 1
    layers = _net(rng, C, K, k, s, res)
    x = rng.standard_normal((N, C, H, H)).astype(np.float32)
    r = rng.standard_normal((N, K, P, P)).astype(np.float32)
    g = build_graph(layers, x.shape, LAM[0], LAM[1], LAM, extra_inputs=[(N, K, P, P)] if res else ())
    g.set_option(SN_OPT_CUDA_GRAPH, 0)
    t = g.cost_table()
    conv = t["n_layers"] - 2
    io = [int(np.flatnonzero((t["layer"] == i))[0]) for i in range(t["n_layers"])]
    tc = [int(c) for c in np.flatnonzero(t["layer"] == conv) if routine_name(int(t["routine"][c])) == "conv2/igemm_tc"
          and t["schema"][c] == 0]
    fused = [c for c in tc if t["out_schema"][c] == 1]
    plain = {int(t["variant"][c]): c for c in tc if t["out_schema"][c] == 0}
    assert fused, "no NCHW-writing candidate"
    ins = [to_device(x, LAM[0])] + ([to_device(r, LAM[0])] if res else [])
    for c in fused:
        outs = []
        for cand in (c, plain[int(t["variant"][c])]):
            path = list(io)
            path[conv] = cand
            g.set_path(path)
            y = g.run_multi(ins)[0] if res else g.run(ins[0])
            torch.cuda.synchronize()
            outs.append(raw_bits(y))
        assert np.array_equal(outs[0], outs[1]), g.candidate_desc(c)
        # the fused path has no adapt launch before the output layer
        path = list(io)
        path[conv] = c
        g.set_path(path)
        n_ops, _ = g.plan_stats()
        assert n_ops == 1


@pytest.mark.parametrize("shape", [(2, 3, 64, 40, 7), (3, 4, 32, 29, 5)])
def test_space_to_depth_stem_reads_and_writes_either_layout(shape):
    """The space-to-depth stem (stride-2 conv of <= 4 channels) reads NCHW or
    NHWC (the layout change fused into its re-layout kernel) and writes NHWC
    or NCHW (its GEMM's TMA store or NCHW epilogue): every (read, written)
    pair of every routine parameter gives the same bits as the NHWC -> NHWC
    candidate of that parameter with the net's adapts around it, and matches
    the oracle."""
    import torch
    from oracle.net import run_layer
    from gpu_helpers import TOL, from_device, maxrel, stored_values
    N, C, K, H, k = shape
    rng = np.random.default_rng(N * 7 + C + K + H + k)
    w = (rng.standard_normal((K, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    b = (rng.standard_normal(K) * 0.1).astype(np.float32)
    layer = {"type": "conv2", "inputs": [-1],
             "params": dict(c_in=C, c_out=K, kh=k, kw=k, sh=2, sw=2, ph=k // 2, pw=k // 2, act="relu"),
             "weight": w, "bias": b}
    x = rng.standard_normal((N, C, H, H)).astype(np.float32)
    ref = run_layer(layer, [stored_values(x, "bf16")], "bf16")
    for io_sch in LAM:  # the net's input and output schema (adapts where a candidate differs)
        g = build_graph([layer], x.shape, io_sch, io_sch, LAM)
        g.set_option(SN_OPT_CUDA_GRAPH, 0)
        t = g.cost_table()
        io = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
        s2d = [int(c) for c in np.flatnonzero(t["layer"] == 1) if routine_name(int(t["routine"][c])) == "conv2/s2d_tc"]
        pairs = {(int(t["schema"][c]), int(t["out_schema"][c])) for c in s2d}
        assert pairs == {(0, 0), (0, 1), (1, 0), (1, 1)}, pairs
        xd = to_device(x, io_sch)
        base = {}
        for c in sorted(s2d, key=lambda c: (t["schema"][c], t["out_schema"][c]) != (0, 0)):
            path = list(io)
            path[1] = c
            g.set_path(path)
            y = g.run(xd)
            torch.cuda.synchronize()
            v = int(t["variant"][c])
            if v not in base:  # the NHWC -> NHWC candidate of this parameter comes first
                base[v] = raw_bits(y)
                assert maxrel(from_device(y, io_sch), ref) <= TOL["bf16"], g.candidate_desc(c)
            assert np.array_equal(raw_bits(y), base[v]), g.candidate_desc(c)
