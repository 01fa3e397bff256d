"""Every conv2/igemm_tc variant the tuner can pick, at the ResNet-50 batch-32
conv shapes (bf16 NHWC, full size), against the oracle on sampled outputs.

For each unique shape (input channels, output channels, input size, kernel,
stride, with or without the fused residual input) the layer runs once per
routine-parameter combination offered for it, and a fixed sample of output
pixels (corners and edges, where the zero padding is read, the last pixel of
the ragged tail, and random ones) is compared, every output channel, with the
oracle's fp64 convolution of the same stored inputs and weights: the receptive
field of each sampled pixel is cut out (zero-padded) and fed to
oracle.conv2d as a one-pixel image.  Bars: normwise max relative error <= 2e-2
(the fp16/bf16 tolerance) and, per element, |got - ref| <= 1e-2 |ref| +
2e-3 max|ref| (one bf16 rounding of the output is 2^-8 relative)."""
import numpy as np
import pytest

import oracle
from paper_2110_06037_gb300 import SN_OPT_CUDA_GRAPH, build_graph, routine_name

from gpu_helpers import from_device, maxrel, stored_values, to_device

pytestmark = pytest.mark.gpu

# (C, K, H_in, k, stride, residual): the unique conv shapes of ResNet-50 v1.5
# at batch 32 (residual: the conv that the residual add is fused into)
SHAPES = [
    (64, 64, 56, 1, 1, False), (64, 64, 56, 3, 1, False), (64, 256, 56, 1, 1, True),
    (256, 64, 56, 1, 1, False), (256, 128, 56, 1, 1, False), (128, 128, 56, 3, 2, False),
    (128, 512, 28, 1, 1, True), (256, 512, 56, 1, 2, True), (512, 128, 28, 1, 1, False),
    (128, 128, 28, 3, 1, False), (512, 256, 28, 1, 1, False), (256, 256, 28, 3, 2, False),
    (256, 1024, 14, 1, 1, True), (512, 1024, 28, 1, 2, True), (1024, 256, 14, 1, 1, False),
    (256, 256, 14, 3, 1, False), (1024, 512, 14, 1, 1, False), (512, 512, 14, 3, 2, False),
    (512, 2048, 7, 1, 1, True), (1024, 2048, 14, 1, 2, True), (2048, 512, 7, 1, 1, False),
    (512, 512, 7, 3, 1, False),
]
N = 32
SCH = ("bf16", "nhwc")


def _layer(rng, C, K, k, s, res):
    pad = k // 2
    w = (rng.standard_normal((K, C, k, k)) * np.sqrt(2.0 / (C * k * k))).astype(np.float32)
    b = (rng.standard_normal(K) * 0.1).astype(np.float32)
    return {"type": "conv2", "inputs": [-1, -2] if res else [-1],
            "params": dict(c_in=C, c_out=K, kh=k, kw=k, sh=s, sw=s, ph=pad, pw=pad, act="relu"),
            "weight": w, "bias": b}


def _sample(rng, P):
    """Output pixels (n, p, q): the four corners of the first and last image,
    edge pixels, the last pixel, and random ones."""
    pts = {(0, 0, 0), (0, 0, P - 1), (0, P - 1, 0), (0, P - 1, P - 1), (N - 1, P - 1, P - 1),
           (N - 1, 0, P // 2), (N // 2, P // 2, 0), (N // 2, P - 1, P // 2)}
    while len(pts) < 48:
        pts.add((int(rng.integers(0, N)), int(rng.integers(0, P)), int(rng.integers(0, P))))
    return sorted(pts)


def _reference(x64, w, b, r64, pts, k, s):
    """The oracle on each sampled pixel's receptive field (a k x k one-pixel image)."""
    pad = k // 2
    C = x64.shape[1]
    xp = np.zeros((N, C, x64.shape[2] + 2 * pad, x64.shape[3] + 2 * pad))
    xp[:, :, pad:pad + x64.shape[2], pad:pad + x64.shape[3]] = x64
    patches = np.stack([xp[n, :, p * s:p * s + k, q * s:q * s + k] for (n, p, q) in pts])
    y = oracle.conv2d(patches, oracle.round_to(w, "bf16"), b, stride=(1, 1), pad=(0, 0), act="none")[:, :, 0, 0]
    if r64 is not None:
        y = y + np.stack([r64[n, :, p, q] for (n, p, q) in pts])
    return np.maximum(y, 0.0)


@pytest.mark.parametrize("shape", SHAPES, ids=lambda t: "%d-%d_%d_k%ds%d%s" % (t[0], t[1], t[2], t[3], t[4],
                                                                            "_res" if t[5] else ""))
def test_every_tensor_core_variant_at_full_size(shape):
    import torch
    C, K, H, k, s, res = shape
    rng = np.random.default_rng(C * 7 + K + H * 13 + k + s)
    P = (H + 2 * (k // 2) - k) // s + 1
    layer = _layer(rng, C, K, k, s, res)
    x = rng.standard_normal((N, C, H, H)).astype(np.float32)
    r = rng.standard_normal((N, K, P, P)).astype(np.float32) if res else None
    g = build_graph([layer], x.shape, SCH, SCH, [SCH], extra_inputs=[(N, K, P, P)] if res else ())
    g.set_option(SN_OPT_CUDA_GRAPH, 0)
    t = g.cost_table()
    io = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
    tc = [int(c) for c in np.flatnonzero(t["layer"] == t["n_layers"] - 2)
          if routine_name(int(t["routine"][c])) == "conv2/igemm_tc"]
    assert tc, "no tensor-core variant offered"
    pts = _sample(rng, P)
    ref = _reference(stored_values(x, "bf16"), layer["weight"], layer["bias"],
                     stored_values(r, "bf16") if res else None, pts, k, s)
    ins = [to_device(x, SCH)] + ([to_device(r, SCH)] if res else [])
    bad = []
    for c in tc:
        path = list(io)
        path[t["n_layers"] - 2] = c
        g.set_path(path)
        y = g.run_multi(ins)[0] if res else g.run(ins[0])
        torch.cuda.synchronize()
        # sampled pixels of the NHWC output, all channels
        idx = torch.tensor(pts, device=y.device)
        got = y[idx[:, 0], idx[:, 1], idx[:, 2], :].float().cpu().numpy().astype(np.float64)
        err = maxrel(got, ref)
        elem = np.abs(got - ref) <= 1e-2 * np.abs(ref) + 2e-3 * np.abs(ref).max()
        if err > 2e-2 or not elem.all():
            bad.append((g.candidate_desc(c), err, int((~elem).sum())))
    assert not bad, bad
