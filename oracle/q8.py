"""Oracle for the qint8 schema (section II-C quantisation; hybrid tuning of
section V-C, Table I).

TEST INFRASTRUCTURE ONLY (see the package docstring).

Section II-C writes a quantised value as q = c + round(x / s) with an
integer offset c and a real scale s, and calls the offset-free form
symmetric.  The qint8 schema here is that symmetric form on 8-bit codes:

  * an activation blob has one scale s > 0; its codes are
        q = clamp(round(x * (1/s)), -127, 127)
    (round half to even, 1/s rounded to fp32 once) and it stands for the
    values q * s;
  * a weight tensor has one scale per output channel,
        s_w[k] = max_j |W[k, j]| / 127   (1 for an all-zero channel),
    and codes clamp(round(W[k, j] / s_w[k]), -127, 127);
  * a qint8 routine sums code products exactly (integers) and then, in fp32
    with every operation rounded to nearest even on its own,
        y = float(acc) * (s_x * s_w[k]) + bias[k]  (+ q_r * s_r: residual)
        y = act(y)
        q_y = clamp(round(y * (1/s_y)), -127, 127).

The paper fixes neither the rounding of each step nor their order; the
reading above (one fp32 rounding per written operation, in the order
written) is what both this oracle and the GPU routines compute, so their
codes agree bit for bit.  numpy float32 arithmetic rounds every operation to
nearest even and never fuses a multiply-add, which is exactly that reading.
Integer sums use int64, which is exact for every size the nets reach.
"""
from __future__ import annotations

import numpy as np

F32 = np.float32
QMAX = 127


def inv_scale(s) -> np.float32:
    """1/s rounded to fp32 (the multiplier every quantising step uses)."""
    return F32(1.0) / F32(s)


def requantize(y, s_out) -> np.ndarray:
    """fp32 values -> int8 codes of scale s_out: clamp(round(y * (1/s)))."""
    y = np.asarray(y, dtype=F32)
    t = y * inv_scale(s_out)
    return np.clip(np.rint(t), -QMAX, QMAX).astype(np.int8)


def quantize(x, s) -> np.ndarray:
    """Quantise adapt (float blob -> qint8 blob of scale s).  x is taken as
    fp32 values (an fp16/bf16 blob widens to fp32 exactly first)."""
    return requantize(np.asarray(x, dtype=F32), s)


def dequantize(q, s) -> np.ndarray:
    """Dequantise adapt: the fp32 values q * s (one rounding)."""
    return np.asarray(q).astype(F32) * F32(s)


def quantize_weights(w):
    """Per-output-channel symmetric weights: (codes int8 like w, s_w fp32 [K])."""
    w = np.asarray(w, dtype=F32)
    k = w.shape[0]
    a = np.abs(w.reshape(k, -1)).max(axis=1)
    s = np.where(a > 0, a / F32(QMAX), F32(1.0)).astype(F32)
    t = w / s.reshape((k,) + (1,) * (w.ndim - 1))
    return np.clip(np.rint(t), -QMAX, QMAX).astype(np.int8), s


def act_f32(y, act: str):
    """The fused activations on fp32 values, one rounding per operation."""
    y = np.asarray(y, dtype=F32)
    if act in (None, "none"):
        return y
    if act == "relu":
        return np.maximum(y, F32(0))
    if act == "relu6":
        return np.minimum(np.maximum(y, F32(0)), F32(6))
    t = np.minimum(np.maximum(y + F32(3), F32(0)), F32(6)) / F32(6)  # hard sigmoid
    if act == "hsigmoid":
        return t
    if act == "hswish":
        return y * t
    raise ValueError(act)


def finish(y, s_out, out_dtype=None):
    """The output of a qint8 routine from its fp32 result y: codes of scale
    s_out, or, for a routine that writes a float schema (dequantisation fused
    into its epilogue), y rounded to nearest even in that dtype (returned as
    fp32 values)."""
    if out_dtype in (None, "qi8"):
        return requantize(y, s_out)
    from . import round_to
    return round_to(np.asarray(y, dtype=F32), out_dtype)


def _epilogue(acc, m, bias, act, s_out, resid=None, out_dtype=None):
    """acc: int64 [N, K, ...]; m: fp32 [K] multipliers s_x * s_w[k]."""
    shape = (1, -1) + (1,) * (acc.ndim - 2)
    y = acc.astype(F32) * m.reshape(shape)
    if bias is not None:
        y = y + np.asarray(bias, dtype=F32).reshape(shape)
    if resid is not None:
        qr, sr = resid
        y = y + dequantize(qr, sr)
    return finish(act_f32(y, act), s_out, out_dtype)


def conv_acc(qx, qw, stride=(1, 1), pad=(0, 0), dil=(1, 1), groups=1) -> np.ndarray:
    """Exact integer cross-correlation sums of int8 NCHW codes with int8
    [K, C/groups, R, S] codes, zero padding: int64 [N, K, P, Q]."""
    qx = np.asarray(qx).astype(np.int64)
    qw = np.asarray(qw).astype(np.int64)
    n, c, h, w = qx.shape
    k, cg, r, s = qw.shape
    sh, sw = stride
    ph, pw = pad
    dh, dw = dil
    p = (h + 2 * ph - dh * (r - 1) - 1) // sh + 1
    q = (w + 2 * pw - dw * (s - 1) - 1) // sw + 1
    xp = np.zeros((n, c, h + 2 * ph, w + 2 * pw), np.int64)
    xp[:, :, ph:ph + h, pw:pw + w] = qx
    kg = k // groups
    out = np.zeros((n, k, p, q), np.int64)
    for g in range(groups):
        xs = xp[:, g * cg:(g + 1) * cg]
        ws = qw[g * kg:(g + 1) * kg]
        for i in range(r):
            for j in range(s):
                win = xs[:, :, i * dh:i * dh + sh * (p - 1) + 1:sh, j * dw:j * dw + sw * (q - 1) + 1:sw]
                out[:, g * kg:(g + 1) * kg] += np.einsum("nchw,kc->nkhw", win, ws[:, :, i, j])
    return out


def conv2d(qx, s_x, qw, s_w, bias, s_out, stride=(1, 1), pad=(0, 0), dil=(1, 1), groups=1,
           act="none", resid=None, out_dtype=None) -> np.ndarray:
    """qint8 conv2 / dwconv2 (groups = C): codes of y = act(conv + bias [+ residual]).
    resid = (codes, scale) of a residual blob shaped like the output."""
    acc = conv_acc(qx, qw, stride, pad, dil, groups)
    m = F32(s_x) * np.asarray(s_w, dtype=F32)
    return _epilogue(acc, m, bias, act, s_out, resid, out_dtype)


def dense(qx, s_x, qw, s_w, bias, s_out, act="none", out_dtype=None) -> np.ndarray:
    """qint8 dense on an N x C (x 1 x 1) blob: y = act(W x + b)."""
    qx = np.asarray(qx)
    shp = qx.shape
    x2 = qx.reshape(shp[0], -1).astype(np.int64)
    acc = x2 @ np.asarray(qw).astype(np.int64).T
    m = F32(s_x) * np.asarray(s_w, dtype=F32)
    y = _epilogue(acc, m, bias, act, s_out, out_dtype=out_dtype)
    return y.reshape((shp[0], -1) + shp[2:]) if len(shp) == 4 else y


def maxpool2d(qx, s_x, s_out, k=(3, 3), stride=(2, 2), pad=(1, 1), out_dtype=None) -> np.ndarray:
    """Max over the window's in-image codes (padding never wins), then the
    maximum's value q * s_x requantised to s_out."""
    qx = np.asarray(qx).astype(np.int64)
    n, c, h, w = qx.shape
    kh, kw = k
    sh, sw = stride
    ph, pw = pad
    p = (h + 2 * ph - kh) // sh + 1
    q = (w + 2 * pw - kw) // sw + 1
    xp = np.full((n, c, h + 2 * ph, w + 2 * pw), -(1 << 20), np.int64)
    xp[:, :, ph:ph + h, pw:pw + w] = qx
    out = np.full((n, c, p, q), -(1 << 20), np.int64)
    for i in range(kh):
        for j in range(kw):
            out = np.maximum(out, xp[:, :, i:i + sh * (p - 1) + 1:sh, j:j + sw * (q - 1) + 1:sw])
    return finish(dequantize(out, s_x), s_out, out_dtype)


def gap(qx, s_x, s_out, out_dtype=None) -> np.ndarray:
    """Global average pool: the exact code sum over H x W, times s_x, divided
    by H*W (two fp32 roundings), requantised.  Output N x C x 1 x 1."""
    qx = np.asarray(qx).astype(np.int64)
    n, c, h, w = qx.shape
    tot = qx.sum(axis=(2, 3)).astype(F32) * F32(s_x)
    y = tot / F32(h * w)
    return finish(y, s_out, out_dtype).reshape(n, c, 1, 1)


def add(qa, s_a, qb, s_b, s_out, act="none", out_dtype=None) -> np.ndarray:
    """y = act(a + b) with a, b dequantised (one rounding each), one rounded add."""
    y = dequantize(qa, s_a) + dequantize(qb, s_b)
    return finish(act_f32(y, act), s_out, out_dtype)


def mul(qx, s_x, qs, s_s, s_out, act="none", out_dtype=None) -> np.ndarray:
    """Squeeze-and-excite scale y[n,c,h,w] = act(x[n,c,h,w] * s[n,c])."""
    x = dequantize(qx, s_x)
    sc = dequantize(np.asarray(qs).reshape(qx.shape[0], qx.shape[1], 1, 1), s_s)
    return finish(act_f32(x * sc, act), s_out, out_dtype)


def absmax_scale(x) -> np.float32:
    """Calibration: max |x| / 127 in fp32 (1 when x is all zero)."""
    a = F32(np.abs(np.asarray(x, dtype=F32)).max()) if np.size(x) else F32(0)
    return a / F32(QMAX) if a > 0 else F32(1.0)


def run_layer(layer: dict, ins: list, s_ins: list, s_out, out_dtype=None) -> np.ndarray:
    """One layer of a net (the dict format of oracle.net) in the qint8 schema:
    ins are int8 NCHW codes with scales s_ins; returns the output codes (or,
    with out_dtype a float dtype, the fused-dequantisation output values)."""
    o = dict(out_dtype=out_dtype)
    t, p = layer["type"], layer.get("params", {})
    act = p.get("act", "none")
    if t in ("conv2", "dwconv2"):
        qw, s_w = quantize_weights(layer["weight"])
        groups = p.get("groups", 1) if t == "conv2" else p["c_in"]
        resid = (ins[1], s_ins[1]) if len(ins) == 2 else None
        return conv2d(ins[0], s_ins[0], qw, s_w, layer.get("bias"), s_out, stride=(p["sh"], p["sw"]),
                      pad=(p["ph"], p["pw"]), dil=(p.get("dh", 1), p.get("dw", 1)), groups=groups,
                      act=act, resid=resid, **o)
    if t == "dense":
        qw, s_w = quantize_weights(layer["weight"])
        return dense(ins[0], s_ins[0], qw, s_w, layer.get("bias"), s_out, act=act, **o)
    if t == "maxpool":
        return maxpool2d(ins[0], s_ins[0], s_out, k=(p["kh"], p["kw"]), stride=(p["sh"], p["sw"]),
                         pad=(p["ph"], p["pw"]), **o)
    if t == "gap":
        return gap(ins[0], s_ins[0], s_out, **o)
    if t == "add":
        return add(ins[0], s_ins[0], ins[1], s_ins[1], s_out, act=act, **o)
    if t == "mul":
        return mul(ins[0], s_ins[0], ins[1], s_ins[1], s_out, act=act, **o)
    raise ValueError(f"unknown layer type {t}")


def calibrate(layers: list, x, dtype: str = "f32"):
    """Per-blob scales from one float forward pass of the fp64 oracle:
    absmax / 127 of the net input and of every layer's output."""
    from .net import run_net
    from . import round_to
    _, outs = run_net(layers, x, dtype, keep=True)
    x0 = round_to(np.asarray(x, np.float32), dtype)
    return absmax_scale(x0), [absmax_scale(o.astype(F32)) for o in outs]


def run_net_q8(layers: list, x, s_in, scales) -> np.ndarray:
    """The whole net in the qint8 schema: the fp32 input is quantised with
    s_in, every layer runs on codes, and the last layer's codes are
    dequantised (fp32 values)."""
    q0 = quantize(np.asarray(x, F32), s_in)
    outs = []
    for i, layer in enumerate(layers):
        ins = [q0 if j < 0 else outs[j] for j in layer["inputs"]]
        s_ins = [s_in if j < 0 else scales[j] for j in layer["inputs"]]
        outs.append(run_layer(layer, ins, s_ins, scales[i]))
    return dequantize(outs[-1], scales[-1])
