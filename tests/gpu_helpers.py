"""Helpers for the GPU parity tests: stored-precision transfers and error metric.

Inputs are rounded to the schema's dtype by the oracle's own RNE cast and
uploaded bit for bit, so the GPU and the oracle see identical stored values.
"""
import numpy as np

import oracle

TOL = {"f32": 1e-4, "f16": 2e-2, "bf16": 2e-2}


def torch_dtype(dt):
    import torch
    return {"f32": torch.float32, "f16": torch.float16, "bf16": torch.bfloat16}[dt]


def to_device(x_nchw, schema):
    """fp32 NCHW values -> a CUDA tensor stored in `schema` (RNE by the oracle)."""
    import torch
    dt, lay = schema
    bits = oracle.to_bits(np.asarray(x_nchw, np.float32), dt)
    if lay == "nhwc":
        bits = oracle.nchw_to_nhwc(bits)
    if dt == "f32":
        return torch.from_numpy(np.ascontiguousarray(bits)).cuda()
    return torch.from_numpy(np.ascontiguousarray(bits).view(np.int16)).cuda().view(torch_dtype(dt))


def stored_values(x_nchw, dt):
    """The values the GPU holds for x in dtype dt, widened exactly (fp64)."""
    return oracle.round_to(np.asarray(x_nchw, np.float32), dt).astype(np.float64)


def from_device(t, schema):
    """CUDA tensor in `schema` -> fp64 NCHW values (exact widening)."""
    import torch
    dt, lay = schema
    if dt == "f32":
        a = t.detach().cpu().numpy()
    else:
        a = t.detach().view(torch.int16).cpu().numpy().view(np.uint16)
        a = oracle.from_bits(a, dt)
    if lay == "nhwc":
        a = oracle.nhwc_to_nchw(a)
    return a.astype(np.float64)


def raw_bits(t):
    import torch
    if t.dtype == torch.float32:
        return t.detach().cpu().numpy().view(np.uint32)
    return t.detach().view(torch.int16).cpu().numpy().view(np.uint16)


def maxrel(got, ref):
    """Normwise max relative error: max|got - ref| / max|ref|."""
    got, ref = np.asarray(got, np.float64), np.asarray(ref, np.float64)
    assert got.shape == ref.shape, (got.shape, ref.shape)
    den = max(float(np.abs(ref).max()), 1e-30)
    return float(np.abs(got - ref).max()) / den


def find_candidate(t, layer, routine_name, variant, schema_index):
    from paper_2110_06037_gb300 import routine_name as rn
    for c in range(len(t["cost"])):
        if (t["layer"][c] == layer and rn(int(t["routine"][c])) == routine_name
                and t["variant"][c] == variant and t["schema"][c] == schema_index):
            return c
    return None
