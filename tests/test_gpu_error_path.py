"""The bounded-wait error path of the tensor-core routine, made to run out on
purpose without any fault: SN_OPT_WAIT_LIMIT shortens every pipeline wait of
the kernel to one SM cycle, so the first wait for a TMA copy expires; the
kernel stops, lets its own copies and MMAs land, frees its tensor memory,
records the cause in the library's error word and returns.  sn_run (with
SN_OPT_CHECK) reports SN_ETIMEOUT and clears the word, and the next run on
the same graph, with the default limit, succeeds with the same output as
before."""
import numpy as np
import pytest

import synth
from paper_2110_06037_gb300 import (SN_OPT_CHECK, SN_OPT_CUDA_GRAPH, SN_OPT_WAIT_LIMIT, SnError, _sn, build_graph,
                                    routine_name)

from gpu_helpers import to_device

pytestmark = pytest.mark.gpu


def _one_cta_variant(g):
    """Layer 1 on a one-CTA tensor-core variant with no K split (no cluster)."""
    t = g.cost_table()
    path = [int(np.flatnonzero(t["layer"] == i)[0]) for i in range(t["n_layers"])]
    for c in np.flatnonzero(t["layer"] == 1):
        d = g.candidate_desc(int(c))
        if (routine_name(int(t["routine"][c])) == "conv2/igemm_tc" and "cta=1" in d and "ksplit=1" in d
                and "csk=1" in d and "bst=0" in d):
            path[1] = int(c)
            break
    else:
        pytest.fail("no one-CTA tensor-core variant")
    g.set_path(path)
    return g.candidate_desc(path[1])


def test_expired_wait_reports_timeout_and_the_graph_recovers():
    import torch
    x, layers = synth.single_conv(2, 14, 64, 128, 3, 1)
    sch = ("bf16", "nhwc")
    g = build_graph(layers, x.shape, sch, sch, [sch])
    _one_cta_variant(g)
    g.set_option(SN_OPT_CHECK, 1)
    g.set_option(SN_OPT_CUDA_GRAPH, 0)
    xd = to_device(x, sch)
    y0 = g.run(xd).clone()
    g.set_option(SN_OPT_WAIT_LIMIT, 1)
    with pytest.raises(SnError) as e:
        g.run(xd)
    assert e.value.status == _sn.SN_ETIMEOUT
    assert b"bounded wait" in _sn.lib().sn_last_error()
    g.set_option(SN_OPT_WAIT_LIMIT, 0)
    y1 = g.run(xd)
    torch.cuda.synchronize()
    assert torch.equal(y0, y1)
    # and again, replayed from a CUDA graph
    g.set_option(SN_OPT_CUDA_GRAPH, 1)
    y2 = g.run(xd)
    torch.cuda.synchronize()
    assert torch.equal(y0, y2)


def test_wait_limit_option_is_validated():
    x, layers = synth.single_conv(1, 8, 64, 64, 1, 1)
    sch = ("bf16", "nhwc")
    g = build_graph(layers, x.shape, sch, sch, [sch])
    with pytest.raises(SnError) as e:
        g.set_option(SN_OPT_WAIT_LIMIT, -5)
    assert e.value.status == _sn.SN_EINVAL
