"""Failure detection without a GPU fault: a device wait that runs out is reported, and the
context keeps working.

The self-test kernel waits on an mbarrier that nothing ever completes, through the same
bounded wait the tensor-core kernels use, with a 2 ms limit. It must give up, record the
timeout in the context's status word and return; ec_check_device reports EC_ERR_TIMEOUT
once and clears it; a full forward + backward afterwards still matches a fresh context.
"""
import numpy as np
import pytest
import torch

import paper_2604_01622_gb300 as ec
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer
from tests._util import dev

pytestmark = pytest.mark.gpu


def test_bounded_wait_times_out_and_context_stays_usable():
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=256, d=128, E=8, d_ff=128, k_base=32)
    inp = I.make_inputs(w)
    L = inp.layers[0]
    args = (dev(inp.X), dev(L.Wr), None, dev(L.Wg), dev(L.Wu), dev(L.Wd))
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype="bf16")
    stream = torch.cuda.current_stream().cuda_stream
    ec.ec_selftest_bounded_wait(lay.ctx, 2_000_000, stream)
    with pytest.raises(ec.ECError) as e:
        lay.check()
    assert e.value.status == ec.EC_ERR_TIMEOUT
    lay.check()                                   # the status word was cleared
    Y1, idx1, _, _ = lay.forward(*args)
    g1 = lay.backward(dev(inp.dY))
    lay.check()
    fresh = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype="bf16")
    Y2, idx2, _, _ = fresh.forward(*args)
    g2 = fresh.backward(dev(inp.dY))
    fresh.check()
    assert torch.equal(idx1, idx2) and torch.equal(Y1, Y2)
    assert torch.equal(g1["dX"], g2["dX"]) and torch.equal(g1["dWg"], g2["dWg"])


def test_selftest_rejects_unbounded_limits():
    w = I.scaled(I.WORKLOADS["tiny_f32"], G=1, L=64)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, [0, 64], [8], dtype="f32")
    with pytest.raises(ec.ECError) as e:
        ec.ec_selftest_bounded_wait(lay.ctx, 60_000_000_000, None)
    assert e.value.status == ec.EC_ERR_INVALID_ARG
