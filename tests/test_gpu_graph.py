"""The layer's forward + backward captured in a CUDA graph replays exactly the eager results.

Every library call is asynchronous on the caller's stream with no host synchronisation or
allocation, so one fwd+bwd step can be captured once and replayed on new input values
written into the same buffers. The kernels are deterministic (no atomics), so the replay
must give bit-identical outputs and gradients to an eager step on the same values.
"""
import numpy as np
import pytest
import torch

from paper_2604_01622_gb300 import inputs as I
from tests._util import dev

pytestmark = pytest.mark.gpu


def _workload(seed):
    return I.Workload("graph_small", G=2, L=512, d=256, E=8, d_ff=256, k_base=96, dtype="bf16",
                      seed=seed, init="std002", x_recipe="rms_unit", router_bias=True)


def _layer(kind, w, inp):
    from paper_2604_01622_gb300.layer import ECMoELayer, TCMoELayer
    if kind == "ec":
        return ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g)
    return TCMoELayer(w.N, w.d, w.E, w.d_ff, 2, 140)


@pytest.mark.parametrize("kind", ["ec", "tc"])
def test_graph_replay_equals_eager(kind):
    w = _workload(31)
    a = I.make_inputs(w)
    b = I.make_inputs(I.scaled(w, seed=32), with_layers=False)
    L = a.layers[0]
    lay = _layer(kind, w, a)
    wts = (dev(L.Wr), torch.from_numpy(L.br).cuda(), dev(L.Wg), dev(L.Wu), dev(L.Wd))
    X, dY = dev(a.X), dev(a.dY)
    Y = torch.empty_like(X)
    g = {"dX": torch.empty_like(X),
         "dWr": torch.empty(w.d, w.E, dtype=torch.float32, device="cuda"),
         "dbr": torch.empty(w.E, dtype=torch.float32, device="cuda"),
         "dWg": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device="cuda"),
         "dWu": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device="cuda"),
         "dWd": torch.empty(w.E, w.d_ff, w.d, dtype=torch.float32, device="cuda")}

    def step():
        lay.forward(X, *wts, Y=Y, outputs=False)
        lay.backward(dY, grads=g)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()                                     # eager warm-up on the inputs of set a
    torch.cuda.current_stream().wait_stream(side)
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    # new values in the same buffers, then replay
    X.copy_(dev(b.X))
    dY.copy_(dev(b.dY))
    graph.replay()
    torch.cuda.synchronize()
    got = {"Y": Y.clone(), **{k: v.clone() for k, v in g.items()}}
    step()                                         # eager on the same values
    lay.check()
    for k, ref in (("Y", Y), *g.items()):
        assert torch.equal(got[k], ref), k
    assert not torch.equal(got["Y"], dev(a.X))     # the replay computed something
    del graph
    lay.close()


def test_graph_with_device_capacity_updates():
    """A captured step that begins with a capacity update from a device array
    (ec_ctx_set_capacity_async) reads the array when it is replayed: new per-sequence
    capacities written into it (same sum) change the step, and the replay equals an eager
    step with those capacities bit for bit."""
    from paper_2604_01622_gb300.layer import ECMoELayer
    w = I.Workload("graph_cap", G=4, L=256, d=256, E=8, d_ff=256, k_base=64, dtype="bf16",
                   seed=33, init="std002", x_recipe="rms_unit", timestep_capacity=True)
    a = I.make_inputs(w)
    L = a.layers[0]
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, a.group_off, a.k_g)
    wts = (dev(L.Wr), None, dev(L.Wg), dev(L.Wu), dev(L.Wd))
    X, dY = dev(a.X), dev(a.dY)
    kg = torch.from_numpy(a.k_g.astype(np.int32)).cuda()
    Y = torch.empty_like(X)
    g = {"dX": torch.empty_like(X),
         "dWr": torch.empty(w.d, w.E, dtype=torch.float32, device="cuda"),
         "dWg": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device="cuda"),
         "dWu": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device="cuda"),
         "dWd": torch.empty(w.E, w.d_ff, w.d, dtype=torch.float32, device="cuda")}

    def step():
        lay.set_capacity_async(kg)
        lay.forward(X, *wts, Y=Y, outputs=False)
        lay.backward(dY, grads=g)

    side = torch.cuda.Stream()
    side.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(side):
        step()
    torch.cuda.current_stream().wait_stream(side)
    torch.cuda.synchronize()
    first = {"Y": Y.clone(), **{k: v.clone() for k, v in g.items()}}
    graph = torch.cuda.CUDAGraph()
    with torch.cuda.graph(graph):
        step()
    new_k = I.timestep_capacity(np.random.default_rng(9).random(w.G), w.k_base, w.L)
    assert int(new_k.sum()) == int(a.k_g.sum()) and not np.array_equal(new_k, a.k_g)
    kg.copy_(torch.from_numpy(new_k.astype(np.int32)))
    graph.replay()
    torch.cuda.synchronize()
    got = {"Y": Y.clone(), **{k: v.clone() for k, v in g.items()}}
    step()                                         # eager with the same capacities
    lay.check()
    for k, ref in (("Y", Y), *g.items()):
        assert torch.equal(got[k], ref), k
    assert not torch.equal(got["Y"], first["Y"])   # the new capacities changed the step
    del graph
    lay.close()
