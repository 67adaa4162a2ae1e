"""Timestep-dependent capacity on the GPU (Sec. 4.2, Table 1): per-sequence masking ratios
drive a capacity schedule, the schedule drives the layer, and every step is compared with
the oracle run at that step's capacities.

Two routes into the layer:
  * ec_capacity_schedule (k_g = round(k(r_g) L_g / E), the sum changes from step to step)
    -> ec_ctx_set_capacity (host array, synchronous);
  * FLOPs-matched capacities (the sum kept at the context's M, as the timestep workloads
    draw them) read from a device array by ec_ctx_set_capacity_async, several steps queued
    on one stream with no host copy between them.
Rules as in the other parity tests: the selection bit-exact on the GPU's own scores, the
layer within 1e-4 (fp32) / 2e-2 (bf16) relative max-norm of the oracle on that selection.
"""
import numpy as np
import pytest
import torch

import paper_2604_01622_gb300 as ec
from oracle import ecmoe as O
from oracle import schedulers as SO
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer
from tests._util import dev, host, relmax, tol

pytestmark = pytest.mark.gpu


def _run(lay, inp, L):
    br = None if L.br is None else torch.from_numpy(L.br).cuda()
    Y, idx, gate, S = lay.forward(dev(inp.X), dev(L.Wr), br, dev(L.Wg), dev(L.Wu), dev(L.Wd))
    g = lay.backward(dev(inp.dY), with_bias=L.br is not None)
    return {"Y": Y, "idx": idx, "gate": gate, "S": S, **g}


def _compare(out, inp, L, k_g):
    """Selection and layer parity of one step run with capacities k_g."""
    S_gpu = host(out["S"]).T
    idx = out["idx"].cpu().numpy()
    assert idx.shape == (inp.w.E, int(k_g.sum()))
    ref_idx, ref_gate = O.ec_select(S_gpu, inp.group_off, k_g)
    assert np.array_equal(idx, ref_idx)
    assert np.array_equal(host(out["gate"]), ref_gate)
    fwd = O.forward(inp.X.f64(), L.Wr.f64(), L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(),
                    inp.group_off, k_g, forced_idx=idx)
    bwd = O.backward(fwd, inp.dY.f64(), L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    ref = {"Y": fwd["Y"], **bwd}
    errs = {k: relmax(host(out[k]), ref[k]) for k in ("Y", "dX", "dWr", "dWg", "dWu", "dWd")}
    assert all(v <= tol(inp.w) for v in errs.values()), errs
    return errs


def _small(dtype):
    if dtype == "f32":
        w = I.scaled(I.WORKLOADS["tiny_f32"], G=4, L=96, d=64, E=8, d_ff=64, k_base=12)
    else:
        w = I.scaled(I.WORKLOADS["ec_timestep_d2048_e64"], G=4, L=256, d=128, E=8, d_ff=128,
                     k_base=32)
    return I.make_inputs(w)


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
@pytest.mark.parametrize("scheduler", ["linear_reverse", "cosine", "gaussian"])
def test_schedule_drives_the_layer_step_after_step(dtype, scheduler):
    inp = _small(dtype)
    w, L = inp.w, inp.layers[0]
    # created at the largest capacity any step can ask for (k_max L / E per sequence)
    k_min, k_max = 2.0, 8.0
    k_cap = np.minimum(np.diff(inp.group_off), int(np.ceil(k_max * w.L / w.E)) + 1)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, k_cap.astype(np.int32), dtype=w.dtype)
    rng = np.random.default_rng(11)
    seen = set()
    for step in range(4):
        r = rng.random(w.G)
        if step == 0:
            r[:2] = [0.0, 1.0]                              # both ends of the schedule
        k_g = ec.ec_capacity_schedule(scheduler, k_min, k_max, w.E, inp.group_off, r)
        assert np.array_equal(k_g, SO.group_capacity(scheduler, r, k_min, k_max, w.E,
                                                     inp.group_off))
        lay.set_capacity(k_g)
        assert lay.M == int(k_g.sum())
        out = _run(lay, inp, L)
        lay.check()
        _compare(out, inp, L, k_g)
        seen.add(tuple(k_g))
    assert len(seen) > 1                                    # the capacities did change
    lay.close()


@pytest.mark.parametrize("dtype", ["f32", "bf16"])
def test_device_capacity_updates_in_stream_order(dtype):
    inp = _small(dtype)
    w, L = inp.w, inp.layers[0]
    T = w.G * w.k_base
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype=w.dtype)
    assert lay.M == T
    # FLOPs-matched capacities for several steps, uploaded once
    rng = np.random.default_rng(5)
    steps = [I.timestep_capacity(rng.random(w.G), w.k_base, w.L) for _ in range(3)]
    steps.append(np.full(w.G, w.k_base, np.int32))
    for k in steps:
        assert int(k.sum()) == T
    kg_dev = torch.from_numpy(np.stack(steps).astype(np.int32)).cuda()
    outs = []
    for i in range(len(steps)):                             # queued back to back
        lay.set_capacity_async(kg_dev[i])
        out = _run(lay, inp, L)
        outs.append({k: v.clone() for k, v in out.items() if v is not None})
    lay.check()
    for k_g, out in zip(steps, outs):
        _compare(out, inp, L, k_g)
    # a rejected update (wrong sum, then a group over its size) leaves the last capacities
    bad = [steps[0].copy(), steps[0].copy()]
    bad[0][0] += 1
    bad[1][0] = w.L + 1
    bad[1][1] -= w.L + 1 - steps[0][0]
    for b in bad:
        lay.set_capacity_async(torch.from_numpy(b.astype(np.int32)).cuda())
        with pytest.raises(ec.ECError) as e:
            lay.check()
        assert e.value.status == ec.EC_ERR_SHAPE
        out = _run(lay, inp, L)
        lay.check()
        _compare(out, inp, L, steps[-1])
    lay.close()
