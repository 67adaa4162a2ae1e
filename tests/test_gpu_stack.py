"""Four stacked layers with residual adds (the wide workload's structure) against the oracle.

Each GPU layer runs with the residual option (Y = X + EC(X), dX = dY + EC input gradient).
Per layer the selection is compared bit-exactly on that layer's GPU scores; the oracle then
runs the whole stack in float64 with those selections and is compared on the stack output,
the input gradient and every layer's weight gradients (relative max-norm 2e-2, bf16).
"""
import numpy as np
import pytest
import torch

from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer
from tests._util import dev, host, relmax

pytestmark = pytest.mark.gpu


def _stack_case(w):
    inp = I.make_inputs(w)
    layers = []
    x = dev(inp.X)
    gpu = []
    for l in range(w.layers):
        L = inp.layers[l]
        lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype=w.dtype)
        lay.set_residual(True)
        br = None if L.br is None else torch.from_numpy(L.br).cuda()
        y, idx, gate, S = lay.forward(x, dev(L.Wr), br, dev(L.Wg), dev(L.Wu), dev(L.Wd))
        gpu.append({"lay": lay, "idx": idx, "gate": gate, "S": S, "x_in": x})
        layers.append((L.Wr.f64(), L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64()))
        x = y
    out = x
    d = dev(inp.dY)
    grads = [None] * w.layers
    for l in range(w.layers - 1, -1, -1):
        grads[l] = gpu[l]["lay"].backward(d, with_bias=inp.layers[l].br is not None)
        d = grads[l]["dX"]
    for g in gpu:
        g["lay"].check()
    return inp, layers, gpu, out, d, grads


def test_four_layer_residual_stack_matches_oracle():
    w = I.scaled(I.WORKLOADS["ec_wide_d4096_e32_x4"], G=2, L=256, d=128, E=8, d_ff=128,
                 k_base=40)
    inp, layers, gpu, out, dx0, grads = _stack_case(w)
    forced = []
    for g in gpu:
        S_gpu = host(g["S"]).T
        ref_idx, _ = O.ec_select(S_gpu, inp.group_off, inp.k_g)
        idx = g["idx"].cpu().numpy()
        assert np.array_equal(idx, ref_idx)
        forced.append(idx)
    xs, fwds = O.stack_forward(inp.X.f64(), layers, inp.group_off, inp.k_g, forced)
    d0, ref_grads = O.stack_backward(fwds, layers, inp.dY.f64())
    errs = {"out": relmax(host(out), xs[-1]), "dX0": relmax(host(dx0), d0)}
    for l in range(w.layers):
        for k in ("dWr", "dWg", "dWu", "dWd"):
            errs[f"{k}[{l}]"] = relmax(host(grads[l][k]), ref_grads[l][k])
    assert max(errs.values()) <= 2e-2, errs
    # residual form: a token no expert of a layer picked passes through that layer unchanged
    x_in = host(gpu[0]["x_in"])
    x_out = host(gpu[1]["x_in"])
    picked = np.zeros(w.N, bool)
    picked[gpu[0]["idx"].cpu().numpy().ravel()] = True
    assert np.array_equal(x_out[~picked], x_in[~picked])
