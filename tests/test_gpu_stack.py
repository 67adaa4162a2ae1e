"""Four stacked layers with residual adds (the wide workload's structure) against the oracle.

Each GPU layer runs with the residual option (Y = X + EC(X), dX = dY + EC input gradient).
Per layer the selection is compared bit-exactly on that layer's GPU scores; the oracle then
runs the whole stack in float64 with those selections and is compared on the stack output,
the input gradient and every layer's weight gradients (relative max-norm 2e-2, bf16).
At the full width of the wide workload (4 x 8192 tokens, d 4096, 32 experts, d_ff 2048, the
launch configuration the bench times) the oracle follows sampled tokens through all four
layers, and checks each layer's weight gradients on one expert's slice of d_ff columns and
the first and last layers' router gradients in full, given that layer's GPU input and the
upstream gradient it received.
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
        gpu[l]["d_in"] = d                       # the upstream gradient layer l receives
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


def test_four_layer_residual_stack_full_width_sampled():
    w = I.WORKLOADS["ec_wide_d4096_e32_x4"]
    inp, layers, gpu, out, dx0, grads = _stack_case(w)
    bound = 2e-2
    idxs = []
    for g in gpu:
        S_gpu = host(g["S"]).T
        ref_idx, ref_gate = O.ec_select(S_gpu, inp.group_off, inp.k_g)
        idx = g["idx"].cpu().numpy()
        assert np.array_equal(idx, ref_idx)
        assert np.array_equal(host(g["gate"]), ref_gate)
        idxs.append(idx)
    rng = np.random.default_rng(77)
    picked0 = np.zeros(w.N, bool)
    picked0[idxs[0].ravel()] = True
    toks = list(rng.choice(np.nonzero(picked0)[0], 20, replace=False))
    toks += list(rng.choice(np.nonzero(~picked0)[0], 4, replace=False)) + [0, w.N - 1]
    toks = [int(t) for t in toks]
    fn = []
    for l in range(w.layers):
        L = inp.layers[l]
        fn.append((L.Wr.f64(), L.br, (lambda e, T=L.Wg: T.f64(e)), (lambda e, T=L.Wu: T.f64(e)),
                   (lambda e, T=L.Wd: T.f64(e))))
    pairs = [O.token_pairs(idx, toks) for idx in idxs]
    X0 = inp.X.f64(np.array(toks))
    dO = inp.dY.f64(np.array(toks))
    xs, d0 = O.stack_tokens({t: X0[i] for i, t in enumerate(toks)},
                            {t: dO[i] for i, t in enumerate(toks)}, fn, pairs)
    out_h, dx0_h = host(out), host(dx0)
    errs = {"out": relmax(np.stack([out_h[t] for t in toks]), np.stack([xs[-1][t] for t in toks])),
            "dX0": relmax(np.stack([dx0_h[t] for t in toks]), np.stack([d0[t] for t in toks]))}
    # each layer's weight gradients on one expert's slice of d_ff columns, given the layer's
    # GPU input and the upstream gradient it received
    for l in range(w.layers):
        Wr, br, Wg, Wu, Wd = fn[l]
        x_in = gpu[l]["x_in"]
        d_in = gpu[l]["d_in"]
        e = int(rng.integers(w.E))
        cols = np.sort(rng.choice(w.d_ff, 64, replace=False))
        rows = torch.from_numpy(idxs[l][e]).cuda()
        H = host(x_in.index_select(0, rows))
        s_col = O.router_scores(H, Wr, br)[:, e]
        dYe = host(d_in.index_select(0, rows))
        dwg, dwu, dwd, _ = O.backward_expert(H, s_col, dYe, Wg(e)[:, cols], Wu(e)[:, cols],
                                             Wd(e)[cols, :])
        errs[f"dWg[{l}]"] = relmax(grads[l]["dWg"][e][:, cols].double().cpu().numpy(), dwg)
        errs[f"dWu[{l}]"] = relmax(grads[l]["dWu"][e][:, cols].double().cpu().numpy(), dwu)
        errs[f"dWd[{l}]"] = relmax(grads[l]["dWd"][e][cols, :].double().cpu().numpy(), dwd)
        if l in (0, w.layers - 1):
            r = O.router_backward_streamed(host(x_in), Wr, br, host(d_in), idxs[l], Wg, Wu, Wd)
            errs[f"dWr[{l}]"] = relmax(host(grads[l]["dWr"]), r["dWr"])
    assert max(errs.values()) <= bound, errs
    for g in gpu:
        g["lay"].close()
