"""Seeded random shapes on the tensor-core path against the oracle (a sweep beyond the
hand-picked cases): ragged groups with random capacities, widths that are and are not
multiples of 512, expert counts from 1 to 40, every tile policy; token choice with random
k and capacity factor. Same rules as the other parity tests: bit-exact selection on the
GPU's scores, then relative max-norm 2e-2 on outputs and gradients."""
import numpy as np
import pytest

from oracle import ecmoe as O
from oracle import token_choice as TC
from paper_2604_01622_gb300 import inputs as I
from tests._util import dev, gpu_layer, host, relmax

pytestmark = pytest.mark.gpu

BOUND = 2e-2


def _ec_case(seed):
    rng = np.random.default_rng(1000 + seed)
    G = int(rng.integers(1, 4))
    L = int(rng.integers(40, 400))
    d = int(rng.choice([64, 128, 192, 256, 512]))
    d_ff = int(rng.choice([64, 128, 256]))
    E = int(rng.integers(1, 41))
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=G, L=L, d=d, E=E, d_ff=d_ff, k_base=1,
                 seed=2000 + seed, router_bias=bool(rng.integers(2)), layers=1)
    inp = I.make_inputs(w)
    sizes = rng.multinomial(G * L - G, [1.0 / G] * G) + 1            # ragged, none empty
    inp.group_off = np.concatenate([[0], np.cumsum(sizes)]).astype(np.int32)
    inp.k_g = np.array([rng.integers(0, min(s, 96) + 1) for s in sizes], np.int32)
    return inp, int(rng.integers(0, 3))


@pytest.mark.parametrize("seed", range(20))
def test_expert_choice_random_shape(seed):
    inp, tiles = _ec_case(seed)
    w = inp.w
    L = inp.layers[0]
    _, out = gpu_layer(inp, tiles=tiles)
    S_gpu = host(out["S"]).T
    idx = out["idx"].cpu().numpy()
    ref_idx, ref_gate = O.ec_select(S_gpu, inp.group_off, inp.k_g)
    assert np.array_equal(idx, ref_idx)
    assert np.array_equal(host(out["gate"]), ref_gate)
    fwd = O.forward(inp.X.f64(), L.Wr.f64(), L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(),
                    inp.group_off, inp.k_g, forced_idx=idx)
    bwd = O.backward(fwd, inp.dY.f64(), L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    errs = {"Y": relmax(host(out["Y"]), fwd["Y"])}
    for k in ("dX", "dWr", "dWg", "dWu", "dWd"):
        errs[k] = relmax(host(out[k]), bwd[k])
    if L.br is not None:
        errs["dbr"] = relmax(host(out["dbr"]), bwd["dbr"])
    assert all(v <= BOUND for v in errs.values()), (w, tiles, errs)


@pytest.mark.parametrize("seed", range(10))
def test_token_choice_random_shape(seed):
    from paper_2604_01622_gb300.layer import TCMoELayer, tc_capacity
    rng = np.random.default_rng(3000 + seed)
    E = int(rng.integers(2, 41))
    k = int(rng.integers(1, min(E, 8) + 1))
    w = I.Workload("tc_random", G=1, L=int(rng.integers(50, 700)),
                   d=int(rng.choice([64, 128, 256, 512])), E=E,
                   d_ff=int(rng.choice([64, 128, 256])), k_base=0, dtype="bf16",
                   seed=4000 + seed, router_bias=bool(rng.integers(2)))
    cf = [None, 0.5, 1.0, 1.5][int(rng.integers(4))]
    inp = I.make_inputs(w)
    L = inp.layers[0]
    cap = tc_capacity(cf, k, w.N, w.E)
    lay = TCMoELayer(w.N, w.d, w.E, w.d_ff, k, cap)
    lay.set_tiles(int(rng.integers(0, 3)))
    import torch
    br = None if L.br is None else torch.from_numpy(L.br).cuda()
    Y, choice, gate, kept, load, S = lay.forward(dev(inp.X), dev(L.Wr), br, dev(L.Wg),
                                                 dev(L.Wu), dev(L.Wd))
    g = lay.backward(dev(inp.dY), with_bias=L.br is not None)
    lay.check()
    ref_c, _, ref_k = TC.tc_select(host(S), k, None if cap < 0 else cap)
    assert np.array_equal(choice.cpu().numpy(), ref_c)
    assert np.array_equal(kept.cpu().numpy().astype(bool), ref_k)
    fwd = TC.tc_forward(inp.X.f64(), L.Wr.f64(), L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(), k,
                        forced=(ref_c, ref_k))
    bwd = TC.tc_backward(fwd, inp.dY.f64(), L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    errs = {"Y": relmax(host(Y), fwd["Y"])}
    for key in ("dX", "dWr", "dWg", "dWu", "dWd"):
        errs[key] = relmax(host(g[key]), bwd[key])
    assert all(v <= BOUND for v in errs.values()), (w, k, cf, errs)
    lay.close()
