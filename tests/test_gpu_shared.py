"""Shared experts (appendix "Token Coverage") on the GPU against the oracle.

The library takes S shared experts of width f as one concatenated SwiGLU FFN of width S*f;
the oracle sums S separate experts. Selection is compared bit-exactly on the GPU's scores,
then Y, dX, the routed gradients and each shared expert's gradients (split back out of the
concatenated ones): 1e-4 (fp32) / 2e-2 (bf16) relative max-norm.
"""
import numpy as np
import pytest
import torch

from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer
from tests._util import dev, host, relmax, tol

pytestmark = pytest.mark.gpu

CASES = {
    "f32": (I.scaled(I.WORKLOADS["tiny_f32"], G=2, L=100, d=36, E=5, d_ff=20, k_base=9), 2, 12),
    "bf16": (I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=256, d=192, E=8, d_ff=128,
                      k_base=40), 2, 64),
    # 2048 tokens: the shared FFN's dWd runs as two split-K halves summed afterwards
    "bf16_split_k": (I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=1024, d=256, E=8, d_ff=128,
                              k_base=64), 2, 128),
}


@pytest.mark.parametrize("name", sorted(CASES))
def test_shared_experts_match_oracle(name):
    w, n_sh, f_sh = CASES[name]
    inp = I.make_inputs(w)
    L = inp.layers[0]
    sh = I.make_shared(w, 0, n_sh, f_sh)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype=w.dtype,
                     d_ff_shared=n_sh * f_sh)
    Y, idx, gate, S = lay.forward(dev(inp.X), dev(L.Wr), None, dev(L.Wg), dev(L.Wu), dev(L.Wd),
                                  shared=(dev(sh.Wg), dev(sh.Wu), dev(sh.Wd)))
    g = lay.backward(dev(inp.dY))
    lay.check()
    idx_h = idx.cpu().numpy()
    ref_idx, _ = O.ec_select(host(S).T, inp.group_off, inp.k_g)
    assert np.array_equal(idx_h, ref_idx)
    experts = [sh.expert(s) for s in range(n_sh)]
    fwd = O.forward(inp.X.f64(), L.Wr.f64(), None, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(),
                    inp.group_off, inp.k_g, forced_idx=idx_h, shared=experts)
    bwd = O.backward(fwd, inp.dY.f64(), L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    errs = {"Y": relmax(host(Y), fwd["Y"])}
    for k in ("dX", "dWr", "dWg", "dWu", "dWd"):
        errs[k] = relmax(host(g[k]), bwd[k])
    for s in range(n_sh):
        c = slice(s * f_sh, (s + 1) * f_sh)
        dwg, dwu, dwd = bwd["dshared"][s]
        errs[f"dWg_s{s}"] = relmax(host(g["dWg_s"])[:, c], dwg)
        errs[f"dWu_s{s}"] = relmax(host(g["dWu_s"])[:, c], dwu)
        errs[f"dWd_s{s}"] = relmax(host(g["dWd_s"])[c, :], dwd)
    assert max(errs.values()) <= tol(w), errs


def test_plain_calls_refuse_a_context_with_shared_experts():
    import paper_2604_01622_gb300 as ec
    w, n_sh, f_sh = CASES["bf16"]
    inp = I.make_inputs(w, with_layers=False)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, d_ff_shared=n_sh * f_sh)
    x = dev(inp.X)
    with pytest.raises(ec.ECError) as e:
        ec.ec_moe_forward(lay.ctx, x.data_ptr(), x.data_ptr(), None, x.data_ptr(), x.data_ptr(),
                          x.data_ptr(), x.data_ptr(), None, None, None, None)
    assert e.value.status == ec.EC_ERR_STATE
