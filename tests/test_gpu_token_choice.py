"""Token-choice routing (arXiv 2604.01622, Sec. 2.2) on the GPU vs the float64 oracle.

The CUDA path runs the router in bf16 with fp32 scores, so, as for expert choice, the
selection is compared bit-exactly against the oracle's top-k and capacity rule applied to
the GPU's own scores; the layer outputs and gradients are then compared with the oracle
run on that selection (relative max-norm 2e-2, bf16 path). At full size the oracle checks
sampled tokens and one sampled expert's weight gradients.
"""
import numpy as np
import pytest
import torch

from oracle import ecmoe as O
from oracle import token_choice as TC
from paper_2604_01622_gb300 import inputs as I
from tests._util import dev, host, relmax

pytestmark = pytest.mark.gpu

BOUND = 2e-2
GRADS = ("Y", "dX", "dWr", "dWg", "dWu", "dWd")


def _run(inp, k, capacity, residual=False, tiles=None):
    from paper_2604_01622_gb300.layer import TCMoELayer
    w = inp.w
    L = inp.layers[0]
    lay = TCMoELayer(w.N, w.d, w.E, w.d_ff, k, capacity)
    if residual:
        lay.set_residual(True)
    if tiles is not None:
        lay.set_tiles(tiles)
    br = None if L.br is None else torch.from_numpy(L.br).cuda()
    Y, choice, gate, kept, load, S = lay.forward(dev(inp.X), dev(L.Wr), br, dev(L.Wg),
                                                 dev(L.Wu), dev(L.Wd))
    g = lay.backward(dev(inp.dY), with_bias=L.br is not None)
    lay.check()
    out = {"Y": Y, "choice": choice, "gate": gate, "kept": kept, "load": load, "S": S, **g}
    return lay, out


def _check_selection(out, k, capacity, E):
    S_gpu = host(out["S"])
    choice = out["choice"].cpu().numpy()
    kept = out["kept"].cpu().numpy().astype(bool)
    ref_c, ref_g, ref_k = TC.tc_select(S_gpu, k, None if capacity < 0 else capacity)
    assert np.array_equal(choice, ref_c)
    assert np.array_equal(kept, ref_k)
    # gates: fp32 division on the GPU, float64 in the oracle
    assert np.max(np.abs(host(out["gate"]) - ref_g)) <= 1e-6
    load = out["load"].cpu().numpy()
    assert np.array_equal(load, np.bincount(choice[kept], minlength=E))
    return S_gpu, choice, kept


CASES = [
    # name, workload overrides, k, capacity factor (None: dropless; 0.0 is a real cap of 0)
    ("dropless_k2", dict(), 2, None),
    ("cf1_k2", dict(), 2, 1.0),
    ("cf05_k2", dict(), 2, 0.5),
    ("k1", dict(), 1, 1.25),
    ("k_eq_E", dict(E=8), 8, None),
    # skewed router bias: experts with several 256-row tiles next to nearly empty ones
    ("skew_dropless", dict(router_bias=True, E=4, L=512), 2, None),
    ("skew_cf1", dict(router_bias=True, E=4, L=512), 2, 1.0),
    # ragged: N = 2 x 350 (not a multiple of the 256-token ranking block), 12 experts (not a
    # multiple of 32 or 64), k = 3, a tight cap
    ("ragged_e12_k3", dict(L=350, E=12, router_bias=True), 3, 0.6),
    # 100 experts over two 64-column router tiles, every expert a tail of 256-row padding
    ("e100_k5", dict(L=384, E=100, d=64, d_ff=64), 5, None),
    # one expert: every token's single choice, normalised gate 1, no router gradient
    ("e1_k1", dict(E=1, L=300), 1, None),
    # the largest routing: 256 experts, each token's 32 best (router tile of 256 columns)
    ("e256_k32", dict(L=256, E=256, d=64, d_ff=64), 32, None),
    # d and 2 d_ff multiples of 512, tile policy EC_TILES_512: the GEMMs take 256 x 512 tiles
    ("wide_tiles", dict(L=300, d=512, d_ff=256, E=6, router_bias=True), 2, 1.0),
]
TILES = {"wide_tiles": 2}


def _workload(over):
    base = I.Workload("tc_small", G=2, L=128, d=128, E=8, d_ff=128, k_base=0, dtype="bf16",
                      seed=11, init="fan_in")
    return I.scaled(base, **over)


@pytest.mark.parametrize("name,over,k,cf", CASES, ids=[c[0] for c in CASES])
def test_tc_layer_parity(name, over, k, cf):
    from paper_2604_01622_gb300.layer import tc_capacity
    w = _workload(over)
    inp = I.make_inputs(w)
    L = inp.layers[0]
    cap = tc_capacity(cf, k, w.N, w.E)
    lay, out = _run(inp, k, cap, tiles=TILES.get(name))
    S_gpu, choice, kept = _check_selection(out, k, cap, w.E)
    Wr, Wg, Wu, Wd = L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64()
    fwd = TC.tc_forward(inp.X.f64(), Wr, L.br, Wg, Wu, Wd, k, forced=(choice, kept))
    bwd = TC.tc_backward(fwd, inp.dY.f64(), Wr, Wg, Wu, Wd)
    ref = {"Y": fwd["Y"], **bwd}
    errs = {g: relmax(host(out[g]), ref[g]) for g in GRADS}
    errs["S"] = relmax(S_gpu, fwd["S"])
    if L.br is not None:
        errs["dbr"] = relmax(host(out["dbr"]), ref["dbr"])
    assert all(v <= BOUND for v in errs.values()), errs
    # experts nobody kept: exactly zero weight gradients
    load = out["load"].cpu().numpy()
    for e in np.nonzero(load == 0)[0]:
        assert not out["dWg"][e].any() and not out["dWd"][e].any()
    # tokens with every pair dropped: exactly zero output
    dropped_all = ~kept.any(axis=1)
    assert np.all(host(out["Y"])[dropped_all] == 0.0)
    lay.close()


@pytest.mark.parametrize("wide", [False, True], ids=["narrow", "wide"])
def test_tc_capacity_zero_drops_everything(wide):
    """Capacity 0: no expert keeps a row, so every GEMM tile has an empty K loop or no rows
    (with 256 x 512 tiles: both accumulator halves are still handed over per tile)."""
    w = _workload(dict(d=512, d_ff=256) if wide else dict())
    inp = I.make_inputs(w)
    lay, out = _run(inp, 2, 0, tiles=2 if wide else None)
    assert not out["kept"].any() and not out["load"].any()
    assert not out["Y"].any() and not out["dX"].any()
    for g in ("dWg", "dWu", "dWd", "dWr"):
        assert not out[g].any(), g
    lay.close()


def test_tc_residual():
    w = _workload(dict())
    inp = I.make_inputs(w)
    lay0, o0 = _run(inp, 2, -1)
    lay1, o1 = _run(inp, 2, -1, residual=True)
    X = host(dev(inp.X))
    # Y1 = X + Y0 and dX1 = dY + dX0, up to the bf16 rounding of the stored sums
    assert relmax(host(o1["Y"]), X + host(o0["Y"])) <= 1e-2
    assert relmax(host(o1["dX"]), inp.dY.f64() + host(o0["dX"])) <= 1e-2
    lay0.close()
    lay1.close()


def test_tc_context_rejects_expert_choice_calls():
    from paper_2604_01622_gb300 import ECError, EC_ERR_STATE, EC_ERR_UNSUPPORTED
    from paper_2604_01622_gb300.layer import TCMoELayer
    lay = TCMoELayer(256, 128, 8, 128, 2, -1)
    with pytest.raises(ECError) as ei:
        lay.set_capacity([4])
    assert ei.value.status == EC_ERR_STATE
    lay.close()
    with pytest.raises(ECError) as ei:
        TCMoELayer(256, 128, 8, 128, 2, -1, dtype="f32")
    assert ei.value.status == EC_ERR_UNSUPPORTED


@pytest.mark.parametrize("cf", [None, 1.0])
def test_tc_full_size_sampled(cf):
    """8 x 4096 tokens, d=2048, 64 experts of d_ff=1024, top-8 token choice (the same
    expert compute as expert choice with 512 tokens per expert and sequence)."""
    from paper_2604_01622_gb300.layer import tc_capacity
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], layers=1)
    inp = I.make_inputs(w)
    _check_full(inp, 8, tc_capacity(cf, 8, w.N, w.E))


def test_tc_large_batch_past_32_bit_offsets():
    """262144 tokens (the bench workload's 32768 repeated 8 times), top-8 dropless: about
    2.1 M padded expert rows, so the gathered rows hold 4.4 G elements, past 32-bit element
    offsets; samples include the last tokens."""
    base = I.scaled(I.WORKLOADS["ec_d2048_e64"], layers=1)
    inp0 = I.make_inputs(base)
    G = 8
    w = I.scaled(base, G=G * base.G)
    X = I.Tensor(np.tile(inp0.X.data, (G, 1)), inp0.X.dtype)
    dY = I.Tensor(np.tile(inp0.dY.data, (G, 1)), inp0.dY.dtype)
    inp = I.Inputs(w, X, dY, (np.arange(w.G + 1) * w.L).astype(np.int32),
                   np.zeros(w.G, np.int32), inp0.layers)
    _check_full(inp, 8, -1, extra=[w.N - 1, w.N - 1000])


def _check_full(inp, k, cap, extra=()):
    w = inp.w
    L = inp.layers[0]
    lay, out = _run(inp, k, cap)
    S_gpu, choice, kept = _check_selection(out, k, cap, w.E)
    Wr = L.Wr.f64()
    rng = np.random.default_rng(99)
    toks = np.union1d(rng.choice(w.N, 16, replace=False), np.array(extra, dtype=np.int64))
    part = ~kept.all(axis=1)
    if part.any():   # tokens with a dropped pair
        toks = np.union1d(toks, rng.choice(np.nonzero(part)[0], min(8, int(part.sum())),
                                           replace=False))
    # Y and dX of a token depend on that token's own pairs only
    fwd = TC.tc_forward(inp.X.f64(toks), Wr, L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(), k,
                        forced=(choice[toks], kept[toks]))
    bwd = TC.tc_backward(fwd, inp.dY.f64(toks), Wr, L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    e_y = relmax(host(out["Y"])[toks], fwd["Y"])
    e_dx = relmax(host(out["dX"])[toks], bwd["dX"])
    assert e_y <= BOUND and e_dx <= BOUND, (e_y, e_dx)
    # one expert's weight gradients over all its kept tokens, on a slice of d_ff columns
    e = int(rng.integers(w.E))
    tok_e, r_e = np.nonzero((choice == e) & kept)
    cols = np.sort(rng.choice(w.d_ff, 64, replace=False))
    H = inp.X.f64(tok_e)
    g_e = TC.tc_gates(O.router_scores(H, Wr, L.br), choice[tok_e])[np.arange(len(tok_e)), r_e]
    dwg, dwu, dwd, _ = O.backward_expert(H, g_e, inp.dY.f64(tok_e), L.Wg.f64(e)[:, cols],
                                         L.Wu.f64(e)[:, cols], L.Wd.f64(e)[cols, :])
    errs = (relmax(host(out["dWg"][e][:, cols]), dwg), relmax(host(out["dWu"][e][:, cols]), dwu),
            relmax(host(out["dWd"][e][cols, :]), dwd))
    assert max(errs) <= BOUND, errs
    # router gradient rows sum to zero (softmax Jacobian)
    dWr = host(out["dWr"])
    assert np.max(np.abs(dWr.sum(axis=1))) <= 1e-3 * np.max(np.abs(dWr))
    lay.close()
