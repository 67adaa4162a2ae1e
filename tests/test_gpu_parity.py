"""CUDA path vs the float64 oracle, through the C ABI.

Rules: the selection is compared bit-exactly when both sides rank the same score tensor
(the GPU's fp32 scores); the layer outputs and gradients are then compared with the
oracle run on that selection: relative max-norm 1e-4 on the fp32 path, 2e-2 on bf16.
"""
import numpy as np
import pytest
import torch

from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I
from tests._util import dev, gpu_layer, host, relmax, tol

pytestmark = pytest.mark.gpu

GRADS = [("Y", "Y"), ("dX", "dX"), ("dWr", "dWr"), ("dWg", "dWg"), ("dWu", "dWu"), ("dWd", "dWd")]


def _oracle_full(inp, layer, idx):
    L = inp.layers[layer]
    fwd = O.forward(inp.X.f64(), L.Wr.f64(), L.br, L.Wg.f64(), L.Wu.f64(), L.Wd.f64(),
                    inp.group_off, inp.k_g, forced_idx=idx)
    bwd = O.backward(fwd, inp.dY.f64(), L.Wr.f64(), L.Wg.f64(), L.Wu.f64(), L.Wd.f64())
    return fwd, bwd


def _check_layer(inp, layer=0, tiles=None):
    w = inp.w
    lay, out = gpu_layer(inp, layer, tiles=tiles)
    S_gpu = host(out["S"]).T                              # [N][E] fp32 values as float64
    idx_gpu = out["idx"].cpu().numpy()
    # selection: bit-exact on the GPU's own scores
    idx_ref, gate_ref = O.ec_select(S_gpu, inp.group_off, inp.k_g)
    assert np.array_equal(idx_gpu, idx_ref)
    assert np.array_equal(host(out["gate"]), gate_ref)
    fwd, bwd = _oracle_full(inp, layer, idx_gpu)
    ref = {"Y": fwd["Y"], **bwd}
    errs = {k: relmax(host(out[k]), ref[r]) for k, r in GRADS}
    if inp.layers[layer].br is not None:
        errs["dbr"] = relmax(host(out["dbr"]), ref["dbr"])
    errs["S"] = relmax(S_gpu, fwd["S"])
    bound = tol(w)
    assert all(v <= bound for v in errs.values()), errs
    # tokens no expert chose: exactly zero output and input gradient
    picked = np.zeros(w.N, bool)
    picked[idx_gpu.ravel()] = True
    assert np.all(host(out["Y"])[~picked] == 0.0)
    assert np.all(host(out["dX"])[~picked] == 0.0)
    return errs


# ------------------------------------------------------------------ selection on given scores
@pytest.mark.parametrize("quant", [None, 8.0, 2.0])
def test_selection_bit_exact_on_given_scores(quant):
    from paper_2604_01622_gb300.layer import ECMoELayer
    rng = np.random.default_rng(7)
    N, E = 3000, 12
    for trial in range(3):
        S = rng.random((N, E)).astype(np.float32)
        if quant is not None:
            S = (np.round(S * quant) / quant).astype(np.float32)
        S[rng.random((N, E)) < 0.03] = np.float32(-0.0)
        S[rng.random((N, E)) < 0.03] = np.float32(0.0)
        S[rng.random((N, E)) < 0.02] *= -1
        group_off = I.random_groups(rng, N, 5)
        sizes = np.diff(group_off)
        k_g = np.array([rng.integers(0, s + 1) for s in sizes], dtype=np.int32)
        k_g[0] = 0
        k_g[-1] = sizes[-1]                                 # k = L edge
        lay = ECMoELayer(N, 64, E, 64, group_off, k_g, dtype="f32")
        ST = torch.from_numpy(np.ascontiguousarray(S.T)).cuda()
        idx, gate, S_out = lay.route(S_in=ST)
        lay.check()
        ref_idx, ref_gate = O.ec_select(S.astype(np.float64), group_off, k_g)
        assert np.array_equal(idx.cpu().numpy(), ref_idx)
        assert np.array_equal(gate.cpu().numpy().astype(np.float64), ref_gate)
        assert np.array_equal(S_out.cpu().numpy(), S.T)


def test_selection_degenerate_columns():
    """Columns the radix select treats specially: all scores equal (no pass), two values,
    one outlier stretching the range to both signs (offsets over 31 bits), subnormals and
    signed zeros, a column whose k-th score is tied across a group boundary; k = 0, k = L."""
    from paper_2604_01622_gb300.layer import ECMoELayer
    rng = np.random.default_rng(9)
    N, E = 2500, 8
    S = np.empty((N, E), np.float32)
    S[:, 0] = 0.25
    S[:, 1] = np.where(rng.random(N) < 0.3, 0.5, 0.125)
    S[:, 2] = (1.0 / 64) * (1 + 0.02 * rng.standard_normal(N))
    S[7, 2] = 3.0e38
    S[11, 2] = -3.0e38
    S[:, 3] = rng.integers(1, 40, N).astype(np.float32) * np.float32(1e-45)
    S[:, 4] = np.where(rng.random(N) < 0.5, np.float32(-0.0), np.float32(0.0))
    S[:, 5] = np.round(rng.random(N) * 4) / 4
    S[:, 6] = -rng.random(N)
    S[:, 7] = rng.random(N)
    group_off = np.array([0, 1000, 1001, 1800, N], np.int32)
    for k_g in (np.array([300, 1, 0, 700], np.int32), np.array([1000, 0, 799, 1], np.int32),
                np.array([999, 1, 1, 350], np.int32)):
        lay = ECMoELayer(N, 64, E, 64, group_off, k_g, dtype="f32")
        idx, gate, _ = lay.route(S_in=torch.from_numpy(np.ascontiguousarray(S.T)).cuda())
        lay.check()
        ref_idx, ref_gate = O.ec_select(S.astype(np.float64), group_off, k_g)
        assert np.array_equal(idx.cpu().numpy(), ref_idx)
        g = gate.cpu().numpy()
        assert np.array_equal(g.astype(np.float64), ref_gate)
        # gates carry the scores bit for bit (the sign of zero included)
        assert np.array_equal(g.view(np.uint32), S.T[np.arange(E)[:, None], ref_idx].view(np.uint32))


def test_selection_long_groups_beyond_shared_memory():
    """Groups longer than the shared-memory key buffer take the global-memory path."""
    from paper_2604_01622_gb300.layer import ECMoELayer
    rng = np.random.default_rng(8)
    N, E = 60000, 3
    S = (np.round(rng.random((N, E)) * 64) / 64).astype(np.float32)
    group_off = np.array([0, 55000, N], np.int32)
    k_g = np.array([7001, 300], np.int32)
    lay = ECMoELayer(N, 64, E, 64, group_off, k_g, dtype="f32")
    idx, gate, _ = lay.route(S_in=torch.from_numpy(np.ascontiguousarray(S.T)).cuda())
    lay.check()
    ref_idx, _ = O.ec_select(S.astype(np.float64), group_off, k_g)
    assert np.array_equal(idx.cpu().numpy(), ref_idx)


# ------------------------------------------------------------------ fp32 path (1e-4)
def test_tiny_f32_layer_matches_oracle():
    _check_layer(I.make_inputs(I.WORKLOADS["tiny_f32"]))


@pytest.mark.parametrize("seed", [11, 12])
def test_f32_ragged_groups_and_capacity_edges(seed):
    # N = 333 tokens, d = 68, d_ff = 36: no size is a multiple of a tile
    w = I.scaled(I.WORKLOADS["tiny_f32"], G=1, L=333, d=68, E=11, d_ff=36, seed=seed,
                 router_bias=True)
    inp = I.make_inputs(w)
    inp.group_off = np.array([0, 0, 150, 151, 333], np.int32)   # an empty and a 1-token group
    inp.k_g = np.array([0, 150, 1, 17], np.int32)                # k = 0 and k = L
    _check_layer(inp)


def test_f32_many_experts():
    """500 experts (the fp32 path takes up to 512): the router softmax and the per-expert
    selection over many columns, 96 tokens, 5 per expert."""
    w = I.scaled(I.WORKLOADS["tiny_f32"], G=1, L=96, d=32, E=500, d_ff=16, k_base=5, seed=20,
                 router_bias=True)
    _check_layer(I.make_inputs(w))


# ------------------------------------------------------------------ bf16 path (2e-2), small shapes
SMALL_BF16 = {
    # d2048/e64-like: ragged M (2*80 = 160 rows: one full 128-row tile and a 32-row tail)
    "ec_d2048_e64": dict(G=2, L=512, d=256, E=8, d_ff=128, k_base=80),
    # timestep capacity with mask-vector ties
    "ec_timestep_d2048_e64": dict(G=4, L=256, d=192, E=8, d_ff=192, k_base=48),
    # many experts with router bias
    "ec_many_small_e128": dict(G=4, L=256, d=128, E=128, d_ff=64, k_base=16),
    # wide, few experts
    "ec_wide_d4096_e32_x4": dict(G=2, L=1024, d=512, E=32, d_ff=256, k_base=64, layers=1),
}


@pytest.mark.parametrize("name", sorted(SMALL_BF16))
def test_bf16_small_layers_match_oracle(name):
    w = I.scaled(I.WORKLOADS[name], **SMALL_BF16[name])
    _check_layer(I.make_inputs(w))


def test_bf16_is_deterministic():
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], **SMALL_BF16["ec_d2048_e64"])
    inp = I.make_inputs(w)
    _, a = gpu_layer(inp)
    _, b = gpu_layer(inp)
    for k in ("Y", "idx", "gate", "dX", "dWr", "dWg", "dWu", "dWd"):
        assert torch.equal(a[k], b[k]), k


def test_set_capacity_matches_fresh_context():
    from paper_2604_01622_gb300.layer import ECMoELayer
    w = I.scaled(I.WORKLOADS["ec_timestep_d2048_e64"], **SMALL_BF16["ec_timestep_d2048_e64"])
    inp = I.make_inputs(w)
    L = inp.layers[0]
    args = (dev(inp.X), dev(L.Wr), None, dev(L.Wg), dev(L.Wu), dev(L.Wd))
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype="bf16")
    k2 = np.array([60, 10, 0, 100], np.int32)          # same total, new split
    lay.set_capacity(k2)
    Y1, idx1, _, _ = lay.forward(*args)
    fresh = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, k2, dtype="bf16")
    Y2, idx2, _, _ = fresh.forward(*args)
    lay.check()
    fresh.check()
    assert torch.equal(idx1, idx2) and torch.equal(Y1, Y2)


# ------------------------------------------------------------------ bf16 edge cases
def test_bf16_ragged_groups_and_capacity_edges():
    """Tensor-core path with an empty group, a one-token group, k = 0 and k = L: 11 experts
    of M = 168 rows (one 128-row tile and a 40-row tail) over 333 tokens."""
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=1, L=333, d=128, E=11, d_ff=64, seed=13,
                 router_bias=True, layers=1)
    inp = I.make_inputs(w)
    inp.group_off = np.array([0, 0, 150, 151, 333], np.int32)
    inp.k_g = np.array([0, 150, 1, 17], np.int32)
    _check_layer(inp)


def _wide_case():
    # d = 512 and 2 d_ff = 512: with EC_TILES_512 every GEMM but dU takes 256 x 512 tiles (two
    # 256-column accumulator halves handed over separately); M = 3 * 70 = 210 rows leaves a
    # ragged row tile, and the short K loops (4 k-slices in the down GEMM, 8 in the others)
    # hold the half-1 MMAs at both ends of a tile at once
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=3, L=256, d=512, E=6, d_ff=256, k_base=70,
                 seed=17, router_bias=True, layers=1)
    return I.make_inputs(w)


def test_bf16_wide_tiles_match_oracle():
    from paper_2604_01622_gb300 import EC_TILES_512
    _check_layer(_wide_case(), tiles=EC_TILES_512)


def test_bf16_wide_tiles_single_k_slice():
    """M = 40 rows per expert: the weight-gradient GEMMs' K loop is one 64-row slice, shorter
    than the 3-slice tail whose half-1 MMAs wait for half 0, so every k-slice is held."""
    from paper_2604_01622_gb300 import EC_TILES_512
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=64, d=512, E=5, d_ff=256, k_base=20,
                 seed=18, layers=1)
    _check_layer(I.make_inputs(w), tiles=EC_TILES_512)


def test_bf16_tile_policies_agree_bit_for_bit():
    """256 x 256 and 256 x 512 tiles issue the same N = 256 MMAs over K in the same order and
    the same epilogue arithmetic per element, so every output is bit-identical."""
    from paper_2604_01622_gb300 import EC_TILES_256, EC_TILES_512
    inp = _wide_case()
    _, a = gpu_layer(inp, tiles=EC_TILES_256)
    _, b = gpu_layer(inp, tiles=EC_TILES_512)
    for k in ("Y", "idx", "gate", "dX", "dWr", "dbr", "dWg", "dWu", "dWd"):
        assert torch.equal(a[k], b[k]), k


def test_bf16_wide_dgrad_up_tiles_match_oracle_and_narrow_tiles():
    """d_ff = 512: the dU GEMM (SwiGLU backward and gate-gradient partials in its epilogue)
    takes 256 x 512 tiles too; M = 2 * 75 rows leaves a ragged row tile and d = 256 a K loop
    of 4 k-slices. The partials cover the same column blocks in both tile forms, so the
    results equal the 256 x 256 ones bit for bit."""
    from paper_2604_01622_gb300 import EC_TILES_256, EC_TILES_512
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=200, d=256, E=5, d_ff=512, k_base=75,
                 seed=23, router_bias=True, layers=1)
    inp = I.make_inputs(w)
    _check_layer(inp, tiles=EC_TILES_512)
    _, a = gpu_layer(inp, tiles=EC_TILES_256)
    _, b = gpu_layer(inp, tiles=EC_TILES_512)
    for k in ("Y", "dX", "dWr", "dbr", "dWg", "dWu", "dWd"):
        assert torch.equal(a[k], b[k]), k


@pytest.mark.parametrize("G,L,E", [(3, 1700, 16), (1, 4868, 64), (2, 2050, 128)])
def test_bf16_router_row_split_uneven(G, L, E):
    """The router splits the tokens over the SMs in 32-row units: 160, 153 and 129 units
    here over at most 152 CTAs, so some CTAs take one unit more than others, tiles of 32 to
    128 rows occur, and the last unit is ragged (none of 5100, 4868, 4100 is a multiple of
    32)."""
    w = I.scaled(I.WORKLOADS["ec_many_small_e128"], G=G, L=L, d=128, E=E, d_ff=64,
                 k_base=max(1, L // 8), seed=29, router_bias=True, layers=1)
    _check_layer(I.make_inputs(w))


@pytest.mark.parametrize("E", [160, 256])
def test_bf16_many_experts_router_widths(E):
    """160 and 256 experts take the router GEMM's 192- and 256-column tiles (softmax over
    the valid columns of a zero-padded score tile); 256 is the largest expert count."""
    w = I.scaled(I.WORKLOADS["ec_many_small_e128"], G=2, L=256, d=128, E=E, d_ff=64, k_base=8,
                 seed=19, router_bias=True, layers=1)
    _check_layer(I.make_inputs(w))


def test_bf16_few_tokens_minimum_widths():
    """Five tokens, d = d_ff = 64 (one k-step, one column block): M = 2 rows per expert."""
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=1, L=5, d=64, E=3, d_ff=64, k_base=2, seed=15,
                 layers=1)
    _check_layer(I.make_inputs(w))


def test_bf16_single_expert_is_a_dense_mlp():
    """E = 1 and k = L: every token goes to the one expert with gate S = 1 (a plain SwiGLU
    MLP), and the router gets no gradient: dZ = S (dS - <dS, S>) is exactly zero."""
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=200, d=64, E=1, d_ff=128, k_base=200,
                 seed=14, layers=1)
    inp = I.make_inputs(w)
    _, out = gpu_layer(inp)
    assert not out["dWr"].any()
    assert torch.equal(out["gate"], torch.ones_like(out["gate"]))
    _check_layer(inp)


def test_bf16_zero_capacity_everywhere():
    """k_g = 0 in every group: no expert rows, so Y, dX and every gradient are exact zeros."""
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=100, d=128, E=4, d_ff=64, k_base=0,
                 seed=16, router_bias=True, layers=1)
    inp = I.make_inputs(w)
    _, out = gpu_layer(inp)
    assert out["idx"].numel() == 0
    for k in ("Y", "dX", "dWr", "dbr", "dWg", "dWu", "dWd"):
        assert not out[k].any(), k
