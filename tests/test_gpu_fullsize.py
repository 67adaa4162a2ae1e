"""Full-size workloads on the GPU, checked against the oracle on samples it can compute.

At full size the oracle cannot run the whole layer in float64 in seconds, so:
  * the selection is compared bit-exactly in full (oracle top-k on the GPU's scores);
  * outputs Y and input gradients dX are compared on sampled tokens (each needs only the
    experts that chose that token);
  * weight gradients are compared on a sampled expert, restricted to a slice of d_ff
    columns (a column slice of the gate/up weights and the matching rows of the down
    weights give exactly that slice of every weight gradient);
  * dWr and dbr are compared element by element with the oracle's router backward computed
    one expert at a time over all pairs (the full layer's dS needs every pair's FFN output,
    seconds of float64 work), besides the properties that hold at any size (softmax
    gradient rows sum to zero); unpicked tokens must give exact zeros.
Tolerance: relative max-norm 2e-2 over each sample (bf16 path).
"""
import numpy as np
import pytest

from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I
from tests._util import gpu_layer, host, relmax, tol

pytestmark = pytest.mark.gpu

FULL = ["ec_d2048_e64", "ec_timestep_d2048_e64", "ec_many_small_e128", "ec_wide_d4096_e32_x4"]


@pytest.mark.parametrize("name", FULL)
def test_full_size_sampled_parity(name):
    w = I.scaled(I.WORKLOADS[name], layers=1)
    _check_sampled(I.make_inputs(w), full_router=True)


def test_large_batch_past_32_bit_offsets():
    """8 sequences of 32768 tokens, 4096 per expert and sequence: 2.1 M expert rows, so the
    gathered rows H and dY[idx] hold 4.4 G elements each, past 32-bit element offsets (and
    about 55 GB are in use on the GPU). The bench workload's 32768 tokens are repeated in
    every sequence; selection is per sequence, so each sequence picks the same positions,
    and the samples include tokens of the last sequence (rows above 2^31 elements)."""
    base = I.scaled(I.WORKLOADS["ec_d2048_e64"], layers=1)
    inp0 = I.make_inputs(base)
    G, L = 8, base.N
    w = I.scaled(base, G=G, L=L, k_base=4096)
    X = I.Tensor(np.tile(inp0.X.data, (G, 1)), inp0.X.dtype)
    dY = I.Tensor(np.tile(inp0.dY.data, (G, 1)), inp0.dY.dtype)
    inp = I.Inputs(w, X, dY, (np.arange(G + 1) * L).astype(np.int32),
                   np.full(G, 4096, np.int32), inp0.layers)
    _check_sampled(inp, extra_tokens=[w.N - 1, w.N - 4097, (G - 1) * L + 123])


def _check_sampled(inp, extra_tokens=(), full_router=False):
    w = inp.w
    L = inp.layers[0]
    lay, out = gpu_layer(inp)
    bound = tol(w)
    S_gpu = host(out["S"]).T
    idx = out["idx"].cpu().numpy()
    # 1. selection, in full, on the GPU's scores
    ref_idx, ref_gate = O.ec_select(S_gpu, inp.group_off, inp.k_g)
    assert np.array_equal(idx, ref_idx)
    assert np.array_equal(host(out["gate"]), ref_gate)
    assert idx.shape == (w.E, int(inp.k_g.sum()))

    Wr = L.Wr.f64()
    rng = np.random.default_rng(2024)
    picked = np.zeros(w.N, bool)
    picked[idx.ravel()] = True
    toks = list(rng.choice(np.nonzero(picked)[0], 24, replace=False)) + list(extra_tokens)
    if (~picked).any():
        toks += list(rng.choice(np.nonzero(~picked)[0], min(4, int((~picked).sum())), replace=False))
    toks = [int(t) for t in toks]
    Xr = inp.X.f64(np.array(toks))
    S_or = O.router_scores(Xr, Wr, L.br)
    rows = {t: Xr[i] for i, t in enumerate(toks)}
    srows = {t: S_or[i] for i, t in enumerate(toks)}
    dyr = {t: inp.dY.f64(np.array([t]))[0] for t in toks}
    pairs = O.token_pairs(idx, toks)
    Wg = lambda e: L.Wg.f64(e)
    Wu = lambda e: L.Wu.f64(e)
    Wd = lambda e: L.Wd.f64(e)
    # 2. sampled outputs and input gradients
    y_ref = O.forward_tokens(rows, srows, pairs, Wg, Wu, Wd)
    dx_ref = O.backward_tokens(rows, srows, dyr, pairs, Wr, Wg, Wu, Wd)
    Y = host(out["Y"])
    dX = host(out["dX"])
    e_y = relmax(np.stack([Y[t] for t in toks]), np.stack([y_ref[t] for t in toks]))
    e_dx = relmax(np.stack([dX[t] for t in toks]), np.stack([dx_ref[t] for t in toks]))
    assert e_y <= bound and e_dx <= bound, (e_y, e_dx)
    for t in toks:
        if not pairs[t]:
            assert np.all(Y[t] == 0.0) and np.all(dX[t] == 0.0)
    # 3. weight gradients of one expert on a slice of d_ff columns
    e = int(rng.integers(w.E))
    cols = np.sort(rng.choice(w.d_ff, 64, replace=False))
    H = inp.X.f64(idx[e])
    s_col = O.router_scores(H, Wr, L.br)[:, e]
    dYe = inp.dY.f64(idx[e])
    dwg, dwu, dwd, _ = O.backward_expert(H, s_col, dYe, Wg(e)[:, cols], Wu(e)[:, cols],
                                         Wd(e)[cols, :])
    g_dwg = out["dWg"][e][:, cols].double().cpu().numpy()
    g_dwu = out["dWu"][e][:, cols].double().cpu().numpy()
    g_dwd = out["dWd"][e][cols, :].double().cpu().numpy()
    errs = (relmax(g_dwg, dwg), relmax(g_dwu, dwu), relmax(g_dwd, dwd))
    assert max(errs) <= bound, errs
    # 4. router gradients: rows of the softmax Jacobian product sum to zero
    dWr = host(out["dWr"])
    assert np.max(np.abs(dWr.sum(axis=1))) <= 1e-3 * np.max(np.abs(dWr))
    if L.br is not None:
        dbr = host(out["dbr"])
        assert abs(dbr.sum()) <= 1e-3 * np.max(np.abs(dbr)) * w.E
    # 5. router gradients in full, element by element
    if full_router:
        r = O.router_backward_streamed(inp.X.f64(), Wr, L.br, inp.dY.f64(), idx, Wg, Wu, Wd)
        errs = {"dWr": relmax(dWr, r["dWr"])}
        if L.br is not None:
            errs["dbr"] = relmax(host(out["dbr"]), r["dbr"])
        assert max(errs.values()) <= bound, errs
    lay.close()
