"""Pins of the float64 oracle against what the paper and the mathematics fix.

No test here retypes an oracle formula: each compares the oracle with an
independent route to the same value (a library routine, a brute-force count,
a reduction to a textbook case, finite differences, automatic differentiation)
or with an invariant the paper states.
"""
import numpy as np
import pytest
import scipy.special
import torch

from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I


def _tiny(seed=0, N=48, d=12, E=5, d_ff=10, groups=(0, 20, 48), k=(6, 9), bias=True):
    rng = np.random.default_rng(seed)
    X = rng.standard_normal((N, d))
    Wr = rng.standard_normal((d, E)) / np.sqrt(d)
    br = rng.standard_normal(E) if bias else None
    Wg = rng.standard_normal((E, d, d_ff)) / np.sqrt(d)
    Wu = rng.standard_normal((E, d, d_ff)) / np.sqrt(d)
    Wd = rng.standard_normal((E, d_ff, d)) / np.sqrt(d_ff)
    return X, Wr, br, Wg, Wu, Wd, np.array(groups), np.array(k)


# --------------------------------------------------------------- router (Sec. 2.2)
def test_softmax_rows_sum_to_one_and_match_library():
    rng = np.random.default_rng(1)
    Z = rng.standard_normal((300, 17)) * 30.0
    S = O.softmax_rows(Z)
    assert np.max(np.abs(S.sum(axis=1) - 1.0)) < 1e-12
    np.testing.assert_allclose(S, scipy.special.softmax(Z, axis=1), rtol=1e-13, atol=1e-300)
    assert np.all(S > 0)


def test_router_single_expert_is_one_and_shift_invariant():
    rng = np.random.default_rng(2)
    X = rng.standard_normal((20, 7))
    assert np.all(O.router_scores(X, rng.standard_normal((7, 1))) == 1.0)
    Wr = rng.standard_normal((7, 4))
    S0 = O.router_scores(X, Wr)
    S1 = O.router_scores(X, Wr, np.full(4, 3.25))
    np.testing.assert_allclose(S0, S1, rtol=1e-13)
    # a bias on one expert raises that expert's score in every row
    S2 = O.router_scores(X, Wr, np.array([0.0, 0.0, 1.0, 0.0]))
    assert np.all(S2[:, 2] > S0[:, 2])


# --------------------------------------------------------------- selection (Sec. 2.2, 4.2, 5.2)
def _brute_force_select(S, group_off, k_g):
    """Token t of group g is chosen by expert e iff fewer than k_g tokens of g
    beat it, where u beats t when S[u,e] > S[t,e] or (equal and u < t).
    Counted pairwise, with no sorting."""
    N, E = S.shape
    sel = np.zeros((N, E), dtype=bool)
    for e in range(E):
        for g in range(len(k_g)):
            lo, hi = group_off[g], group_off[g + 1]
            for t in range(lo, hi):
                beaten_by = 0
                for u in range(lo, hi):
                    if S[u, e] > S[t, e] or (S[u, e] == S[t, e] and u < t):
                        beaten_by += 1
                sel[t, e] = beaten_by < k_g[g]
    return sel


@pytest.mark.parametrize("quant", [None, 4.0, 1.0])
def test_selection_matches_brute_force(quant):
    rng = np.random.default_rng(3)
    N, E = 60, 6
    for trial in range(6):
        S = rng.random((N, E))
        if quant is not None:  # forced ties
            S = np.round(S * quant) / quant
        S[rng.random((N, E)) < 0.05] = -0.0 if trial % 2 else 0.0
        group_off = I.random_groups(rng, N, 4)
        k_g = np.array([rng.integers(0, group_off[g + 1] - group_off[g] + 1) for g in range(4)])
        idx, gate = O.ec_select(S, group_off, k_g)
        sel = _brute_force_select(S + 0.0, group_off, k_g)
        for e in range(E):
            assert np.array_equal(np.sort(idx[e]), np.nonzero(sel[:, e])[0])
            assert np.array_equal(gate[e], S[idx[e], e])


def test_selection_invariants_and_edges():
    rng = np.random.default_rng(4)
    N, E = 64, 5
    S = rng.random((N, E))
    group_off = np.array([0, 10, 10, 40, 64])      # includes an empty group
    k_g = np.array([3, 0, 30, 7])                  # k = 0 and k = L
    idx, gate = O.ec_select(S, group_off, k_g)
    M = k_g.sum()
    assert idx.shape == (E, M)                     # every expert has the same load M
    for e in range(E):
        pos = 0
        for g in range(4):
            blk = idx[e, pos:pos + k_g[g]]
            assert len(set(blk.tolist())) == k_g[g]            # no duplicates
            assert np.all(np.diff(blk) > 0)                    # ascending
            assert np.all((blk >= group_off[g]) & (blk < group_off[g + 1]))
            pos += k_g[g]
        # k = L takes the whole group
        assert np.array_equal(idx[e, 3:33], np.arange(10, 40))


def test_expert_choice_balance_six_by_three():
    """Fig. 2 setting: 6 tokens, 3 experts, capacity 2 -> loads 2/2/2 and
    E*c = 6 pairs, the same count as token-choice top-1 over 6 tokens."""
    rng = np.random.default_rng(5)
    for _ in range(20):
        S = O.softmax_rows(rng.standard_normal((6, 3)))
        idx, _ = O.ec_select(S, [0, 6], [2])
        loads = [len(idx[e]) for e in range(3)]
        assert loads == [2, 2, 2]
        assert sum(loads) == 6 * 1
        # TC top-1 on the same scores: a per-row argmax, whose loads vary
        tc = np.bincount(S.argmax(axis=1), minlength=3)
        assert tc.sum() == 6


# --------------------------------------------------------------- forward (Sec. 2.2, App. "Experimental Setup")
def test_silu_and_grad_match_torch():
    a = np.linspace(-30, 30, 601)
    ta = torch.tensor(a, dtype=torch.float64, requires_grad=True)
    ts = torch.nn.functional.silu(ta)
    ts.sum().backward()
    np.testing.assert_allclose(O.silu(a), ts.detach().numpy(), rtol=1e-14, atol=1e-300)
    np.testing.assert_allclose(O.silu_grad(a), ta.grad.numpy(), rtol=1e-12, atol=1e-300)


def test_single_expert_full_capacity_is_textbook_swiglu_mlp():
    """E = 1 and k = L: S == 1, every token chosen once, so Y = SwiGLU-MLP(X)."""
    rng = np.random.default_rng(6)
    N, d, f = 40, 9, 13
    X = rng.standard_normal((N, d))
    Wr = rng.standard_normal((d, 1))
    Wg, Wu = rng.standard_normal((1, d, f)), rng.standard_normal((1, d, f))
    Wd = rng.standard_normal((1, f, d))
    out = O.forward(X, Wr, None, Wg, Wu, Wd, [0, 25, 40], [25, 15])
    tx = torch.tensor(X)
    mlp = (torch.nn.functional.silu(tx @ torch.tensor(Wg[0])) * (tx @ torch.tensor(Wu[0]))) \
        @ torch.tensor(Wd[0])
    np.testing.assert_allclose(out["Y"], mlp.numpy(), rtol=1e-12, atol=1e-12)


def test_full_capacity_reduces_to_dense_soft_moe():
    """k_g = L for all groups: Y = sum_e S[:, e] * FFN_e(X), no gather or scatter."""
    X, Wr, br, Wg, Wu, Wd, groups, _ = _tiny(7)
    L = np.diff(groups)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, L)
    S = scipy.special.softmax(X @ Wr + br, axis=1)
    Y = np.zeros_like(X)
    for e in range(Wr.shape[1]):
        A = np.einsum("nd,df->nf", X, Wg[e])
        B = np.einsum("nd,df->nf", X, Wu[e])
        Y += S[:, e:e + 1] * np.einsum("nf,fd->nd", scipy.special.expit(A) * A * B, Wd[e])
    np.testing.assert_allclose(out["Y"], Y, rtol=1e-12, atol=1e-12)


def test_unpicked_tokens_get_exact_zero():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(8, k=(2, 3))
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    picked = np.zeros(X.shape[0], bool)
    picked[out["idx"].ravel()] = True
    assert (~picked).sum() > 0
    assert np.all(out["Y"][~picked] == 0.0)
    bw = O.backward(out, np.random.default_rng(0).standard_normal(X.shape), Wr, Wg, Wu, Wd)
    assert np.all(bw["dX"][~picked] == 0.0)
    assert np.all(bw["dZ"][~picked] == 0.0)
    assert O.drop_ratio(out["idx"], X.shape[0]) == pytest.approx((~picked).mean())


def test_token_permutation_within_group_is_equivariant():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(9)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    rng = np.random.default_rng(1)
    perm = np.arange(X.shape[0])
    perm[0:20] = rng.permutation(20)
    perm[20:48] = 20 + rng.permutation(28)
    out_p = O.forward(X[perm], Wr, br, Wg, Wu, Wd, groups, k)
    np.testing.assert_allclose(out_p["Y"], out["Y"][perm], rtol=1e-12, atol=1e-13)


# --------------------------------------------------------------- backward (chain rule)
def _objective(X, Wr, br, Wg, Wu, Wd, groups, k, dY, ref_idx):
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    return float(np.sum(dY * out["Y"])), np.array_equal(out["idx"], ref_idx)


def test_backward_matches_central_finite_differences():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(10)
    rng = np.random.default_rng(11)
    dY = rng.standard_normal(X.shape)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    g = O.backward(out, dY, Wr, Wg, Wu, Wd)
    params = {"X": X, "Wr": Wr, "br": br, "Wg": Wg, "Wu": Wu, "Wd": Wd}
    grads = {"X": g["dX"], "Wr": g["dWr"], "br": g["dbr"], "Wg": g["dWg"], "Wu": g["dWu"],
             "Wd": g["dWd"]}
    h = 1e-6
    checked = 0
    for name in params:
        for trial in range(4):
            V = rng.standard_normal(params[name].shape)
            plus = dict(params)
            minus = dict(params)
            plus[name] = params[name] + h * V
            minus[name] = params[name] - h * V
            fp, same_p = _objective(**plus, groups=groups, k=k, dY=dY, ref_idx=out["idx"])
            fm, same_m = _objective(**minus, groups=groups, k=k, dY=dY, ref_idx=out["idx"])
            if not (same_p and same_m):
                continue  # the perturbation moved the selection: not differentiable here
            fd = (fp - fm) / (2 * h)
            an = float(np.sum(grads[name] * V))
            assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (name, fd, an)
            checked += 1
    assert checked >= 20


def test_backward_matches_torch_autograd_with_fixed_selection():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(12, E=4)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    dY = np.random.default_rng(13).standard_normal(X.shape)
    g = O.backward(out, dY, Wr, Wg, Wu, Wd)
    t = {n: torch.tensor(v, requires_grad=True) for n, v in
         dict(X=X, Wr=Wr, br=br, Wg=Wg, Wu=Wu, Wd=Wd).items()}
    S = torch.softmax(t["X"] @ t["Wr"] + t["br"], dim=1)
    Y = torch.zeros_like(t["X"])
    idx = torch.tensor(out["idx"])
    for e in range(Wr.shape[1]):
        h = t["X"][idx[e]]
        o = (torch.nn.functional.silu(h @ t["Wg"][e]) * (h @ t["Wu"][e])) @ t["Wd"][e]
        Y = Y.index_add(0, idx[e], S[idx[e], e:e + 1] * o)
    (Y * torch.tensor(dY)).sum().backward()
    for name, key in [("X", "dX"), ("Wr", "dWr"), ("br", "dbr"), ("Wg", "dWg"), ("Wu", "dWu"),
                      ("Wd", "dWd")]:
        np.testing.assert_allclose(g[key], t[name].grad.numpy(), rtol=1e-10, atol=1e-12)


def test_router_gradient_rows_sum_to_zero():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(14)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    g = O.backward(out, np.random.default_rng(0).standard_normal(X.shape), Wr, Wg, Wu, Wd)
    assert np.max(np.abs(g["dZ"].sum(axis=1))) < 1e-13
    assert abs(g["dbr"].sum()) < 1e-12
    assert np.max(np.abs(g["dWr"].sum(axis=1))) < 1e-12


# --------------------------------------------------------------- sampled forms agree with full forms
def test_sampled_forms_match_full_layer():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(15)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    dY = np.random.default_rng(16).standard_normal(X.shape)
    g = O.backward(out, dY, Wr, Wg, Wu, Wd)
    toks = [0, 5, 19, 20, 33, 47]
    pairs = O.token_pairs(out["idx"], toks)
    rows = {t: X[t] for t in toks}
    srows = {t: out["S"][t] for t in toks}
    dyr = {t: dY[t] for t in toks}
    yt = O.forward_tokens(rows, srows, pairs, lambda e: Wg[e], lambda e: Wu[e], lambda e: Wd[e])
    dxt = O.backward_tokens(rows, srows, dyr, pairs, Wr, lambda e: Wg[e], lambda e: Wu[e],
                            lambda e: Wd[e])
    for t in toks:
        np.testing.assert_allclose(yt[t], out["Y"][t], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(dxt[t], g["dX"][t], rtol=1e-11, atol=1e-12)
    for e in range(Wr.shape[1]):
        idx = out["idx"][e]
        dwg, dwu, dwd, dgate = O.backward_expert(X[idx], out["gate"][e], dY[idx], Wg[e], Wu[e], Wd[e])
        np.testing.assert_allclose(dwg, g["dWg"][e], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(dwu, g["dWu"][e], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(dwd, g["dWd"][e], rtol=1e-11, atol=1e-12)
        np.testing.assert_allclose(dgate, g["dgate"][e], rtol=1e-11, atol=1e-12)


@pytest.mark.parametrize("bias", [True, False])
def test_streamed_router_backward_matches_full_backward(bias):
    """The expert-at-a-time form used at full size gives the full backward's dS, dZ, dWr, dbr
    (which finite differences and autograd pin)."""
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(17, bias=bias)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    dY = np.random.default_rng(18).standard_normal(X.shape)
    g = O.backward(out, dY, Wr, Wg, Wu, Wd)
    r = O.router_backward_streamed(X, Wr, br, dY, out["idx"], lambda e: Wg[e], lambda e: Wu[e],
                                   lambda e: Wd[e])
    for key in ("dS", "dZ", "dWr", "dbr"):
        np.testing.assert_allclose(r[key], g[key], rtol=1e-11, atol=1e-13)


def test_per_token_stack_matches_full_stack():
    """Per-token composition through stacked layers equals the full stack on those rows."""
    X, *_rest, groups, k = _tiny(23, N=40, d=8, E=4, d_ff=6, groups=(0, 17, 40), k=(5, 7))
    layers = []
    for l in range(3):
        _, Wr, br, Wg, Wu, Wd, _, _ = _tiny(40 + l, N=40, d=8, E=4, d_ff=6, groups=(0, 17, 40),
                                            bias=l != 1)
        layers.append((Wr, br, Wg, Wu, Wd))
    dOut = np.random.default_rng(24).standard_normal(X.shape)
    xs, fwds = O.stack_forward(X, layers, groups, k)
    d0, _ = O.stack_backward(fwds, layers, dOut)
    toks = [0, 3, 16, 17, 29, 39]
    pairs = [O.token_pairs(f["idx"], toks) for f in fwds]
    fn = [(Wr, br, (lambda e, W=Wg: W[e]), (lambda e, W=Wu: W[e]), (lambda e, W=Wd: W[e]))
          for (Wr, br, Wg, Wu, Wd) in layers]
    xt, dt = O.stack_tokens({t: X[t] for t in toks}, {t: dOut[t] for t in toks}, fn, pairs)
    for t in toks:
        for l in range(len(layers) + 1):
            np.testing.assert_allclose(xt[l][t], xs[l][t], rtol=1e-12, atol=1e-13)
        np.testing.assert_allclose(dt[t], d0[t], rtol=1e-11, atol=1e-12)


def test_residual_stack_backward_matches_finite_differences():
    rng = np.random.default_rng(21)
    X, *_rest, groups, k = _tiny(22, N=30, d=6, E=3, d_ff=5, groups=(0, 14, 30), k=(4, 6))
    layers = []
    for l in range(2):
        _, Wr, br, Wg, Wu, Wd, _, _ = _tiny(30 + l, N=30, d=6, E=3, d_ff=5, groups=(0, 14, 30))
        layers.append((Wr, br, Wg, Wu, Wd))
    dOut = rng.standard_normal(X.shape)
    xs, fwds = O.stack_forward(X, layers, groups, k)
    # one layer of the stack is the layer plus its input
    f0 = O.forward(X, *layers[0], groups, k)
    np.testing.assert_allclose(xs[1], X + f0["Y"], rtol=0, atol=0)
    dX, _ = O.stack_backward(fwds, layers, dOut)
    idx_ref = [f["idx"] for f in fwds]
    h = 1e-6
    for _ in range(4):
        V = rng.standard_normal(X.shape)
        xp, fp = O.stack_forward(X + h * V, layers, groups, k)
        xm, fm = O.stack_forward(X - h * V, layers, groups, k)
        if not all(np.array_equal(a["idx"], b) and np.array_equal(c["idx"], b)
                   for a, c, b in zip(fp, fm, idx_ref)):
            continue
        fd = (np.sum(dOut * xp[-1]) - np.sum(dOut * xm[-1])) / (2 * h)
        an = float(np.sum(dX * V))
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an))


# --------------------------------------------------------------- shared experts (appendix "Token Coverage")
def _shared(seed, d, f, S=2):
    rng = np.random.default_rng(seed)
    return [(rng.standard_normal((d, f)) / np.sqrt(d), rng.standard_normal((d, f)) / np.sqrt(d),
             rng.standard_normal((f, d)) / np.sqrt(f)) for _ in range(S)]


def test_shared_experts_sum_equals_one_concatenated_swiglu():
    """Two shared experts of width f act like one SwiGLU FFN of width 2f (hidden units are
    independent), computed here with torch on concatenated weights."""
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(40)
    sh = _shared(41, X.shape[1], 7)
    with_sh = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k, shared=sh)
    without = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k)
    tx = torch.tensor(X)
    Wgc = torch.tensor(np.concatenate([s[0] for s in sh], axis=1))
    Wuc = torch.tensor(np.concatenate([s[1] for s in sh], axis=1))
    Wdc = torch.tensor(np.concatenate([s[2] for s in sh], axis=0))
    ffn = (torch.nn.functional.silu(tx @ Wgc) * (tx @ Wuc)) @ Wdc
    np.testing.assert_allclose(with_sh["Y"] - without["Y"], ffn.numpy(), rtol=1e-11, atol=1e-12)
    # unpicked tokens now carry only the shared output
    picked = np.zeros(X.shape[0], bool)
    picked[with_sh["idx"].ravel()] = True
    np.testing.assert_allclose(with_sh["Y"][~picked], ffn.numpy()[~picked], rtol=1e-11, atol=1e-12)


def test_shared_experts_backward_matches_finite_differences():
    X, Wr, br, Wg, Wu, Wd, groups, k = _tiny(42)
    sh = _shared(43, X.shape[1], 6)
    rng = np.random.default_rng(44)
    dY = rng.standard_normal(X.shape)
    out = O.forward(X, Wr, br, Wg, Wu, Wd, groups, k, shared=sh)
    g = O.backward(out, dY, Wr, Wg, Wu, Wd)
    h = 1e-6

    def f(X_, sh_):
        o = O.forward(X_, Wr, br, Wg, Wu, Wd, groups, k, shared=sh_)
        return float(np.sum(dY * o["Y"])), np.array_equal(o["idx"], out["idx"])
    checked = 0
    for trial in range(3):
        V = rng.standard_normal(X.shape)
        (fp, okp), (fm, okm) = f(X + h * V, sh), f(X - h * V, sh)
        if okp and okm:
            an = float(np.sum(g["dX"] * V))
            assert abs((fp - fm) / (2 * h) - an) <= 1e-6 * max(1.0, abs(an))
            checked += 1
        for s_i in range(2):
            for w_i in range(3):
                Vw = rng.standard_normal(sh[s_i][w_i].shape)
                shp = [list(t) for t in sh]
                shm = [list(t) for t in sh]
                shp[s_i][w_i] = sh[s_i][w_i] + h * Vw
                shm[s_i][w_i] = sh[s_i][w_i] - h * Vw
                fd = (f(X, shp)[0] - f(X, shm)[0]) / (2 * h)
                an = float(np.sum(g["dshared"][s_i][w_i] * Vw))
                assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), (s_i, w_i)
                checked += 1
    assert checked >= 12
