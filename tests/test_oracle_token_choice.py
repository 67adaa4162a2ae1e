"""Pins of the token-choice oracle (Sec. 2.2): brute-force top-k, the capacity rule, the
dense reduction shared with expert choice, finite differences and torch autograd."""
import numpy as np
import pytest
import torch

from oracle import ecmoe as O
from oracle import token_choice as T
from tests.test_oracle_pins import _tiny


def test_topk_rows_match_brute_force_with_ties():
    rng = np.random.default_rng(50)
    S = np.round(rng.random((80, 9)) * 4) / 4                   # many ties
    for k in (1, 2, 4, 9):
        choices, gates, kept = T.tc_select(S, k)
        for t in range(80):
            beats = lambda u, j: S[t, u] > S[t, j] or (S[t, u] == S[t, j] and u < j)
            ranked = sorted(range(9), key=lambda j: sum(beats(u, j) for u in range(9)))
            assert list(choices[t]) == ranked[:k]
        np.testing.assert_allclose(gates.sum(axis=1), 1.0, rtol=1e-13)
        assert kept.all()


def test_capacity_keeps_first_tokens_and_bounds_loads():
    rng = np.random.default_rng(51)
    S = O.softmax_rows(rng.standard_normal((200, 6)) + np.array([2.0, 0, 0, 0, 0, -1]))
    k, E, N = 2, 6, 200
    C = T.tc_capacity(1.0, k, N, E)
    assert C == int(np.ceil(1.0 * k * N / E))
    choices, gates, kept = T.tc_select(S, k, C)
    loads = np.bincount(choices[kept], minlength=E)
    assert loads.max() <= C and (~kept).any()
    for e in range(E):                                           # kept = first C in token order
        rows = [t for t in range(N) if e in choices[t]]
        kept_rows = [t for t in range(N) for r in range(k) if choices[t, r] == e and kept[t, r]]
        assert kept_rows == rows[:C]
    assert T.tc_capacity(None, k, N, E) is None and T.tc_capacity(0, k, N, E) is None


def test_all_experts_dropless_equals_expert_choice_dense_reduction():
    """k = E and no cap: every token uses every expert with gate S / 1, the same dense
    soft-MoE as expert choice with k_g = L."""
    X, Wr, br, Wg, Wu, Wd, groups, _ = _tiny(52, E=4)
    tc = T.tc_forward(X, Wr, br, Wg, Wu, Wd, k=4)
    ec = O.forward(X, Wr, br, Wg, Wu, Wd, groups, np.diff(groups))
    np.testing.assert_allclose(tc["Y"], ec["Y"], rtol=1e-11, atol=1e-12)


def test_backward_matches_finite_differences_and_autograd():
    X, Wr, br, Wg, Wu, Wd, groups, _ = _tiny(53, N=40, E=5)
    k, C = 2, 14
    rng = np.random.default_rng(54)
    dY = rng.standard_normal(X.shape)
    fwd = T.tc_forward(X, Wr, br, Wg, Wu, Wd, k, C)
    assert (~fwd["kept"]).any()
    g = T.tc_backward(fwd, dY, Wr, Wg, Wu, Wd)
    forced = (fwd["choices"], fwd["kept"])
    params = {"X": X, "Wr": Wr, "br": br, "Wg": Wg, "Wu": Wu, "Wd": Wd}
    keys = {"X": "dX", "Wr": "dWr", "br": "dbr", "Wg": "dWg", "Wu": "dWu", "Wd": "dWd"}
    h = 1e-6
    for name in params:
        V = rng.standard_normal(params[name].shape)
        p_, m_ = dict(params), dict(params)
        p_[name] = params[name] + h * V
        m_[name] = params[name] - h * V
        fp = T.tc_forward(p_["X"], p_["Wr"], p_["br"], p_["Wg"], p_["Wu"], p_["Wd"], k, C)
        fm = T.tc_forward(m_["X"], m_["Wr"], m_["br"], m_["Wg"], m_["Wu"], m_["Wd"], k, C)
        if not (np.array_equal(fp["choices"], fwd["choices"]) and
                np.array_equal(fm["choices"], fwd["choices"])):
            continue
        fd = (np.sum(dY * fp["Y"]) - np.sum(dY * fm["Y"])) / (2 * h)
        an = float(np.sum(g[keys[name]] * V))
        assert abs(fd - an) <= 1e-6 * max(1.0, abs(an)), name
    # autograd of the same layer with the selection fixed
    t = {n: torch.tensor(v, requires_grad=True) for n, v in params.items()}
    S = torch.softmax(t["X"] @ t["Wr"] + t["br"], dim=1)
    ch = torch.tensor(fwd["choices"])
    sel = torch.gather(S, 1, ch)
    gates = sel / sel.sum(dim=1, keepdim=True)
    Y = torch.zeros_like(t["X"])
    for tok in range(X.shape[0]):
        for r in range(k):
            if fwd["kept"][tok, r]:
                e = int(ch[tok, r])
                h_ = t["X"][tok]
                o = (torch.nn.functional.silu(h_ @ t["Wg"][e]) * (h_ @ t["Wu"][e])) @ t["Wd"][e]
                Y = Y.index_add(0, torch.tensor([tok]), (gates[tok, r] * o)[None])
    (Y * torch.tensor(dY)).sum().backward()
    for n, key in keys.items():
        np.testing.assert_allclose(g[key], t[n].grad.numpy(), rtol=1e-9, atol=1e-11)
