"""Token-choice (TC) routing, float64 oracle (test infrastructure only).

Only tests/ and bench.py's CPU baseline leg use this module; it shares no code with the
CUDA library. Passage followed (arXiv 2604.01622, Sec. 2.2, "Token-choice"): each token i
selects its top-k experts, E_i = TopK_j(S_ij, k), and y_i = sum_{j in E_i} g_ij FFN_j(x_i)
with normalised gates; a capacity factor CF caps each expert at ceil(CF k N / E) tokens and
the overflow is dropped; dropless TC has no cap.

Readings where the paper is silent (shared with the CUDA path):
  * ties in TopK go to the lower expert index; a token's choices are listed best first;
  * normalised gates: g_ij = S_ij / sum_{j' in E_i} S_ij' (over the k chosen experts);
  * an expert over capacity keeps its tokens in ascending token order (the first C tokens
    that chose it); a dropped pair contributes nothing, the other gates are unchanged;
  * the capacity pool is the whole batch of N tokens.
"""
from __future__ import annotations

import math

import numpy as np

from .ecmoe import router_scores, silu, silu_grad, swiglu_ffn


def tc_capacity(cf: float | None, k: int, N: int, E: int):
    """Sec. 2.2: ceil(CF k N / E); None (dropless) when cf is None or <= 0."""
    if cf is None or cf <= 0:
        return None
    return int(math.ceil(cf * k * N / E))


def tc_gates(S, choices):
    """Normalised gates g_tj = S_tj / sum_{j' in E_t} S_tj' of the given choices [N][k]."""
    sel = np.take_along_axis(np.asarray(S, np.float64), np.asarray(choices), axis=1)
    return sel / sel.sum(axis=1, keepdims=True)


def tc_select(S, k, capacity=None):
    """Returns (choices [N][k] expert ids best first, gates [N][k], kept [N][k] bool)."""
    S = np.asarray(S, np.float64)
    N, E = S.shape
    choices = np.zeros((N, k), dtype=np.int64)
    for t in range(N):
        order = np.lexsort((np.arange(E), -(S[t] + 0.0)))     # score desc, expert index asc
        choices[t] = order[:k]
    gates = tc_gates(S, choices)
    kept = np.ones((N, k), dtype=bool)
    if capacity is not None:
        load = np.zeros(E, dtype=np.int64)
        for t in range(N):                                       # token order decides who stays
            for r in range(k):
                e = choices[t, r]
                kept[t, r] = load[e] < capacity
                load[e] += 1
    return choices, gates, kept


def tc_forward(X, Wr, br, Wg, Wu, Wd, k, capacity=None, forced=None):
    """Layer forward under token choice. forced = (choices, kept) replaces the selection."""
    X = np.asarray(X, np.float64)
    N, d = X.shape
    S = router_scores(X, Wr, br)
    if forced is None:
        choices, gates, kept = tc_select(S, k, capacity)
    else:
        choices, kept = (np.asarray(a) for a in forced)
        gates = tc_gates(S, choices)
    Y = np.zeros((N, d))
    cache = {}
    for t in range(N):
        for r in range(k):
            if not kept[t, r]:
                continue
            e = int(choices[t, r])
            a, b, u, o = swiglu_ffn(X[t:t + 1], Wg[e], Wu[e], Wd[e])
            cache[(t, r)] = (a[0], b[0], u[0], o[0])
            Y[t] += gates[t, r] * o[0]
    return {"S": S, "choices": choices, "gates": gates, "kept": kept, "Y": Y, "X": X,
            "cache": cache}


def tc_backward(fwd, dY, Wr, Wg, Wu, Wd):
    """Gradients of <dY, Y>; the selection is held fixed, the gate normalisation is not:
    for j in E_t, dS_tj = (dg_tj - sum_{j' kept} dg_tj' g_tj') / Z_t with dg_tj = <dY_t, o_tj>
    (0 for a dropped pair) and Z_t = sum_{j in E_t} S_tj; then the softmax Jacobian."""
    dY = np.asarray(dY, np.float64)
    X, S, choices, gates, kept = fwd["X"], fwd["S"], fwd["choices"], fwd["gates"], fwd["kept"]
    N, d = X.shape
    E = S.shape[1]
    k = choices.shape[1]
    dX = np.zeros_like(X)
    dWg = np.zeros((E,) + np.asarray(Wg).shape[1:])
    dWu = np.zeros_like(dWg)
    dWd = np.zeros((E,) + np.asarray(Wd).shape[1:])
    dS = np.zeros((N, E))
    for t in range(N):
        dg = np.zeros(k)
        for r in range(k):
            if not kept[t, r]:
                continue
            e = int(choices[t, r])
            a, b, u, o = fwd["cache"][(t, r)]
            dg[r] = float(dY[t] @ o)
            dO = gates[t, r] * dY[t]
            dU = np.asarray(Wd[e], np.float64) @ dO
            dA = dU * b * silu_grad(a)
            dB = dU * silu(a)
            dX[t] += np.asarray(Wg[e], np.float64) @ dA + np.asarray(Wu[e], np.float64) @ dB
            dWd[e] += np.outer(u, dO)
            dWg[e] += np.outer(X[t], dA)
            dWu[e] += np.outer(X[t], dB)
        Z = float(np.sum(S[t, choices[t]]))
        common = float(np.sum(dg * gates[t]))
        for r in range(k):
            dS[t, int(choices[t, r])] = (dg[r] - common) / Z
    dZ = S * (dS - np.sum(dS * S, axis=1, keepdims=True))
    Wr64 = np.asarray(Wr, np.float64)
    dX += dZ @ Wr64.T
    return {"dX": dX, "dWr": X.T @ dZ, "dbr": dZ.sum(axis=0), "dWg": dWg, "dWu": dWu,
            "dWd": dWd, "dS": dS, "dZ": dZ}
