"""Float64 CPU oracle of the expert-choice (EC) MoE layer, forward and backward.

TEST INFRASTRUCTURE. Only tests/, __graft_entry__.smoke() and bench.py's CPU
baseline leg may import this module. The CUDA library never calls it and the
two share no code: this file is a plain, slow restatement of what arXiv
2604.01622 defines, written so a reader can check it against the paper by eye.

Paper passages followed (section / equation of arXiv 2604.01622):
  * Sec. 2.2, "Mixture-of-Experts Routing": a router gives a score matrix
    S in R^{N x E}; under expert choice each expert j takes its top-c tokens,
    T_j = TopC_i(S_ij, c), and y_i = sum_{j: i in T_j} g_ij FFN_j(x_i).
    Every expert processes exactly c tokens.
  * Sec. 4.2, "Scheduling Strategies": capacity varies per denoising step
    (a per-sequence capacity k_g is therefore an input array).
  * Sec. 5.2, "Inference-Time Properties" (single-sample decoding): each
    expert selects from the pool of one L-token sequence (one selection group
    per sequence).
  * Appendix "Experimental Setup": the expert FFNs use SwiGLU activations.
  * Appendix "Token Coverage in Expert-Choice Routing": a token no routed
    expert selects gets nothing from the routed path.

Readings where the paper is silent (each listed in the design notes):
  * router activation: softmax over the E experts of logits X.Wr (+ bias br);
  * EC gate g_ij = S_ij, not renormalised;
  * ties in TopC go to the lower token index; -0.0 equals +0.0;
  * the selected tokens of one (expert, group) are listed in ascending index;
  * SwiGLU: FFN(x) = (silu(x Wg) * (x Wu)) Wd with silu(a) = a / (1 + e^-a);
  * the selection is piecewise constant in S, so the backward pass treats it as
    fixed and sends the gate gradient through the softmax Jacobian.

Parity status: pinned by invariants, brute-force selection, finite
differences, the dense soft-MoE reduction and the textbook SwiGLU MLP
(tests/test_oracle_*.py).
"""
from __future__ import annotations

import numpy as np


# ----------------------------------------------------------------------------
# Router: Sec. 2.2 score matrix S in R^{N x E}; softmax over experts (reading).
# ----------------------------------------------------------------------------
def softmax_rows(Z: np.ndarray) -> np.ndarray:
    """Row softmax, the plain definition: exp(z - max z) / sum exp(z - max z)."""
    Z = np.asarray(Z, dtype=np.float64)
    ex = np.exp(Z - Z.max(axis=1, keepdims=True))
    return ex / ex.sum(axis=1, keepdims=True)


def router_scores(X: np.ndarray, Wr: np.ndarray, br: np.ndarray | None = None) -> np.ndarray:
    """S = softmax(X Wr + br) row by row; X [N][d], Wr [d][E] -> S [N][E]."""
    Z = np.asarray(X, np.float64) @ np.asarray(Wr, np.float64)
    if br is not None:
        Z = Z + np.asarray(br, np.float64)[None, :]
    return softmax_rows(Z)


# ----------------------------------------------------------------------------
# Expert-choice selection: Sec. 2.2 T_j = TopC_i(S_ij, c), per group (Sec. 5.2),
# with capacity k_g per group (Sec. 4.2).
# ----------------------------------------------------------------------------
def ec_select(S: np.ndarray, group_off, k_g):
    """For every expert e and group g, the k_g tokens of g with the largest S[t, e].

    Order of preference: larger score first, then lower token index. The chosen
    tokens of (e, g) are returned in ascending token index, groups in order, so
    row e of `idx` holds M = sum_g k_g token indices. gate[e, m] = S[idx[e, m], e].
    """
    S = np.asarray(S)
    N, E = S.shape
    group_off = [int(v) for v in group_off]
    k_g = [int(v) for v in k_g]
    M = sum(k_g)
    idx = np.zeros((E, M), dtype=np.int64)
    for e in range(E):
        pos = 0
        for g in range(len(k_g)):
            lo, hi = group_off[g], group_off[g + 1]
            toks = np.arange(lo, hi)
            score = S[lo:hi, e].astype(np.float64) + 0.0   # + 0.0 turns -0.0 into +0.0
            # np.lexsort sorts by the last key first: score descending, then index ascending
            order = np.lexsort((toks, -score))
            chosen = np.sort(toks[order[:k_g[g]]])
            idx[e, pos:pos + k_g[g]] = chosen
            pos += k_g[g]
    gate = np.take_along_axis(np.asarray(S, np.float64).T, idx, axis=1)
    return idx, gate


# ----------------------------------------------------------------------------
# SwiGLU expert FFN (appendix "Experimental Setup")
# ----------------------------------------------------------------------------
def sigmoid(a):
    a = np.asarray(a, np.float64)
    with np.errstate(over="ignore"):
        return 1.0 / (1.0 + np.exp(-a))


def silu(a):
    a = np.asarray(a, np.float64)
    return a * sigmoid(a)


def silu_grad(a):
    """d silu / da = sigma(a) (1 + a (1 - sigma(a)))."""
    s = sigmoid(a)
    return s * (1.0 + a * (1.0 - s))


def swiglu_ffn(h, Wg, Wu, Wd):
    """FFN(h) = (silu(h Wg) * (h Wu)) Wd for the rows of h; returns (a, b, u, o)."""
    h = np.asarray(h, np.float64)
    a = h @ np.asarray(Wg, np.float64)
    b = h @ np.asarray(Wu, np.float64)
    u = silu(a) * b
    o = u @ np.asarray(Wd, np.float64)
    return a, b, u, o


# ----------------------------------------------------------------------------
# Layer forward: Sec. 2.2 y_i = sum_{j: i in T_j} g_ij FFN_j(x_i)
# ----------------------------------------------------------------------------
def forward(X, Wr, br, Wg, Wu, Wd, group_off, k_g, forced_idx=None, shared=None):
    """Whole-layer forward.

    X [N][d]; Wr [d][E]; br [E] or None; Wg, Wu [E][d][d_ff]; Wd [E][d_ff][d].
    forced_idx [E][M] replaces the selection (used when the scores being ranked
    are another implementation's, after the selection itself was compared).
    shared: optional list of (Wg_s, Wu_s, Wd_s), one SwiGLU expert each that every
    token passes through (appendix "Token Coverage"); their outputs add to Y.
    Returns a dict holding S, idx, gate, Y and what the backward pass needs.
    """
    X = np.asarray(X, np.float64)
    N, d = X.shape
    E = np.asarray(Wr).shape[1]
    S = router_scores(X, Wr, br)
    if forced_idx is None:
        idx, gate = ec_select(S, group_off, k_g)
    else:
        idx = np.asarray(forced_idx, dtype=np.int64)
        gate = np.take_along_axis(S.T, idx, axis=1)
    Y = np.zeros((N, d))
    per_expert = []
    for e in range(E):
        h = X[idx[e]]                                  # gather the chosen tokens
        a, b, u, o = swiglu_ffn(h, Wg[e], Wu[e], Wd[e])
        per_expert.append((h, a, b, u, o))
        for m in range(idx.shape[1]):                  # scatter-add, experts in ascending order
            Y[idx[e, m]] += gate[e, m] * o[m]
    shared_cache = []
    for (Wg_s, Wu_s, Wd_s) in (shared or []):         # shared experts: every token, no gate
        a, b, u, o = swiglu_ffn(X, Wg_s, Wu_s, Wd_s)
        shared_cache.append((a, b, u))
        Y += o
    return {"S": S, "idx": idx, "gate": gate, "Y": Y, "per_expert": per_expert,
            "X": X, "group_off": np.asarray(group_off), "k_g": np.asarray(k_g),
            "shared": list(shared or []), "shared_cache": shared_cache}


def drop_ratio(idx, N):
    """Fraction of the N tokens that no expert selected (appendix "Token Coverage")."""
    picked = np.zeros(N, dtype=bool)
    picked[np.asarray(idx).ravel()] = True
    return 1.0 - picked.mean()


# ----------------------------------------------------------------------------
# Layer backward: chain rule through the forward above, selection held fixed.
# ----------------------------------------------------------------------------
def backward(fwd, dY, Wr, Wg, Wu, Wd):
    """Gradients of <dY, Y> with respect to X, Wr, br, Wg, Wu, Wd.

    Per selected pair (e, m) with token t = idx[e, m]:
      dO = gate * dY_t;  dgate = <dY_t, O>;
      dU = dO Wd^T;  dA = dU * B * silu'(A);  dB = dU * silu(A);
      dH = dA Wg^T + dB Wu^T;  dX_t += dH;
      dWd += U^T dO;  dWg += H^T dA;  dWu += H^T dB.
    Through the router: dS[t, e] = dgate of the pair (zero if (t, e) was not
    selected); the softmax Jacobian gives dZ = S * (dS - <dS, S>_row);
    dX += dZ Wr^T; dWr = X^T dZ; dbr = sum_t dZ.
    """
    dY = np.asarray(dY, np.float64)
    X, S, idx, gate = fwd["X"], fwd["S"], fwd["idx"], fwd["gate"]
    N, d = X.shape
    E, M = idx.shape
    dX = np.zeros_like(X)
    dS = np.zeros((N, E))
    dWg = np.zeros((E,) + np.asarray(Wg).shape[1:])
    dWu = np.zeros_like(dWg)
    dWd = np.zeros((E,) + np.asarray(Wd).shape[1:])
    dgate = np.zeros((E, M))
    for e in range(E):
        h, a, b, u, o = fwd["per_expert"][e]
        dYt = dY[idx[e]]
        dgate[e] = np.sum(dYt * o, axis=1)
        dO = gate[e][:, None] * dYt
        dU = dO @ np.asarray(Wd[e], np.float64).T
        dA = dU * b * silu_grad(a)
        dB = dU * silu(a)
        dH = dA @ np.asarray(Wg[e], np.float64).T + dB @ np.asarray(Wu[e], np.float64).T
        dWd[e] = u.T @ dO
        dWg[e] = h.T @ dA
        dWu[e] = h.T @ dB
        for m in range(M):
            dX[idx[e, m]] += dH[m]
            dS[idx[e, m], e] = dgate[e, m]
    dZ = S * (dS - np.sum(dS * S, axis=1, keepdims=True))
    Wr64 = np.asarray(Wr, np.float64)
    dX += dZ @ Wr64.T
    dWr = X.T @ dZ
    dbr = dZ.sum(axis=0)
    dshared = []
    for (Wg_s, Wu_s, Wd_s), (a, b, u) in zip(fwd.get("shared", []), fwd.get("shared_cache", [])):
        dU = dY @ np.asarray(Wd_s, np.float64).T       # the shared output enters Y ungated
        dA = dU * b * silu_grad(a)
        dB = dU * silu(a)
        dX += dA @ np.asarray(Wg_s, np.float64).T + dB @ np.asarray(Wu_s, np.float64).T
        dshared.append((X.T @ dA, X.T @ dB, u.T @ dY))
    return {"dX": dX, "dWr": dWr, "dbr": dbr, "dWg": dWg, "dWu": dWu, "dWd": dWd,
            "dgate": dgate, "dS": dS, "dZ": dZ, "dshared": dshared}


# ----------------------------------------------------------------------------
# Sampled forms for large workloads: the same definitions restricted to a few
# tokens or experts, given a selection that was already compared in full.
# ----------------------------------------------------------------------------
def token_pairs(idx, tokens):
    """For each token, the (e, m) pairs that selected it, experts ascending."""
    idx = np.asarray(idx)
    want = {int(t): [] for t in tokens}
    E, M = idx.shape
    for e in range(E):
        row = idx[e]
        for t in want:
            hit = np.nonzero(row == t)[0]
            for m in hit:
                want[t].append((e, int(m)))
    return want


def forward_tokens(X_rows, S_rows, pairs, Wg, Wu, Wd):
    """Y_t for sampled tokens: sum over the experts that chose t of S[t,e] FFN_e(x_t).

    X_rows, S_rows: dict token -> row of X (float64) and row of S (float64).
    pairs: token -> list of (e, m). Wg/Wu/Wd: callables e -> float64 matrix.
    """
    out = {}
    for t, plist in pairs.items():
        y = np.zeros_like(X_rows[t])
        for e, _m in plist:
            _, _, _, o = swiglu_ffn(X_rows[t][None, :], Wg(e), Wu(e), Wd(e))
            y += S_rows[t][e] * o[0]
        out[t] = y
    return out


def backward_tokens(X_rows, S_rows, dY_rows, pairs, Wr, Wg, Wu, Wd):
    """dX_t for sampled tokens (the definition in `backward`, for one row each).

    dS_t only involves the pairs of token t, so dX_t needs no other token.
    """
    Wr64 = np.asarray(Wr, np.float64)
    out = {}
    for t, plist in pairs.items():
        x = X_rows[t][None, :]
        s = S_rows[t]
        dy = dY_rows[t][None, :]
        dx = np.zeros(x.shape[1])
        ds = np.zeros(s.shape[0])
        for e, _m in plist:
            a, b, u, o = swiglu_ffn(x, Wg(e), Wu(e), Wd(e))
            ds[e] = float(np.sum(dy * o))
            dO = s[e] * dy
            dU = dO @ Wd(e).T
            dA = dU * b * silu_grad(a)
            dB = dU * silu(a)
            dx += (dA @ Wg(e).T + dB @ Wu(e).T)[0]
        dz = s * (ds - np.sum(ds * s))
        dx += dz @ Wr64.T
        out[t] = dx
    return out


def backward_expert(H, S_col, dY_rows, Wg_e, Wu_e, Wd_e):
    """Weight gradients of one expert from all its M selected rows.

    H [M][d]: the expert's gathered inputs; S_col [M]: its gates; dY_rows [M][d].
    Returns (dWg_e, dWu_e, dWd_e, dgate_e).
    """
    a, b, u, o = swiglu_ffn(H, Wg_e, Wu_e, Wd_e)
    dgate = np.sum(dY_rows * o, axis=1)
    dO = np.asarray(S_col, np.float64)[:, None] * dY_rows
    dU = dO @ np.asarray(Wd_e, np.float64).T
    dA = dU * b * silu_grad(a)
    dB = dU * silu(a)
    return H.T @ dA, H.T @ dB, u.T @ dO, dgate


def router_backward_streamed(X, Wr, br, dY, idx, Wg, Wu, Wd):
    """The router part of `backward` (dS, dZ, dWr, dbr) for a layer too large to hold the
    per-expert activations: the same definitions, computed one expert at a time.

    X, dY [N][d] float64; idx [E][M] the selection; Wg/Wu/Wd: callables e -> float64
    matrix of expert e. For every selected pair (e, m), t = idx[e, m]:
    dS[t, e] = <dY_t, FFN_e(x_t)>; then dZ = S * (dS - <dS, S>_row), dWr = X^T dZ,
    dbr = sum_t dZ, with S the router scores of X.
    """
    X = np.asarray(X, np.float64)
    dY = np.asarray(dY, np.float64)
    idx = np.asarray(idx)
    S = router_scores(X, Wr, br)
    N, E = S.shape
    dS = np.zeros((N, E))
    for e in range(E):
        rows = idx[e]
        _, _, _, o = swiglu_ffn(X[rows], Wg(e), Wu(e), Wd(e))
        dS[rows, e] = np.sum(dY[rows] * o, axis=1)
    dZ = S * (dS - np.sum(dS * S, axis=1, keepdims=True))
    return {"S": S, "dS": dS, "dZ": dZ, "dWr": X.T @ dZ, "dbr": dZ.sum(axis=0)}


# ----------------------------------------------------------------------------
# Stacked layers with residual adds, x_{l+1} = x_l + EC_l(x_l): how the four-layer
# wide workload composes the layer (the transformer residual stream around each MoE
# layer). A composition of `forward`/`backward` above, nothing more.
# ----------------------------------------------------------------------------
def stack_forward(X, layers, group_off, k_g, forced_idx=None):
    """layers: list of (Wr, br, Wg, Wu, Wd). Returns (xs, fwds) with xs[l+1] = xs[l] + Y_l."""
    xs = [np.asarray(X, np.float64)]
    fwds = []
    for l, (Wr, br, Wg, Wu, Wd) in enumerate(layers):
        f = forward(xs[-1], Wr, br, Wg, Wu, Wd, group_off, k_g,
                    None if forced_idx is None else forced_idx[l])
        fwds.append(f)
        xs.append(xs[-1] + f["Y"])
    return xs, fwds


def stack_backward(fwds, layers, dOut):
    """Gradients of <dOut, x_L>: returns (dX_0, per-layer gradient dicts)."""
    d = np.asarray(dOut, np.float64)
    grads = [None] * len(layers)
    for l in range(len(layers) - 1, -1, -1):
        Wr, br, Wg, Wu, Wd = layers[l]
        g = backward(fwds[l], d, Wr, Wg, Wu, Wd)
        grads[l] = g
        d = d + g["dX"]
    return d, grads


def stack_tokens(X_rows, dOut_rows, layers, pairs):
    """Stack output and input gradient of sampled tokens, one token at a time.

    With each layer's selection fixed, layer l's output for token t depends on x_{l,t} alone
    (its gate is S[t, e] of that row), so x_{l+1,t} = x_{l,t} + Y_l(x_{l,t}) and
    d_{l,t} = d_{l+1,t} + (input gradient of layer l at token t, given d_{l+1,t}) follow
    `forward_tokens` / `backward_tokens` row by row.
    X_rows, dOut_rows: token -> float64 row; layers: list of (Wr, br, Wg, Wu, Wd) with
    Wg/Wu/Wd callables e -> float64 matrix; pairs: per layer, token -> [(e, m), ...].
    Returns (xs, d0): xs[l][t] the input of layer l (xs[-1] the stack output), d0[t].
    """
    xs = [dict(X_rows)]
    for l, (Wr, br, Wg, Wu, Wd) in enumerate(layers):
        x = xs[-1]
        toks = list(x)
        S = router_scores(np.stack([x[t] for t in toks]), Wr, br)
        srows = {t: S[i] for i, t in enumerate(toks)}
        y = forward_tokens(x, srows, pairs[l], Wg, Wu, Wd)
        xs.append({t: x[t] + y[t] for t in toks})
    d = dict(dOut_rows)
    for l in range(len(layers) - 1, -1, -1):
        Wr, br, Wg, Wu, Wd = layers[l]
        x = xs[l]
        toks = list(x)
        S = router_scores(np.stack([x[t] for t in toks]), Wr, br)
        srows = {t: S[i] for i, t in enumerate(toks)}
        dx = backward_tokens(x, srows, d, pairs[l], Wr, Wg, Wu, Wd)
        d = {t: d[t] + dx[t] for t in toks}
    return xs, d
