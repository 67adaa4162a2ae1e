"""Planted mistakes in the oracle (on the CPU) must be caught by its pins.

Each case patches one step of the oracle with a plausible slip (a dropped
term, a wrong sign, a swapped operand, a reversed tie rule) and runs the pin
that should catch it; the pin must fail.
"""
import math

import numpy as np
import pytest

from oracle import ecmoe as O
from tests import test_oracle_pins as P


def _fails(pin, *args):
    try:
        pin(*args)
    except AssertionError:
        return True
    return False


def test_reversed_tie_rule_is_caught(monkeypatch):
    real = O.ec_select

    def wrong(S, group_off, k_g):  # ties to the HIGHER token index
        S = np.asarray(S)
        N = S.shape[0]
        idx, gate = real(S[::-1], [N - v for v in group_off[::-1]], list(k_g)[::-1])
        idx = np.sort(N - 1 - idx, axis=1)
        return idx, np.take_along_axis(S.T, idx, axis=1)

    monkeypatch.setattr(O, "ec_select", wrong)
    assert _fails(P.test_selection_matches_brute_force, 1.0)


def test_dropped_gate_in_combine_is_caught(monkeypatch):
    real = O.router_scores
    monkeypatch.setattr(O, "router_scores", lambda X, Wr, br=None: np.ones_like(real(X, Wr, br)))
    assert _fails(P.test_full_capacity_reduces_to_dense_soft_moe)


def test_wrong_silu_is_caught(monkeypatch):
    monkeypatch.setattr(O, "silu", lambda a: np.asarray(a, np.float64) * O.sigmoid(2 * np.asarray(a)))
    assert _fails(P.test_single_expert_full_capacity_is_textbook_swiglu_mlp)


def test_wrong_softmax_backward_sign_is_caught(monkeypatch):
    real = O.backward

    def wrong(fwd, dY, Wr, Wg, Wu, Wd):
        out = real(fwd, dY, Wr, Wg, Wu, Wd)
        S = fwd["S"]
        dZ = S * (out["dS"] + np.sum(out["dS"] * S, axis=1, keepdims=True))  # sign slip
        out["dX"] = out["dX"] - out["dZ"] @ Wr.T + dZ @ Wr.T
        out["dWr"] = fwd["X"].T @ dZ
        out["dbr"] = dZ.sum(axis=0)
        out["dZ"] = dZ
        return out

    monkeypatch.setattr(O, "backward", wrong)
    assert _fails(P.test_backward_matches_central_finite_differences)


def test_missing_silu_derivative_term_is_caught(monkeypatch):
    monkeypatch.setattr(O, "silu_grad", lambda a: O.sigmoid(a))  # drops the a(1-s) term
    assert _fails(P.test_backward_matches_central_finite_differences)


def test_transposed_down_projection_gradient_is_caught(monkeypatch):
    real = O.backward

    def wrong(fwd, dY, Wr, Wg, Wu, Wd):
        out = real(fwd, dY, Wr, Wg, Wu, Wd)
        E = out["dWd"].shape[0]
        # accumulate dWd with operands swapped (dO^T U, transposed back to shape)
        for e in range(E):
            _h, _a, _b, u, _o = fwd["per_expert"][e]
            dO = fwd["gate"][e][:, None] * np.asarray(dY)[fwd["idx"][e]]
            out["dWd"][e] = (dO.T @ u).T[::-1]
        return out

    monkeypatch.setattr(O, "backward", wrong)
    assert _fails(P.test_backward_matches_central_finite_differences)


def _wrong_capacity(rule):
    import math
    from oracle import schedulers as SO

    def group_capacity(name, r, k_min, k_max, E, group_off, sigma=0.22):
        out = []
        for g in range(len(r)):
            L = int(group_off[g + 1]) - int(group_off[g])
            k = SO.k_of_r(name, float(r[g]), k_min, k_max, sigma)
            out.append(min(max(rule(k, L, E, int(group_off[-1])), 0), L))
        return np.array(out, dtype=np.int32)
    return group_capacity


@pytest.mark.parametrize("rule", [
    lambda k, L, E, N: math.floor(k * L + 0.5),          # the / E dropped
    lambda k, L, E, N: math.floor(k * L / E),            # rounded down, not half up
    lambda k, L, E, N: math.floor(k * N / E + 0.5),      # the whole batch as the pool
])
def test_wrong_group_capacity_is_caught(monkeypatch, rule):
    from oracle import schedulers as SO
    from tests import test_schedulers as TS
    monkeypatch.setattr(SO, "group_capacity", _wrong_capacity(rule))
    assert (_fails(TS.test_group_capacity_exact_where_no_rounding_is_in_play)
            or _fails(TS.test_group_capacity_rounding_and_clipping))
