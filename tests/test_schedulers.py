"""Capacity schedulers (Sec. 4.2, Table 1): the oracle against the paper's Table 7 and closed
forms, and the library's host function against the oracle (CPU only)."""
import math
import os

import numpy as np
import pytest

import paper_2604_01622_gb300 as ec
from oracle import schedulers as SO

GOLDEN = os.path.join(os.path.dirname(__file__), "golden", "scheduler_expectations_table7.txt")


def _table7():
    rows = {}
    for line in open(GOLDEN):
        line = line.strip()
        if line and not line.startswith("#"):
            name, es, ek = line.split()
            rows[name] = (float(es), float(ek))
    return rows


def test_expectations_match_table7():
    """E[s(r)] as printed (4 decimals), and E[k(r)] = 8 + 24 E[s(r)] derived the way the
    appendix prints it, from the 4-decimal E[s] ("8 + 24 x 0.5010 = 20.02"): the exact
    Gaussian value 20.025 sits on the 2-decimal rounding boundary."""
    for name, (es, ek) in _table7().items():
        got = SO.expected_s(name)
        assert round(got, 4) == pytest.approx(es, abs=1e-12), (name, got)
        assert round(8 + 24 * round(got, 4), 2) == pytest.approx(ek, abs=1e-12), (name, got)
        assert abs(8 + 24 * got - ek) <= 0.0051


def test_closed_forms_and_endpoints():
    # E[s] = 1/2 exactly for the linear and cosine families (the appendix's integrals)
    for name in ("linear", "linear_reverse", "cosine", "cosine_reverse"):
        assert SO.expected_s(name) == pytest.approx(0.5, abs=1e-12)
    # normalized Gaussian: 0 at both ends, 1 at the middle, symmetric
    assert SO.gaussian_normalized(0.0) == pytest.approx(0.0, abs=1e-15)
    assert SO.gaussian_normalized(1.0) == pytest.approx(0.0, abs=1e-15)
    assert SO.gaussian_normalized(0.5) == pytest.approx(1.0, abs=1e-15)
    for r in np.linspace(0, 1, 17):
        assert SO.gaussian_normalized(r) == pytest.approx(SO.gaussian_normalized(1 - r), abs=1e-14)
    # the reverse schedulers mirror the forward ones; every s stays in [0, 1]
    for r in np.linspace(0, 1, 33):
        assert SO.s_of_r("linear", r) + SO.s_of_r("linear_reverse", r) == pytest.approx(1.0)
        assert SO.s_of_r("cosine", r) == pytest.approx(SO.s_of_r("cosine_reverse", 1 - r))
        for name in SO.SCHEDULERS:
            assert -1e-15 <= SO.s_of_r(name, r) <= 1 + 1e-15
    # linear-reverse puts k_max at r = 0 (fully unmasked) and k_min at r = 1
    assert SO.k_of_r("linear_reverse", 0.0, 8, 32) == 32
    assert SO.k_of_r("linear_reverse", 1.0, 8, 32) == 8


@pytest.mark.parametrize("name", SO.SCHEDULERS)
def test_library_capacities_match_oracle(name):
    rng = np.random.default_rng(hash(name) % 1000)
    G = 64
    group_off = np.concatenate([[0], np.cumsum(rng.integers(1, 5000, G))]).astype(np.int32)
    r = rng.random(G)
    r[:3] = [0.0, 1.0, 0.5]
    for (kmin, kmax, E) in [(8, 32, 512), (2, 14, 64), (0, 16, 64)]:
        got = ec.ec_capacity_schedule(name, kmin, kmax, E, group_off, r)
        ref = SO.group_capacity(name, r, kmin, kmax, E, group_off)
        assert np.array_equal(got, ref), (name, kmin, kmax, E)
        assert np.all(got >= 0) and np.all(got <= np.diff(group_off))


def test_library_rejects_bad_arguments():
    off = np.array([0, 10], np.int32)
    with pytest.raises(ec.ECError):
        ec.ec_capacity_schedule(9, 8, 32, 64, off, [0.5])
    with pytest.raises(ec.ECError):
        ec.ec_capacity_schedule("linear", 8, 32, 64, off, [1.5])
    with pytest.raises(ec.ECError):
        ec.ec_capacity_schedule("linear", 32, 8, 64, off, [0.5])
    with pytest.raises(ec.ECError):
        ec.ec_capacity_schedule("gaussian", 8, 32, 64, off, [0.5], sigma=0.0)


def test_group_capacity_exact_where_no_rounding_is_in_play():
    """Sec. 2.2: capacity c = k N / E per selection pool. With L_g / E = 64 and k(r) an integer
    (the schedule's ends and middle), c_g is that product exactly: values written out by hand."""
    E, L = 64, 4096
    off = np.arange(4 + 1, dtype=np.int32) * L
    k_min, k_max = 8, 32
    cases = {
        "static": ([0.0, 0.3, 0.5, 1.0], [1280, 1280, 1280, 1280]),          # k = 20
        "linear": ([0.0, 0.5, 1.0, 0.25], [512, 1280, 2048, 896]),          # k = 8, 20, 32, 14
        "linear_reverse": ([0.0, 0.5, 1.0, 0.75], [2048, 1280, 512, 896]),
        "cosine": ([0.0, 0.5, 1.0, 0.5], [512, 1280, 2048, 1280]),
        "cosine_reverse": ([0.0, 0.5, 1.0, 1.0], [2048, 1280, 512, 512]),
        "gaussian": ([0.0, 0.5, 1.0, 0.5], [512, 2048, 512, 2048]),         # g~ = 0, 1, 0
        "gaussian_reverse": ([0.0, 0.5, 1.0, 0.0], [2048, 512, 2048, 2048]),
    }
    for name, (r, want) in cases.items():
        got = SO.group_capacity(name, np.array(r), k_min, k_max, E, off)
        assert got.tolist() == want, name
        assert ec.ec_capacity_schedule(name, k_min, k_max, E, off, r).tolist() == want, name


def test_group_capacity_rounding_and_clipping():
    """The reading where the paper is silent: k L_g / E rounded half up, then clipped to
    [0, L_g]. Hand-computed: 9*32/64 = 4.5 -> 5, 7*32/64 = 3.5 -> 4, 9*16/64 = 2.25 -> 2,
    11*16/64 = 2.75 -> 3, 3*16/64 = 0.75 -> 1, 1*16/64 = 0.25 -> 0; with k = 8 and E = 4
    the product 2 L_g is clipped to L_g."""
    E = 64
    for k, L, want in ((9, 32, 5), (7, 32, 4), (9, 16, 2), (11, 16, 3), (3, 16, 1), (1, 16, 0)):
        off = np.array([0, L], np.int32)
        # a static schedule with k_min = k_max = k gives k(r) = k for every r
        assert SO.group_capacity("static", [0.4], k, k, E, off).tolist() == [want], (k, L)
        assert ec.ec_capacity_schedule("static", k, k, E, off, [0.4]).tolist() == [want], (k, L)
    off = np.array([0, 10, 30, 30], np.int32)                  # includes an empty group
    assert SO.group_capacity("static", [0.5] * 3, 8, 8, 4, off).tolist() == [10, 20, 0]
    assert ec.ec_capacity_schedule("static", 8, 8, 4, off, [0.5] * 3).tolist() == [10, 20, 0]


@pytest.mark.parametrize("name", ["linear", "linear_reverse", "cosine", "cosine_reverse",
                                  "gaussian", "gaussian_reverse"])
def test_group_capacity_matches_static_flops_on_a_symmetric_grid(name):
    """Table 7 / appendix "Scheduler Definitions and FLOPs Equivalence": over masking ratios
    spread evenly on [0, 1] a schedule spends the static schedule's FLOPs, E[k(r)] = 20 for
    k in [8, 32] (19.98 and 20.02 for the Gaussian pair, as printed). Each c_g is rounded
    once, so the total differs from G E[k] L / E by at most G / 2 (plus the quadrature gap
    of the grid)."""
    E, L, G = 64, 1024, 400
    off = np.arange(G + 1, dtype=np.int32) * L
    r = (np.arange(G) + 0.5) / G
    ek = {n: float(v[1]) for n, v in _table7().items()}[name]
    c = SO.group_capacity(name, r, 8, 32, E, off)
    assert abs(int(c.sum()) - G * ek * L / E) <= G / 2 + 0.01 * G * L / E
    if name in ("linear", "linear_reverse", "cosine", "cosine_reverse"):
        # symmetric grid: s(r) + s(1 - r) = 1 pairs the ratios exactly, so sum k(r_g) = 20 G
        assert abs(int(c.sum()) - 20 * G * L // E) <= G / 2
    assert np.array_equal(c, ec.ec_capacity_schedule(name, 8, 32, E, off, r))
