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
