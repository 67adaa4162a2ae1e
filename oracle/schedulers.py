"""Timestep-dependent capacity schedulers (float64 oracle; test infrastructure only).

Only tests/ use this module. Passages followed (arXiv 2604.01622):
  * Sec. 4.2 "Scheduling Strategies": k(r) = clamp(k_min + (k_max - k_min) s(r), k_min, k_max)
    for masking ratio r in [0, 1];
  * Table 1: s(r) = r (linear), 1 - r (linear-reverse), (1 - cos(pi r))/2 (cosine),
    (1 + cos(pi r))/2 (cosine-reverse), g~(r) (Gaussian), 1 - g~(r) (Gaussian-reverse);
    the static baseline uses the constant k = (k_min + k_max)/2, i.e. s(r) = 1/2;
  * appendix "Scheduler Definitions and FLOPs Equivalence": g~(r) = (g(r) - g(0)) / (1 - g(0)),
    g(r) = exp(-(r - 1/2)^2 / (2 sigma^2)), sigma = 0.22;
  * Sec. 2.2: capacity c = k N / E gives E c = k N token-expert pairs; applied per selection
    group (one sequence of L_g tokens, Sec. 5.2) this is c_g = k(r_g) L_g / E.
Reading where the paper is silent: c_g is rounded half up, floor(k L_g / E + 1/2), and
clipped to [0, L_g].
"""
from __future__ import annotations

import math

import numpy as np

SCHEDULERS = ("static", "linear", "linear_reverse", "cosine", "cosine_reverse", "gaussian",
              "gaussian_reverse")


def gaussian_normalized(r, sigma=0.22):
    g = lambda x: math.exp(-((x - 0.5) ** 2) / (2.0 * sigma * sigma))
    g0 = g(0.0)
    return (g(r) - g0) / (1.0 - g0)


def s_of_r(name: str, r: float, sigma: float = 0.22) -> float:
    if name == "static":
        return 0.5
    if name == "linear":
        return r
    if name == "linear_reverse":
        return 1.0 - r
    if name == "cosine":
        return 0.5 * (1.0 - math.cos(math.pi * r))
    if name == "cosine_reverse":
        return 0.5 * (1.0 + math.cos(math.pi * r))
    if name == "gaussian":
        return gaussian_normalized(r, sigma)
    if name == "gaussian_reverse":
        return 1.0 - gaussian_normalized(r, sigma)
    raise ValueError(name)


def k_of_r(name, r, k_min, k_max, sigma=0.22):
    """Sec. 4.2: clamp(k_min + (k_max - k_min) s(r), k_min, k_max)."""
    k = k_min + (k_max - k_min) * s_of_r(name, r, sigma)
    return min(max(k, k_min), k_max)


def expected_s(name, sigma=0.22):
    """E[s(r)] for r ~ U(0, 1), by adaptive quadrature."""
    from scipy.integrate import quad
    return quad(lambda r: s_of_r(name, r, sigma), 0.0, 1.0, epsabs=1e-13, epsrel=1e-13)[0]


def group_capacity(name, r, k_min, k_max, E, group_off, sigma=0.22):
    """Per-group capacities c_g = floor(k(r_g) L_g / E + 1/2), clipped to [0, L_g]."""
    out = []
    for g in range(len(r)):
        L = int(group_off[g + 1]) - int(group_off[g])
        c = math.floor(k_of_r(name, float(r[g]), k_min, k_max, sigma) * L / E + 0.5)
        out.append(min(max(c, 0), L))
    return np.array(out, dtype=np.int32)
