"""Seeded synthetic workloads for the expert-choice (EC) MoE layer.

This module holds none of the layer's arithmetic. It only draws random numbers,
rounds them to bf16, and applies the per-sequence capacity recipe of the
timestep-capacity workloads (a property of the input, not of the layer: the
layer takes k_g as an input array). Both the CUDA path (tests, bench) and the
float64 oracle's tests consume the arrays made here.

Workloads stand in for one MoE layer of the paper's EC-vs-TC model (d=2048,
64 fine-grained experts; appendix "Experimental Setup"); the paper's training data
is not used.

Random numbers come from numpy's counter-based Philox bit generator with a
fixed 128-bit key per (workload seed, layer, tensor), so every machine
(x86 or Arm) draws the same values.
"""
from __future__ import annotations

import math
from dataclasses import dataclass, field

import numpy as np

# tensor ids folded into the Philox key
_T_X, _T_WR, _T_BR, _T_WG, _T_WU, _T_WD, _T_DY, _T_MASK, _T_T, _T_PERM = range(10)


@dataclass(frozen=True)
class Workload:
    """Shape and recipe of one synthetic EC-MoE workload.

    G sequences of L tokens each form the selection groups (one group per
    sequence). k_base is the uniform per-expert, per-sequence capacity; with
    timestep_capacity the per-sequence k_g are redistributed by mask ratio
    while their sum stays G*k_base.
    """
    name: str
    G: int
    L: int
    d: int
    E: int
    d_ff: int
    k_base: int
    dtype: str                  # "f32" or "bf16"
    seed: int
    timestep_capacity: bool = False
    router_bias: bool = False
    layers: int = 1
    init: str = "fan_in"        # "fan_in": N(0,1/d) / N(0,1/d_ff); "std002": N(0, 0.02^2)
    x_recipe: str = "normal"    # "normal": N(0,1); "rms_unit": rmsnorm(z)/sqrt(d)

    @property
    def N(self) -> int:
        return self.G * self.L

    @property
    def M(self) -> int:
        return self.G * self.k_base


WORKLOADS = {
    # 2 x 128 tokens, fp32, the small case the oracle finishes in seconds
    "tiny_f32": Workload("tiny_f32", G=2, L=128, d=64, E=8, d_ff=128, k_base=16,
                         dtype="f32", seed=1),
    # 8 x 4096 tokens, d=2048, 64 experts of d_ff=1024, k_g=512 (top-8 equivalent)
    "ec_d2048_e64": Workload("ec_d2048_e64", G=8, L=4096, d=2048, E=64, d_ff=1024,
                             k_base=512, dtype="bf16", seed=2, init="std002",
                             x_recipe="rms_unit"),
    # same shape, per-sequence mask ratio and timestep-dependent capacity
    "ec_timestep_d2048_e64": Workload("ec_timestep_d2048_e64", G=8, L=4096, d=2048, E=64,
                                      d_ff=1024, k_base=512, dtype="bf16", seed=3,
                                      timestep_capacity=True, init="std002",
                                      x_recipe="rms_unit"),
    # 16 x 2048 tokens, d=1024, 128 experts of d_ff=512, k_g=128, skewed router bias
    "ec_many_small_e128": Workload("ec_many_small_e128", G=16, L=2048, d=1024, E=128,
                                   d_ff=512, k_base=128, dtype="bf16", seed=4,
                                   router_bias=True, init="std002", x_recipe="rms_unit"),
    # 4 x 8192 tokens, d=4096, 32 experts of d_ff=2048, k_g=512 base, timestep capacity,
    # four layers stacked with residual adds
    "ec_wide_d4096_e32_x4": Workload("ec_wide_d4096_e32_x4", G=4, L=8192, d=4096, E=32,
                                     d_ff=2048, k_base=512, dtype="bf16", seed=5,
                                     timestep_capacity=True, layers=4, init="std002",
                                     x_recipe="rms_unit"),
}


def scaled(w: Workload, **kw) -> Workload:
    """Copy of a workload with some fields replaced (smaller parity cases)."""
    fields = {f: getattr(w, f) for f in w.__dataclass_fields__}
    fields.update(kw)
    return Workload(**fields)


def _rng(seed: int, layer: int, tensor: int) -> np.random.Generator:
    key = (int(seed) << 64) | (int(layer) << 32) | int(tensor)
    return np.random.Generator(np.random.Philox(key=key))


def bf16_bits(x: np.ndarray) -> np.ndarray:
    """Round float32 values to bf16 (round to nearest, ties to even); returns uint16 bits."""
    u = np.ascontiguousarray(x, dtype=np.float32).view(np.uint32)
    rounding = np.uint32(0x7FFF) + ((u >> np.uint32(16)) & np.uint32(1))
    return ((u + rounding) >> np.uint32(16)).astype(np.uint16)


def bf16_to_f64(bits: np.ndarray) -> np.ndarray:
    """Exact value of bf16 bits as float64."""
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32).astype(np.float64)


def bf16_to_f32(bits: np.ndarray) -> np.ndarray:
    return (bits.astype(np.uint32) << np.uint32(16)).view(np.float32)


@dataclass
class Tensor:
    """One input tensor in the workload's storage type.

    `data` is float32 for fp32 workloads and uint16 bf16 bits for bf16 ones.
    """
    data: np.ndarray
    dtype: str

    @property
    def shape(self):
        return self.data.shape

    def f64(self, index=None) -> np.ndarray:
        a = self.data if index is None else self.data[index]
        if self.dtype == "bf16":
            return bf16_to_f64(a)
        return np.asarray(a, dtype=np.float64)

    def f32(self) -> np.ndarray:
        if self.dtype == "bf16":
            return bf16_to_f32(self.data)
        return self.data


def _store(x32: np.ndarray, dtype: str) -> Tensor:
    if dtype == "bf16":
        return Tensor(bf16_bits(x32), "bf16")
    return Tensor(np.ascontiguousarray(x32, dtype=np.float32), "f32")


def _normal(rng, shape, std) -> np.ndarray:
    x = rng.standard_normal(size=shape, dtype=np.float32)
    if std != 1.0:
        x *= np.float32(std)
    return x


def _rms_unit_rows(z: np.ndarray) -> np.ndarray:
    """rmsnorm(z)/sqrt(d) row by row: every row ends with Euclidean norm 1."""
    z64 = z.astype(np.float64)
    rms = np.sqrt(np.mean(z64 * z64, axis=-1, keepdims=True))
    return (z64 / rms / math.sqrt(z.shape[-1])).astype(np.float32)


def mask_ratios(w: Workload) -> np.ndarray:
    """Per-sequence mask ratio t_g ~ U(0,1) (timestep workloads only)."""
    return _rng(w.seed, 0, _T_T).random(w.G)


def timestep_capacity(t: np.ndarray, k_base: int, L: int) -> np.ndarray:
    """Per-sequence capacity of the timestep workloads (input recipe).

    Weight w(t) = 2(1 - t) per sequence, renormalised so the integer k_g sum to
    exactly G*k_base: k_g = floor(T*w_g/sum(w)), and the T - sum(floor) leftover
    units go one each to the largest fractional parts (ties to the lower g).
    Clipped to [0, L]. If every weight is zero the split is uniform.
    """
    G = len(t)
    T = G * k_base
    w = 2.0 * (1.0 - np.asarray(t, dtype=np.float64))
    if w.sum() <= 0.0:
        w = np.ones(G)
    raw = T * w / w.sum()
    k = np.floor(raw).astype(np.int64)
    left = int(T - k.sum())
    frac = raw - k
    order = sorted(range(G), key=lambda g: (-frac[g], g))
    for g in order[:left]:
        k[g] += 1
    return np.clip(k, 0, L).astype(np.int32)


@dataclass
class LayerInputs:
    """Inputs of one EC-MoE layer (weights in storage type)."""
    Wr: Tensor            # [d][E]
    br: np.ndarray | None  # [E] float32 or None
    Wg: Tensor            # [E][d][d_ff]
    Wu: Tensor            # [E][d][d_ff]
    Wd: Tensor            # [E][d_ff][d]


@dataclass
class Inputs:
    w: Workload
    X: Tensor             # [N][d]
    dY: Tensor            # [N][d]
    group_off: np.ndarray  # [G+1] int32
    k_g: np.ndarray        # [G] int32
    layers: list = field(default_factory=list)
    t: np.ndarray | None = None
    masked: np.ndarray | None = None  # [N] bool, positions holding the mask vector


def make_layer(w: Workload, layer: int, experts: slice | None = None) -> LayerInputs:
    """Weights of one layer. `experts` restricts Wg/Wu/Wd to a slice of experts
    (the draws are made per expert so a slice equals the full tensor's slice)."""
    d, E, d_ff = w.d, w.E, w.d_ff
    if w.init == "fan_in":
        s_in, s_ff, s_r = 1.0 / math.sqrt(d), 1.0 / math.sqrt(d_ff), 1.0 / math.sqrt(d)
    else:
        s_in = s_ff = s_r = 0.02
    Wr = _store(_normal(_rng(w.seed, layer, _T_WR), (d, E), s_r), w.dtype)
    br = None
    if w.router_bias:
        br = _normal(_rng(w.seed, layer, _T_BR), (E,), 1.0)
    ex = range(E) if experts is None else range(E)[experts]

    def per_expert(tid, shape, std):
        out = []
        for e in ex:
            r = _rng(w.seed, layer, tid * 4096 + e + 16)
            out.append(_normal(r, shape, std))
        return _store(np.stack(out) if out else np.zeros((0,) + shape, np.float32), w.dtype)

    Wg = per_expert(_T_WG, (d, d_ff), s_in)
    Wu = per_expert(_T_WU, (d, d_ff), s_in)
    Wd = per_expert(_T_WD, (d_ff, d), s_ff)
    return LayerInputs(Wr, br, Wg, Wu, Wd)


@dataclass
class SharedInputs:
    """Shared experts in concatenated form: expert s owns columns s*f .. s*f+f-1 of Wg, Wu
    ([d][S*f]) and the same rows of Wd ([S*f][d])."""
    n: int
    f: int
    Wg: Tensor
    Wu: Tensor
    Wd: Tensor

    def expert(self, s: int):
        """float64 (Wg_s, Wu_s, Wd_s) of shared expert s."""
        c = slice(s * self.f, (s + 1) * self.f)
        return self.Wg.f64()[:, c], self.Wu.f64()[:, c], self.Wd.f64()[c, :]


_T_SHARED = 3000


def make_shared(w: Workload, layer: int, n: int, f: int) -> SharedInputs:
    """n shared experts of width f, drawn like the routed experts' weights."""
    d = w.d
    if w.init == "fan_in":
        s_in, s_ff = 1.0 / math.sqrt(d), 1.0 / math.sqrt(f)
    else:
        s_in = s_ff = 0.02
    g, u, dn = [], [], []
    for s in range(n):
        g.append(_normal(_rng(w.seed, layer, _T_SHARED + 3 * s), (d, f), s_in))
        u.append(_normal(_rng(w.seed, layer, _T_SHARED + 3 * s + 1), (d, f), s_in))
        dn.append(_normal(_rng(w.seed, layer, _T_SHARED + 3 * s + 2), (f, d), s_ff))
    return SharedInputs(n, f, _store(np.concatenate(g, axis=1), w.dtype),
                        _store(np.concatenate(u, axis=1), w.dtype),
                        _store(np.concatenate(dn, axis=0), w.dtype))


def make_inputs(w: Workload, with_layers: bool = True) -> Inputs:
    """All inputs of a workload: tokens X, upstream gradient dY, groups, k_g, weights."""
    N, d, L, G = w.N, w.d, w.L, w.G
    z = _normal(_rng(w.seed, 0, _T_X), (N, d), 1.0)
    x = _rms_unit_rows(z) if w.x_recipe == "rms_unit" else z
    t = masked = None
    if w.timestep_capacity:
        t = mask_ratios(w)
        mz = _normal(_rng(w.seed, 0, _T_MASK), (1, d), 1.0)
        mvec = _rms_unit_rows(mz)[0] if w.x_recipe == "rms_unit" else mz[0]
        masked = np.zeros(N, dtype=bool)
        prng = _rng(w.seed, 0, _T_PERM)
        for g in range(G):
            n_mask = int(math.floor(t[g] * L + 0.5))
            perm = prng.permutation(L)
            masked[g * L + perm[:n_mask]] = True
        x[masked] = mvec
        k_g = timestep_capacity(t, w.k_base, L)
    else:
        k_g = np.full(G, w.k_base, dtype=np.int32)
    X = _store(x, w.dtype)
    dY = _store(_normal(_rng(w.seed, 0, _T_DY), (N, d), 1.0), w.dtype)
    group_off = (np.arange(G + 1, dtype=np.int64) * L).astype(np.int32)
    inp = Inputs(w, X, dY, group_off, k_g, [], t, masked)
    if with_layers:
        inp.layers = [make_layer(w, l) for l in range(w.layers)]
    return inp


def random_groups(rng: np.random.Generator, N: int, G: int) -> np.ndarray:
    """Ragged group offsets: G groups covering N tokens with random sizes (>=0)."""
    cuts = np.sort(rng.integers(0, N + 1, size=G - 1))
    return np.concatenate([[0], cuts, [N]]).astype(np.int32)
