"""Seeded input generators: determinism, bf16 rounding, capacity recipe."""
import numpy as np
import torch

from paper_2604_01622_gb300 import inputs as I


def test_bf16_rounding_matches_torch():
    rng = np.random.default_rng(0)
    x = np.concatenate([rng.standard_normal(100000).astype(np.float32) * 10,
                        np.array([0.0, -0.0, 1.0, -1.0, 3.0e38, 1e-40], np.float32)])
    ours = I.bf16_bits(x)
    ref = torch.from_numpy(x).to(torch.bfloat16).view(torch.int16).numpy().view(np.uint16)
    assert np.array_equal(ours, ref)
    np.testing.assert_array_equal(I.bf16_to_f64(ours),
                                  torch.from_numpy(x).to(torch.bfloat16).double().numpy())


def test_timestep_capacity_sums_to_uniform_total():
    rng = np.random.default_rng(1)
    # the sum is exact whenever G*k_base <= L (then no k_g can exceed L), as in
    # both timestep workloads (8*512 = 4096 = L and 4*512 <= 8192)
    for G, kb, L in [(8, 512, 4096), (4, 512, 8192), (3, 5, 15), (16, 1, 16)]:
        for _ in range(50):
            t = rng.random(G)
            k = I.timestep_capacity(t, kb, L)
            assert k.sum() == G * kb
            assert np.all((k >= 0) & (k <= L))
            # more capacity at lower mask ratio (weights 2(1-t) are decreasing in t)
            order = np.argsort(t)
            assert np.all(np.diff(k[order]) <= 1)
    assert np.array_equal(I.timestep_capacity(np.ones(4), 3, 10), np.full(4, 3))
    assert np.all(I.timestep_capacity(rng.random(3), 5, 7) <= 7)   # clipped to L


def test_tiny_workload_is_deterministic_and_shaped():
    w = I.WORKLOADS["tiny_f32"]
    a = I.make_inputs(w)
    b = I.make_inputs(w)
    assert np.array_equal(a.X.data, b.X.data)
    assert np.array_equal(a.layers[0].Wg.data, b.layers[0].Wg.data)
    assert a.X.shape == (256, 64) and a.layers[0].Wg.shape == (8, 64, 128)
    assert a.layers[0].Wd.shape == (8, 128, 64) and a.layers[0].Wr.shape == (64, 8)
    assert list(a.k_g) == [16, 16] and list(a.group_off) == [0, 128, 256]
    # per-expert draws: a slice of experts equals the slice of the full tensor
    part = I.make_layer(w, 0, slice(2, 5))
    assert np.array_equal(part.Wu.data, a.layers[0].Wu.data[2:5])


def test_timestep_workload_masks_and_capacity():
    w = I.scaled(I.WORKLOADS["ec_timestep_d2048_e64"], G=4, L=256, d=64, E=8, d_ff=64, k_base=16)
    inp = I.make_inputs(w, with_layers=False)
    X = inp.X.f64()
    for g in range(w.G):
        m = inp.masked[g * w.L:(g + 1) * w.L]
        assert m.sum() == int(np.floor(inp.t[g] * w.L + 0.5))
    rows = X[inp.masked]
    assert np.all(rows == rows[0])
    assert inp.k_g.sum() == w.G * w.k_base
    # rmsnorm(z)/sqrt(d): unit rows (before bf16 rounding)
    assert np.allclose(np.linalg.norm(X, axis=1), 1.0, atol=1e-2)
