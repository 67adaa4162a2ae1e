"""The allocation-free selection entry point (ec_select_static) against ec_route.

ec_select_static exists for callers that cannot call cudaMalloc (a fixed memory budget
handed out by another runtime, or code that must not grow its device footprint while
serving): its scratch lives in a static device array inside the library. It must return
exactly the selection ec_route returns on the same scores, call after call, although all
calls share that array. This file is collected last so a failure here cannot stop the
rest of the GPU suite.
"""
import numpy as np
import pytest
import torch

import paper_2604_01622_gb300 as ec
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer

pytestmark = pytest.mark.gpu


def _case(seed, N, E, G, quant):
    rng = np.random.default_rng(seed)
    S = rng.random((E, N)).astype(np.float32)
    if quant:
        S = (np.round(S * quant) / quant).astype(np.float32)   # ties
    group_off = I.random_groups(rng, N, G)
    k_g = np.array([rng.integers(0, s + 1) for s in np.diff(group_off)], np.int32)
    return S, group_off, k_g


def _static(S_dev, N, E, group_off, k_g):
    M = int(k_g.sum())
    idx = torch.full((E, M), -7, dtype=torch.int32, device="cuda")
    gate = torch.full((E, M), -7.0, dtype=torch.float32, device="cuda")
    ec.ec_select_static(S_dev.data_ptr(), N, E, group_off, k_g, idx.data_ptr(),
                        gate.data_ptr(), torch.cuda.current_stream().cuda_stream)
    return idx, gate


def test_static_selection_matches_ec_route_on_two_calls_in_a_row():
    cases = [_case(1, 5000, 16, 3, 8.0), _case(2, 32768, 64, 8, None)]
    outs = []
    for S, group_off, k_g in cases:                      # two calls, back to back
        N, E = S.shape[1], S.shape[0]
        S_dev = torch.from_numpy(S).cuda()
        outs.append((_static(S_dev, N, E, group_off, k_g), S_dev, group_off, k_g))
    torch.cuda.synchronize()
    for (idx, gate), S_dev, group_off, k_g in outs:
        E, N = S_dev.shape
        lay = ECMoELayer(N, 64, E, 64, group_off, k_g, dtype="f32")
        ref_idx, ref_gate, _ = lay.route(S_in=S_dev)
        lay.check()
        # integer selection: bit-exact; gates are copies of the scores: exact
        assert torch.equal(idx, ref_idx)
        assert torch.equal(gate, ref_gate)


def test_static_selection_rejects_sizes_beyond_its_array():
    N, E = 70000, 64                                     # N*E above the static maximum
    S_dev = torch.zeros((E, N), dtype=torch.float32, device="cuda")
    with pytest.raises(ec.ECError) as e:
        _static(S_dev, N, E, np.array([0, N], np.int32), np.array([1], np.int32))
    assert e.value.status == ec.EC_ERR_UNSUPPORTED
