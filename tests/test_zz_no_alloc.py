"""The allocation-free selection entry point (ec_select_static) against ec_route and the oracle.

ec_select_static exists for callers that cannot call cudaMalloc (a fixed memory budget
handed out by another runtime, or code that must not grow its device footprint while
serving): its scratch lives in a static device array inside the library. It must return
exactly the selection ec_route returns on the same scores, and the one the oracle's TopC
defines (Sec. 2.2: each expert keeps its top-k_g tokens of every group), call after call,
although all calls share that array. This file is collected last so a failure here cannot
stop the rest of the GPU suite.
"""
import numpy as np
import pytest
import torch

import paper_2604_01622_gb300 as ec
from oracle import ecmoe as O
from paper_2604_01622_gb300 import inputs as I
from paper_2604_01622_gb300.layer import ECMoELayer

pytestmark = pytest.mark.gpu

MAX_SCORES = 4194304    # EC_STATIC_SELECT_MAX_SCORES in include/ecmoe.h
MAX_GROUPS = 4096       # EC_STATIC_SELECT_MAX_GROUPS


def _case(seed, N, E, G, quant, kmax_frac=1.0):
    rng = np.random.default_rng(seed)
    S = rng.random((E, N)).astype(np.float32)
    if quant:
        S = (np.round(S * quant) / quant).astype(np.float32)   # ties
    group_off = I.random_groups(rng, N, G)
    k_g = np.array([rng.integers(0, int(s * kmax_frac) + 1) for s in np.diff(group_off)],
                   np.int32)
    return S, group_off, k_g


def _static(S_dev, N, E, group_off, k_g, stream=None):
    M = int(np.asarray(k_g).sum())
    idx = torch.full((E, M), -7, dtype=torch.int32, device="cuda")
    gate = torch.full((E, M), -7.0, dtype=torch.float32, device="cuda")
    st = stream or torch.cuda.current_stream()
    ec.ec_select_static(S_dev.data_ptr(), N, E, group_off, k_g, idx.data_ptr(),
                        gate.data_ptr(), st.cuda_stream)
    return idx, gate


def _check(idx, gate, S, S_dev, group_off, k_g):
    """Bit-exact against ec_route on the same device scores and against the oracle's TopC."""
    E, N = S.shape
    lay = ECMoELayer(N, 64, E, 64, group_off, k_g, dtype="f32")
    ref_idx, ref_gate, _ = lay.route(S_in=S_dev)
    lay.check()
    # integer selection: bit-exact; gates are copies of the scores: exact
    assert torch.equal(idx, ref_idx)
    assert torch.equal(gate, ref_gate)
    o_idx, o_gate = O.ec_select(S.T.astype(np.float64), group_off, k_g)
    assert np.array_equal(idx.cpu().numpy(), o_idx)
    assert np.array_equal(gate.double().cpu().numpy(), o_gate)
    lay.close()


def test_static_selection_matches_ec_route_and_oracle_on_two_calls_in_a_row():
    cases = [_case(1, 5000, 16, 3, 8.0), _case(2, 32768, 64, 8, None)]
    outs = []
    for S, group_off, k_g in cases:                      # two calls, back to back
        N, E = S.shape[1], S.shape[0]
        S_dev = torch.from_numpy(S).cuda()
        outs.append((_static(S_dev, N, E, group_off, k_g), S, S_dev, group_off, k_g))
    torch.cuda.synchronize()
    for (idx, gate), S, S_dev, group_off, k_g in outs:
        _check(idx, gate, S, S_dev, group_off, k_g)


def test_static_selection_at_its_limits():
    """N*E exactly at the array's maximum (the slot map fills the whole array), then the
    largest number of groups (the group tables fill theirs), also at the score maximum."""
    for seed, N, E, G, quant in ((3, 65536, 64, 8, 16.0), (4, 65536, 64, MAX_GROUPS, 4.0)):
        assert N * E == MAX_SCORES
        S, group_off, k_g = _case(seed, N, E, G, quant, kmax_frac=0.25)
        assert len(k_g) == G
        S_dev = torch.from_numpy(S).cuda()
        idx, gate = _static(S_dev, N, E, group_off, k_g)
        torch.cuda.synchronize()
        _check(idx, gate, S, S_dev, group_off, k_g)


def test_static_selection_host_arrays_reusable_on_return():
    """Pinned host tables may be overwritten as soon as the call returns."""
    S, group_off, k_g = _case(5, 20000, 32, 16, 8.0)
    N, E = S.shape[1], S.shape[0]
    S_dev = torch.from_numpy(S).cuda()
    g_pin = torch.from_numpy(group_off.astype(np.int32)).pin_memory()
    k_pin = torch.from_numpy(k_g.astype(np.int32)).pin_memory()
    busy = torch.cuda.current_stream()
    torch.cuda._sleep(50_000_000)                        # keep the stream busy for a while
    idx, gate = _static(S_dev, N, E, g_pin.numpy(), k_pin.numpy(), stream=busy)
    g_pin.fill_(0)                                       # the caller reuses its arrays at once
    k_pin.fill_(0)
    torch.cuda.synchronize()
    _check(idx, gate, S, S_dev, group_off, k_g)


def test_static_selection_refuses_a_capturing_stream():
    S, group_off, k_g = _case(6, 4096, 8, 2, None)
    S_dev = torch.from_numpy(S).cuda()
    torch.cuda.synchronize()
    side = torch.cuda.Stream()
    graph = torch.cuda.CUDAGraph()
    status = None
    with torch.cuda.stream(side):
        graph.capture_begin()
        try:
            _static(S_dev, 4096, 8, group_off, k_g, stream=side)
        except ec.ECError as e:
            status = e.status
        finally:
            graph.capture_end()
    assert status == ec.EC_ERR_UNSUPPORTED
    # outside the capture the same call works
    idx, gate = _static(S_dev, 4096, 8, group_off, k_g)
    torch.cuda.synchronize()
    _check(idx, gate, S, S_dev, group_off, k_g)


def test_static_selection_rejects_sizes_beyond_its_array():
    N, E = 70000, 64                                     # N*E above the static maximum
    S_dev = torch.zeros((E, N), dtype=torch.float32, device="cuda")
    with pytest.raises(ec.ECError) as e:
        _static(S_dev, N, E, np.array([0, N], np.int32), np.array([1], np.int32))
    assert e.value.status == ec.EC_ERR_UNSUPPORTED
    G = MAX_GROUPS + 1                                   # more groups than its tables hold
    off = np.arange(G + 1, dtype=np.int32)
    S_dev = torch.zeros((4, G), dtype=torch.float32, device="cuda")
    with pytest.raises(ec.ECError) as e:
        _static(S_dev, G, 4, off, np.ones(G, np.int32))
    assert e.value.status == ec.EC_ERR_UNSUPPORTED
