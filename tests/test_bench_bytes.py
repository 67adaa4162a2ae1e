"""The bench's algorithmic byte counts for the memory-bound kernels (the routing figure).

A stack's residual adds are fused into the combine (which then also reads X) and the dX
scatter (which also reads the incoming gradient); shared experts add their output to the
combine and their input gradient to the scatter. Those reads are part of the work, so they
are counted; a single layer without shared experts reads neither.
"""
import bench
from paper_2604_01622_gb300 import inputs as I


def _sizes(w):
    P = w.E * int(w.G * w.k_base)
    return P, w.N * w.d * 2, P * w.d * 2


def test_single_layer_counts():
    w = I.WORKLOADS["ec_d2048_e64"]
    P, nd, pd = _sizes(w)
    m = bench._mem_bytes(w, P, tc=False)
    assert m["gather"] == nd + pd == m["gather_dy"]
    assert m["combine"] == pd + nd
    assert m["dx_combine"] == pd + 2 * nd
    assert m["router_gemm_softmax"] == nd + 3 * w.N * w.E * 4


def test_stack_and_shared_experts_add_their_reads():
    w = I.WORKLOADS["ec_wide_d4096_e32_x4"]
    assert w.layers > 1
    P, nd, pd = _sizes(w)
    m = bench._mem_bytes(w, P, tc=False)
    assert m["combine"] == pd + 2 * nd           # O rows, X (residual); Y
    assert m["dx_combine"] == pd + 3 * nd        # dH rows, router dX part, dY (residual); dX
    m2 = bench._mem_bytes(w, P, tc=False, shared=True)
    assert m2["combine"] == m["combine"] + nd
    assert m2["dx_combine"] == m["dx_combine"] + nd
    one = I.scaled(w, layers=1)
    m1 = bench._mem_bytes(one, P, tc=False, shared=True)
    assert m1["combine"] == pd + 2 * nd and m1["dx_combine"] == pd + 3 * nd


def test_gemm_rooflines_from_the_work_of_each_phase():
    """FLOPs per phase sum to the 18 P d d_ff of a step; dU (the SwiGLU backward reads A and B
    and writes dA and dB) has the lowest intensity, and an intensity below the ridge caps the
    attainable rate at intensity x bandwidth."""
    w = I.WORKLOADS["ec_d2048_e64"]
    P = w.E * w.G * w.k_base
    kms = {k: 1.0 for k in ("gemm_gate_up_swiglu", "gemm_down", "gemm_dgrad_up_swiglu",
                            "gemm_dgrad_h", "gemm_wgrad")}
    r = bench._gemm_rooflines(w, P, kms, hbm=6681.8, burst=1909.7)
    tf = sum(v["tflops"] for v in r.values())      # 1 ms each: TFLOP/s = GFLOP per phase / 1e3
    assert abs(tf - 18 * P * w.d * w.d_ff / 1e9) < 1.0
    low = min(r, key=lambda k: r[k]["flop_per_byte"])
    assert low == "gemm_dgrad_up_swiglu"
    small = I.WORKLOADS["ec_many_small_e128"]
    Ps = small.E * small.G * small.k_base
    rs = bench._gemm_rooflines(small, Ps, kms, hbm=6681.8, burst=1909.7)
    du = rs["gemm_dgrad_up_swiglu"]
    assert du["flop_per_byte"] < 1909.7e3 / 6681.8
    assert abs(du["attainable_tflops"] / (du["flop_per_byte"] * 6.6818) - 1) < 1e-3
    assert bench._gemm_rooflines(I.WORKLOADS["tiny_f32"], 32, kms, 6681.8, 1909.7) is None
