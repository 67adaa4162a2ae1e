#!/usr/bin/env python3
"""EC-MoE layer forward + backward throughput on GB300 (tokens/s).

Default workload: 8 sequences x 4096 tokens (N = 32768), d_model 2048, 64 SwiGLU experts
of d_ff 1024, capacity k_g = 512 per expert per sequence (top-8 equivalent), bf16 with
fp32 accumulation, seeded synthetic inputs. One step = ec_moe_forward + ec_moe_backward
through the C ABI on inputs resident in HBM. Inputs and saved activations (GBs) are far
larger than the 129 MB L2, so no explicit flush is done between steps.

  python bench.py [--gpus N] [--steps K] [--warmup W] [--impl ours|reference]

With N > 1 (torchrun) every rank runs its own replica of the workload on its own GPU
(the layer needs no exchange in the forward pass and this benchmark does not all-reduce
weight gradients); value = tokens of all ranks / max over ranks of the step time.
`--impl reference` times the float64 CPU oracle on the host cores instead.
`--routing tc --tc-k K [--tc-cf CF]` runs the same shape under token-choice routing (each
token takes its K best experts, capacity ceil(CF K N / E) per expert, dropless without
--tc-cf), the comparison baseline of the paper's Sec. 2.2.
"""
from __future__ import annotations

import argparse
import hashlib
import json
import math
import os
import subprocess
import sys
import tempfile
import time

ROOT = os.path.dirname(os.path.abspath(__file__))
sys.path.insert(0, ROOT)

METRIC = "EC-MoE layer fwd+bwd tokens/sec on 1 GB300; expert-GEMM % BF16 peak; routing HBM GB/s"
METRIC_TC = "TC-MoE layer fwd+bwd tokens/sec on 1 GB300 (token-choice comparison routing)"
UNIT = "tokens/s"

# DRAM traffic per launch of the grouped-GEMM kernels (dram__bytes_read.sum +
# dram__bytes_write.sum, mean of the six expert-GEMM launches of one step), keyed by the hash
# of the kernel source it was taken on; a changed kernel reports null until re-captured. The
# counters were taken on 1, 2 and 4 of the workload's 8 sequences (captures of a few GB); each
# launch's traffic is affine in the sequences (within 1.4%) and is extrapolated to 8.
TILE_POLICY = {"auto": 0, "256": 1, "512": 2}   # EC_TILES_AUTO / EC_TILES_256 / EC_TILES_512
TRAFFIC = {"d35aded7c71d": 2865896485}


def _peaks():
    p = os.path.join(ROOT, "MEASURED_PEAKS.json")
    if os.path.exists(p):
        d = json.load(open(p))
        return d["hbm_gbs"], d["bf16_tflops"], d["bf16_tflops_sustained"], "measured"
    return 6800.0, 1900.0, 1700.0, "fallback"


def _src_hash(path):
    return hashlib.sha1(open(path, "rb").read()).hexdigest()[:12]


def _cores():
    for v in ("OPENBLAS_NUM_THREADS", "OMP_NUM_THREADS"):
        if os.environ.get(v, "").isdigit():
            return int(os.environ[v])
    try:
        return len(os.sched_getaffinity(0))
    except AttributeError:
        return os.cpu_count()


# ------------------------------------------------------------------ clocks
class Clocks:
    """nvidia-smi sampler running during the timed region."""
    Q = ("timestamp,clocks.sm,clocks.max.sm,power.draw,utilization.gpu,clocks_event_reasons.active,"
         "clocks_event_reasons.hw_slowdown,clocks_event_reasons.hw_thermal_slowdown,"
         "clocks_event_reasons.sw_thermal_slowdown,clocks_event_reasons.sw_power_cap")

    def __init__(self, index):
        self.index = index
        self.proc = None
        self.f = tempfile.NamedTemporaryFile("w+", suffix=".csv", delete=False)

    def start(self):
        self.t_begin = None
        self.t_end = None
        try:
            self.proc = subprocess.Popen(
                ["nvidia-smi", f"--id={self.index}", f"--query-gpu={self.Q}",
                 "--format=csv,noheader,nounits", "-lms", "100"],
                stdout=self.f, stderr=subprocess.DEVNULL)
        except OSError:
            self.proc = None

    def mark_begin(self):
        self.t_begin = time.time()

    def mark_end(self):
        self.t_end = time.time()

    def stop(self, window=None):
        """Summary of the samples between mark_begin and mark_end (or the given (t0, t1))."""
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        time.sleep(0.25)
        self.proc.terminate()
        self.proc.wait()
        self.f.flush()
        self.rows = [r.split(",") for r in open(self.f.name).read().strip().splitlines() if r]
        os.unlink(self.f.name)
        return self.summary((self.t_begin, self.t_end) if window is None else window)

    def summary(self, window):
        import datetime
        if self.proc is None:
            return {"sm_mhz": None, "sm_max_mhz": None, "reasons": ["nvidia-smi unavailable"]}
        t_begin, t_end = window
        names = ["hw_slowdown", "hw_thermal_slowdown", "sw_thermal_slowdown", "sw_power_cap"]
        sm, smax, reasons, load = [], [], set(), []
        for r in self.rows:
            r = [x.strip() for x in r]
            if len(r) < 10:
                continue
            try:
                ts = datetime.datetime.strptime(r[0], "%Y/%m/%d %H:%M:%S.%f").timestamp()
                if t_begin and t_end and not (t_begin - 0.05 <= ts <= t_end + 0.05):
                    continue
                sm.append(float(r[1]))
                smax.append(float(r[2]))
                load.append(float(r[4]))
            except ValueError:
                continue
            for n, v in zip(names, r[6:10]):
                if v.lower() == "active":
                    reasons.add(n)
        busy = [s for s, u in zip(sm, load) if u >= 50] or sm
        busy.sort()
        return {"sm_mhz": busy[len(busy) // 2] if busy else None,
                "sm_max_mhz": max(smax) if smax else None,
                "reasons": sorted(reasons), "samples": len(sm)}


class NvmlClocks:
    """SM clock and clock-event reasons read through NVML every few milliseconds, so a timed
    region of a tenth of a second still gets tens of samples (reads only; nothing is set)."""
    BITS = {0x4: "sw_power_cap", 0x8: "hw_slowdown", 0x20: "sw_thermal_slowdown",
            0x40: "hw_thermal_slowdown", 0x80: "hw_power_brake_slowdown"}

    def __init__(self, index, period_s=0.004):
        import ctypes
        import threading
        self.period = period_s
        self.samples = []
        self.lib = None
        self.stop_flag = threading.Event()
        self.thread = None
        try:
            lib = ctypes.CDLL("libnvidia-ml.so.1")
            if lib.nvmlInit_v2() != 0:
                return
            h = ctypes.c_void_p()
            if lib.nvmlDeviceGetHandleByIndex_v2(ctypes.c_uint(index), ctypes.byref(h)) != 0:
                return
            self.h = h
            self.reasons_fn = getattr(lib, "nvmlDeviceGetCurrentClocksEventReasons", None) or \
                getattr(lib, "nvmlDeviceGetCurrentClocksThrottleReasons")
            mx = ctypes.c_uint()
            self.max_mhz = (float(mx.value) if lib.nvmlDeviceGetMaxClockInfo(h, 1, ctypes.byref(mx)) == 0
                            else None)
            self.lib = lib
        except (OSError, AttributeError):
            self.lib = None

    def _run(self):
        import ctypes
        mhz = ctypes.c_uint()
        bits = ctypes.c_ulonglong()
        while not self.stop_flag.is_set():
            t = time.time()
            ok = self.lib.nvmlDeviceGetClockInfo(self.h, 1, ctypes.byref(mhz)) == 0   # SM clock
            ok = ok and self.reasons_fn(self.h, ctypes.byref(bits)) == 0
            if ok:
                self.samples.append((t, float(mhz.value), int(bits.value)))
            time.sleep(self.period)

    def start(self):
        import threading
        if self.lib is None:
            return
        self.stop_flag.clear()
        self.thread = threading.Thread(target=self._run, daemon=True)
        self.thread.start()

    def stop(self):
        if self.thread is not None:
            self.stop_flag.set()
            self.thread.join()
            self.thread = None

    def summary(self, window):
        if self.lib is None:
            return None
        t0, t1 = window
        sel = [(m, b) for (t, m, b) in self.samples if t0 <= t <= t1]
        if not sel:
            return None
        mhz = sorted(m for m, _ in sel)
        reasons = sorted({name for m, b in sel for bit, name in self.BITS.items() if b & bit})
        return {"sm_mhz": mhz[len(mhz) // 2], "sm_max_mhz": self.max_mhz, "reasons": reasons,
                "samples": len(sel)}


def _clock_record(smi, nvml, window):
    """nvidia-smi's record of the window (the profiling recipe's query), with NVML's denser
    samples of the same window taking over the median and adding their reasons."""
    rec = smi.summary(window)
    nv = nvml.summary(window) if nvml is not None else None
    if nv:
        rec = dict(rec)
        rec["nvidia_smi_samples"] = rec.get("samples")
        rec["sm_mhz"] = nv["sm_mhz"]
        rec["sm_max_mhz"] = nv["sm_max_mhz"] or rec.get("sm_max_mhz")
        rec["reasons"] = sorted(set(rec.get("reasons", [])) | set(nv["reasons"]))
        rec["samples"] = nv["samples"]
        rec["source"] = "NVML every 4 ms (median SM clock, clock-event reasons) + nvidia-smi every 100 ms"
    return rec


# ------------------------------------------------------------------ CPU oracle sample
class OracleSample:
    """A bounded sample of the workload for the float64 oracle (as it stands): whole
    sequences of the workload when `tokens` >= its sequence length, else one shorter
    sequence with the capacity scaled to keep the workload's capacity factor. Shared
    experts are included when configured; for a stack of layers one layer is timed and the
    rate divided by the number of layers (the layers have equal shapes)."""

    def __init__(self, tokens: int, w, shared_experts: int = 0, shared_dff: int = 0):
        from paper_2604_01622_gb300 import inputs as I
        if tokens >= w.L:
            G, L, k = max(1, tokens // w.L), w.L, w.k_base
        else:
            G, L, k = 1, tokens, max(1, w.k_base * tokens // w.L)
        self.tokens = G * L
        self.layers = w.layers
        ws = I.scaled(w, G=G, L=L, k_base=k, timestep_capacity=False, layers=1)
        inp = I.make_inputs(ws)
        Ld = inp.layers[0]
        self.args = (inp.X.f64(), Ld.Wr.f64(), Ld.br, Ld.Wg.f64(), Ld.Wu.f64(), Ld.Wd.f64(),
                     inp.group_off, inp.k_g)
        self.dY = inp.dY.f64()
        self.shared = None
        if shared_experts:
            sh = I.make_shared(ws, 0, shared_experts, shared_dff)
            g, u, dn, f = sh.Wg.f64(), sh.Wu.f64(), sh.Wd.f64(), shared_dff
            self.shared = [(g[:, i * f:(i + 1) * f], u[:, i * f:(i + 1) * f],
                            dn[i * f:(i + 1) * f, :]) for i in range(shared_experts)]
        self.desc = (f"{G} sequence(s) x {L} tokens of the workload (k_g={k}, capacity factor "
                     f"{w.E * k / L:g}, E={w.E}, d={w.d}, d_ff={w.d_ff}"
                     + (f", {shared_experts} shared experts of d_ff {shared_dff}"
                        if shared_experts else "")
                     + (f"; one of the {w.layers} layers timed" if w.layers > 1 else "")
                     + "), oracle fwd+bwd")

    def run(self):
        """Returns (tokens/s through the whole stack, seconds of the timed layer)."""
        from oracle import ecmoe as O
        X, Wr, br, Wg, Wu, Wd, goff, kg = self.args
        t0 = time.perf_counter()
        f = O.forward(X, Wr, br, Wg, Wu, Wd, goff, kg, shared=self.shared)
        O.backward(f, self.dY, Wr, Wg, Wu, Wd)
        dt = time.perf_counter() - t0
        return self.tokens / dt / self.layers, dt


class TCOracleSample:
    """A bounded sample for the token-choice oracle: `tokens` tokens of the workload's
    first sequence under the same k and capacity factor."""

    def __init__(self, tokens: int, w, k: int, cf):
        from paper_2604_01622_gb300 import inputs as I
        L = min(tokens, w.L)
        ws = I.scaled(w, G=1, L=L, timestep_capacity=False, layers=1)
        inp = I.make_inputs(ws)
        Ld = inp.layers[0]
        self.tokens, self.k = L, k
        self.cap = None if cf is None else int(math.ceil(cf * k * L / w.E))
        self.args = (inp.X.f64(), Ld.Wr.f64(), Ld.br, Ld.Wg.f64(), Ld.Wu.f64(), Ld.Wd.f64())
        self.dY = inp.dY.f64()
        self.desc = (f"{L} tokens of one sequence of the workload, token choice k={k}, "
                     f"capacity {'none' if cf is None else self.cap}, E={w.E}, d={w.d}, "
                     f"d_ff={w.d_ff}, oracle fwd+bwd")

    def run(self):
        from oracle import token_choice as TC
        X, Wr, br, Wg, Wu, Wd = self.args
        t0 = time.perf_counter()
        f = TC.tc_forward(X, Wr, br, Wg, Wu, Wd, self.k, self.cap)
        TC.tc_backward(f, self.dY, Wr, Wg, Wu, Wd)
        dt = time.perf_counter() - t0
        return self.tokens / dt, dt


# ------------------------------------------------------------------ distributed
def _dist():
    ws = int(os.environ.get("WORLD_SIZE", "1"))
    rank = int(os.environ.get("RANK", "0"))
    local = int(os.environ.get("LOCAL_RANK", "0"))
    return ws, rank, local


def _max_over_ranks(x: float, ws: int, device) -> float:
    if ws == 1:
        return x
    import torch
    import torch.distributed as dist
    t = torch.tensor([x], dtype=torch.float64, device=device)
    dist.all_reduce(t, op=dist.ReduceOp.MAX)
    return float(t.item())


def _barrier(ws):
    if ws > 1:
        import torch.distributed as dist
        dist.barrier()


# ------------------------------------------------------------------ our arm
NOMINAL = {"bf16_tflops": 2250.0, "hbm_gbs": 7900.0,
           "source": "GB300 nominal dense BF16 tensor rate and HBM3e bandwidth"}
# the other workloads timed beside the headline one (single-GPU runs of the default line)
EXTRA_WORKLOADS = ("tiny_f32", "ec_timestep_d2048_e64", "ec_many_small_e128",
                   "ec_wide_d4096_e32_x4")


def _mem_bytes(w, P, tc, shared=False, splits_hint=None):
    """Algorithmic bytes per launch of the memory-bound kernels (routing, gathers, combine,
    router backward) of one layer: what each must read and write at least, with the gathers
    counted token-major ((N + P) d b: each token row read once, P rows written). In a stack
    (residual adds) the combine also reads X and the dX scatter the incoming gradient; with
    shared experts they also read the shared FFN's output and its input gradient."""
    b = 2 if w.dtype == "bf16" else 4
    N, d, E = w.N, w.d, w.E
    Ep = (E + 63) // 64 * 64
    parts = math.ceil(w.d_ff / 256) if w.dtype == "bf16" else 1   # gate-gradient partials
    fused_rb = E % 4 == 0 and E <= 128 and not tc   # one router-backward kernel
    dz = 2 * N * Ep * 2 if w.dtype == "bf16" else N * E * 4     # dZ (bf16 hi + lo, or fp32)
    extra = ((1 if w.layers > 1 else 0) + (1 if shared else 0)) * N * d * b
    return {
        # X, S and S^T; expert choice also sets the slot map [N][E] to -1 there
        "router_gemm_softmax": N * d * b + 2 * N * E * 4 + (0 if tc else N * E * 4),
        "topk": N * E * 4 + 3 * P * 4,      # S^T read; idx, gate and the selected slots
        "tc_route": 2 * N * E * 4 + 3 * P * 4,
        "gather": (N + P) * d * b,          # token-major: each X row read once, P rows written
        "combine": P * d * b + N * d * b + extra,
        "bwd_gather_scale": 3 * P * d * b,
        "gather_dy": (N + P) * d * b,
        # slot map and S read, gate-gradient partials read, dZ planes (bf16) or dZ (fp32)
        "softmax_bwd": (2 * N * E * 4 + parts * P * 4 + dz) if fused_rb else 3 * N * E * 4,
        "dgate_reduce": (parts + 1) * P * 4,
        "router_dgrad_gemm": dz + N * d * b,        # dZ read, the router's dX part written
        "dx_combine": P * d * b + 2 * N * d * b + extra,   # dH rows; router's dX part; dX
        "router_wgrad_gemm": N * d * b + dz,       # X and dZ read (split-K partials aside)
        "router_wgrad_reduce": d * E * 4,          # dWr written
    }


def _gemm_rooflines(w, P, kms, hbm, burst):
    """Each expert-GEMM phase against its own roofline: FLOPs and algorithmic DRAM bytes per
    step (operands, weights and outputs once each; fp32 weight gradients), their ratio, the
    attainable rate min(burst peak, ratio x copy bandwidth) and the fraction of it reached.
    Only for the tensor-core (bf16) path."""
    if w.dtype != "bf16":
        return None
    b, d, F, E, L = 2, w.d, w.d_ff, w.E, w.layers
    work = {   # phase: (FLOP, bytes) per layer
        "gemm_gate_up_swiglu": (4 * P * d * F, P * d * b + 2 * E * d * F * b + 3 * P * F * b),
        "gemm_down": (2 * P * d * F, P * F * b + E * F * d * b + P * d * b),
        "gemm_dgrad_up_swiglu": (2 * P * d * F, P * d * b + E * F * d * b + 4 * P * F * b),
        "gemm_dgrad_h": (4 * P * d * F, 2 * P * F * b + 2 * E * d * F * b + P * d * b),
        "gemm_wgrad": (6 * P * d * F, (P * d * b + 2 * P * F * b + 2 * E * d * F * 4)
                       + (P * F * b + P * d * b + E * F * d * 4)),
    }
    out = {}
    for k, (fl, by) in work.items():
        ms = kms.get(k)
        if not ms:
            continue
        fl, by = fl * L, by * L
        att = min(burst, fl / by * hbm / 1e3)   # TFLOP/s (hbm in GB/s)
        ach = fl / (ms * 1e-3) / 1e12
        out[k] = {"ms": ms, "tflops": round(ach, 1), "gbytes": round(by / 1e9, 3),
                  "flop_per_byte": round(fl / by, 1), "attainable_tflops": round(att, 1),
                  "frac_of_attainable": round(ach / att, 3)}
    return out


def _timestep_schedule(w, n, seed=12345):
    """Per-step capacities of a timestep workload: each step draws a new masking ratio per
    sequence and takes k_g by the workload's FLOPs-matched rule (the sum stays G k_base)."""
    import numpy as np
    from paper_2604_01622_gb300 import inputs as I
    rng = np.random.default_rng(seed)
    return np.stack([I.timestep_capacity(rng.random(w.G), w.k_base, w.L) for _ in range(n)])


def measure(w, args, device, ws, local, headline):
    """Build one workload's layers on the device and time fwd+bwd steps. Returns a dict of
    the line's keys for it (the headline also gets the CUDA-graph leg and token coverage)."""
    import numpy as np
    import torch
    from paper_2604_01622_gb300 import inputs as I
    from paper_2604_01622_gb300.layer import ECMoELayer, TCMoELayer, tc_capacity
    tc = args.routing == "tc"
    if tc and args.shared_experts:
        raise SystemExit("--routing tc has no shared experts")
    inp = I.make_inputs(w)

    def to_dev(t):
        if t.dtype == "bf16":
            return torch.from_numpy(t.data.view(np.int16)).to(device).view(torch.bfloat16)
        return torch.from_numpy(t.data).to(device)

    X, dY = to_dev(inp.X), to_dev(inp.dY)
    stack = []          # one context per layer; several layers stack with residual adds
    Fs = args.shared_experts * args.shared_dff if headline else 0
    tc_cap = None
    for li, Ld in enumerate(inp.layers):
        wts = (to_dev(Ld.Wr), None if Ld.br is None else torch.from_numpy(Ld.br).to(device),
               to_dev(Ld.Wg), to_dev(Ld.Wu), to_dev(Ld.Wd))
        shared = None
        if Fs:
            sh = I.make_shared(w, li, args.shared_experts, args.shared_dff)
            shared = (to_dev(sh.Wg), to_dev(sh.Wu), to_dev(sh.Wd))
        if tc:
            tc_cap = tc_capacity(args.tc_cf, args.tc_k, w.N, w.E)
            lay_l = TCMoELayer(w.N, w.d, w.E, w.d_ff, args.tc_k, tc_cap, dtype=w.dtype,
                               device=device)
        else:
            lay_l = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype=w.dtype,
                               device=device, d_ff_shared=Fs)
        if w.layers > 1:
            lay_l.set_residual(True)
        lay_l.set_tiles(TILE_POLICY[args.tiles])
        g = {"dX": torch.empty_like(X),
             "dWr": torch.empty(w.d, w.E, dtype=torch.float32, device=device),
             "dbr": None if Ld.br is None else torch.empty(w.E, dtype=torch.float32,
                                                           device=device),
             "dWg": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device=device),
             "dWu": torch.empty(w.E, w.d, w.d_ff, dtype=torch.float32, device=device),
             "dWd": torch.empty(w.E, w.d_ff, w.d, dtype=torch.float32, device=device)}
        if Fs:
            g.update(dWg_s=torch.empty(w.d, Fs, dtype=torch.float32, device=device),
                     dWu_s=torch.empty(w.d, Fs, dtype=torch.float32, device=device),
                     dWd_s=torch.empty(Fs, w.d, dtype=torch.float32, device=device))
        stack.append((lay_l, wts, [torch.empty_like(X)], g, shared))
    lay = stack[0][0]
    Y = stack[-1][2][0]
    grads = stack[0][3]
    stream = torch.cuda.current_stream(device)
    # Timestep workloads (Sec. 4.2): a new capacity per sequence every step, read by the
    # layers from a device array uploaded once (ec_ctx_set_capacity_async), so the step has
    # no host copy and no synchronisation for it.
    dyn = w.timestep_capacity and not tc and not args.static_capacity
    kg_dev = None
    if dyn:
        kg_dev = torch.from_numpy(_timestep_schedule(w, 16).astype(np.int32)).to(device)
    step_no = [0]

    def run_stack(x, dy, y_last, dx_first, st=None):
        """Forward through every layer, then backward in reverse; returns nothing."""
        kg = None
        if dyn:
            kg = kg_dev[step_no[0] % kg_dev.shape[0]]
            step_no[0] += 1
        h = x
        for i, (l_, wts, ybuf, g, shared) in enumerate(stack):
            out = y_last if i == len(stack) - 1 else ybuf[0]
            if kg is not None:
                l_.set_capacity_async(kg, stream=st)
            l_.forward(h, *wts, Y=out, outputs=False, stream=st, shared=shared)
            h = out
        d = dy
        for i in range(len(stack) - 1, -1, -1):
            l_, wts, ybuf, g, _sh = stack[i]
            gi = dict(g)
            if i == 0:
                gi["dX"] = dx_first
            l_.backward(d, grads=gi, stream=st)
            d = gi["dX"]

    def step(x=X, dy=dY, y=Y, g=grads):
        run_stack(x, dy, y, g["dX"])

    for _ in range(args.warmup):
        step()
    lay.check()
    # ---- device-timed steps (inputs resident), per-kernel events on the same stream
    for l_ in stack:
        l_[0].set_profiling(True)
    launches0 = sum(l_[0].launches for l_ in stack)
    clocks = Clocks(local)
    nvml = NvmlClocks(local)
    clocks.start()
    nvml.start()
    time.sleep(0.5)       # let the samplers come up before the timed region
    _barrier(ws)
    torch.cuda.synchronize(device)
    clocks.mark_begin()
    e0 = torch.cuda.Event(enable_timing=True)
    e1 = torch.cuda.Event(enable_timing=True)
    e0.record(stream)
    for _ in range(args.steps):
        step()
    e1.record(stream)
    torch.cuda.synchronize(device)
    clocks.mark_end()
    dev_window = (clocks.t_begin, clocks.t_end)
    _barrier(ws)
    launches = sum(l_[0].launches for l_ in stack) - launches0
    phases = [ph for l_ in stack for ph in l_[0].profile()]
    for l_ in stack:
        l_[0].set_profiling(False)
        l_[0].check()
    ms = e0.elapsed_time(e1) / args.steps
    ms_max = _max_over_ranks(ms, ws, device)

    graph_ms = None
    if headline:
        # ---- the same step captured once in a CUDA graph and replayed (no per-kernel
        # events): the launch-free form of the step
        side = torch.cuda.Stream(device)
        side.wait_stream(stream)
        with torch.cuda.stream(side):
            step()
        stream.wait_stream(side)
        graph = torch.cuda.CUDAGraph()
        with torch.cuda.graph(graph):
            step()
        for _ in range(2):
            graph.replay()
        _barrier(ws)
        torch.cuda.synchronize(device)
        g0 = torch.cuda.Event(enable_timing=True)
        g1 = torch.cuda.Event(enable_timing=True)
        g0.record(stream)
        for _ in range(args.steps):
            graph.replay()
        g1.record(stream)
        torch.cuda.synchronize(device)
        graph_ms = _max_over_ranks(g0.elapsed_time(g1) / args.steps, ws, device)
        for l_ in stack:
            l_[0].check()
        del graph

    # ---- end to end: every step copies its inputs in from pinned host memory and its
    # results (Y, dX) out, through the public API. Copies run on their own streams with
    # NB-deep buffering, so a step's transfers may take up to NB - 1 steps of compute (the
    # boxes' host link is shared and its rate varies); the timed region spans the first input
    # copy to the last output copy.
    NB = 3
    hX = torch.empty(X.shape, dtype=X.dtype, pin_memory=True)
    hdY = torch.empty(dY.shape, dtype=dY.dtype, pin_memory=True)
    hX.copy_(X)
    hdY.copy_(dY)
    hY = [torch.empty(Y.shape, dtype=Y.dtype, pin_memory=True) for _ in range(NB)]
    hdX = [torch.empty(X.shape, dtype=X.dtype, pin_memory=True) for _ in range(NB)]
    Xe = [torch.empty_like(X) for _ in range(NB)]
    dYe = [torch.empty_like(dY) for _ in range(NB)]
    Ye = [torch.empty_like(Y) for _ in range(NB)]
    # the weight gradients stay on the device (shared by the buffers); dX is copied out
    ge = [dict(grads, dX=torch.empty_like(grads["dX"])) for _ in range(NB)]
    s_in = torch.cuda.Stream(device)
    s_out = torch.cuda.Stream(device)
    ev = lambda: torch.cuda.Event()
    in_ready = [ev() for _ in range(NB)]
    computed = [ev() for _ in range(NB)]
    copied_out = [ev() for _ in range(NB)]

    def e2e_pass(n):
        """n pipelined steps; returns ms from the first input copy to the last output copy."""
        _barrier(ws)
        torch.cuda.synchronize(device)
        t0 = torch.cuda.Event(enable_timing=True)
        t1 = torch.cuda.Event(enable_timing=True)
        t0.record(s_in)
        for i in range(n):
            b = i % NB
            with torch.cuda.stream(s_in):
                if i >= NB:
                    s_in.wait_event(computed[b])         # step i-NB no longer reads Xe[b]
                Xe[b].copy_(hX, non_blocking=True)
                dYe[b].copy_(hdY, non_blocking=True)
                in_ready[b].record(s_in)
            stream.wait_event(in_ready[b])
            if i >= NB:
                stream.wait_event(copied_out[b])        # Ye[b], dX[b] of step i-NB copied out
            run_stack(Xe[b], dYe[b], Ye[b], ge[b]["dX"], st=stream)
            computed[b].record(stream)
            with torch.cuda.stream(s_out):
                s_out.wait_event(computed[b])
                hY[b].copy_(Ye[b], non_blocking=True)
                hdX[b].copy_(ge[b]["dX"], non_blocking=True)
                copied_out[b].record(s_out)
        s_out.wait_event(computed[(n - 1) % NB])
        t1.record(s_out)
        torch.cuda.synchronize(device)
        return t0.elapsed_time(t1)

    e_steps = max(4, args.steps // 2)
    e2e_pass(min(args.warmup, 4))      # untimed: first copies through the pinned buffers
    e2e_t0 = time.time()
    e2e_total = e2e_pass(e_steps)
    e2e_window = (e2e_t0, time.time())
    nvml.stop()
    clocks.stop(dev_window)
    clk = _clock_record(clocks, nvml, dev_window)
    clk_e2e = _clock_record(clocks, nvml, e2e_window)
    e2e_ms = _max_over_ranks(e2e_total / e_steps, ws, device)
    for l_ in stack:
        l_[0].check()

    # (after all timed work, so profiler launch counts of the timed steps are unaffected)
    # expert rows per layer: E x sum(k_g) under expert choice (the same every step, also
    # with per-step capacities, whose sum is fixed); the kept (token, expert) pairs under
    # token choice (read once from a forward with outputs)
    if tc:
        rows = []
        h = X
        for l_, wts, ybuf, g, _sh in stack:
            o = l_.forward(h, *wts, Y=ybuf[0], outputs=True)
            rows.append(int(o[4].cpu().numpy().sum()))
            h = ybuf[0]
    else:
        rows = [w.E * int(inp.k_g.sum())] * w.layers
    coverage = None
    if headline:
        # token coverage of the first layer: tokens no expert picked (expert choice) or
        # token-expert pairs dropped by the capacity (token choice)
        if tc:
            coverage = {"pairs_dropped_frac": round(1.0 - rows[0] / (w.N * args.tc_k), 6)}
        else:
            l0, wts0, ybuf0 = stack[0][0], stack[0][1], stack[0][2]
            if dyn:
                l0.set_capacity(inp.k_g)
            idx0 = l0.forward(X, *wts0, Y=ybuf0[0], outputs=True, shared=stack[0][4])[1]
            picked = np.zeros(w.N, dtype=bool)
            picked[idx0.cpu().numpy().ravel()] = True
            coverage = {"tokens_unpicked_frac": round(1.0 - float(picked.mean()), 6)}

    # ---- roofline of the dominant kernel (the tcgen05 grouped GEMM)
    hbm, bf16_burst, bf16_sust, peak_src = _peaks()
    per = {}
    for name, t in phases:
        per.setdefault(name, []).append(t)
    gemm = {k: v for k, v in per.items() if k.startswith("gemm_")}
    shared_ms = sum(sum(v) for k, v in per.items() if k.startswith("shared_")) / args.steps
    gemm_launches = sum(len(v) for v in gemm.values()) + len(per.get("gemm_wgrad", []))
    gemm_ms_step = sum(sum(v) for v in gemm.values()) / args.steps
    P = sum(rows) / len(rows)
    flops_step = 18.0 * sum(rows) * w.d * w.d_ff
    gemm_tflops = flops_step / (gemm_ms_step * 1e-3) / 1e12 if gemm_ms_step > 0 else None
    gemm_per_launch = flops_step / max(1, gemm_launches / args.steps)
    kms = {k: round(sum(v) / args.steps, 4) for k, v in per.items()}
    mem_bytes = {k: v for k, v in _mem_bytes(w, P, tc, shared=Fs > 0).items() if k in per}
    # from the rounded per-kernel times of the line, so the figure can be recomputed from it
    mem_ms = sum(kms[k] for k in mem_bytes)
    mem_gbs = (w.layers * sum(mem_bytes.values()) / (mem_ms * 1e-3) / 1e9 if mem_ms > 0
               else None)
    r = {
        "ms_per_step": round(ms_max, 4),
        "value": round(ws * w.N / (ms_max * 1e-3), 1),
        "e2e": {"value": round(ws * w.N / (e2e_ms * 1e-3), 1), "unit": UNIT,
                "h2d_bytes_per_step": int(X.numel() * X.element_size() * 2),
                "d2h_bytes_per_step": int(X.numel() * X.element_size() * 2),
                "ms_per_step": round(e2e_ms, 4), "steps": e_steps,
                "sm_mhz": clk_e2e.get("sm_mhz")},
        "gemm_tflops": gemm_tflops, "gemm_per_launch": gemm_per_launch,
        "expert_gemm_pct_bf16_peak": (None if gemm_tflops is None
                                      else round(100 * gemm_tflops / bf16_burst, 2)),
        "routing_hbm_gbs": None if mem_gbs is None else round(mem_gbs, 1),
        "routing_hbm_frac": None if mem_gbs is None else round(mem_gbs / hbm, 4),
        "routing_bytes_per_step": w.layers * sum(mem_bytes.values()),
        "routing_kernels": sorted(mem_bytes),
        "gpu_launches": int(launches),
        "kernel_ms_per_step": kms,
        "gemm_rooflines": _gemm_rooflines(w, P, kms, hbm, bf16_burst),
        "clocks": clk,
        "graph_ms": graph_ms, "coverage": coverage, "rows": rows, "tc_cap": tc_cap,
        "shared_ms": shared_ms, "Fs": Fs,
        "dynamic_capacity": bool(dyn),
    }
    for l_ in stack:
        l_[0].close()
    return r


def run_ours(args):
    import gc
    import torch
    ws, rank, local = _dist()
    if ws > 1:
        import torch.distributed as dist
        dist.init_process_group("nccl", init_method="env://")
    torch.cuda.set_device(local)
    device = torch.device("cuda", local)

    from paper_2604_01622_gb300 import build as B
    if rank == 0 or ws == 1:
        B.build()
    _barrier(ws)
    from paper_2604_01622_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    tc = args.routing == "tc"
    if args.seqs:
        w = I.scaled(w, G=args.seqs)
    res = measure(w, args, device, ws, local, headline=True)
    hbm, bf16_burst, bf16_sust, peak_src = _peaks()
    gemm_tflops = res["gemm_tflops"]
    src = os.path.join(ROOT, "paper_2604_01622_gb300", "csrc", "gemm_tc.cu")
    tr = TRAFFIC.get(_src_hash(src))
    roofline = {
        "kernel": "tc_gemm_kernel (tcgen05 grouped expert GEMMs: gate/up, down, dU, dH, dW)",
        "bound": "tensor", "achieved": round(gemm_tflops, 1),
        "peak": bf16_sust, "unit": "TFLOP/s", "frac": round(gemm_tflops / bf16_sust, 4),
        "peak_kind": f"bf16 sustained, {peak_src}",
        "frac_of_burst": round(gemm_tflops / bf16_burst, 4),
        "frac_of_nominal": round(gemm_tflops / NOMINAL["bf16_tflops"], 4),
        "flops_per_launch": res["gemm_per_launch"],
        "traffic": tr,
    }
    out = {
        "metric": METRIC_TC if tc else METRIC, "value": res["value"], "unit": UNIT, "n_gpus": ws,
        "steps": args.steps, "warmup": args.warmup, "ms_per_step": res["ms_per_step"],
        "higher_is_better": True, "scaling": "weak", "vs_baseline": None, "dtype": w.dtype,
        "data": "synthetic",
        "config": {"workload": w.name, "sequences": w.G, "seq_len": w.L, "tokens": w.N,
                   "d_model": w.d, "experts": w.E, "d_ff": w.d_ff, "k_per_seq": w.k_base,
                   "layers": w.layers, "shared_experts": args.shared_experts,
                   "tiles": args.tiles,
                   "parallelism": f"replicas{ws}" if ws > 1 else "single",
                   "l2": "inputs and activations larger than L2 (no flush)"},
    }
    if res["dynamic_capacity"]:
        out["config"]["capacity"] = ("per-sequence k_g redrawn every step from a device "
                                     "array (ec_ctx_set_capacity_async), sum fixed")
    if tc:
        out["config"].update(routing="token_choice", k=args.tc_k, capacity=res["tc_cap"],
                             capacity_factor=args.tc_cf, expert_rows=res["rows"])
    out["expert_gemm_pct_bf16_peak"] = res["expert_gemm_pct_bf16_peak"]
    out["routing_hbm_gbs"] = res["routing_hbm_gbs"]
    out["routing_hbm_frac"] = res["routing_hbm_frac"]
    out["routing_hbm_frac_of_nominal"] = (None if res["routing_hbm_gbs"] is None else
                                          round(res["routing_hbm_gbs"] / NOMINAL["hbm_gbs"], 4))
    out["routing_bytes_per_step"] = res["routing_bytes_per_step"]
    out["routing_kernels"] = res["routing_kernels"]
    out["nominal_peaks"] = NOMINAL
    out["e2e"] = res["e2e"]
    out["roofline"] = roofline
    if res["Fs"]:
        sh_flops = 18.0 * w.N * w.d * res["Fs"] * w.layers
        out["shared_experts"] = {"experts": args.shared_experts, "d_ff_each": args.shared_dff,
                                 "gemm_ms_per_step": round(res["shared_ms"], 4),
                                 "tflops": round(sh_flops / (res["shared_ms"] * 1e-3) / 1e12, 1)}
    out["graph"] = {"ms_per_step": round(res["graph_ms"], 4),
                    "value": round(ws * w.N / (res["graph_ms"] * 1e-3), 1), "unit": UNIT,
                    "note": "same step captured in one CUDA graph, replayed; no per-kernel events"}
    out["coverage"] = res["coverage"]
    out["gpu_launches"] = res["gpu_launches"]
    out["kernel_ms_per_step"] = res["kernel_ms_per_step"]
    out["gemm_rooflines"] = res["gemm_rooflines"]
    out["clocks"] = res["clocks"]
    # the other workloads, each in the same run (single GPU, default expert-choice line)
    extra = [] if (ws > 1 or tc or args.shared_experts or args.seqs
                   or args.workloads == "none") else \
        [n for n in (EXTRA_WORKLOADS if args.workloads == "all" else args.workloads.split(","))
         if n != w.name]
    if extra:
        out["workloads"] = {}
    for name in extra:
        del res
        gc.collect()
        torch.cuda.empty_cache()
        wx = I.WORKLOADS[name]
        res = measure(wx, args, device, ws, local, headline=False)
        gt = res["gemm_tflops"]
        out["workloads"][name] = {
            "config": {"sequences": wx.G, "seq_len": wx.L, "tokens": wx.N, "d_model": wx.d,
                       "experts": wx.E, "d_ff": wx.d_ff, "k_per_seq": wx.k_base,
                       "layers": wx.layers, "dtype": wx.dtype,
                       "capacity": ("per-sequence, redrawn every step (device array)"
                                    if res["dynamic_capacity"] else "fixed")},
            "ms_per_step": res["ms_per_step"], "tokens_per_s": res["value"],
            "e2e_tokens_per_s": res["e2e"]["value"], "e2e_ms_per_step": res["e2e"]["ms_per_step"],
            "expert_gemm_tflops": None if gt is None else round(gt, 1),
            "expert_gemm_frac_of_burst": None if gt is None else round(gt / bf16_burst, 4),
            "expert_gemm_frac_of_sustained": None if gt is None else round(gt / bf16_sust, 4),
            "routing_hbm_gbs": res["routing_hbm_gbs"], "routing_hbm_frac": res["routing_hbm_frac"],
            "gpu_launches": res["gpu_launches"],
            "kernel_ms_per_step": res["kernel_ms_per_step"],
            "gemm_rooflines": res["gemm_rooflines"],
            "clocks": res["clocks"],
        }
    if rank == 0 and not args.no_cpu_baseline:
        smp = (TCOracleSample(args.tc_cpu_tokens, w, args.tc_k, args.tc_cf) if tc
               else OracleSample(args.cpu_tokens, w, args.shared_experts, args.shared_dff))
        n, total, t_end = 0, 0.0, time.perf_counter() + args.cpu_seconds
        while n == 0 or time.perf_counter() < t_end:
            total += smp.run()[1]
            n += 1
        total *= getattr(smp, "layers", 1)   # one of the stack's equal layers was timed
        out["cpu_baseline"] = {"value": round(n * smp.tokens / total, 2), "unit": UNIT,
                               "cores": _cores(), "kind": "oracle",
                               "sample": f"{smp.desc}, run {n} time(s)",
                               "seconds": round(total, 2)}
    if rank == 0:
        print(json.dumps(out), flush=True)
    if ws > 1:
        import torch.distributed as dist
        dist.destroy_process_group()


# ------------------------------------------------------------------ reference arm (oracle)
def run_reference(args):
    ws, rank, local = _dist()
    if rank != 0:
        return
    from paper_2604_01622_gb300 import inputs as I
    w = I.WORKLOADS[args.workload]
    tc = args.routing == "tc"
    smp = (TCOracleSample(args.tc_cpu_tokens, w, args.tc_k, args.tc_cf) if tc
           else OracleSample(args.cpu_tokens, w, args.shared_experts, args.shared_dff))
    for _ in range(args.warmup):
        smp.run()
    total_t = 0.0
    for _ in range(args.steps):
        total_t += smp.run()[1]
    desc = smp.desc
    total_t *= getattr(smp, "layers", 1)   # one of the stack's equal layers was timed
    v = args.steps * smp.tokens / total_t
    out = {"impl": "reference", "metric": METRIC_TC if tc else METRIC, "value": round(v, 2),
           "unit": UNIT,
           "n_gpus": 1, "steps": args.steps, "warmup": args.warmup,
           "ms_per_step": round(1e3 * total_t / args.steps, 2), "higher_is_better": True,
           "scaling": "weak", "vs_baseline": None, "dtype": "f64", "data": "synthetic",
           "config": {"workload": w.name, "sequences": w.G, "seq_len": w.L, "tokens": w.N,
                      "d_model": w.d, "experts": w.E, "d_ff": w.d_ff, "k_per_seq": w.k_base,
                      "layers": w.layers, "shared_experts": args.shared_experts,
                      "parallelism": "host cores",
                      **({"routing": "token_choice", "k": args.tc_k,
                          "capacity_factor": args.tc_cf} if tc else {})},
           "cpu_baseline": {"value": round(v, 2), "unit": UNIT, "cores": _cores(),
                            "kind": "oracle", "sample": desc + " per step"},
           "e2e": {"value": round(v, 2), "unit": UNIT, "h2d_bytes_per_step": 0,
                   "d2h_bytes_per_step": 0}}
    print(json.dumps(out), flush=True)


def main():
    ap = argparse.ArgumentParser(description=__doc__.split("\n")[0])
    ap.add_argument("--gpus", type=int, default=1)
    ap.add_argument("--steps", type=int, default=50)
    ap.add_argument("--warmup", type=int, default=5)
    ap.add_argument("--impl", choices=["ours", "reference"], default="ours")
    ap.add_argument("--workload", default="ec_d2048_e64")
    ap.add_argument("--seqs", type=int, default=0,
                    help="run only this many sequences of the workload (small profiling cases)")
    ap.add_argument("--shared-experts", type=int, default=0,
                    help="add this many shared SwiGLU experts per layer (the paper's block has 2)")
    ap.add_argument("--shared-dff", type=int, default=1024, help="width of each shared expert")
    ap.add_argument("--routing", choices=["ec", "tc"], default="ec",
                    help="expert choice (the paper's method) or token choice (its baseline)")
    ap.add_argument("--tc-k", type=int, default=8, help="experts per token under --routing tc")
    ap.add_argument("--tc-cf", type=float, default=None,
                    help="token-choice capacity factor (default: dropless)")
    ap.add_argument("--tc-cpu-tokens", type=int, default=32,
                    help="tokens of the token-choice oracle's CPU sample (both arms)")
    ap.add_argument("--tiles", choices=sorted(TILE_POLICY), default="auto",
                    help="expert-GEMM tile policy (bf16 path): auto, 256 or 512 columns")
    ap.add_argument("--no-cpu-baseline", action="store_true")
    ap.add_argument("--cpu-tokens", type=int, default=4096,
                    help="tokens of the oracle's sample (whole sequences of the workload): the "
                         "cpu_baseline leg and every step of the reference arm")
    ap.add_argument("--cpu-seconds", type=float, default=10.0,
                    help="the cpu_baseline leg repeats its sample for at least this long")
    ap.add_argument("--workloads", default="all",
                    help="other workloads timed in the same run: all, none, or a comma list")
    ap.add_argument("--static-capacity", action="store_true",
                    help="timestep workloads keep their first capacities every step")
    args = ap.parse_args()
    if args.warmup < 3 and args.impl == "ours":
        ap.error("--warmup must be at least 3")
    if args.impl == "reference":
        run_reference(args)
    else:
        run_ours(args)


if __name__ == "__main__":
    main()
