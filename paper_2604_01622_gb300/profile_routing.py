"""Routing kernels alone on a workload's token shape, for profilers.

`--phase router` runs `ec_route` (router GEMM + softmax, then the top-k) on the workload's
tokens and router weights with a capacity of 8 per sequence, so the context's workspace
stays small (under 300 MB for the bench workload, whose X of 134 MB is still larger than
the 129 MB L2); the router kernel's work does not depend on the capacity.
`--phase topk` computes the scores that way once, then selects with the workload's own
capacities from those scores (`ec_route` with S_in) on a context of the same tokens, experts
and groups but d_model = d_ff = 64, so the top-k kernel sees the real scores and shapes
while the workspace stays small. A handful of launches of each, so a profiler capture of
one of them ends within seconds.

  python -m paper_2604_01622_gb300.profile_routing [--workload NAME] [--phase router|topk]
                                                   [--calls N]
"""
from __future__ import annotations

import argparse

import numpy as np
import torch

from . import inputs as I
from .layer import ECMoELayer


def main():
    ap = argparse.ArgumentParser()
    ap.add_argument("--workload", default="ec_d2048_e64")
    ap.add_argument("--phase", choices=["router", "topk"], default="router")
    ap.add_argument("--calls", type=int, default=4)
    a = ap.parse_args()
    w = I.scaled(I.WORKLOADS[a.workload], layers=1)
    inp = I.make_inputs(w)
    L = inp.layers[0]

    def dev(t):
        return torch.from_numpy(t.data.view(np.int16)).cuda().view(torch.bfloat16)

    small_k = np.minimum(np.diff(inp.group_off), 8).astype(np.int32)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, small_k, dtype=w.dtype)
    X, Wr = dev(inp.X), dev(L.Wr)
    br = None if L.br is None else torch.from_numpy(L.br).cuda()
    if a.phase == "router":
        for _ in range(a.calls):
            lay.route(X, Wr, br)
        lay.check()
        mb = lay.ws_bytes // 2**20
    else:
        _, _, S = lay.route(X, Wr, br)
        lay.check()
        sel = ECMoELayer(w.N, 64, w.E, 64, inp.group_off, inp.k_g, dtype="f32")
        for _ in range(a.calls):
            sel.route(S_in=S)
        sel.check()
        mb = (lay.ws_bytes + sel.ws_bytes) // 2**20
    print(f"{a.phase}: {a.calls} calls on {w.name} (workspace {mb} MB)")


if __name__ == "__main__":
    main()
