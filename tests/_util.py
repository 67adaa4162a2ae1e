"""Helpers shared by the GPU parity tests: tensor transfer, error norms, layer runs."""
from __future__ import annotations

import numpy as np
import torch

from paper_2604_01622_gb300 import inputs as I


def relmax(a, b) -> float:
    """Relative max-norm error ||a - b||_inf / max(||b||_inf, tiny)."""
    a = np.asarray(a, np.float64)
    b = np.asarray(b, np.float64)
    if a.size == 0:
        return 0.0
    return float(np.max(np.abs(a - b)) / max(np.max(np.abs(b)), 1e-30))


def dev(t: I.Tensor, device="cuda"):
    """Input tensor in its storage type on the device (bf16 bits reinterpret exactly)."""
    if t.dtype == "bf16":
        return torch.from_numpy(t.data.view(np.int16)).to(device).view(torch.bfloat16)
    return torch.from_numpy(np.ascontiguousarray(t.data)).to(device)


def host(x) -> np.ndarray:
    """Device tensor -> float64 numpy (bf16 values are exact in float64)."""
    return x.detach().to(torch.float64).cpu().numpy()


def tol(w: I.Workload) -> float:
    """Parity bound: 1e-4 on the fp32 path, 2e-2 on the bf16 path (relative max-norm)."""
    return 1e-4 if w.dtype == "f32" else 2e-2


def gpu_layer(inp: I.Inputs, layer: int = 0, X=None, dY=None, backward=True, tiles=None):
    """Run one layer on the GPU through the C ABI; returns (layer, outputs dict of tensors).
    `tiles`: an expert-GEMM tile policy (EC_TILES_*), else the library's choice."""
    from paper_2604_01622_gb300.layer import ECMoELayer
    w = inp.w
    L = inp.layers[layer]
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype=w.dtype)
    if tiles is not None:
        lay.set_tiles(tiles)
    Xd = dev(inp.X) if X is None else X
    br = None if L.br is None else torch.from_numpy(L.br).cuda()
    Y, idx, gate, S = lay.forward(Xd, dev(L.Wr), br, dev(L.Wg), dev(L.Wu), dev(L.Wd))
    out = {"Y": Y, "idx": idx, "gate": gate, "S": S}
    if backward:
        g = lay.backward(dev(inp.dY) if dY is None else dY, with_bias=L.br is not None)
        out.update(g)
    lay.check()
    return lay, out
