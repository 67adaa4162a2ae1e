"""Out-of-bounds write check (stands in for a memory sanitizer, which is not available here).

The workspace and every output buffer of a call are placed between 64 KB guard regions
filled with a byte pattern; after forward and backward the guards must be untouched and the
outputs finite. Shapes are ragged (group sizes, expert counts, token counts that are not
multiples of any tile), where an indexing slip would land outside a buffer.
"""
import numpy as np
import pytest
import torch

import paper_2604_01622_gb300 as ec
from paper_2604_01622_gb300 import inputs as I
from tests._util import dev

pytestmark = pytest.mark.gpu

G = 1 << 16
PAT = 0xA5


class Guarded:
    def __init__(self, shape, dtype):
        n = int(np.prod(shape)) * torch.empty((), dtype=dtype).element_size()
        self.n = n
        self.raw = torch.full((n + 2 * G,), PAT, dtype=torch.uint8, device="cuda")
        self.t = self.raw[G:G + n].view(dtype).view(*shape) if n else torch.empty(
            shape, dtype=dtype, device="cuda")

    def intact(self):
        return bool((self.raw[:G] == PAT).all()) and bool((self.raw[G + self.n:] == PAT).all())

    @property
    def ptr(self):
        return self.t.data_ptr() if self.n else None


def _guard_workspace(lay):
    ws = Guarded((lay.ws_bytes,), torch.uint8)
    ec.ec_ctx_set_workspace(lay.ctx, ws.ptr, lay.ws_bytes)
    lay.ws = ws.raw   # keep it alive with the layer
    return ws


def _grads(w, dt):
    return {"dX": Guarded((w.N, w.d), dt), "dWr": Guarded((w.d, w.E), torch.float32),
            "dbr": Guarded((w.E,), torch.float32),
            "dWg": Guarded((w.E, w.d, w.d_ff), torch.float32),
            "dWu": Guarded((w.E, w.d, w.d_ff), torch.float32),
            "dWd": Guarded((w.E, w.d_ff, w.d), torch.float32)}


def _check(bufs):
    for name, b in bufs.items():
        assert b.intact(), f"write outside {name}"
        if b.t.is_floating_point():
            assert torch.isfinite(b.t.float()).all(), name


# (dtype, d, d_ff, tile policy): fp32 SIMT path; bf16 with 256-column tiles (d = 192 leaves a
# ragged column tile); bf16 with 256 x 512 tiles (d and 2 d_ff multiples of 512)
EC_SHAPES = [("f32", 68, 36, 0), ("bf16", 192, 128, 1), ("bf16", 512, 256, 2)]


@pytest.mark.parametrize("dtype,d,d_ff,tiles", EC_SHAPES, ids=["f32", "bf16", "bf16_wide"])
def test_expert_choice_writes_stay_inside_buffers(dtype, d, d_ff, tiles):
    from paper_2604_01622_gb300.layer import ECMoELayer
    base = I.WORKLOADS["tiny_f32"] if dtype == "f32" else I.WORKLOADS["ec_d2048_e64"]
    w = I.scaled(base, G=3, L=200, d=d, E=12, d_ff=d_ff, k_base=40, router_bias=True, layers=1)
    inp = I.make_inputs(w)
    group_off = np.array([0, 137, 137 + 263, 600], np.int32)   # ragged, N = 600
    k_g = np.array([40, 0, 70], np.int32)
    L = inp.layers[0]
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, group_off, k_g, dtype=dtype)
    lay.set_tiles(tiles)
    ws = _guard_workspace(lay)
    dt = lay.tdtype
    M = lay.M
    out = {"Y": Guarded((w.N, w.d), dt), "idx": Guarded((w.E, M), torch.int32),
           "gate": Guarded((w.E, M), torch.float32), "S": Guarded((w.E, w.N), torch.float32)}
    X, Wr, Wg, Wu, Wd = dev(inp.X), dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd)
    br = torch.from_numpy(L.br).cuda()
    s = torch.cuda.current_stream().cuda_stream
    ec.ec_moe_forward(lay.ctx, X.data_ptr(), Wr.data_ptr(), br.data_ptr(), Wg.data_ptr(),
                      Wu.data_ptr(), Wd.data_ptr(), out["Y"].ptr, out["idx"].ptr,
                      out["gate"].ptr, out["S"].ptr, s)
    g = _grads(w, dt)
    dY = dev(inp.dY)
    ec.ec_moe_backward(lay.ctx, dY.data_ptr(), g["dX"].ptr, g["dWr"].ptr, g["dbr"].ptr,
                       g["dWg"].ptr, g["dWu"].ptr, g["dWd"].ptr, s)
    lay.check()
    _check({"workspace": ws, **out, **g})
    lay.close()


@pytest.mark.parametrize("d,d_ff,tiles", [(128, 192, 1), (512, 256, 2)], ids=["narrow", "wide"])
def test_token_choice_writes_stay_inside_buffers(d, d_ff, tiles):
    from paper_2604_01622_gb300.layer import TCMoELayer
    w = I.Workload("guard_tc", G=1, L=700, d=d, E=12, d_ff=d_ff, k_base=0, dtype="bf16",
                   seed=21, router_bias=True)
    inp = I.make_inputs(w)
    L = inp.layers[0]
    k, cap = 3, 150
    lay = TCMoELayer(w.N, w.d, w.E, w.d_ff, k, cap)
    lay.set_tiles(tiles)
    ws = _guard_workspace(lay)
    out = {"Y": Guarded((w.N, w.d), torch.bfloat16), "choice": Guarded((w.N, k), torch.int32),
           "gate": Guarded((w.N, k), torch.float32), "kept": Guarded((w.N, k), torch.int32),
           "load": Guarded((w.E,), torch.int32), "S": Guarded((w.N, w.E), torch.float32)}
    X, Wr, Wg, Wu, Wd = dev(inp.X), dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd)
    br = torch.from_numpy(L.br).cuda()
    s = torch.cuda.current_stream().cuda_stream
    ec.ec_tc_forward(lay.ctx, X.data_ptr(), Wr.data_ptr(), br.data_ptr(), Wg.data_ptr(),
                     Wu.data_ptr(), Wd.data_ptr(), out["Y"].ptr, out["choice"].ptr,
                     out["gate"].ptr, out["kept"].ptr, out["load"].ptr, out["S"].ptr, s)
    g = _grads(w, torch.bfloat16)
    dY = dev(inp.dY)
    ec.ec_tc_backward(lay.ctx, dY.data_ptr(), g["dX"].ptr, g["dWr"].ptr, g["dbr"].ptr,
                      g["dWg"].ptr, g["dWu"].ptr, g["dWd"].ptr, s)
    lay.check()
    _check({"workspace": ws, **out, **g})
    assert int(out["load"].t.max()) <= cap
    lay.close()


def test_shared_experts_writes_stay_inside_buffers():
    """Shared experts over 2048 tokens: their FFN buffers and the two split-K halves of their
    dWd (summed afterwards) stay inside the workspace; the shared gradients inside theirs."""
    from paper_2604_01622_gb300.layer import ECMoELayer
    w = I.scaled(I.WORKLOADS["ec_d2048_e64"], G=2, L=1024, d=512, E=6, d_ff=256, k_base=96,
                 router_bias=True, layers=1)
    n_sh, f_sh = 2, 256
    inp = I.make_inputs(w)
    L = inp.layers[0]
    sh = I.make_shared(w, 0, n_sh, f_sh)
    lay = ECMoELayer(w.N, w.d, w.E, w.d_ff, inp.group_off, inp.k_g, dtype="bf16",
                     d_ff_shared=n_sh * f_sh)
    ws = _guard_workspace(lay)
    M, Fs = lay.M, n_sh * f_sh
    out = {"Y": Guarded((w.N, w.d), torch.bfloat16), "idx": Guarded((w.E, M), torch.int32),
           "gate": Guarded((w.E, M), torch.float32), "S": Guarded((w.E, w.N), torch.float32)}
    X, Wr, Wg, Wu, Wd = dev(inp.X), dev(L.Wr), dev(L.Wg), dev(L.Wu), dev(L.Wd)
    Wgs, Wus, Wds = dev(sh.Wg), dev(sh.Wu), dev(sh.Wd)
    br = torch.from_numpy(L.br).cuda()
    s = torch.cuda.current_stream().cuda_stream
    ec.ec_moe_forward_shared(lay.ctx, X.data_ptr(), Wr.data_ptr(), br.data_ptr(), Wg.data_ptr(),
                             Wu.data_ptr(), Wd.data_ptr(), Wgs.data_ptr(), Wus.data_ptr(),
                             Wds.data_ptr(), out["Y"].ptr, out["idx"].ptr, out["gate"].ptr,
                             out["S"].ptr, s)
    g = _grads(w, torch.bfloat16)
    g.update({"dWg_s": Guarded((w.d, Fs), torch.float32), "dWu_s": Guarded((w.d, Fs), torch.float32),
              "dWd_s": Guarded((Fs, w.d), torch.float32)})
    dY = dev(inp.dY)
    ec.ec_moe_backward_shared(lay.ctx, dY.data_ptr(), g["dX"].ptr, g["dWr"].ptr, g["dbr"].ptr,
                              g["dWg"].ptr, g["dWu"].ptr, g["dWd"].ptr, g["dWg_s"].ptr,
                              g["dWu_s"].ptr, g["dWd_s"].ptr, s)
    lay.check()
    _check({"workspace": ws, **out, **g})
    lay.close()
