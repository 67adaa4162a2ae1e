"""Torch-facing wrapper of one EC-MoE layer context (argument marshalling only).

PyTorch supplies device memory and the current stream; every step of the layer runs in
libecmoe.so. Tensor layouts are those of include/ecmoe.h.
"""
from __future__ import annotations

import torch

from . import (EC_BF16, EC_F32, ec_check_device, ec_ctx_create, ec_ctx_destroy,
               ec_ctx_profile, ec_ctx_set_capacity, ec_ctx_set_profiling, ec_ctx_set_residual,
               ec_ctx_set_tiles,
               ec_ctx_set_shared, ec_ctx_set_workspace, ec_kernel_launches,
               ec_moe_backward, ec_moe_backward_shared, ec_moe_forward, ec_moe_forward_shared,
               ec_ctx_set_capacity_async, ec_route, ec_rows_per_expert, ec_tc_backward,
               ec_tc_capacity, ec_tc_ctx_create, ec_tc_forward, ec_workspace_bytes)

_DT = {"f32": (EC_F32, torch.float32), "bf16": (EC_BF16, torch.bfloat16)}


def _p(t):
    return None if t is None else t.data_ptr()


def _stream(stream):
    return (stream or torch.cuda.current_stream()).cuda_stream


class ECMoELayer:
    """One layer shape: N tokens in groups `group_off`, E experts, capacities k_g."""

    def __init__(self, N, d, E, d_ff, group_off, k_g, dtype="bf16", device="cuda",
                 d_ff_shared=0):
        self.N, self.d, self.E, self.d_ff = int(N), int(d), int(E), int(d_ff)
        self.G = len(group_off) - 1
        self.code, self.tdtype = _DT[dtype]
        self.device = torch.device(device)
        self.d_ff_shared = int(d_ff_shared)
        self.ctx = ec_ctx_create(self.N, self.d, self.E, self.d_ff, self.G, group_off, k_g,
                                 self.code)
        if self.d_ff_shared:
            ec_ctx_set_shared(self.ctx, self.d_ff_shared)
        self.ws_bytes = ec_workspace_bytes(self.ctx)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=self.device)
        ec_ctx_set_workspace(self.ctx, self.ws.data_ptr(), self.ws_bytes)

    @property
    def M(self) -> int:
        return ec_rows_per_expert(self.ctx)

    def set_capacity(self, k_g):
        ec_ctx_set_capacity(self.ctx, k_g)

    def set_capacity_async(self, k_g_dev, stream=None):
        """k_g from an int32 device tensor [G] in stream order (sum must keep M)."""
        ec_ctx_set_capacity_async(self.ctx, k_g_dev.data_ptr(), _stream(stream))

    def set_residual(self, on: bool):
        """Y = X + EC(X) and dX = dY + EC input gradient (stacked layers)."""
        ec_ctx_set_residual(self.ctx, on)

    def set_tiles(self, policy: int):
        """Expert-GEMM tile policy: EC_TILES_AUTO, EC_TILES_256 or EC_TILES_512."""
        ec_ctx_set_tiles(self.ctx, policy)

    def _empty(self, *shape, dtype=None):
        return torch.empty(*shape, dtype=dtype or self.tdtype, device=self.device)

    def route(self, X=None, Wr=None, br=None, S_in=None, stream=None):
        """Selection only. Returns (idx [E][M] int32, gate [E][M] f32, S [E][N] f32)."""
        idx = self._empty(self.E, self.M, dtype=torch.int32)
        gate = self._empty(self.E, self.M, dtype=torch.float32)
        S = self._empty(self.E, self.N, dtype=torch.float32)
        ec_route(self.ctx, _p(X), _p(Wr), _p(br), _p(S_in), _p(S), _p(idx), _p(gate),
                 _stream(stream))
        return idx, gate, S

    def forward(self, X, Wr, br, Wg, Wu, Wd, Y=None, stream=None, outputs=True, shared=None):
        """Y = EC-MoE(X) (+ shared experts). Returns (Y, idx, gate, S); idx/gate/S are None if
        outputs=False. shared = (Wg_s, Wu_s, Wd_s) in concatenated form when configured."""
        Y = self._empty(self.N, self.d) if Y is None else Y
        idx = gate = S = None
        if outputs:
            idx = self._empty(self.E, self.M, dtype=torch.int32)
            gate = self._empty(self.E, self.M, dtype=torch.float32)
            S = self._empty(self.E, self.N, dtype=torch.float32)
        if self.d_ff_shared:
            Wgs, Wus, Wds = shared
            ec_moe_forward_shared(self.ctx, _p(X), _p(Wr), _p(br), _p(Wg), _p(Wu), _p(Wd),
                                  _p(Wgs), _p(Wus), _p(Wds), _p(Y), _p(idx), _p(gate), _p(S),
                                  _stream(stream))
        else:
            ec_moe_forward(self.ctx, _p(X), _p(Wr), _p(br), _p(Wg), _p(Wu), _p(Wd), _p(Y),
                           _p(idx), _p(gate), _p(S), _stream(stream))
        # the backward pass reads these through the pointers the context remembered
        self._keep = (X, Wr, br, Wg, Wu, Wd, shared)
        return Y, idx, gate, S

    def backward(self, dY, grads=None, stream=None, with_bias=False):
        """Gradients of <dY, Y> for the last forward. Returns a dict of tensors."""
        g = grads or {
            "dX": self._empty(self.N, self.d),
            "dWr": self._empty(self.d, self.E, dtype=torch.float32),
            "dbr": self._empty(self.E, dtype=torch.float32) if with_bias else None,
            "dWg": self._empty(self.E, self.d, self.d_ff, dtype=torch.float32),
            "dWu": self._empty(self.E, self.d, self.d_ff, dtype=torch.float32),
            "dWd": self._empty(self.E, self.d_ff, self.d, dtype=torch.float32),
        }
        if self.d_ff_shared:
            for k, shape in (("dWg_s", (self.d, self.d_ff_shared)),
                             ("dWu_s", (self.d, self.d_ff_shared)),
                             ("dWd_s", (self.d_ff_shared, self.d))):
                if g.get(k) is None:
                    g[k] = self._empty(*shape, dtype=torch.float32)
            ec_moe_backward_shared(self.ctx, _p(dY), _p(g["dX"]), _p(g["dWr"]), _p(g.get("dbr")),
                                   _p(g["dWg"]), _p(g["dWu"]), _p(g["dWd"]), _p(g["dWg_s"]),
                                   _p(g["dWu_s"]), _p(g["dWd_s"]), _stream(stream))
        else:
            ec_moe_backward(self.ctx, _p(dY), _p(g["dX"]), _p(g["dWr"]), _p(g.get("dbr")),
                            _p(g["dWg"]), _p(g["dWu"]), _p(g["dWd"]), _stream(stream))
        return g

    def set_profiling(self, on: bool):
        ec_ctx_set_profiling(self.ctx, on)

    def profile(self):
        """[(kernel, ms)] of every launch since profiling was switched on."""
        return ec_ctx_profile(self.ctx)

    @property
    def launches(self) -> int:
        return ec_kernel_launches(self.ctx)

    def check(self, stream=None):
        """Synchronise and raise if a kernel reported a device-side timeout."""
        ec_check_device(self.ctx, _stream(stream))

    def close(self):
        if self.ctx is not None:
            ec_ctx_destroy(self.ctx)
            self.ctx = None

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


def tc_capacity(cf, k, N, E) -> int:
    """Token-choice expert capacity for a capacity factor (computed by the library's
    ec_tc_capacity); -1 (no cap, dropless) when cf is None or <= 0."""
    return ec_tc_capacity(cf, k, N, E)


class TCMoELayer(ECMoELayer):
    """Token-choice layer of the same shape (bf16): every token takes its k best experts,
    each expert keeps at most `capacity` tokens (-1: dropless)."""

    def __init__(self, N, d, E, d_ff, k, capacity=-1, dtype="bf16", device="cuda"):
        self.N, self.d, self.E, self.d_ff = int(N), int(d), int(E), int(d_ff)
        self.k, self.capacity = int(k), int(capacity)
        self.G = 1
        self.code, self.tdtype = _DT[dtype]
        self.device = torch.device(device)
        self.d_ff_shared = 0
        self.ctx = None
        self.ctx = ec_tc_ctx_create(self.N, self.d, self.E, self.d_ff, self.k, self.capacity,
                                    self.code)
        self.ws_bytes = ec_workspace_bytes(self.ctx)
        self.ws = torch.empty(self.ws_bytes, dtype=torch.uint8, device=self.device)
        ec_ctx_set_workspace(self.ctx, self.ws.data_ptr(), self.ws_bytes)

    def route(self, *a, **kw):
        raise NotImplementedError("token choice routes inside forward()")

    def forward(self, X, Wr, br, Wg, Wu, Wd, Y=None, stream=None, outputs=True, shared=None):
        """Y = TC-MoE(X). Returns (Y, choice [N][k], gate [N][k], kept [N][k], load [E],
        S [N][E]); all but Y are None if outputs=False."""
        if shared is not None:
            raise ValueError("token-choice layers have no shared experts")
        Y = self._empty(self.N, self.d) if Y is None else Y
        outs = [None] * 5
        if outputs:
            outs = [self._empty(self.N, self.k, dtype=torch.int32),
                    self._empty(self.N, self.k, dtype=torch.float32),
                    self._empty(self.N, self.k, dtype=torch.int32),
                    self._empty(self.E, dtype=torch.int32),
                    self._empty(self.N, self.E, dtype=torch.float32)]
        ec_tc_forward(self.ctx, _p(X), _p(Wr), _p(br), _p(Wg), _p(Wu), _p(Wd), _p(Y),
                      *[_p(t) for t in outs], _stream(stream))
        self._keep = (X, Wr, br, Wg, Wu, Wd)
        return (Y, *outs)

    def backward(self, dY, grads=None, stream=None, with_bias=False):
        g = grads or {
            "dX": self._empty(self.N, self.d),
            "dWr": self._empty(self.d, self.E, dtype=torch.float32),
            "dbr": self._empty(self.E, dtype=torch.float32) if with_bias else None,
            "dWg": self._empty(self.E, self.d, self.d_ff, dtype=torch.float32),
            "dWu": self._empty(self.E, self.d, self.d_ff, dtype=torch.float32),
            "dWd": self._empty(self.E, self.d_ff, self.d, dtype=torch.float32),
        }
        ec_tc_backward(self.ctx, _p(dY), _p(g["dX"]), _p(g["dWr"]), _p(g.get("dbr")),
                       _p(g["dWg"]), _p(g["dWu"]), _p(g["dWd"]), _stream(stream))
        return g
