"""GB300-native expert-choice (EC) MoE layer, forward and backward (arXiv 2604.01622).

Thin ctypes binding of the C ABI in include/ecmoe.h: every function here has the name of
the C entry point it calls and only marshals arguments (device pointers as Python ints,
a CUDA stream handle, host int32 arrays). All compute runs in libecmoe.so's CUDA kernels;
there is no fallback. `ECMoELayer` (layer.py) wraps a context with torch-allocated
buffers for convenience.
"""
from __future__ import annotations

import ctypes
import os

import numpy as np

_PKG = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(_PKG, "libecmoe.so")

EC_OK, EC_ERR_INVALID_ARG, EC_ERR_SHAPE, EC_ERR_UNSUPPORTED = 0, 1, 2, 3
EC_ERR_CUDA, EC_ERR_TIMEOUT, EC_ERR_WORKSPACE, EC_ERR_STATE = 4, 5, 6, 7
EC_F32, EC_BF16 = 0, 1

# C entry points declared in include/ecmoe.h
EXPORTS = (
    "ec_ctx_create", "ec_ctx_destroy", "ec_ctx_set_capacity", "ec_rows_per_expert",
    "ec_workspace_bytes", "ec_ctx_set_workspace", "ec_route", "ec_moe_forward",
    "ec_moe_backward", "ec_check_device", "ec_last_error", "ec_status_string",
    "ec_ctx_set_profiling", "ec_ctx_profile", "ec_kernel_launches", "ec_select_static",
    "ec_selftest_bounded_wait", "ec_ctx_set_residual", "ec_capacity_schedule",
    "ec_ctx_set_shared", "ec_moe_forward_shared", "ec_moe_backward_shared",
    "ec_tc_ctx_create", "ec_tc_forward", "ec_tc_backward", "ec_ctx_set_tiles",
    "ec_ctx_set_capacity_async", "ec_get_last_error", "ec_tc_capacity",
)
EC_TILES_AUTO, EC_TILES_256, EC_TILES_512 = 0, 1, 2

EC_SCHEDULERS = {"static": 0, "linear": 1, "linear_reverse": 2, "cosine": 3,
                 "cosine_reverse": 4, "gaussian": 5, "gaussian_reverse": 6}

_lib = None


class ECError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{status_string(status)}: {msg}")
        self.status = status


def load():
    """Load libecmoe.so (built by build.py). Raises if it is missing: there is no fallback."""
    global _lib
    if _lib is not None:
        return _lib
    if not os.path.exists(LIB_PATH):
        raise RuntimeError(f"{LIB_PATH} is missing: run paper_2604_01622_gb300.build.build() "
                           "(the EC-MoE layer has no non-CUDA implementation)")
    lib = ctypes.CDLL(LIB_PATH)
    vp, i32, i64, sz = ctypes.c_void_p, ctypes.c_int32, ctypes.c_int64, ctypes.c_size_t
    P32 = ctypes.POINTER(ctypes.c_int32)
    sig = {
        "ec_ctx_create": (i32, [ctypes.POINTER(vp), i32, i32, i32, i32, i32, P32, P32, i32]),
        "ec_ctx_destroy": (None, [vp]),
        "ec_ctx_set_capacity": (i32, [vp, P32]),
        "ec_ctx_set_capacity_async": (i32, [vp, vp, vp]),
        "ec_get_last_error": (i32, [vp, ctypes.c_char_p, sz]),
        "ec_tc_capacity": (i64, [ctypes.c_double, i32, i32, i32]),
        "ec_rows_per_expert": (i64, [vp]),
        "ec_workspace_bytes": (sz, [vp]),
        "ec_ctx_set_workspace": (i32, [vp, vp, sz]),
        "ec_route": (i32, [vp, vp, vp, vp, vp, vp, vp, vp, vp]),
        "ec_moe_forward": (i32, [vp] * 12),
        "ec_moe_backward": (i32, [vp] * 9),
        "ec_check_device": (i32, [vp, vp]),
        "ec_last_error": (ctypes.c_char_p, [vp]),
        "ec_status_string": (ctypes.c_char_p, [i32]),
        "ec_ctx_set_profiling": (i32, [vp, i32]),
        "ec_ctx_profile": (i32, [vp, ctypes.POINTER(ctypes.c_char_p),
                                 ctypes.POINTER(ctypes.c_float), i32]),
        "ec_kernel_launches": (i64, [vp]),
        "ec_select_static": (i32, [vp, i32, i32, i32, P32, P32, vp, vp, vp]),
        "ec_selftest_bounded_wait": (i32, [vp, ctypes.c_uint64, vp]),
        "ec_ctx_set_residual": (i32, [vp, i32]),
        "ec_ctx_set_tiles": (i32, [vp, i32]),
        "ec_ctx_set_shared": (i32, [vp, i32]),
        "ec_moe_forward_shared": (i32, [vp] * 15),
        "ec_moe_backward_shared": (i32, [vp] * 12),
        "ec_tc_ctx_create": (i32, [ctypes.POINTER(vp), i32, i32, i32, i32, i32, i32, i32]),
        "ec_tc_forward": (i32, [vp] * 14),
        "ec_tc_backward": (i32, [vp] * 9),
        "ec_capacity_schedule": (i32, [i32, ctypes.c_double, ctypes.c_double, ctypes.c_double,
                                       i32, i32, P32, ctypes.POINTER(ctypes.c_double), P32]),
    }
    for name, (res, args) in sig.items():
        fn = getattr(lib, name)
        fn.restype = res
        fn.argtypes = args
    _lib = lib
    return lib


def status_string(status: int) -> str:
    return load().ec_status_string(int(status)).decode()


def _check(ctx, status: int):
    if status != EC_OK:
        msg = load().ec_last_error(ctx).decode() if ctx else ""
        raise ECError(status, msg)


def _i32(a):
    arr = np.ascontiguousarray(np.asarray(a, dtype=np.int32))
    return arr, arr.ctypes.data_as(ctypes.POINTER(ctypes.c_int32))


def ec_ctx_create(N, d, E, d_ff, G, group_off, k_g, dtype):
    lib = load()
    ctx = ctypes.c_void_p()
    g_arr, g_ptr = _i32(group_off)
    k_arr, k_ptr = _i32(k_g)
    st = lib.ec_ctx_create(ctypes.byref(ctx), N, d, E, d_ff, G, g_ptr, k_ptr, dtype)
    if st != EC_OK:
        raise ECError(st, "ec_ctx_create rejected the sizes")
    return ctx


def ec_ctx_destroy(ctx):
    load().ec_ctx_destroy(ctx)


def ec_ctx_set_capacity(ctx, k_g):
    k_arr, k_ptr = _i32(k_g)
    _check(ctx, load().ec_ctx_set_capacity(ctx, k_ptr))


def ec_ctx_set_capacity_async(ctx, k_g_dev: int, stream):
    """k_g from a device array (int32 [G]) on `stream`; sum(k_g) must keep the context's M."""
    _check(ctx, load().ec_ctx_set_capacity_async(ctx, k_g_dev, stream))


def ec_ctx_set_residual(ctx, on: bool):
    _check(ctx, load().ec_ctx_set_residual(ctx, 1 if on else 0))


def ec_ctx_set_tiles(ctx, policy: int):
    _check(ctx, load().ec_ctx_set_tiles(ctx, int(policy)))


def ec_rows_per_expert(ctx) -> int:
    return int(load().ec_rows_per_expert(ctx))


def ec_workspace_bytes(ctx) -> int:
    return int(load().ec_workspace_bytes(ctx))


def ec_ctx_set_workspace(ctx, ptr: int, nbytes: int):
    _check(ctx, load().ec_ctx_set_workspace(ctx, ptr, nbytes))


def ec_route(ctx, X, Wr, br, S_in, S_out, idx, gate, stream):
    _check(ctx, load().ec_route(ctx, X, Wr, br, S_in, S_out, idx, gate, stream))


def ec_moe_forward(ctx, X, Wr, br, Wg, Wu, Wd, Y, idx, gate, S_out, stream):
    _check(ctx, load().ec_moe_forward(ctx, X, Wr, br, Wg, Wu, Wd, Y, idx, gate, S_out, stream))


def ec_moe_backward(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, stream):
    _check(ctx, load().ec_moe_backward(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, stream))


def ec_ctx_set_shared(ctx, d_ff_shared: int):
    _check(ctx, load().ec_ctx_set_shared(ctx, int(d_ff_shared)))


def ec_moe_forward_shared(ctx, X, Wr, br, Wg, Wu, Wd, Wg_s, Wu_s, Wd_s, Y, idx, gate, S_out,
                          stream):
    _check(ctx, load().ec_moe_forward_shared(ctx, X, Wr, br, Wg, Wu, Wd, Wg_s, Wu_s, Wd_s, Y, idx,
                                             gate, S_out, stream))


def ec_moe_backward_shared(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, dWg_s, dWu_s, dWd_s, stream):
    _check(ctx, load().ec_moe_backward_shared(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, dWg_s, dWu_s,
                                              dWd_s, stream))


def ec_tc_ctx_create(N, d, E, d_ff, k, capacity, dtype):
    """Token-choice context: k experts per token, `capacity` tokens per expert (< 0: none)."""
    lib = load()
    ctx = ctypes.c_void_p()
    st = lib.ec_tc_ctx_create(ctypes.byref(ctx), N, d, E, d_ff, k, int(capacity), dtype)
    if st != EC_OK:
        raise ECError(st, "ec_tc_ctx_create rejected the sizes")
    return ctx


def ec_tc_forward(ctx, X, Wr, br, Wg, Wu, Wd, Y, choice, gate, kept, load_out, S_out, stream):
    _check(ctx, load().ec_tc_forward(ctx, X, Wr, br, Wg, Wu, Wd, Y, choice, gate, kept, load_out,
                                     S_out, stream))


def ec_tc_backward(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, stream):
    _check(ctx, load().ec_tc_backward(ctx, dY, dX, dWr, dbr, dWg, dWu, dWd, stream))


def ec_check_device(ctx, stream):
    _check(ctx, load().ec_check_device(ctx, stream))


def ec_ctx_set_profiling(ctx, on: bool):
    _check(ctx, load().ec_ctx_set_profiling(ctx, 1 if on else 0))


def ec_ctx_profile(ctx, cap: int = 4096):
    """[(kernel name, ms), ...] of the phases recorded since profiling was switched on."""
    names = (ctypes.c_char_p * cap)()
    ms = (ctypes.c_float * cap)()
    n = load().ec_ctx_profile(ctx, names, ms, cap)
    if n < 0:
        raise ECError(EC_ERR_CUDA, "ec_ctx_profile: CUDA error while reading events")
    return [(names[i].decode(), float(ms[i])) for i in range(min(n, cap))]


def ec_kernel_launches(ctx) -> int:
    return int(load().ec_kernel_launches(ctx))


def ec_select_static(S, N, E, group_off, k_g, idx, gate, stream):
    """Selection with no workspace (scratch in the library's static device array)."""
    g_arr, g_ptr = _i32(group_off)
    k_arr, k_ptr = _i32(k_g)
    st = load().ec_select_static(S, N, E, len(g_arr) - 1, g_ptr, k_ptr, idx, gate, stream)
    if st != EC_OK:
        raise ECError(st, "ec_select_static rejected the call")


def ec_selftest_bounded_wait(ctx, limit_ns: int, stream):
    _check(ctx, load().ec_selftest_bounded_wait(ctx, int(limit_ns), stream))


def ec_capacity_schedule(scheduler, k_min, k_max, E, group_off, r, sigma=0.22):
    """Per-group capacities k_g for masking ratios r (host computation in the library)."""
    g_arr, g_ptr = _i32(group_off)
    r_arr = np.ascontiguousarray(np.asarray(r, dtype=np.float64))
    G = len(g_arr) - 1
    if len(r_arr) != G:
        raise ValueError("one masking ratio per group")
    out = np.zeros(G, dtype=np.int32)
    code = EC_SCHEDULERS[scheduler] if isinstance(scheduler, str) else int(scheduler)
    st = load().ec_capacity_schedule(code, float(k_min), float(k_max), float(sigma), int(E), G,
                                     g_ptr, r_arr.ctypes.data_as(ctypes.POINTER(ctypes.c_double)),
                                     out.ctypes.data_as(ctypes.POINTER(ctypes.c_int32)))
    if st != EC_OK:
        raise ECError(st, "ec_capacity_schedule rejected its arguments")
    return out


def ec_last_error(ctx) -> str:
    return load().ec_last_error(ctx).decode()


def ec_get_last_error(ctx, n: int = 512):
    """(status of the last failed call, its message truncated to n-1 bytes)."""
    buf = ctypes.create_string_buffer(n) if n > 0 else None
    st = load().ec_get_last_error(ctx, buf, n)
    return int(st), (buf.value.decode() if buf is not None else "")


def ec_tc_capacity(capacity_factor, k: int, N: int, E: int) -> int:
    """Token-choice capacity ceil(CF k N / E) computed by the library; -1 (dropless) when
    capacity_factor is None or <= 0."""
    if capacity_factor is None:
        return -1
    v = int(load().ec_tc_capacity(float(capacity_factor), int(k), int(N), int(E)))
    if v < -1:
        raise ECError(EC_ERR_SHAPE, "ec_tc_capacity rejected its arguments")
    return v
