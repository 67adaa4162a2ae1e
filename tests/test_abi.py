"""The C ABI library loads on a machine without a GPU and exports every declared entry
point; host-side argument checks work without touching the device."""
import ctypes
import os
import re

import pytest

import paper_2604_01622_gb300 as ec
from paper_2604_01622_gb300 import build as B

ROOT = os.path.dirname(os.path.dirname(os.path.abspath(__file__)))


@pytest.fixture(scope="module")
def lib():
    if not os.path.exists(ec.LIB_PATH):
        B.build()
    return ec.load()


def _declared():
    names = set()
    for f in os.listdir(os.path.join(ROOT, "include")):
        if f.endswith(".h"):
            src = open(os.path.join(ROOT, "include", f)).read()
            src = re.sub(r"/\*.*?\*/", "", src, flags=re.S)
            names |= set(re.findall(r"^\s*(?:[\w\s\*]+?)\b(ec_\w+)\s*\(", src, flags=re.M))
    return names


def test_header_declares_the_boundary():
    names = _declared()
    for n in ("ec_route", "ec_moe_forward", "ec_moe_backward", "ec_ctx_create"):
        assert n in names
    assert names == set(ec.EXPORTS)


def test_library_exports_every_declared_symbol(lib):
    handle = ctypes.CDLL(ec.LIB_PATH)
    for name in _declared():
        assert hasattr(handle, name), name


def test_status_strings(lib):
    assert ec.status_string(ec.EC_OK) == "EC_OK"
    assert ec.status_string(ec.EC_ERR_TIMEOUT) == "EC_ERR_TIMEOUT"


def test_host_validation_without_device(lib):
    # k_g larger than its group
    with pytest.raises(ec.ECError) as e:
        ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 256], [16, 129], ec.EC_F32)
    assert e.value.status == ec.EC_ERR_SHAPE
    # group offsets not covering N
    with pytest.raises(ec.ECError):
        ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 255], [16, 16], ec.EC_F32)
    # bf16 path needs d, d_ff multiples of 64
    with pytest.raises(ec.ECError) as e:
        ec.ec_ctx_create(256, 96, 8, 128, 2, [0, 128, 256], [16, 16], ec.EC_BF16)
    assert e.value.status == ec.EC_ERR_UNSUPPORTED
    ctx = ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 256], [16, 16], ec.EC_F32)
    try:
        assert ec.ec_rows_per_expert(ctx) == 32
        assert ec.ec_workspace_bytes(ctx) > 0
        # capacities may change per step but not exceed the workspace's
        ec.ec_ctx_set_capacity(ctx, [0, 20])
        assert ec.ec_rows_per_expert(ctx) == 20
        with pytest.raises(ec.ECError) as e:
            ec.ec_ctx_set_capacity(ctx, [20, 20])
        assert e.value.status == ec.EC_ERR_SHAPE
        # compute calls without a workspace are refused before any launch
        with pytest.raises(ec.ECError) as e:
            ec.ec_route(ctx, 16, 16, None, None, None, 16, 16, None)
        assert e.value.status == ec.EC_ERR_WORKSPACE
        with pytest.raises(ec.ECError) as e:
            ec.ec_ctx_set_workspace(ctx, 0x1001, 1 << 40)
        assert e.value.status == ec.EC_ERR_WORKSPACE
        # tile policies: the three named ones, nothing else
        for policy in (ec.EC_TILES_256, ec.EC_TILES_512, ec.EC_TILES_AUTO):
            ec.ec_ctx_set_tiles(ctx, policy)
        for policy in (-1, 3):
            with pytest.raises(ec.ECError) as e:
                ec.ec_ctx_set_tiles(ctx, policy)
            assert e.value.status == ec.EC_ERR_INVALID_ARG
    finally:
        ec.ec_ctx_destroy(ctx)


def test_token_choice_host_validation_without_device(lib):
    # bf16 only; 1 <= k <= min(E, 32); at most 256 experts; d, d_ff multiples of 64
    for args, status in (((256, 64, 8, 128, 2, -1, ec.EC_F32), ec.EC_ERR_UNSUPPORTED),
                         ((256, 64, 8, 128, 0, -1, ec.EC_BF16), ec.EC_ERR_SHAPE),
                         ((256, 64, 8, 128, 9, -1, ec.EC_BF16), ec.EC_ERR_SHAPE),
                         ((256, 64, 64, 128, 33, -1, ec.EC_BF16), ec.EC_ERR_SHAPE),
                         ((256, 64, 300, 128, 2, -1, ec.EC_BF16), ec.EC_ERR_UNSUPPORTED),
                         ((256, 96, 8, 128, 2, -1, ec.EC_BF16), ec.EC_ERR_UNSUPPORTED)):
        with pytest.raises(ec.ECError) as e:
            ec.ec_tc_ctx_create(*args)
        assert e.value.status == status, args
    ctx = ec.ec_tc_ctx_create(1000, 64, 12, 128, 3, 250, ec.EC_BF16)
    try:
        # the padded rows (N k + 255 E, in 256-row blocks) make the workspace larger than an
        # expert-choice one of the same shape and capacity
        ec_ctx = ec.ec_ctx_create(1000, 64, 12, 128, 1, [0, 1000], [250], ec.EC_BF16)
        assert ec.ec_workspace_bytes(ctx) > ec.ec_workspace_bytes(ec_ctx)
        ec.ec_ctx_destroy(ec_ctx)
        # expert-choice calls are refused on a token-choice context
        with pytest.raises(ec.ECError) as e:
            ec.ec_ctx_set_capacity(ctx, [4])
        assert e.value.status == ec.EC_ERR_STATE
        with pytest.raises(ec.ECError) as e:
            ec.ec_ctx_set_shared(ctx, 64)
        assert e.value.status == ec.EC_ERR_STATE
        # and compute calls need a workspace first
        with pytest.raises(ec.ECError) as e:
            ec.ec_tc_forward(ctx, 16, 16, None, 16, 16, 16, 16, None, None, None, None, None,
                             None)
        assert e.value.status == ec.EC_ERR_WORKSPACE
    finally:
        ec.ec_ctx_destroy(ctx)
    # token-choice calls are refused on an expert-choice context (after the workspace check)
    ctx = ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 256], [16, 16], ec.EC_F32)
    try:
        with pytest.raises(ec.ECError) as e:
            ec.ec_tc_backward(ctx, 16, 16, 16, None, 16, 16, 16, None)
        assert e.value.status == ec.EC_ERR_WORKSPACE
    finally:
        ec.ec_ctx_destroy(ctx)


def test_get_last_error_copies_the_message(lib):
    ctx = ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 256], [16, 16], ec.EC_F32)
    try:
        assert ec.ec_get_last_error(ctx) == (ec.EC_OK, "")
        with pytest.raises(ec.ECError):
            ec.ec_ctx_set_capacity(ctx, [200, 1])        # k_g above its group's 128 tokens
        status, msg = ec.ec_get_last_error(ctx)
        assert status == ec.EC_ERR_SHAPE and msg == ec.ec_last_error(ctx) and "k_g[0]" in msg
        # truncated to n - 1 bytes plus the terminating NUL; n = 0 writes nothing
        assert ec.ec_get_last_error(ctx, 6) == (ec.EC_ERR_SHAPE, msg[:5])
        assert ec.ec_get_last_error(ctx, 0) == (ec.EC_ERR_SHAPE, "")
        # a NULL buffer with room claimed is an argument error
        assert lib.ec_get_last_error(ctx, None, 8) == ec.EC_ERR_INVALID_ARG
    finally:
        ec.ec_ctx_destroy(ctx)
    assert lib.ec_get_last_error(None, None, 0) == ec.EC_ERR_INVALID_ARG


def test_async_capacity_needs_a_workspace_and_an_aligned_array(lib):
    ctx = ec.ec_ctx_create(256, 64, 8, 128, 2, [0, 128, 256], [16, 16], ec.EC_F32)
    try:
        with pytest.raises(ec.ECError) as e:
            ec.ec_ctx_set_capacity_async(ctx, 0x1000, None)
        assert e.value.status == ec.EC_ERR_WORKSPACE
    finally:
        ec.ec_ctx_destroy(ctx)
    ctx = ec.ec_tc_ctx_create(1000, 64, 12, 128, 3, 250, ec.EC_BF16)
    try:
        with pytest.raises(ec.ECError):
            ec.ec_ctx_set_capacity_async(ctx, 0x1000, None)
    finally:
        ec.ec_ctx_destroy(ctx)


def test_tc_capacity_in_the_library_matches_the_oracle(lib):
    from oracle import token_choice as T
    for cf in (0.5, 1.0, 1.25, 1.5, 2.0, 1.0 / 3.0, 7.3):
        for (k, N, E) in ((8, 32768, 64), (1, 1000, 12), (2, 333, 7), (32, 262144, 256)):
            assert ec.ec_tc_capacity(cf, k, N, E) == T.tc_capacity(cf, k, N, E)
    for cf in (None, 0, -1.0, float("nan")):
        assert ec.ec_tc_capacity(cf, 8, 1024, 64) == -1
    assert lib.ec_tc_capacity(1.0, 0, 1024, 64) == -2
    assert lib.ec_tc_capacity(1.0, 8, 1024, 0) == -2
