"""The C-ABI library builds for sm_103a, loads, and exports every entry point
include/xpress.h declares.  Host-side argument checks are exercised without a
GPU (they return before any CUDA call)."""
import ctypes as C

import pytest

from paper_2608_02438_gb300 import binding as X
from paper_2608_02438_gb300 import build as BLD


@pytest.fixture(scope="module")
def lib():
    BLD.build()
    return X.load()


def test_exports_every_declared_symbol(lib):
    names = X.declared_symbols()
    assert {"xpress_refine_block", "xpress_accept", "xpress_refiner_create"} <= set(names)
    for n in names:
        assert hasattr(lib, n), n


def test_version_and_status_strings(lib):
    assert lib.xpress_version() >= 1
    for code in (0, -1, -2, -3, -4, -5, -6):
        assert lib.xpress_status_string(code)


def test_null_arguments_are_rejected_without_touching_the_gpu(lib):
    h = C.c_void_p()
    assert lib.xpress_refiner_create(None, None, C.byref(h)) == X.XPRESS_ERR_INVALID_ARG
    w = X.XpressWeights(4096, 151936, 256, 16, X.XPRESS_BF16, 0)   # weight pointers NULL
    assert lib.xpress_refiner_create(C.byref(w), None, C.byref(h)) == X.XPRESS_ERR_INVALID_ARG
    assert lib.xpress_refine_workspace_size(None, 4) == 0
    assert lib.xpress_accept_workspace_size(None, 4) == 0
    blk_in, blk_out = X.XpressBlockIn(), X.XpressBlockOut()
    assert lib.xpress_refine_block(None, C.byref(blk_in), C.byref(blk_out), None, 0, None) == X.XPRESS_ERR_INVALID_ARG
    acc = X.XpressAcceptIn()
    assert lib.xpress_accept(None, C.byref(acc), None, None, None, 0, None) == X.XPRESS_ERR_INVALID_ARG
    v = C.c_int32()
    assert lib.xpress_get_device_status(None, None, C.byref(v)) == X.XPRESS_ERR_INVALID_ARG


def test_unsupported_shapes_are_rejected(lib):
    h = C.c_void_p()
    dummy = [C.c_void_p(16)] * 8   # never dereferenced: the shape check fails first
    for H, V, r, B in [(4096, 151936, 128, 16), (4096, 151937, 256, 16), (4096, 151936, 256, 33),
                       (4100 + 1, 151936, 256, 16)]:
        w = X.XpressWeights(H, V, r, B, X.XPRESS_BF16, 0, *dummy)
        assert lib.xpress_refiner_create(C.byref(w), None, C.byref(h)) == X.XPRESS_ERR_UNSUPPORTED


def test_wait_limit_argument_checks(lib):
    assert lib.xpress_set_wait_limit(None, 1000) == X.XPRESS_ERR_INVALID_ARG
