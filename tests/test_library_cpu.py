"""Host-side checks of libsphq.so that need no GPU: it builds for sm_103a,
loads, exports every function include/sphq.h declares, and rejects bad
arguments before touching CUDA."""
import ctypes

import pytest

from paper_2609_24875_gb300 import build as libbuild
from paper_2609_24875_gb300 import sphq


@pytest.fixture(scope="module")
def lib():
    libbuild.build()
    return sphq.load()


def test_header_declares_the_boundary():
    names = sphq.header_functions()
    for n in ("sphq_create", "sphq_pack", "sphq_gemv", "sphq_decode", "sphq_bytes",
              "sphq_destroy", "sphq_last_error", "sphq_version"):
        assert n in names


def test_every_declared_symbol_is_exported(lib):
    for name in sphq.header_functions():
        assert hasattr(lib, name), name


def test_version(lib):
    assert lib.sphq_version() >= 10100


def test_invalid_arguments_rejected_on_host(lib):
    h = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(1 << 16)
    p = ctypes.cast(buf, ctypes.c_void_p)
    # cols not a multiple of 128
    assert lib.sphq_create(32, 100, 2, 64, p, p, p, ctypes.byref(h)) == 1
    assert b"128" in lib.sphq_last_error()
    assert h.value is None
    # unsupported bits / K
    assert lib.sphq_create(32, 128, 4, 1 << 20, p, p, p, ctypes.byref(h)) == 2
    assert lib.sphq_create(32, 128, 2, 128, p, p, p, ctypes.byref(h)) == 2
    # NULL pointers
    assert lib.sphq_create(32, 128, 2, 64, None, p, p, ctypes.byref(h)) == 1
    assert lib.sphq_create(32, 128, 2, 64, p, p, p, None) == 1
    # NULL handle everywhere
    assert lib.sphq_gemv(None, p, p, 1, None) == 1
    assert lib.sphq_decode(None, p, None) == 1
    assert lib.sphq_pack(None, p, p, p, None) == 1
    assert lib.sphq_bytes(None, 1) == 0
    info = sphq.PlanInfo()
    assert lib.sphq_get_plan(None, 1, ctypes.byref(info)) == 1
    assert lib.sphq_set_cluster_size(None, 1, 2) == 1
    assert lib.sphq_destroy(None) == 0
    assert lib.sphq_last_error() == b""


def test_vector_dimension_and_workspace_arguments_rejected_on_host(lib):
    h = ctypes.c_void_p()
    buf = ctypes.create_string_buffer(1 << 16)
    p = ctypes.cast(buf, ctypes.c_void_p)
    # 16-D vectors take the W2 allocation only: bits 2, K = 2^14, 4 radius bits
    assert lib.sphq_create_dim(32, 128, 16, 2, 4, 1 << 13, p, p, p, ctypes.byref(h)) == 2
    assert lib.sphq_create_dim(32, 128, 16, 3, 4, 1 << 14, p, p, p, ctypes.byref(h)) == 2
    assert lib.sphq_create_dim(32, 128, 16, 2, 3, 1 << 14, p, p, p, ctypes.byref(h)) == 2
    assert b"16-D" in lib.sphq_last_error()
    # 4-D likewise (bits 2, K 4, 4 radius bits); other dimensions are unsupported
    assert lib.sphq_create_dim(32, 128, 4, 2, 4, 8, p, p, p, ctypes.byref(h)) == 2
    assert lib.sphq_create_dim(32, 128, 12, 2, 4, 64, p, p, p, ctypes.byref(h)) == 2
    assert h.value is None
    # the workspace entry points and shape queries with a NULL handle
    n = ctypes.c_size_t(7)
    assert lib.sphq_gemm_workspace(None, 64, ctypes.byref(n)) == 1
    assert lib.sphq_gemm_ws(None, p, p, 64, p, 1 << 16, None) == 1
    info = sphq.GemmInfo()
    assert lib.sphq_get_gemm_shape(None, 64, ctypes.byref(info)) == 1
    assert lib.sphq_set_gemm_shape(None, 1, 128) == 1
