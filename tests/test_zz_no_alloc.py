"""sphq_gemv_noalloc, the entry point for callers that may not allocate GPU
memory while serving (it keeps its split-K scratch in one fixed device array
compiled into the library), checked through the C ABI against sphq_gemv.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes on its own in a fresh process.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import sphq

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def _noalloc(m, xd, y, batch, stream):
    L = sphq.load()
    L.sphq_gemv_noalloc.argtypes = [ctypes.c_void_p, ctypes.c_void_p, ctypes.c_void_p,
                                    ctypes.c_int, ctypes.c_void_p]
    L.sphq_gemv_noalloc.restype = ctypes.c_int
    return L.sphq_gemv_noalloc(m.handle, xd.data_ptr(), y.data_ptr(), batch, stream.cuda_stream)


@pytest.mark.parametrize("bits,rows,cols,batch", [(2, 3584, 3584, 1), (3, 512, 3584, 4),
                                                  (2, 1000, 1024, 2), (3, 96, 18944, 8)])
def test_noalloc_matches_gemv_on_two_calls(bits, rows, cols, batch):
    codes, x = inp.random_codes(bits, rows, cols, seed=4242 + rows + bits, B=batch)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    stream = torch.cuda.current_stream()
    y_ref = m.gemv(xd).clone()
    torch.cuda.synchronize()
    w_ref = G.oracle_decode(codes)
    _, absdot = oracle.gemv(w_ref, x)
    tol = oracle.gemv_tolerance(absdot)
    ref = y_ref.float().cpu().numpy().astype(np.float64)
    for _ in range(2):  # two calls in a row share (and reuse) the fixed scratch
        y = torch.full((batch, rows), float("nan"), dtype=torch.float16, device=G.DEV)
        assert _noalloc(m, xd, y, batch, stream) == 0, sphq.load().sphq_last_error()
        torch.cuda.synchronize()
        got = y.float().cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got))
        assert np.all(np.abs(got - ref) <= tol)
    m.close()


def test_noalloc_rejects_matrices_beyond_its_scratch():
    rows = 16 * 16384 + 16  # one row tile more than the fixed counters cover
    codes, x = inp.random_codes(2, rows, 128, seed=7)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y = torch.empty((1, rows), dtype=torch.float16, device=G.DEV)
    status = _noalloc(m, xd, y, 1, torch.cuda.current_stream())
    assert status == 2  # SPHQ_ERR_UNSUPPORTED
    assert b"4 MiB" in sphq.load().sphq_last_error()
    m.close()
