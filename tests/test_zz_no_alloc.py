"""sphq_gemv_noalloc, the entry point for callers that may not allocate GPU
memory while serving (it keeps any split-K scratch in one fixed device array
compiled into the library), checked through the C ABI against sphq_gemv.

Both entry points launch the same deterministic kernel (on-chip reduction in a
fixed order), so their outputs must agree bit for bit; the oracle's tolerance
is checked as well.  The free device memory must not change across calls.

This file is collected last so that a run stopping at the first failure has
already run every other test; it also passes on its own in a fresh process.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import sphq

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def _noalloc(m, xd, y, batch, stream):
    return sphq.load().sphq_gemv_noalloc(m.handle, xd.data_ptr(), y.data_ptr(), batch,
                                         stream.cuda_stream)


def _bits16(t):
    return t.cpu().view(torch.int16).numpy()


@pytest.mark.parametrize("bits,rows,cols,batch,wrapper",
                         [(2, 3584, 3584, 1, False), (3, 512, 3584, 4, False),
                          (2, 1000, 1024, 2, True), (3, 96, 18944, 8, False),
                          (3, 300, 1024, 16, False)])
def test_noalloc_matches_gemv_on_two_calls(bits, rows, cols, batch, wrapper):
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
    ys = [torch.full((batch, rows), float("nan"), dtype=torch.float16, device=G.DEV)
          for _ in range(2)]
    torch.cuda.synchronize()
    free0 = None
    for y in ys:  # two calls in a row share (and reuse) the fixed scratch
        if wrapper:
            m.gemv_noalloc(xd, y)
        else:
            assert _noalloc(m, xd, y, batch, stream) == 0, sphq.load().sphq_last_error()
        torch.cuda.synchronize()
        free = torch.cuda.mem_get_info()[0]
        if free0 is None:
            free0 = free
        else:
            assert free == free0, "a call changed the free device memory"
        got = y.float().cpu().numpy().astype(np.float64)
        assert np.all(np.isfinite(got))
        assert np.array_equal(_bits16(y), _bits16(y_ref)), "differs from sphq_gemv"
        assert np.all(np.abs(got - ref) <= tol)
    m.close()


def test_noalloc_takes_shapes_beyond_the_scratch_limit_of_a_scratch_plan():
    # 16385 row tiles: beyond what a plan that reduced through the fixed array
    # could cover; the current plans reduce on chip, so the call is accepted
    rows = 16 * 16384 + 16
    codes, x = inp.random_codes(2, rows, 128, seed=7)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y_ref = m.gemv(xd).clone()
    y = torch.empty((1, rows), dtype=torch.float16, device=G.DEV)
    assert _noalloc(m, xd, y, 1, torch.cuda.current_stream()) == 0, sphq.load().sphq_last_error()
    torch.cuda.synchronize()
    assert np.array_equal(_bits16(y), _bits16(y_ref))
    m.close()


def test_noalloc_wrapper_checks_dtypes():
    codes, x = inp.random_codes(2, 64, 128, seed=9)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    with pytest.raises(ValueError):
        m.gemv_noalloc(xd.float(), torch.empty((1, 64), dtype=torch.float16, device=G.DEV))
    with pytest.raises(ValueError):
        m.gemv_noalloc(xd, torch.empty((1, 64), dtype=torch.float32, device=G.DEV))
    m.close()
