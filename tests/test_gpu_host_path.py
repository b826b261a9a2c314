"""sphq_gemv_host through the C ABI: pinned (mapped) host buffers, which the
kernel reads and writes directly, and pageable buffers, which go through the
handle's staging copies; both must give the device GEMV's result exactly
(same kernel, same launch shape) and agree with the oracle."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


@pytest.mark.parametrize("bits,rows,cols,batch", [(2, 1000, 2048, 1), (3, 512, 3584, 2),
                                                  (2, 96, 4096, 5), (3, 80, 1024, 8)])
@pytest.mark.parametrize("pinned", [True, False])
def test_host_buffers_match_device_gemv(bits, rows, cols, batch, pinned):
    codes, x = inp.random_codes(bits, rows, cols, seed=3100 + rows + bits + batch, B=batch)
    m = G.make_matrix(codes)
    y_dev = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    xh = torch.from_numpy(np.ascontiguousarray(x.view(np.int16))).view(torch.float16)
    yh = torch.full((batch, rows), float("nan"), dtype=torch.float16)
    if pinned:
        xh = xh.pin_memory()
        yh = yh.pin_memory()
    stream = torch.cuda.current_stream()
    for _ in range(2):
        yh.fill_(float("nan"))
        m.gemv_host(xh, yh, stream=stream)
        stream.synchronize()
        assert torch.equal(yh, y_dev.cpu())
    w = G.oracle_decode(codes)
    ref, absdot = oracle.gemv(w, x)
    got = yh.float().numpy().astype(np.float64)
    assert np.all(np.abs(got - ref) <= oracle.gemv_tolerance(absdot))
    m.close()


def test_host_buffer_at_an_offset_into_a_pinned_allocation():
    codes, x = inp.random_codes(2, 64, 1024, seed=3300)
    m = G.make_matrix(codes)
    y_dev = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    big_x = torch.zeros(3 * 1024 + 8, dtype=torch.float16).pin_memory()
    big_y = torch.zeros(3 * 64 + 2, dtype=torch.float16).pin_memory()
    xh = big_x[1024:2048].view(1, 1024)  # 2048-byte offset: still 16-byte aligned
    yh = big_y[2:66].view(1, 64)         # 4-byte offset
    xh.copy_(torch.from_numpy(np.ascontiguousarray(x.view(np.int16))).view(torch.float16).view(1, 1024))
    m.gemv_host(xh, yh)
    torch.cuda.synchronize()
    assert torch.equal(yh, y_dev.cpu())
    assert torch.count_nonzero(big_y[:2]) == 0 and torch.count_nonzero(big_y[66:]) == 0
    m.close()
