"""sphq_gemm_ws, the two-pass form of the prefill product: W_hat decoded into a
caller-provided workspace (exactly sphq_decode's output), then a dense
tensor-core pass that loads W_hat and X tiles with TMA.  Products, their
order of accumulation and the output rounding are those of the fused kernel,
so Y must equal sphq_gemm's bit for bit; the fused kernel is checked against
the float64 oracle in test_gpu_gemm.py, and one shape per format is checked
against the oracle here as well.
"""
import ctypes

import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, sphq

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

FORMATS = [(2, 4, 64), (3, 4, 8192), (3, 3, 8192), (2, 2, 256), (2, 3, 64)]
FIDS = ["W2", "W3", "W3V3", "8-8-2", "8-6-3"]
SHAPES = [(1, 128), (1, 256), (2, 256)]


def _ws(m):
    return torch.empty(m.rows * m.cols, dtype=torch.float16, device="cuda")


def _bits(t):
    return t.contiguous().view(torch.int16)


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
@pytest.mark.parametrize("shape", SHAPES, ids=[f"mt{m}-bn{n}" for m, n in SHAPES])
def test_equals_fused_bit_for_bit(fmt, shape):
    bits, v, K = fmt
    mt, bn = shape
    # ragged in every dimension: rows not a multiple of 16 or of the weight
    # tile, batch past one activation tile, several radius groups
    rows, cols, batch = 531, 640, 300
    codes, x = inp.random_codes(bits, rows, cols, seed=1700 + 10 * mt + bn + v, B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    m.set_gemm_shape(mt, bn)
    xd = G.x_dev(x)
    ws = _ws(m)
    y_fused = m.gemm(xd)
    y_two = m.gemm_ws(xd, ws)
    torch.cuda.synchronize()
    assert torch.equal(_bits(y_fused), _bits(y_two))
    # the workspace holds W_hat exactly as sphq_decode writes it
    w_dec = m.decode()
    torch.cuda.synchronize()
    assert torch.equal(_bits(ws.view(rows, cols)), _bits(w_dec))
    m.check()
    m.close()


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
def test_against_oracle(fmt):
    bits, v, K = fmt
    rows, cols, batch = 257, 384, 130
    codes, x = inp.random_codes(bits, rows, cols, seed=1800 + v + bits, B=batch, radius_bits=v, K=K)
    m = G.make_matrix(codes)
    y = m.gemm_ws(G.x_dev(x), _ws(m))
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().astype(np.float64)
    y_ref, absdot = oracle.gemv(G.oracle_decode(codes, np.arange(rows)), x)
    err = np.abs(y - y_ref)
    tol = oracle.gemv_tolerance(absdot)
    assert np.all(np.isfinite(y))
    assert np.all(err <= tol), f"max err/tol = {float(np.max(err / tol)):.3g}"
    m.check()
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:3], ids=FIDS[:3])
def test_report_size_equals_fused(fmt):
    # the size the report times: every output compared on the device
    bits, v, K = fmt
    rows, cols, batch = 8192, 8192, 4096
    codes, _ = inp.random_codes(bits, rows, cols, seed=1900 + v + bits, B=1, radius_bits=v, K=K)
    m = G.make_matrix(codes)
    g = torch.Generator(device="cpu").manual_seed(7)
    xd = torch.randn((batch, cols), generator=g).to(torch.float16).cuda()
    ws = _ws(m)
    y_fused = m.gemm(xd)
    y_two = m.gemm_ws(xd, ws)
    torch.cuda.synchronize()
    assert torch.equal(_bits(y_fused), _bits(y_two))
    m.check()
    m.close()
    del ws
    torch.cuda.empty_cache()


def test_workspace_advice_and_errors():
    bits, v, K = 3, 4, 8192
    codes, x = inp.random_codes(bits, 256, 512, seed=1950, B=200, radius_bits=v, K=K)
    m = G.make_matrix(codes)
    need = m.rows * m.cols * 2
    for batch in (1, 8, 200, 4096):
        # W_hat for the two-pass form, the partials of the split-K form, or none
        assert m.gemm_workspace(batch) in (0, need) or m.gemm_shape(batch)["ksplit"] > 1
    big = G.make_matrix(inp.random_codes(3, 8192, 8192, seed=1951, B=1)[0])
    assert big.gemm_workspace(4096) == 8192 * 8192 * 2  # the 8192-entry table at prefill size
    big.close()
    xd = G.x_dev(x)
    L = sphq.load()
    y = torch.empty((200, m.rows), dtype=torch.float16, device="cuda")
    ws = _ws(m)
    stream = torch.cuda.current_stream().cuda_stream
    # too small a workspace, a misaligned one
    assert L.sphq_gemm_ws(m.handle, xd.data_ptr(), y.data_ptr(), 200, ws.data_ptr(), need - 2,
                          stream) == 1
    assert b"workspace" in L.sphq_last_error()
    assert L.sphq_gemm_ws(m.handle, xd.data_ptr(), y.data_ptr(), 200, ws.data_ptr() + 2, need,
                          stream) == 1
    # NULL workspace: the fused kernel
    y_null = m.gemm_ws(xd, None)
    y_fused = m.gemm(xd)
    torch.cuda.synchronize()
    assert torch.equal(_bits(y_null), _bits(y_fused))
    with pytest.raises(SphqError):
        m.gemm_ws(xd, _ws(m)[: m.rows])
    n = ctypes.c_size_t(5)
    assert L.sphq_gemm_workspace(m.handle, 0, ctypes.byref(n)) == 2
    assert n.value == 0
    m.check()
    m.close()


def test_graph_capture_and_side_stream():
    # both passes captured in a CUDA graph on a side stream; replays equal the
    # eager call bit for bit, and so does a batch of 12 (two GEMV launches)
    codes, x = inp.random_codes(3, 384, 512, seed=1960, B=160)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    ws = _ws(m)
    y_ref = m.gemm_ws(xd, ws)
    y12_ref = m.gemm(xd[:12].contiguous())
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    y = torch.empty_like(y_ref)
    x12 = xd[:12].contiguous()
    y12 = torch.empty_like(y12_ref)
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        m.gemm_ws(xd, ws, y=y, stream=s)
        m.gemm(x12, y=y12, stream=s)
    for _ in range(2):
        y.zero_()
        y12.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(_bits(y), _bits(y_ref))
        assert torch.equal(_bits(y12), _bits(y12_ref))
    m.check()
    m.close()


@pytest.mark.parametrize("rows,cols,batch", [(1, 128, 1), (1, 128, 129), (17, 256, 200),
                                             (300, 128, 64)])
def test_tiny_and_ragged_shapes(rows, cols, batch):
    # one row, one radius group, a batch of one: the W_hat and X tiles read
    # zeros past the matrix and the batch; equal to the fused kernel and
    # within the oracle's tolerance
    codes, x = inp.random_codes(3, rows, cols, seed=1970 + rows + batch, B=batch)
    m = G.make_matrix(codes)
    m.set_gemm_shape(1, 128)  # the tensor-core kernel for every batch size
    xd = G.x_dev(x)
    y_fused = m.gemm(xd)
    y_two = m.gemm_ws(xd, _ws(m))
    torch.cuda.synchronize()
    assert torch.equal(_bits(y_fused), _bits(y_two))
    y = y_two.float().cpu().numpy().astype(np.float64)
    y_ref, absdot = oracle.gemv(G.oracle_decode(codes, np.arange(rows)), x)
    assert np.all(np.abs(y - y_ref) <= oracle.gemv_tolerance(absdot))
    m.check()
    m.close()


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
@pytest.mark.parametrize("rows,cols,batch", [(8000, 4096, 48), (1000, 8192, 200), (300, 4096, 41),
                                             (3584, 18944, 256)])
def test_split_k(fmt, rows, cols, batch):
    # batches of 41-256 with a workspace and at least 16 radius groups per
    # share: the output tiles' columns are shared by several CTAs whose fp32
    # partials the tile's last CTA sums in share order (ragged rows, ragged
    # batch); against the oracle and repeatable bit for bit
    bits, v, K = fmt
    codes, x = inp.random_codes(bits, rows, cols, seed=2000 + rows + batch + v + bits, B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    info = m.gemm_shape(batch)
    assert info["ksplit"] >= 2
    need = m.gemm_workspace(batch)  # the split-K partials and counters
    assert need > 0
    ws = torch.empty(need, dtype=torch.uint8, device="cuda")
    xd = G.x_dev(x)
    y1 = m.gemm_ws(xd, ws)
    y2 = m.gemm_ws(xd, ws)
    torch.cuda.synchronize()
    assert torch.equal(_bits(y1), _bits(y2))
    sel = np.arange(rows) if rows <= 1000 else G.sample_rows(rows, 300, seed=batch)
    y = y1.float().cpu().numpy().astype(np.float64)
    y_ref, absdot = oracle.gemv(G.oracle_decode(codes, sel), x)
    err = np.abs(y[:, sel] - y_ref)
    tol = oracle.gemv_tolerance(absdot)
    assert np.all(np.isfinite(y[:, sel]))
    assert np.all(err <= tol), f"max err/tol = {float(np.max(err / tol)):.3g}"
    # a workspace too small for the partials (and for W_hat) is refused
    with pytest.raises(SphqError):
        m.gemm_ws(xd, ws[: need // 2])
    # a fixed shape turns the split off
    m.set_gemm_shape(1, 128)
    assert m.gemm_shape(batch)["ksplit"] == 1
    m.set_gemm_shape(0, 0)
    m.check()
    m.close()


def test_split_k_graph_capture():
    # the counter memset and the split-K launch captured in a CUDA graph on a
    # side stream: replays equal the eager call bit for bit
    codes, x = inp.random_codes(3, 300, 4096, seed=2050, B=64)
    m = G.make_matrix(codes)
    assert m.gemm_shape(64)["ksplit"] >= 2
    ws = torch.empty(m.gemm_workspace(64), dtype=torch.uint8, device="cuda")
    xd = G.x_dev(x)
    y_ref = m.gemm_ws(xd, ws)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    y = torch.empty_like(y_ref)
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        m.gemm_ws(xd, ws, y=y, stream=s)
    for _ in range(3):
        y.zero_()
        g.replay()
        torch.cuda.synchronize()
        assert torch.equal(_bits(y), _bits(y_ref))
    m.check()
    m.close()
