"""16-D vectors (Tab. 7 at the W2 allocation: 16 sign bits, a 14-bit index into
K = 16384 directions, a 4-bit radius code; 2.125 bits per weight, the 512 KiB
codebook gathered from global memory) through the C ABI against the float64
oracle (oracle.decode_dim): decode bit-exact, the GEMV within
1e-3 * sum_j |w_hat_j||x_j| + 2^-24 at batch 1..16, every cluster size,
ragged shapes, edge codes, the decoder projections, the host-buffer and
no-allocation entry points, export / import, code validation and the entry
points that take 8-D vectors only."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

K16 = 1 << 14


def make16(codes, pack=True):
    m = SphqMatrix(codes.rows, codes.cols, 2, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset), radius_bits=4, K=K16, dim=16)
    if pack:
        m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    return m


def ref_decode(codes, rows=None):
    c = codes
    if rows is not None:
        c = inp.CodesDim(16, 2, codes.codebook, codes.scale[rows], codes.offset[rows],
                         codes.sign[rows], codes.idx[rows], codes.rcode[rows])
    return oracle.decode_dim(c.codebook, c.scale, c.offset, c.sign, c.idx, c.rcode)


def check(m, codes, x, rows=None, y=None):
    if y is None:
        y = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().astype(np.float64)
    if rows is None:
        rows = np.arange(codes.rows)
    y_ref, absdot = oracle.gemv(ref_decode(codes, rows), x)
    err = np.abs(y[:, rows] - y_ref)
    tol = oracle.gemv_tolerance(absdot)
    assert np.all(np.isfinite(y[:, rows]))
    assert np.all(err <= tol), f"max err/tol = {float(np.max(err / tol)):.3g}"


@pytest.mark.parametrize("rows,cols", [(1, 128), (15, 256), (33, 384), (257, 640), (1000, 2048)])
def test_small_shapes_decode_and_gemv(rows, cols):
    codes, x = inp.random_codes_dim(16, 2, rows, cols, seed=5000 + rows + cols, B=16)
    m = make16(codes)
    assert np.array_equal(G.decoded_bits(m), ref_decode(codes))
    for B in (1, 2, 3, 5, 8, 9, 16):
        check(m, codes, x[:B])
    m.check()
    m.close()


def test_edge_codes():
    # every sign bit set and clear, the first and last directions, radius codes
    # 0 and 15 (both halves of the split code), zero and subnormal scales,
    # zero offsets, zero codebook coordinates (+-0 after the sign)
    codes, x = inp.random_codes_dim(16, 2, 80, 512, seed=55, B=4)
    codes.codebook[:2, 5] = 0
    codes.codebook[K16 - 1, :] = codes.codebook[K16 - 1, ::-1]
    codes.sign[:8] = 0xFFFF
    codes.sign[8:16] = 0
    codes.idx[16:24] = K16 - 1
    codes.idx[24:32, ::2] = 0
    codes.idx[24:32, 1::2] = 1
    codes.rcode[32:40] = 15
    codes.rcode[40:48] = 0
    codes.rcode[48:56] = 3
    codes.rcode[56:60] = 12
    codes.scale[60:68] = 0
    codes.offset[68:72] = 0
    codes.scale[72:80] = 0x0001
    m = make16(codes)
    assert np.array_equal(G.decoded_bits(m), ref_decode(codes))
    check(m, codes, x)
    m.close()


@pytest.mark.parametrize("rows,cols", [(1000, 1024), (48, 3584), (5, 128)])
def test_every_cluster_size(rows, cols):
    codes, x = inp.random_codes_dim(16, 2, rows, cols, seed=56 + rows, B=8)
    m = make16(codes)
    ng = cols // 128
    for cs in (1, 2, 4, 8):
        if cs > ng:
            with pytest.raises(SphqError):
                m.set_cluster_size(1, cs)
            continue
        for B in (1, 3, 8):
            m.set_cluster_size(B, cs)
            assert m.plan(B)["cluster_size"] == cs
            check(m, codes, x[:B])
            y1 = m.gemv(G.x_dev(x[:B]))
            y2 = m.gemv(G.x_dev(x[:B]))
            torch.cuda.synchronize()
            assert torch.equal(y1, y2)  # fixed summation order
    m.check()
    m.close()


def test_decoder_projections_sampled_rows():
    for rows, cols in ((512, 3584), (3584, 3584), (3584, 18944), (18944, 3584)):
        codes, x = inp.random_codes_dim(16, 2, rows, cols, seed=57 + rows % 89 + cols % 97, B=8)
        m = make16(codes)
        rs = G.sample_rows(rows, 96, seed=rows)
        assert np.array_equal(G.decoded_bits(m, rs), ref_decode(codes, rs))
        for B in (1, 8):
            check(m, codes, x[:B], rs)
        m.check()
        m.close()
        torch.cuda.empty_cache()


def test_8192_square_every_row_and_bytes():
    n = 8192
    codes, x = inp.random_codes_dim(16, 2, n, n, seed=58, B=4)
    m = make16(codes)
    for B in (1, 4):
        check(m, codes, x[:B])
    # 34 bits per 16-D vector + 4 B per 128 weights + the 512 KiB codebook + x and y
    assert m.bytes(1) == n * n // 16 * 34 // 8 + n * (n // 128) * 4 + K16 * 32 + 2 * (n + n)
    m.check()
    m.close()


def test_host_path_no_alloc_export_import():
    rows, cols, B = 700, 1536, 5
    codes, x = inp.random_codes_dim(16, 2, rows, cols, seed=59, B=B)
    m = make16(codes)
    xd = G.x_dev(x)
    y_dev = m.gemv(xd)
    xh = torch.from_numpy(x.view(np.int16)).view(torch.float16).pin_memory()
    yh = torch.empty((B, rows), dtype=torch.float16).pin_memory()
    m.gemv_host(xh, yh)
    y_na = torch.empty((B, rows), dtype=torch.float16, device="cuda")
    m.gemv_noalloc(xd, y_na)
    torch.cuda.synchronize()
    assert torch.equal(y_dev.cpu().view(torch.int16), yh.view(torch.int16))
    assert torch.equal(y_dev.view(torch.int16), y_na.view(torch.int16))
    check(m, codes, x, y=y_dev)
    m2 = SphqMatrix.from_blob(m.export())
    assert m2.dim == 16
    assert torch.equal(m2.gemv(xd).view(torch.int16), y_dev.view(torch.int16))
    m.close()
    m2.close()


def test_graph_capture_with_pdl():
    codes, x = inp.random_codes_dim(16, 2, 512, 1024, seed=60, B=2)
    mats = [make16(codes) for _ in range(3)]
    xd = G.x_dev(x)
    ys = [torch.empty((2, 512), dtype=torch.float16, device="cuda") for _ in mats]
    ref = mats[0].gemv(xd)
    torch.cuda.synchronize()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for m, y in zip(mats, ys):
            m.gemv(xd, y=y, stream=s)
    g.replay()
    torch.cuda.synchronize()
    for y in ys:
        assert torch.equal(y.view(torch.int16), ref.view(torch.int16))
    for m in mats:
        m.close()


def test_code_validation_and_unsupported_entry_points():
    codes, x = inp.random_codes_dim(16, 2, 32, 256, seed=61)
    m = make16(codes, pack=False)
    for key, val in (("idx", K16), ("rcode", 16)):
        bad = {k: getattr(codes, k).copy() for k in ("sign", "idx", "rcode")}
        bad[key][3, 5] = val
        with pytest.raises(SphqError) as e:
            m.pack(G.to_dev(bad["sign"]), G.to_dev(bad["idx"]), G.to_dev(bad["rcode"]))
        assert e.value.status == 1
    with pytest.raises(ValueError):  # 16 sign bits need 2-byte signs
        m.pack(G.to_dev(codes.sign.astype(np.uint8)), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    check(m, codes, x)
    with pytest.raises(SphqError) as e:
        m.gemm(G.x_dev(np.zeros((16, 256), np.uint16)))
    assert e.value.status == 2
    with pytest.raises(SphqError):
        m.set_cluster_size(12, 1)  # batches above 8 are two launches
    m.close()
    # the W2 allocation only: K = 2^14, 2 bits, 4 radius bits
    sc = inp.to_f16_bits(np.ones((16, 1)))
    cb = inp.to_f16_bits(np.full((1 << 13, 16), 0.25))
    with pytest.raises(SphqError) as e:
        SphqMatrix(16, 128, 2, G.to_dev(cb), G.to_dev(sc), G.to_dev(sc), K=1 << 13, dim=16)
    assert e.value.status == 2
