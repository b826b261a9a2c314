"""4-D vectors (Tab. 7 at the W2 allocation: 4 sign bits, a 2-bit index into
K = 4 directions, a 4-bit radius code; 2.5 bits per weight) through the C ABI
against the float64 oracle (oracle.decode_dim): decode bit-exact, the GEMV
within 1e-3 * sum_j |w_hat_j||x_j| + 2^-24, batch 1..8, every cluster size,
ragged shapes, code validation, and the entry points that do not take 4-D."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def make4(codes, pack=True):
    m = SphqMatrix(codes.rows, codes.cols, 2, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset), radius_bits=4, K=4, dim=4)
    if pack:
        m.pack(G.to_dev(codes.sign.astype(np.uint8)), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    return m


def ref_decode(codes, rows=None):
    c = codes
    if rows is not None:
        c = inp.CodesDim(4, 2, codes.codebook, codes.scale[rows], codes.offset[rows],
                         codes.sign[rows], codes.idx[rows], codes.rcode[rows])
    return oracle.decode_dim(c.codebook, c.scale, c.offset, c.sign, c.idx, c.rcode)


def check(m, codes, x, rows=None):
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


@pytest.mark.parametrize("rows,cols", [(1, 128), (31, 256), (33, 384), (257, 640), (1000, 2048)])
def test_small_shapes_decode_and_gemv(rows, cols):
    codes, x = inp.random_codes_dim(4, 2, rows, cols, seed=4000 + rows + cols, B=8)
    m = make4(codes)
    assert np.array_equal(G.decoded_bits(m), ref_decode(codes))
    for B in (1, 2, 3, 5, 8):
        check(m, codes, x[:B])
    m.close()


def test_edge_codes():
    codes, x = inp.random_codes_dim(4, 2, 64, 512, seed=44, B=4)
    codes.codebook[:2, 3] = 0                  # zero coordinates -> +-0
    codes.sign[:8] = 15
    codes.sign[8:16] = 0
    codes.idx[16:24] = 3
    codes.rcode[24:32] = 15
    codes.rcode[32:40] = 0
    codes.scale[40:48] = 0
    codes.offset[48:56] = 0
    codes.scale[56:64] = 0x0001
    m = make4(codes)
    assert np.array_equal(G.decoded_bits(m), ref_decode(codes))
    check(m, codes, x)
    m.close()


def test_every_cluster_size():
    codes, x = inp.random_codes_dim(4, 2, 1000, 1024, seed=45, B=5)
    m = make4(codes)
    for cs in (1, 2, 4, 8):
        for B in (1, 2, 5):
            m.set_cluster_size(B, cs)
            assert m.plan(B)["cluster_size"] == cs
            check(m, codes, x[:B])
    m.close()


def test_large_sampled_rows_and_bytes():
    n = 4096
    codes, x = inp.random_codes_dim(4, 2, n, n, seed=46, B=4)
    m = make4(codes)
    rs = G.sample_rows(n, 96, seed=3)
    assert np.array_equal(G.decoded_bits(m, rs), ref_decode(codes, rs))
    for B in (1, 2, 4):
        check(m, codes, x[:B], rs)
    # 10 bits per 4-D vector + 4 B per 128 weights + 32 B codebook + x and y
    assert m.bytes(1) == n * n // 4 * 10 // 8 + n * (n // 128) * 4 + 32 + 2 * (n + n)
    blob = m.export()
    m2 = SphqMatrix.from_blob(blob)
    assert m2.dim == 4
    xd = G.x_dev(x)
    assert torch.equal(m.gemv(xd).view(torch.int16), m2.gemv(xd).view(torch.int16))
    m.close()
    m2.close()


def test_code_validation_and_unsupported_entry_points():
    codes, x = inp.random_codes_dim(4, 2, 32, 256, seed=47)
    m = make4(codes, pack=False)
    for key, val in (("sign", 16), ("idx", 4), ("rcode", 16)):
        bad = {k: getattr(codes, k).copy() for k in ("sign", "idx", "rcode")}
        bad[key][3, 5] = val
        with pytest.raises(SphqError) as e:
            m.pack(G.to_dev(bad["sign"].astype(np.uint8)), G.to_dev(bad["idx"]),
                   G.to_dev(bad["rcode"]))
        assert e.value.status == 1
    m.pack(G.to_dev(codes.sign.astype(np.uint8)), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    check(m, codes, x)
    with pytest.raises(SphqError) as e:
        m.gemm(G.x_dev(np.zeros((16, 256), np.uint16)))
    assert e.value.status == 2
    m.close()


def test_8192_square_sampled_rows():
    n = 8192
    codes, x = inp.random_codes_dim(4, 2, n, n, seed=48, B=4)
    m = make4(codes)
    rs = G.sample_rows(n, 64, seed=5)
    assert np.array_equal(G.decoded_bits(m, rs), ref_decode(codes, rs))
    for B in (1, 4):
        check(m, codes, x[:B], rs)
    m.close()
