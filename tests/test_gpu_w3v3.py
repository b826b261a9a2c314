"""The W3 bit split with 3-bit radius codes (8 + 13 + 3 = 24 bits per 8-D
vector, 3.00 bits per weight; §3.1 and Eq. (7) with V = 3, the 3.00-bit W3
row of Tab. 12) against the float64 oracle through the C ABI.

The decode formula is the one of the V = 4 formats (Eq. (7) then Eq. (4)), so
the oracle's decode applies unchanged; only the code range (q < 8) and the
device layout differ.  Decode is bit-exact, the GEMV within
1e-3 * sum_j |w_hat_j||x_j| + 2^-24 per output.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

V = 3


def codes3(rows, cols, seed, B=1, codebook=None):
    return inp.random_codes(3, rows, cols, seed=seed, B=B, codebook=codebook, radius_bits=V)


@pytest.mark.parametrize("rows,cols", [(1, 128), (31, 256), (33, 384), (100, 1024), (257, 640),
                                       (1000, 2048)])
def test_small_shapes_decode_and_gemv(rows, cols):
    codes, x = codes3(rows, cols, seed=3000 + rows + cols, B=8)
    assert int(codes.rcode.max()) <= 7
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    for B in (1, 2, 3, 5, 8):
        G.check_gemv(m, codes, x[:B])
    m.close()


def test_edge_codes():
    rows, cols = 64, 512
    codes, x = codes3(rows, cols, seed=79, B=4)
    K = codes.K
    codes.codebook[: K // 2, 5] = 0          # zero coordinates -> +-0 weights
    codes.sign[:8] = 0xFF
    codes.sign[8:16] = 0
    codes.idx[16:24] = K - 1                 # every index bit set (bits 8-12 in the extra bytes)
    codes.idx[24:28] = 0x1F00                # only the five high index bits
    codes.idx[28:32] = 0x00FF                # only the eight low index bits
    codes.rcode[32:36] = 7                   # largest radius code
    codes.rcode[36:40] = 0
    codes.scale[40:48] = 0                   # Delta = 0 -> r_hat = r_min
    codes.offset[48:56] = 0                  # r_min = 0
    codes.scale[56:64] = 0x0001              # subnormal Delta
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    G.check_gemv(m, codes, x)
    m.close()


def test_pack_rejects_radius_codes_above_seven():
    codes, x = codes3(32, 256, seed=4)
    m = SphqMatrix(32, 256, 3, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset), radius_bits=V)
    bad = codes.rcode.copy()
    bad[5, 9] = 8
    with pytest.raises(SphqError) as e:
        m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(bad))
    assert e.value.status == 1
    with pytest.raises(SphqError) as e:
        m.gemv(G.x_dev(x))
    assert e.value.status == 3  # left unpacked
    m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    G.check_gemv(m, codes, x)
    m.close()


def test_unsupported_splits_are_refused():
    codes, _ = inp.random_codes(2, 16, 128, seed=1)
    for bits, vb in ((3, 2), (3, 5), (2, 0), (2, 5)):
        cb = codes.codebook if bits == 2 else inp.random_codes(3, 16, 128, seed=1)[0].codebook
        with pytest.raises(SphqError) as e:
            SphqMatrix(16, 128, bits, G.to_dev(cb), G.to_dev(codes.scale),
                       G.to_dev(codes.offset), radius_bits=vb)
        assert e.value.status == 2


def test_bytes_count_three_bits_per_weight():
    rows, cols = 4096, 4096
    codes, _ = codes3(rows, cols, seed=2)
    m = G.make_matrix(codes)
    codes4, _ = inp.random_codes(3, rows, cols, seed=2)
    m4 = G.make_matrix(codes4)
    for B in (1, 8):
        io = 2 * B * (rows + cols)
        params = 4 * rows * (cols // 128)
        cb = 8192 * 16
        assert m.bytes(B) == rows * cols * 3 // 8 + params + cb + io
        assert m.bytes(B) == int(rows * cols * oracle.payload_bits_per_weight(3, V)) // 8 \
            + params + cb + io
        assert m4.bytes(B) - m.bytes(B) == rows * cols // 8 // 8  # one bit per vector less
    m.close()
    m4.close()


def test_every_cluster_size():
    codes, x = codes3(1000, 1024, seed=31, B=5)
    m = G.make_matrix(codes)
    for cs in (1, 2, 4, 8):
        for B in (1, 2, 5):
            m.set_cluster_size(B, cs)
            assert m.plan(B)["cluster_size"] == cs
            G.check_gemv(m, codes, x[:B])
    m.close()


@pytest.mark.parametrize("n", [4096, 8192])
def test_encoded_square(n):
    # Sampled rows carry codes from the oracle's encoder at V = 3 (Gaussian
    # weights with outliers); the other rows are seeded random V = 3 codes.
    seed = inp.seed_for(1, 10 + n // 4096)
    rs = G.sample_rows(n, 128, seed=n + 33)
    w = inp.gaussian_weights(n, n, seed=seed)[rs]
    cb, x = inp.encoded_inputs_rng(3, n, seed=seed, B=8)
    e = oracle.encode(w, cb, V=V, chunk=4096)
    assert int(e["rcode"].max()) <= 7
    codes, _ = codes3(n, n, seed=seed + 1, codebook=cb)
    for key in ("sign", "idx", "rcode", "scale", "offset"):
        getattr(codes, key)[rs] = e[key]
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
    for B in (1, 2, 4, 8):
        G.check_gemv(m, codes, x[:B], rs)
    m.close()


def test_decoder_projections_batch1_and_4():
    for name, rows, cols in inp.DECODER_PROJ_FUSED:
        codes, x = codes3(rows, cols, seed=500 + rows + cols, B=4)
        rs = G.sample_rows(rows, 96, seed=rows)
        m = G.make_matrix(codes)
        assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
        for B in (1, 4):
            G.check_gemv(m, codes, x[:B], rs)
        m.close()


def test_deterministic_and_graph_capturable():
    codes, x = codes3(3584, 3584, seed=22, B=2)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y1 = m.gemv(xd).clone()
    torch.cuda.synchronize()
    y = torch.empty((2, 3584), dtype=torch.float16, device=G.DEV)
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        m.gemv(xd, y, stream=s)                  # warm up outside capture
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        m.gemv(xd, y, stream=s)
    y.zero_()
    g.replay()
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y.view(torch.int16))
    m.close()
