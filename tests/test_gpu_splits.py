"""The small-codebook bit splits of Tab. 4 (8 sign bits / D-bit direction
index, K = 2^D / V-bit radius code: 8/6/2, 8/6/3, 8/7/2, 8/8/2, plus 8/7/3,
and the W2 split 8/6/4 itself) against the float64 oracle through the C ABI.

Decode follows Eq. (7) and Eq. (4) for every split, so the oracle's decode
applies unchanged with the split's codebook size and code range.  Decode is
bit-exact; the GEMV stays within 1e-3 * sum_j |w_hat_j||x_j| + 2^-24.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

# (direction index bits D, radius bits V)
SPLITS = [(6, 2), (6, 3), (7, 2), (7, 3), (8, 2), (6, 4)]
IDS = [f"8-{d}-{v}" for d, v in SPLITS]


def codes_for(d, v, rows, cols, seed, B=1, codebook=None):
    return inp.random_codes(2, rows, cols, seed=seed, B=B, codebook=codebook, radius_bits=v,
                            K=1 << d)


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
@pytest.mark.parametrize("rows,cols", [(1, 128), (33, 384), (257, 640), (1000, 2048)])
def test_small_shapes_decode_and_gemv(d, v, rows, cols):
    codes, x = codes_for(d, v, rows, cols, seed=7000 + 10 * d + v + rows + cols, B=8)
    assert codes.K == 1 << d and int(codes.rcode.max()) < 1 << v
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    for B in (1, 2, 3, 8):
        G.check_gemv(m, codes, x[:B])
    m.close()


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
def test_edge_codes(d, v):
    rows, cols = 64, 512
    codes, x = codes_for(d, v, rows, cols, seed=90 + 10 * d + v, B=4)
    K = codes.K
    codes.codebook[: K // 2, 5] = 0          # zero coordinates -> +-0 weights
    codes.sign[:8] = 0xFF                    # every sign bit, incl. the pairs kept in records
    codes.sign[8:12] = 0xC0                  # only sign bits 6, 7
    codes.sign[12:16] = 0x3F
    codes.idx[16:24] = K - 1                 # every index bit
    codes.rcode[24:32] = (1 << v) - 1        # largest radius code
    codes.rcode[32:40] = 0
    codes.scale[40:48] = 0                   # Delta = 0 -> r_hat = r_min
    codes.offset[48:56] = 0                  # r_min = 0
    codes.scale[56:64] = 0x0001              # subnormal Delta
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    G.check_gemv(m, codes, x)
    m.close()


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
def test_out_of_range_codes_rejected(d, v):
    codes, x = codes_for(d, v, 32, 256, seed=5 + d + v)
    m = SphqMatrix(32, 256, 2, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset), radius_bits=v, K=1 << d)
    bad_r = codes.rcode.copy()
    bad_r[3, 4] = 1 << v
    bad_k = codes.idx.copy()
    bad_k[7, 1] = 1 << d
    for sg, ix, rc in ((codes.sign, codes.idx, bad_r), (codes.sign, bad_k, codes.rcode)):
        with pytest.raises(SphqError) as e:
            m.pack(G.to_dev(sg), G.to_dev(ix), G.to_dev(rc))
        assert e.value.status == 1
    m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    G.check_gemv(m, codes, x)
    m.close()


def test_unsupported_splits_refused():
    for d, v in ((7, 4), (8, 3), (8, 4), (5, 2), (9, 2), (6, 1), (6, 5)):
        K = 1 << d
        cb = inp.to_f16_bits(np.full((K, 8), 0.25))
        sc = inp.to_f16_bits(np.ones((16, 1)))
        with pytest.raises(SphqError) as e:
            SphqMatrix(16, 128, 2, G.to_dev(cb), G.to_dev(sc), G.to_dev(sc), radius_bits=v, K=K)
        assert e.value.status == 2


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
def test_bytes_follow_the_split(d, v):
    rows, cols = 2048, 4096
    codes, _ = codes_for(d, v, rows, cols, seed=3)
    m = G.make_matrix(codes)
    for B in (1, 8):
        payload = rows * cols * (8 + d + v) // 64
        assert payload == int(rows * cols * oracle.split_bits_per_weight(d, v)) // 8
        assert m.bytes(B) == payload + 4 * rows * (cols // 128) + (1 << d) * 16 + 2 * B * (rows + cols)
    m.close()


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
def test_every_cluster_size(d, v):
    codes, x = codes_for(d, v, 1000, 1024, seed=40 + d + v, B=5)
    m = G.make_matrix(codes)
    for cs in (1, 2, 4, 8):
        for B in (1, 2, 5):
            m.set_cluster_size(B, cs)
            assert m.plan(B)["cluster_size"] == cs
            G.check_gemv(m, codes, x[:B])
    m.close()


@pytest.mark.parametrize("d,v", SPLITS, ids=IDS)
def test_encoded_square_4096(d, v):
    # Sampled rows carry codes from the oracle's encoder (Gaussian weights with
    # outliers, a K-entry codebook, V-bit radius codes); the other rows random.
    n = 4096
    seed = inp.seed_for(1, 20 + 10 * d + v)
    rs = G.sample_rows(n, 96, seed=n + d + v)
    w = inp.gaussian_weights(n, n, seed=seed)[rs]
    rng = np.random.Generator(np.random.PCG64(seed))
    cb = inp.make_codebook(rng, 1 << d)
    x = inp.make_x(rng, 8, n)
    e = oracle.encode(w, cb, V=v, chunk=4096)
    assert int(e["rcode"].max()) < 1 << v and int(e["idx"].max()) < 1 << d
    codes, _ = codes_for(d, v, n, n, seed=seed + 1, codebook=cb)
    for key in ("sign", "idx", "rcode", "scale", "offset"):
        getattr(codes, key)[rs] = e[key]
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
    for B in (1, 2, 8):
        G.check_gemv(m, codes, x[:B], rs)
    m.close()


def test_gate_projection_batch1_and_4():
    rows, cols = 18944, 3584
    for d, v in SPLITS[:-1]:
        codes, x = codes_for(d, v, rows, cols, seed=600 + 10 * d + v, B=4)
        rs = G.sample_rows(rows, 64, seed=rows + d)
        m = G.make_matrix(codes)
        assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
        for B in (1, 4):
            G.check_gemv(m, codes, x[:B], rs)
        m.close()
        torch.cuda.empty_cache()
