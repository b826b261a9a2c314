"""sphq_encode, the GPU encoder (§3.1: Eqs. (3), (5), (6), (7)), against the
single-precision oracle encoder (oracle.encode_fp32): sign bits, direction
indices, radius codes and group parameters bit for bit, for every codebook
size, on Gaussian weights with outliers and on the degenerate cases (zero
vectors, ties between duplicate entries, vectors along an entry), with ragged
vector counts; the packed result then decodes as the oracle decodes the
oracle's codes."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

# (bits, radius bits, K)
FORMATS = [(2, 4, 64), (3, 4, 8192), (3, 3, 8192), (2, 2, 256), (2, 3, 128)]
FIDS = ["W2", "W3", "W3V3", "8-8-2", "8-7-3"]


def _codebook(K, seed):
    return inp.make_codebook(np.random.Generator(np.random.PCG64(seed)), K)


def _matrix(bits, v, K, rows, cols, cb):
    ng = cols // 128
    ones = inp.to_f16_bits(np.ones((rows, ng)))
    return SphqMatrix(rows, cols, bits, G.to_dev(cb), G.to_dev(ones), G.to_dev(ones),
                      radius_bits=v, K=K)


def _check(m, w, cb, v, rows=None):
    wd = torch.from_numpy(w).to(G.DEV)
    sign, idx, rcode, scale, offset = m.encode(wd)
    torch.cuda.synchronize()
    got = dict(sign=sign.cpu().numpy(), idx=idx.cpu().numpy().view(np.uint16),
               rcode=rcode.cpu().numpy(), scale=scale.cpu().numpy().view(np.uint16),
               offset=offset.cpu().numpy().view(np.uint16))
    sel = slice(None) if rows is None else rows
    ref = oracle.encode_fp32(w[sel], cb, v)
    for key in ("sign", "idx", "rcode", "scale", "offset"):
        a, b = got[key][sel], ref[key]
        assert np.array_equal(a, b), f"{key}: {int(np.sum(a != b))} of {a.size} differ"
    return got


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
def test_gaussian_weights_bit_exact_and_decodable(fmt):
    bits, v, K = fmt
    rows, cols = 48, 1024
    cb = _codebook(K, 3 + K + v)
    w = inp.gaussian_weights(rows, cols, seed=K + v).astype(np.float32)
    m = _matrix(bits, v, K, rows, cols, cb)
    got = _check(m, w, cb, v)
    # the handle is packed with the encoded codes and parameters
    codes = inp.Codes(bits, cb, got["scale"], got["offset"], got["sign"], got["idx"],
                      got["rcode"], v)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    _, x = inp.random_codes(bits, 16, cols, seed=1, B=2)
    G.check_gemv(m, codes, x)
    m.check()
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:2], ids=FIDS[:2])
def test_degenerate_vectors_and_ragged_counts(fmt):
    bits, v, K = fmt
    rows, cols = 33, 384                       # 1584 vectors: not a multiple of 128
    cb = _codebook(K, 9)
    cb[K - 1] = cb[5]                          # a duplicate entry: ties -> index 5
    C = oracle.half_to_double(cb)
    rng = np.random.default_rng(2)
    w = inp.gaussian_weights(rows, cols, seed=4).astype(np.float32)
    w[0] = 0.0                                 # zero vectors (every score ties)
    w[1, :8] = -0.0
    w[2] = np.tile(C[5] * 2.5, cols // 8)      # along the duplicated entry
    ks = rng.choice(K - 1, size=cols // 8, replace=False) if K > cols // 8 else \
        rng.choice(K - 1, size=cols // 8)
    w[3] = (C[ks] * rng.uniform(0.5, 2, size=(cols // 8, 1))).reshape(-1)
    w[4] *= 1e-30                              # tiny magnitudes
    m = _matrix(bits, v, K, rows, cols, cb)
    got = _check(m, w, cb, v)
    assert np.all(got["idx"][0] == 0) and np.all(got["idx"][2] == 5)
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:3], ids=FIDS[:3])
def test_4096_square_sampled_rows(fmt):
    bits, v, K = fmt
    n = 4096
    cb = _codebook(K, 11 + v)
    w = inp.gaussian_weights(n, n, seed=inp.seed_for(1, 3)).astype(np.float32)
    m = _matrix(bits, v, K, n, n, cb)
    _check(m, w, cb, v, rows=G.sample_rows(n, 24, seed=n + bits))
    m.close()


def test_argument_errors():
    cb = _codebook(64, 1)
    m = _matrix(2, 4, 64, 16, 128, cb)
    w = torch.zeros((16, 128), dtype=torch.float64, device=G.DEV)
    with pytest.raises(ValueError):
        m.encode(w)
    m.close()


def test_8192_square_w3_sampled_rows():
    # the size `bench.py --report` times (encode), checked on sampled rows
    bits, v, K = 3, 4, 8192
    n = 8192
    cb = _codebook(K, 12)
    w = inp.gaussian_weights(n, n, seed=inp.seed_for(1, 4)).astype(np.float32)
    m = _matrix(bits, v, K, n, n, cb)
    _check(m, w, cb, v, rows=G.sample_rows(n, 12, seed=n))
    m.close()
