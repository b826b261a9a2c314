"""Pins of the decode for 4-D and 16-D vectors (oracle.decode_dim; §3.1 with
k = 4, 16, the configurations of Tab. 7): it reduces to the pinned 8-D decode
for k = 8, and gives the closed-form values of Eq. (7) / Eq. (4) on exactly
representable inputs; the bit budget of Tab. 7 (codebook bytes) is pinned in
tests/golden/bit_budget.txt."""
import numpy as np
import pytest

import oracle
import sphq_inputs as inp


def test_dim8_reduces_to_the_8d_decode():
    codes, _ = inp.random_codes(2, 40, 512, seed=9)
    w8 = oracle.decode(codes.codebook, codes.scale, codes.offset, codes.sign, codes.idx,
                       codes.rcode)
    wd = oracle.decode_dim(codes.codebook, codes.scale, codes.offset,
                           codes.sign.astype(np.uint16), codes.idx, codes.rcode)
    assert np.array_equal(w8, wd)


@pytest.mark.parametrize("dim", [4, 16])
def test_closed_form(dim):
    # c = (1, 1/2, 1/4, ..., 2^-(dim-1)) (exact), Delta = 1/4, r_min = 1, q = 4:
    # r_hat = 2 exactly; w_hat_j = 2^(1-j), negated where the sign bit is set
    K = 4
    c = np.zeros((K, dim))
    c[2] = [2.0 ** -j for j in range(dim)]
    cb = inp.to_f16_bits(c)
    rows, cols = 1, 128
    nv = cols // dim
    scale = inp.to_f16_bits(np.full((rows, 1), 0.25))
    offset = inp.to_f16_bits(np.full((rows, 1), 1.0))
    sign = np.zeros((rows, nv), np.uint16)
    sign[0, 0] = 0b0101 | (1 << (dim - 1))
    idx = np.full((rows, nv), 2, np.uint16)
    rcode = np.full((rows, nv), 4, np.uint8)
    w = oracle.half_to_double(oracle.decode_dim(cb, scale, offset, sign, idx, rcode)).reshape(-1)
    expect = np.array([2.0 ** (1 - j) for j in range(dim)])
    assert np.array_equal(w[dim:2 * dim], expect)            # vector 1: no signs
    e0 = expect.copy()
    e0[[0, 2, dim - 1]] *= -1
    assert np.array_equal(w[:dim], e0)
    # V = 4: q = 16 is out of range
    rcode[0, 3] = 16
    with pytest.raises(ValueError):
        oracle.decode_dim(cb, scale, offset, sign, idx, rcode)


def test_radius_groups_span_128_scalars():
    dim = 4
    cb = inp.to_f16_bits(np.full((4, dim), 0.5))
    rows, cols = 1, 256
    nv = cols // dim
    scale = inp.to_f16_bits(np.array([[1.0, 2.0]]))
    offset = inp.to_f16_bits(np.array([[0.0, 0.0]]))
    z = np.zeros((rows, nv), np.uint16)
    w = oracle.half_to_double(oracle.decode_dim(cb, scale, offset, z, z,
                                                np.ones((rows, nv), np.uint8)))
    assert np.all(w[0, :128] == 0.5) and np.all(w[0, 128:] == 1.0)


def test_budget_of_the_dimensions():
    # (dim - 1) B - dim index bits at B = 2: 2 (4-D), 6 (8-D), 14 (16-D)
    assert [oracle.direction_index_bits(2, d) for d in (4, 8, 16)] == [2, 6, 14]
    assert oracle.payload_bits_per_weight(2, 4, dim=4) == 2.5
    assert oracle.payload_bits_per_weight(2, 4, dim=16) == 2.125
