"""Pins of the oracle's decode (Eq. (7) radius, Eq. (4) reconstruction) against
numpy's independent float16 rounding, closed-form special cases, the paper's
worked example and hand-derived fixtures."""
import os

import numpy as np
import pytest

import oracle
import sphq_inputs as inp

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _np_decode(codes):
    """Same definition computed through numpy: exact float64 arithmetic and
    numpy's float64 -> float16 conversion (a separate implementation of RN16)."""
    C = codes.codebook.view(np.float16).astype(np.float64)
    D = codes.scale.view(np.float16).astype(np.float64)
    M = codes.offset.view(np.float16).astype(np.float64)
    rows, nv = codes.sign.shape
    g = np.arange(nv) // (inp.GROUP_COLS // inp.VEC)
    q = codes.rcode.astype(np.float64)
    r = (q * D[:, g] + M[:, g]).astype(np.float16).astype(np.float64)   # Eq. (7)
    c = C[codes.idx.astype(np.int64)]                                    # (rows, nv, 8)
    w = (r[..., None] * c).astype(np.float16).view(np.uint16)            # Eq. (4)
    neg = (codes.sign[..., None] >> np.arange(8, dtype=np.uint8)) & 1
    w = w ^ (neg.astype(np.uint16) << 15)
    return w.reshape(rows, nv * 8)


def _decode(codes):
    return oracle.decode(codes.codebook, codes.scale, codes.offset, codes.sign,
                         codes.idx, codes.rcode)


@pytest.mark.parametrize("bits,rows,cols", [(2, 16, 256), (2, 5, 1024), (3, 7, 384)])
def test_decode_matches_numpy_definition(bits, rows, cols):
    codes, _ = inp.random_codes(bits, rows, cols, seed=11 + rows)
    assert np.array_equal(_decode(codes), _np_decode(codes))


def test_decode_matches_numpy_on_wide_parameter_ranges():
    # parameters spanning subnormal to large radii, to exercise every rounding regime
    rng = np.random.default_rng(3)
    codes, _ = inp.random_codes(2, 32, 256, seed=5)
    mag = np.exp2(rng.uniform(-20, 10, size=codes.scale.shape))
    codes.scale = inp.to_f16_bits(mag * rng.uniform(0.5, 1.5, size=mag.shape))
    codes.offset = inp.to_f16_bits(np.exp2(rng.uniform(-24, 10, size=mag.shape)))
    assert np.array_equal(_decode(codes), _np_decode(codes))


def _read_decode_fixture():
    radii, blocks = [], []
    with open(os.path.join(GOLDEN, "decode_examples.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            if line.startswith("R"):
                p = line.split()
                radii.append((int(p[1]), int(p[2], 16), int(p[3], 16), int(p[4], 16)))
            elif line.startswith("W"):
                head, cb, exp = line[1:].split("|")
                h = head.split()
                blocks.append((int(h[0], 16), int(h[1]), int(h[2], 16), int(h[3], 16),
                               [int(t, 16) for t in cb.split()],
                               [int(t, 16) for t in exp.split()]))
    return radii, blocks


def test_radius_fixture():
    radii, _ = _read_decode_fixture()
    assert radii
    for q, d, m, expected in radii:
        assert oracle.radius(q, d, m) == expected, (q, hex(d), hex(m))


def test_block_fixture():
    _, blocks = _read_decode_fixture()
    assert blocks
    for sign, q, d, m, cb, expected in blocks:
        # a one-group matrix whose first vector is the fixture block
        codes = inp.Codes(2, np.array([cb], np.uint16), np.array([[d]], np.uint16),
                          np.array([[m]], np.uint16), np.zeros((1, 16), np.uint8),
                          np.zeros((1, 16), np.uint16), np.zeros((1, 16), np.uint8))
        codes.sign[0, 0] = sign
        codes.rcode[0, 0] = q
        w = _decode(codes)
        assert [int(v) for v in w[0, :8]] == expected


def test_worked_example_radius():
    """§1: (1,...,1) has radius 2*sqrt(2); (1,1,1,1,5,1,1,1) has radius 4*sqrt(2)."""
    with open(os.path.join(GOLDEN, "worked_example_radius.txt")) as f:
        rows = [l.split() for l in f if l.strip() and not l.startswith("#")]
    for r in rows:
        w = np.array([float(t) for t in r[:8]])
        _, wp, radius, d = oracle.decompose(w)
        assert radius == pytest.approx(float(r[8]) * np.sqrt(2), rel=1e-15)
        # the direction is a non-negative unit vector (§3.1: d in S^7_+)
        assert np.all(d >= 0) and np.linalg.norm(d) == pytest.approx(1.0, rel=1e-15)


def test_zero_delta_gives_offset_radius():
    codes, _ = inp.random_codes(2, 8, 256, seed=9)
    codes.scale[:] = 0
    w = oracle.half_to_double(_decode(codes)).reshape(8, -1, 8)
    r = oracle.half_to_double(codes.offset)[:, np.arange(32) // 16]
    C = oracle.half_to_double(codes.codebook)[codes.idx.astype(np.int64)]
    s = 1.0 - 2.0 * ((codes.sign[..., None] >> np.arange(8)) & 1)
    # power-of-two-free check: |w| equals the binary16 rounding of r*c
    expect = oracle.half_to_double(oracle.round_half(r[..., None] * C)) * s
    assert np.array_equal(w, expect)


def test_power_of_two_radius_is_exact():
    """With r_hat = 2^e no product rounds (for normal results): w = s * 2^e * c."""
    codes, _ = inp.random_codes(2, 4, 128, seed=13)
    codes.scale[:] = 0
    codes.offset[:] = 0x4400  # 4.0
    w = oracle.half_to_double(_decode(codes)).reshape(4, -1, 8)
    C = oracle.half_to_double(codes.codebook)[codes.idx.astype(np.int64)]
    s = 1.0 - 2.0 * ((codes.sign[..., None] >> np.arange(8)) & 1)
    normal = np.abs(4.0 * C) >= 2.0 ** -14
    assert np.array_equal(w[normal], (4.0 * C * s)[normal])


def test_sign_bits_and_negative_zero():
    codes, _ = inp.random_codes(2, 2, 128, seed=17)
    codes.codebook[:, 3] = 0            # coordinate 3 of every direction is +0
    codes.sign[:] = 0xFF                # every coordinate negative
    w = _decode(codes).reshape(2, -1, 8)
    assert np.all(w[..., 3] == 0x8000)  # -0 keeps its sign bit
    assert np.all((w >> 15) == 1)
    codes.sign[:] = 0
    w = _decode(codes).reshape(2, -1, 8)
    assert np.all((w >> 15) == 0)


def test_reconstruction_invariants_on_random_codes():
    codes, _ = inp.random_codes(2, 16, 512, seed=21)
    C = oracle.half_to_double(codes.codebook)
    # the generated codebook is a set of positive-orthant unit vectors (§3.1, S^7_+),
    # up to binary16 rounding of each coordinate
    assert np.all(C >= 0)
    assert np.all(np.abs(np.linalg.norm(C, axis=1) - 1) <= 8 * 2.0 ** -11)
    w = oracle.half_to_double(_decode(codes)).reshape(16, -1, 8)
    g = np.arange(64) // 16
    r = oracle.half_to_double(np.array(
        [[oracle.radius(int(q), int(codes.scale[i, gg]), int(codes.offset[i, gg]))
          for q, gg in zip(codes.rcode[i], g)] for i in range(16)], np.uint16))
    c = C[codes.idx.astype(np.int64)]
    s = 1.0 - 2.0 * ((codes.sign[..., None] >> np.arange(8)) & 1)
    # Eq. (4): every block equals r_hat * s (.) c within one binary16 rounding
    assert np.all(np.abs(w - r[..., None] * s * c) <= np.abs(r[..., None] * c) * 2.0 ** -11
                  + 2.0 ** -25)
    # ||w_hat|| ~= r_hat * ||c||
    assert np.allclose(np.linalg.norm(w, axis=-1), r * np.linalg.norm(c, axis=-1),
                       rtol=2e-3, atol=1e-6)
    # signs of nonzero weights are the stored signs
    nz = w != 0
    assert np.array_equal(np.signbit(w)[nz], (s < 0)[nz])


def test_out_of_range_code_is_rejected():
    codes, _ = inp.random_codes(2, 2, 128, seed=3)
    codes.idx[0, 0] = 64
    with pytest.raises(ValueError):
        _decode(codes)
