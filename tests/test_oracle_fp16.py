"""Pins of the oracle's IEEE binary16 layer against things other than itself:
numpy's independent float16 conversions, the rounding definition checked by
brute force on neighbours, and hand-derived fixtures (tests/golden)."""
import os

import numpy as np
import pytest

import oracle

GOLDEN = os.path.join(os.path.dirname(__file__), "golden")


def _read_rounding_fixture():
    rows = []
    with open(os.path.join(GOLDEN, "fp16_rounding.txt")) as f:
        for line in f:
            if line.startswith("#") or not line.strip():
                continue
            parts = line.split()
            rows.append((float.fromhex(parts[0]), int(parts[1], 16)))
    return rows


def test_half_to_double_all_patterns_match_numpy():
    bits = np.arange(1 << 16, dtype=np.uint32).astype(np.uint16)
    ours = oracle.half_to_double(bits)
    ref = bits.view(np.float16).astype(np.float64)
    nan = np.isnan(ref)
    assert np.array_equal(np.isnan(ours), nan)
    assert np.array_equal(ours[~nan], ref[~nan])
    # signed zeros keep their sign
    assert np.signbit(ours[0x8000]) and not np.signbit(ours[0])


def test_rounding_fixture():
    for v, expected in _read_rounding_fixture():
        got = int(oracle.round_half(np.array([v]))[0])
        assert got == expected, f"{v!r}: got 0x{got:04X} expected 0x{expected:04X}"


def _random_doubles(rng, n):
    # magnitudes from deep underflow to past overflow, both signs
    e = rng.uniform(-30, 17, size=n)
    m = rng.uniform(1, 2, size=n)
    s = rng.choice([-1.0, 1.0], size=n)
    return s * m * np.exp2(np.floor(e))


def _midpoints(rng, n):
    # exact midpoints between consecutive finite binary16 values (ties)
    h = rng.integers(0, 0x7BFF, size=n).astype(np.uint16)
    a = h.view(np.float16).astype(np.float64)
    b = (h + 1).astype(np.uint16).view(np.float16).astype(np.float64)
    return (a + b) / 2.0  # exact in float64


def test_round_half_matches_numpy_conversion():
    rng = np.random.default_rng(1)
    v = np.concatenate([_random_doubles(rng, 400_000), _midpoints(rng, 100_000),
                        -_midpoints(rng, 50_000)])
    ours = oracle.round_half(v)
    with np.errstate(over="ignore"):
        ref = v.astype(np.float16).view(np.uint16)
    bad = np.nonzero(ours != ref)[0]
    assert bad.size == 0, [(v[i], hex(ours[i]), hex(ref[i])) for i in bad[:5]]


def test_round_half_is_nearest_ties_even_by_definition():
    """Independent of numpy's conversion: the result is at least as close as both
    binary16 neighbours, and on a tie its significand is even."""
    rng = np.random.default_rng(2)
    v = np.abs(np.concatenate([_random_doubles(rng, 20_000), _midpoints(rng, 5_000)]))
    v = v[v < 65504.0]
    h = oracle.round_half(v).astype(np.int64)
    val = oracle.half_to_double(h.astype(np.uint16))
    up = oracle.half_to_double(np.minimum(h + 1, 0x7BFF).astype(np.uint16))
    dn = oracle.half_to_double(np.maximum(h - 1, 0).astype(np.uint16))
    err = np.abs(v - val)
    assert np.all(err <= np.abs(v - up))
    assert np.all(err <= np.abs(v - dn))
    tie = (err == np.abs(v - up)) & (h != 0x7BFF) | (err == np.abs(v - dn)) & (h != 0)
    tie &= err > 0
    assert np.all(h[tie] % 2 == 0)


def test_round_half_overflow_and_signed_zero():
    v = np.array([65519.99, 65520.0, 1e6, -1e6, -0.0, 0.0, np.inf, -np.inf])
    h = oracle.round_half(v)
    assert list(h) == [0x7BFF, 0x7C00, 0x7C00, 0xFC00, 0x8000, 0x0000, 0x7C00, 0xFC00]
    assert (int(oracle.round_half(np.array([np.nan]))[0]) & 0x7C00) == 0x7C00


@pytest.mark.parametrize("bits", [0x0001, 0x03FF, 0x0400, 0x3C00, 0x7BFF, 0x8001, 0xFBFF])
def test_round_half_identity_on_representable(bits):
    v = oracle.half_to_double(np.array([bits], np.uint16))
    assert int(oracle.round_half(v)[0]) == bits
