"""Pins of the single-precision encoder (oracle.encode_fp32: Eqs. (3), (5),
(6), (7) with every decision in IEEE binary32), the reference a GPU encoder
must match bit for bit.

It is pinned to the float64 encoder (itself pinned in test_oracle_encoder.py)
wherever single precision cannot change a decision, and to the special cases
the equations fix: zero vectors, ties (lowest index), exact codebook
directions, negative zero, constant groups.
"""
import numpy as np
import pytest

import oracle
import sphq_inputs as inp


def _cb(K, seed):
    return inp.make_codebook(np.random.Generator(np.random.PCG64(seed)), K)


@pytest.mark.parametrize("K,V", [(64, 4), (8192, 4), (8192, 3), (256, 2)])
def test_agrees_with_float64_encoder_away_from_ties(K, V):
    w = inp.gaussian_weights(24, 512, seed=K + V).astype(np.float32)
    cb = _cb(K, 7 + V)
    e32 = oracle.encode_fp32(w, cb, V)
    e64 = oracle.encode(w.astype(np.float64), cb, V=V)
    assert np.array_equal(e32["sign"], e64["sign"])
    # an index may differ only where the float64 scores of the two choices are
    # within single-precision error of each other
    C = oracle.half_to_double(cb)
    _, _, _, d = oracle.decompose(w.astype(np.float64).reshape(24, -1, 8))
    diff = np.argwhere(e32["idx"] != e64["idx"])
    for i, t in diff:
        s32 = float(d[i, t] @ C[int(e32["idx"][i, t])])
        s64 = float(d[i, t] @ C[int(e64["idx"][i, t])])
        assert s64 - s32 < 1e-5
    assert len(diff) <= 0.001 * e32["idx"].size
    same = (e32["idx"] == e64["idx"]).reshape(24, -1, 16).all(axis=-1)
    assert np.mean(e32["scale"][same] == e64["scale"][same]) > 0.999
    assert np.mean(e32["offset"][same] == e64["offset"][same]) > 0.999


def test_zero_vectors_ties_and_negative_zero():
    cb = _cb(64, 3)
    w = np.zeros((2, 128), np.float32)
    w[1, :8] = -0.0
    e = oracle.encode_fp32(w, cb, 4)
    assert np.all(e["idx"] == 0)          # all scores 0: the lowest index wins
    assert np.all(e["sign"] == 0)         # -0.0 is not negative
    assert np.all(e["rcode"] == 0)        # constant group: Delta = 0 -> q = 0
    assert np.all(e["scale"] == 0) and np.all(e["offset"] == 0)


def test_duplicate_entries_take_the_lowest_index():
    cb = _cb(64, 4)
    cb[40] = cb[9]                        # an exact duplicate of entry 9
    c9 = oracle.half_to_double(cb[9]).astype(np.float32)
    w = np.tile(np.concatenate([c9 * 3.0, -c9 * 0.5]), (1, 8)).astype(np.float32)
    e = oracle.encode_fp32(w, cb, 4)
    assert np.all(e["idx"] == 9)
    assert np.all(e["sign"][0, 1::2] == 0xFF)


def test_exact_directions_and_radius_bound():
    K, V = 8192, 4
    cb = _cb(K, 5)
    rng = np.random.default_rng(0)
    C = oracle.half_to_double(cb)
    ks = rng.choice(K, size=64, replace=False)
    r = rng.uniform(0.1, 2.0, size=64)
    w = (C[ks] * r[:, None]).astype(np.float32).reshape(4, 128)
    e = oracle.encode_fp32(w, cb, V)
    # a vector along an entry picks that entry (entries are distinct here)
    assert np.array_equal(e["idx"].reshape(-1), ks)
    # Eq. (7): the dequantised radius is within half a step (plus fp16 rounding)
    # of r~ = <w+, c_z>
    rt = np.sum(np.abs(w.reshape(-1, 8)) * C[ks], axis=-1).reshape(4, 16)
    D = oracle.half_to_double(e["scale"])
    M = oracle.half_to_double(e["offset"])
    rhat = e["rcode"].astype(np.float64) * D + M
    assert np.all(np.abs(rhat - rt) <= 0.5 * D + 2e-3 * rt + 1e-6)
    assert int(e["rcode"].max()) <= (1 << V) - 1
