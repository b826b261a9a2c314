"""Pins of the reference encoder (Eqs. (3), (5), (6), (7)) used to produce the
encoded configuration's codes: brute-force argmax, the least-squares radius's
orthogonality, the radius quantisation bound, sign consistency and the
degenerate cases (zero vectors, constant groups)."""
import numpy as np
import pytest

import oracle
import sphq_inputs as inp


@pytest.fixture(scope="module")
def encoded():
    rows, cols = 24, 512
    w = inp.gaussian_weights(rows, cols, seed=101)
    cb, _ = inp.encoded_inputs_rng(2, cols, seed=101)
    return w, cb, oracle.encode(w, cb)


def test_argmax_is_true_argmax(encoded):
    w, cb, e = encoded
    C = oracle.half_to_double(cb)
    _, _, _, d = oracle.decompose(w.reshape(24, -1, 8))
    for i in range(0, 24, 5):
        for t in range(0, 64, 7):
            scores = [sum(d[i, t, j] * C[k, j] for j in range(8)) for k in range(C.shape[0])]
            best = max(scores)
            # the chosen entry attains the maximum cosine (up to summation order)
            assert scores[int(e["idx"][i, t])] >= best - 1e-12


def test_least_squares_radius(encoded):
    w, cb, e = encoded
    C = oracle.half_to_double(cb)
    wp = np.abs(w.reshape(24, -1, 8))
    c = C[e["idx"].astype(np.int64)]
    rt = e["r_tilde"]
    # Eq. (6): r_tilde = <w_+, c_z>
    assert np.allclose(rt, np.sum(wp * c, axis=-1), rtol=1e-14)
    # the residual w_+ - r_tilde c_z is orthogonal to c_z up to ||c_z|| != 1 by fp16 rounding
    res = np.sum((wp - rt[..., None] * c) * c, axis=-1)
    nrm = np.sum(c * c, axis=-1)
    assert np.all(np.abs(res) <= np.abs(rt * (1 - nrm)) + 1e-12)


def test_radius_quantisation_bound(encoded):
    w, cb, e = encoded
    D = oracle.half_to_double(e["scale"])[:, np.arange(64) // 16]
    M = oracle.half_to_double(e["offset"])[:, np.arange(64) // 16]
    q = e["rcode"].astype(np.float64)
    rt = e["r_tilde"]
    assert e["rcode"].max() <= 15
    rhat = M + q * D
    inside = (rt >= M) & (rt <= M + 15 * D)
    # Eq. (7): nearest level, so the error is at most half a step (plus the
    # binary16 rounding of Delta and r_min)
    assert np.all(np.abs(rhat - rt)[inside] <= D[inside] / 2 + 1e-12)
    # every group minimum maps to level 0 or 1 (r_min is rounded to fp16)
    g = rt.reshape(24, 4, 16)
    qg = e["rcode"].reshape(24, 4, 16)
    amin = np.argmin(g, axis=-1)
    assert np.all(np.take_along_axis(qg, amin[..., None], -1) <= 1)


def test_signs_match_weights(encoded):
    w, cb, e = encoded
    dec = oracle.half_to_double(oracle.decode(cb, e["scale"], e["offset"], e["sign"],
                                              e["idx"], e["rcode"]))
    nz = (dec != 0) & (w != 0)
    assert np.array_equal(np.signbit(dec)[nz], (w < 0)[nz])


def test_reconstruction_error_is_bounded(encoded):
    w, cb, e = encoded
    dec = oracle.half_to_double(oracle.decode(cb, e["scale"], e["offset"], e["sign"],
                                              e["idx"], e["rcode"]))
    err = np.linalg.norm(dec - w) / np.linalg.norm(w)
    assert err < 0.9
    # reconstructing with the unquantised least-squares radius is at least as good
    # as with the quantised one, block by block in aggregate
    C = oracle.half_to_double(cb)[e["idx"].astype(np.int64)]
    s = np.where(w.reshape(24, -1, 8) < 0, -1.0, 1.0)
    ls = (e["r_tilde"][..., None] * s * C).reshape(w.shape)
    assert np.linalg.norm(ls - w) <= np.linalg.norm(dec - w) * (1 + 1e-9)


def test_degenerate_zero_vectors_and_constant_groups():
    cb, _ = inp.encoded_inputs_rng(2, 128, seed=5)
    w = np.zeros((2, 128))
    e = oracle.encode(w, cb)
    assert np.all(e["idx"] == 0)          # d = 0 scores 0 everywhere: lowest index
    assert np.all(e["rcode"] == 0)        # Delta = 0 -> q = 0
    assert np.all(e["scale"] == 0) and np.all(e["offset"] == 0)
    dec = oracle.decode(cb, e["scale"], e["offset"], e["sign"], e["idx"], e["rcode"])
    assert np.all(oracle.half_to_double(dec) == 0)
    # sign(0) is + : no sign bit for zero coordinates, including -0.0
    e2 = oracle.encode(-np.zeros((1, 128)), cb)
    assert np.all(e2["sign"] == 0)
