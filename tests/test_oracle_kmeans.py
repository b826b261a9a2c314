"""Pins of the oracle's radius-weighted sampling and spherical k-means step
(§3.1: directions drawn with probability proportional to r^2, assignment by
largest cosine, Eq. (5); centres the normalised means of their members)."""
import numpy as np

import oracle


def _brute_step(D, C):
    S, K = D.shape[0], C.shape[0]
    z, best = [], []
    for i in range(S):
        bk, bs = 0, None
        for k in range(K):
            s = 0.0
            for j in range(8):
                s = s + D[i, j] * C[k, j] if j else D[i, 0] * C[k, 0]
            if bs is None or s > bs:
                bk, bs = k, s
        z.append(bk)
        best.append(bs)
    out = C.copy()
    for k in range(K):
        m = [i for i in range(S) if z[i] == k]
        if not m:
            continue
        v = np.zeros(8)
        for i in m:
            v = v + D[i]
        out[k] = v / np.sqrt(np.sum(v * v))
    return out, np.array(z), float(np.mean(best))


def test_kmeans_step_matches_brute_force():
    rng = np.random.default_rng(3)
    D = np.abs(rng.standard_normal((40, 8)))
    D /= np.linalg.norm(D, axis=1, keepdims=True)
    C = np.abs(rng.standard_normal((6, 8)))
    C /= np.linalg.norm(C, axis=1, keepdims=True)
    C[5] = 0.0  # a centre nothing is closest to keeps its value
    C[5, 0] = -1.0
    got = oracle.kmeans_step(D, C, chunk=7)
    ref = _brute_step(D, C)
    assert np.array_equal(got[1], ref[1])
    assert np.allclose(got[0], ref[0], rtol=0, atol=1e-15)
    assert abs(got[2] - ref[2]) < 1e-15
    assert np.array_equal(got[0][5], C[5])  # empty cluster unchanged


def test_kmeans_step_hand_case():
    # two centres on the axes; samples on either side of the diagonal
    e0, e1 = np.eye(8)[0], np.eye(8)[1]
    a = np.array([3.0, 1.0, 0, 0, 0, 0, 0, 0]) / np.sqrt(10.0)
    b = np.array([1.0, 3.0, 0, 0, 0, 0, 0, 0]) / np.sqrt(10.0)
    d = np.array([1.0, 1.0, 0, 0, 0, 0, 0, 0]) / np.sqrt(2.0)  # tie: lowest index
    C, z, obj = oracle.kmeans_step(np.stack([a, b, d, e0]), np.stack([e0, e1]))
    assert list(z) == [0, 1, 0, 0]
    s0 = a + d + e0
    assert np.allclose(C[0], s0 / np.linalg.norm(s0), atol=1e-15)
    assert np.allclose(C[1], b, atol=1e-15)
    assert abs(obj - (3 / np.sqrt(10) + 3 / np.sqrt(10) + 1 / np.sqrt(2) + 1) / 4) < 1e-15


def test_sample_directions_inverse_transform_hand_case():
    # radii^2 1, 0, 3 (exact in binary): P = [1, 1, 4], total 4
    w = np.zeros((1, 24), np.float32)
    w[0, 0] = 1.0
    w[0, 16:19] = [-1.0, 1.0, 1.0]
    u = np.array([0.0, 0.2, 0.25, 0.24999999, 0.5, 0.999999])
    d, idx = oracle.sample_directions(w, u)
    # a pick is the first P_i > u * 4: u = 0.25 lands exactly on P_0 = P_1 = 1
    # and goes past both (vector 1 has zero radius and is never drawn)
    assert list(idx) == [0, 0, 2, 0, 2, 2]
    assert np.array_equal(d[0], np.eye(8)[0])
    ref = np.array([1.0, 1.0, 1.0, 0, 0, 0, 0, 0]) / np.sqrt(3.0)
    assert np.array_equal(d[2], ref)
    assert np.all(d >= 0)


def test_sample_directions_top_of_range():
    # radii^2 1, 2, 0: P = [1, 3, 3], total 3.  The largest double below 1,
    # u = 1 - 2^-53, gives u * 3 = 3 - 3 * 2^-53, which rounds to 3 - 2^-51
    # (spacing 2^-51 on [2, 4)): still below the total, so the pick is the
    # first P_i above it, index 1, never the zero-radius vector 2.  u = 1
    # itself reaches the total and takes the same last nonzero vector.
    u_top = 1.0 - 2.0 ** -53
    assert u_top * 3.0 == 3.0 - 2.0 ** -51
    w = np.zeros((1, 24), np.float32)
    w[0, 0] = 1.0
    w[0, 8:10] = [1.0, -1.0]
    d, idx = oracle.sample_directions(w, np.array([u_top, 1.0, 0.5, 1.0 / 3.0]))
    # 0.5 * 3 = 1.5 lies in [P_0, P_1); (1/3) * 3 rounds to exactly 1 = P_0
    assert list(idx) == [1, 1, 1, 1]
    assert np.array_equal(d[0], np.array([1.0, 1.0, 0, 0, 0, 0, 0, 0]) / np.sqrt(2.0))
    # a trailing zero-radius vector after a total that is a power of two:
    # P = [1, 2, 2]; 2 * (1 - 2^-53) = 2 - 2^-52 is exact and below 2
    w[0, 8:10] = [1.0, 0.0]
    _, idx = oracle.sample_directions(w, np.array([u_top, 1.0]))
    assert list(idx) == [1, 1]


def test_sample_directions_frequencies_follow_squared_radius():
    rng = np.random.default_rng(11)
    w = (rng.standard_normal((1, 40)) * np.array([1, 1, 1, 1, 1, 1, 1, 1] * 5)).astype(np.float32)
    w[0, 8:16] *= 3.0   # vector 1 nine times the weight of a unit-scale vector
    w[0, 24:32] = 0.0   # vector 3 never drawn
    r2 = np.sum(w.astype(np.float64).reshape(5, 8) ** 2, axis=1)
    n = 200000
    _, idx = oracle.sample_directions(w, rng.random(n))
    counts = np.bincount(idx, minlength=5)
    assert counts[3] == 0
    expect = n * r2 / r2.sum()
    chi2 = np.sum((counts - expect) ** 2 / np.where(expect > 0, expect, 1))
    assert chi2 < 25.0  # 4 degrees of freedom; far in the tail if the weights were wrong


def test_sampled_directions_are_unit_and_nonnegative():
    rng = np.random.default_rng(5)
    w = rng.standard_normal((16, 64)).astype(np.float32)
    d, idx = oracle.sample_directions(w, rng.random(500))
    assert np.all(d >= 0)
    assert np.allclose(np.linalg.norm(d, axis=1), 1.0, atol=1e-15)
    v = np.abs(w.reshape(-1, 8)[idx].astype(np.float64))
    assert np.allclose(d * np.linalg.norm(v, axis=1, keepdims=True), v, atol=1e-15)
