"""Pins of the quantize-side codebook constructions in the oracle: the
angle-parameterised codebook of §3.3 (Eqs. sph-angle-codebook /
sph-angle-logits) and the radius-weighted spherical k-means of §3.1."""
import numpy as np

import oracle


def test_angle_codebook_is_nonnegative_and_unit_norm():
    rng = np.random.default_rng(1)
    phi = np.concatenate([rng.normal(0, 3, (4096, 7)), np.full((2, 7), 50.0), np.full((2, 7), -50.0)])
    c = oracle.angle_codebook(phi)
    assert c.shape == (4100, 8)
    assert np.all(c >= 0)
    assert np.allclose(np.sum(c * c, axis=1), 1.0, atol=1e-14)


def test_angle_codebook_closed_form_at_pi_over_4():
    # phi = 0 -> theta = eps + (pi/2 - 2 eps)/2 = pi/4 exactly: c_i = 2^{-i/2}
    # for i = 1..7 and c_8 = 2^{-7/2}
    c = oracle.angle_codebook(np.zeros(7))
    want = np.array([2 ** (-i / 2) for i in range(1, 8)] + [2 ** (-7 / 2)])
    assert np.allclose(c, want, rtol=0, atol=1e-15)


def test_angle_codebook_limits_are_axes():
    # phi -> -inf: theta -> eps, the first axis; phi -> +inf: theta -> pi/2 - eps,
    # the last axis (all weight in c_8)
    lo = oracle.angle_codebook(np.full(7, -60.0), eps=1e-6)
    hi = oracle.angle_codebook(np.full(7, 60.0), eps=1e-6)
    assert abs(lo[0] - 1.0) < 1e-10 and np.all(lo[1:] < 1e-5)
    assert abs(hi[7] - 1.0) < 1e-10 and np.all(hi[:7] < 1e-5)


def test_angles_round_trip():
    rng = np.random.default_rng(2)
    phi = rng.normal(0, 2, (1000, 7))
    eps = 1e-4
    theta = eps + (np.pi / 2 - 2 * eps) / (1 + np.exp(-phi))
    back = oracle.codebook_angles(oracle.angle_codebook(phi, eps))
    assert np.allclose(back, theta, atol=1e-12)


def _planted(K=16, per=400, noise=0.01, seed=3):
    rng = np.random.default_rng(seed)
    centres = np.abs(rng.normal(size=(K, 8)))
    centres /= np.linalg.norm(centres, axis=1, keepdims=True)
    d = np.repeat(centres, per, axis=0) + noise * rng.normal(size=(K * per, 8))
    d = np.abs(d)
    d /= np.linalg.norm(d, axis=1, keepdims=True)
    radii = rng.uniform(0.5, 2.0, K * per)
    signs = rng.choice([-1.0, 1.0], size=d.shape)
    w = (signs * d * radii[:, None]).reshape(-1, 128)
    return centres, w


def test_kmeans_centres_are_positive_unit_and_objective_is_monotone():
    _, w = _planted()
    c, hist = oracle.kmeans_codebook(w, 16, samples=4096, iters=12, seed=0)
    assert c.shape == (16, 8)
    assert np.all(c >= 0)
    assert np.allclose(np.linalg.norm(c, axis=1), 1.0, atol=1e-12)
    assert all(b >= a - 1e-12 for a, b in zip(hist, hist[1:]))


def test_kmeans_recovers_well_separated_planted_centres():
    planted, w = _planted(K=8, per=600, noise=0.005, seed=4)
    # spherical k-means from data-point seeds can merge clusters; with more
    # centres than clusters every planted centre still gets a close match
    c, _ = oracle.kmeans_codebook(w, 24, samples=8192, iters=20, seed=1)
    best = np.max(planted @ c.T, axis=1)
    assert np.all(best > 0.999)


def test_kmeans_samples_proportional_to_squared_radius():
    # half the vectors have radius 0: they can never be drawn, so every centre
    # is a direction of the non-zero half (all of which point along e_1)
    w = np.zeros((64, 128))
    w[:32, 0::8] = 3.0
    c, _ = oracle.kmeans_codebook(w, 4, samples=1000, iters=3, seed=5)
    assert np.allclose(c, np.eye(8)[0], atol=1e-12)


def test_kmeans_codebook_feeds_the_encoder():
    _, w = _planted(K=8, per=256, seed=6)
    c, _ = oracle.kmeans_codebook(w, 64, samples=4096, iters=5, seed=2)
    cb16 = oracle.round_half(c)
    codes = oracle.encode(w, cb16, V=4)
    assert codes["idx"].max() < 64
