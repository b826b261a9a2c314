"""GPU codebook construction (§3.1 radius-weighted sampling and spherical
k-means, §3.3 angle-parameterised codebook) against the oracle.

Every k-means step is compared from identical inputs: the assignment must be
identical (both sides take the float64 argmax of the same fixed-order dots),
the centres equal within 1e-12 (float64 sums of unit vectors in different
orders) and the objective within 1e-12.  Sampled indices must be identical
except where the uniform lands within 1e-12 of a step of the r^2 cumulative
distribution (prefix sums in different orders), where the other neighbour
is checked to be a valid pick.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import sphq

pytestmark = pytest.mark.gpu

DEV = torch.device("cuda", 0)


def _weights(rows, cols, seed):
    return inp.gaussian_weights(rows, cols, seed=seed).astype(np.float32)


@pytest.mark.parametrize("rows,cols,S", [(64, 256, 3000), (1024, 1024, 65536), (333, 128, 700)])
def test_sample_directions_matches_oracle(rows, cols, S):
    w = _weights(rows, cols, seed=rows + cols)
    u = np.random.default_rng(S).random(S)
    u[:5] = [0.0, 0.5, 1.0 - 2.0 ** -53, 0.25, 1.0]
    d_gpu, i_gpu = sphq.sample_directions(torch.from_numpy(w).to(DEV),
                                          torch.from_numpy(u).to(DEV))
    torch.cuda.synchronize()
    d_gpu, i_gpu = d_gpu.cpu().numpy(), i_gpu.cpu().numpy().astype(np.int64)
    d_ref, i_ref = oracle.sample_directions(w, u)
    same = i_gpu == i_ref
    if not np.all(same):
        # only near a step of the CDF: |u * total - P| tiny for the pick
        w64 = w.astype(np.float64).reshape(-1, 8)
        P = np.cumsum(np.sum(w64 * w64, axis=1))
        t = u[~same] * P[-1]
        near = np.minimum(np.abs(P[i_ref[~same]] - t), np.abs(P[np.maximum(i_ref[~same] - 1, 0)] - t))
        assert np.all(near <= 1e-12 * P[-1]), "sampled indices differ away from a CDF step"
        assert np.all(np.abs(i_gpu[~same] - i_ref[~same]) == 1)
    assert np.array_equal(d_gpu[same], d_ref[same])  # bit-identical directions
    assert np.all(d_gpu >= 0)


def _step_case(K, S, seed):
    rng = np.random.default_rng(seed)
    w = _weights(256, 2048, seed)
    D, _ = oracle.sample_directions(w, rng.random(S))
    C = D[rng.choice(S, size=K, replace=False)].copy()
    return D, C


@pytest.mark.parametrize("K,S", [(64, 65536), (8192, 9000), (100, 1000)])
def test_kmeans_steps_match_oracle(K, S):
    D, C = _step_case(K, S, seed=K + S)
    Dd = torch.from_numpy(D).to(DEV)
    c = C
    for it in range(3):
        c_gpu, z_gpu, obj_gpu = sphq.kmeans_step(Dd, torch.from_numpy(c).to(DEV))
        torch.cuda.synchronize()
        c_ref, z_ref, obj_ref = oracle.kmeans_step(D, c)
        assert np.array_equal(z_gpu.cpu().numpy().astype(np.int64), z_ref), f"assignment, step {it}"
        c_gpu = c_gpu.cpu().numpy()
        assert np.max(np.abs(c_gpu - c_ref)) <= 1e-12, f"centres, step {it}"
        assert abs(float(obj_gpu.item()) - obj_ref) <= 1e-12
        c = c_gpu  # next step from the GPU's centres, the oracle fed the same


def test_kmeans_full_run_properties_and_encoder():
    # the paper's settings: 65,536 samples, 20 iterations; a W2 codebook
    w = _weights(2048, 4096, seed=5)
    S, K = 65536, 64
    u = np.random.default_rng(9).random(S)
    dirs, _ = sphq.sample_directions(torch.from_numpy(w).to(DEV), torch.from_numpy(u).to(DEV))
    init = dirs[torch.from_numpy(np.random.default_rng(10).choice(S, K, replace=False)).to(DEV)]
    c, hist = sphq.kmeans(dirs, init.contiguous(), iters=20)
    torch.cuda.synchronize()
    c, hist = c.cpu().numpy(), hist.cpu().numpy()
    assert np.all(c >= 0)
    assert np.allclose(np.linalg.norm(c, axis=1), 1.0, atol=1e-14)
    assert np.all(np.diff(hist) >= -1e-14)  # Lloyd steps never lower the objective
    # the same run on the oracle, step by step from the same start
    D, _ = oracle.sample_directions(w, u)
    cr = D[np.random.default_rng(10).choice(S, K, replace=False)].copy()
    for _ in range(20):
        cr, _, _ = oracle.kmeans_step(D, cr)
    assert np.max(np.abs(c - cr)) <= 1e-9
    # the fp16 codebook feeds sphq_create / sphq_encode
    cb16 = torch.from_numpy(oracle.round_half(c).astype(np.uint16).view(np.int16)).to(DEV)
    from paper_2609_24875_gb300 import SphqMatrix
    zero = torch.zeros((256, 4096 // 128), dtype=torch.int16, device=DEV)
    m = SphqMatrix(256, 4096, 2, cb16, zero, zero)
    m.encode(torch.from_numpy(w[:256]).to(DEV))
    m.check()
    m.close()


@pytest.mark.parametrize("K", [1, 64, 8192])
def test_angle_codebook_matches_oracle(K):
    rng = np.random.default_rng(K)
    phi = (rng.standard_normal((K, 7)) * 3).astype(np.float32)
    phi[0] = 0.0
    c64, c16 = sphq.angle_codebook(torch.from_numpy(phi).to(DEV), eps=1e-4)
    torch.cuda.synchronize()
    c64 = c64.cpu().numpy()
    ref = oracle.angle_codebook(phi.astype(np.float64), eps=1e-4)
    assert np.max(np.abs(c64 - ref)) <= 1e-13
    assert np.all(c64 >= 0)
    assert np.allclose(np.linalg.norm(c64, axis=1), 1.0, atol=1e-13)
    h = c16.cpu().view(torch.int16).numpy().view(np.uint16)
    r16 = oracle.round_half(ref)
    diff = h != r16
    if np.any(diff):  # only where the float64 value sits on an fp16 rounding boundary
        lo = oracle.round_half(ref[diff] - 1e-13)
        hi = oracle.round_half(ref[diff] + 1e-13)
        assert np.all((h[diff] == lo) | (h[diff] == hi))
