"""Every-row parity at the benchmark's full sizes, in the launch configuration
the benchmark times (the automatic plan).

The kernel's hard paths depend on where a row tile sits in the work split:
the one-tile strip at the end of an odd range, the owner CTA of a tile
(tile mod cluster size), the last cluster's short range.  Sampled rows can
miss them, so one full-size shape per format family is checked on every row:
decode bit-exact against the oracle, and the GEMV within
|y - W_hat x| <= 1e-3 * sum_j |w_hat_j||x_j| + 2^-24 at batch 1, 4 and 8.

The factored batch 1-2 path skips the per-product binary16 rounding of
r_hat * c (up to 2^-11 relative), so its margin to the tolerance is recorded
on the longest rows (18944 columns) and held to at most half the tolerance.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


def _gemv_all_rows(m, codes, x):
    """GPU output of every row against the oracle's decode + matvec; returns
    the largest err/tol over all outputs."""
    y = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().astype(np.float64)
    y_ref, absdot = oracle.decode_gemv(codes.codebook, codes.scale, codes.offset, codes.sign,
                                       codes.idx, codes.rcode, x)
    tol = oracle.gemv_tolerance(absdot)
    err = np.abs(y - y_ref)
    assert np.all(np.isfinite(y))
    ratio = float(np.max(err / tol))
    bad = np.argwhere(err > tol)
    assert bad.size == 0, f"{len(bad)} outputs out of tolerance, first (batch, row) {bad[0]}"
    return ratio


@pytest.mark.parametrize("bits,rows,cols,seed", [(2, 8192, 8192, inp.seed_for(1, 1)),
                                                 (3, 8192, 8192, inp.seed_for(1, 3)),
                                                 (3, 3584, 18944, inp.seed_for(3, 6))])
def test_every_row_full_size(bits, rows, cols, seed):
    codes, x = inp.random_codes(bits, rows, cols, seed=seed, B=8)
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    for B in (1, 4, 8):
        ratio = _gemv_all_rows(m, codes, x[:B])
        print(f"W{bits} {rows}x{cols} batch {B}: max err/tol over all rows {ratio:.4f}")
    m.close()


def test_every_row_encoded_w2_8192():
    # the encoded configuration at full size: codes from the oracle's encoder
    # (K = 64 keeps the float64 encoder fast enough for all 8192 rows)
    seed = inp.seed_for(1, 1)
    w = inp.gaussian_weights(8192, 8192, seed=seed)
    cb, x = inp.encoded_inputs_rng(2, 8192, seed=seed)
    e = oracle.encode(w, cb, chunk=1 << 16)
    codes = inp.Codes(2, cb, e["scale"], e["offset"], e["sign"], e["idx"], e["rcode"])
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    ratio = _gemv_all_rows(m, codes, x)
    print(f"encoded W2 8192x8192 batch 1: max err/tol over all rows {ratio:.4f}")
    m.close()


@pytest.mark.parametrize("bits", [2, 3])
def test_factored_path_margin_on_long_rows(bits):
    # the down projection (3584 x 18944): the longest rows of the workload
    rows, cols = 3584, 18944
    codes, x = inp.random_codes(bits, rows, cols, seed=inp.seed_for(2 if bits == 2 else 3, 6),
                                B=2)
    m = G.make_matrix(codes)
    for B in (1, 2):
        ratio = _gemv_all_rows(m, codes, x[:B])
        print(f"factored path W{bits} {rows}x{cols} batch {B}: max err/tol {ratio:.4f}")
        assert ratio <= 0.5, f"factored path uses {ratio:.3f} of the tolerance"
    m.close()
