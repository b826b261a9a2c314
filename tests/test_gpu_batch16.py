"""The GEMV at 9-16 activation rows: each decoded block of W_hat feeds two
tensor-core products, one per batch half of 8 rows (8-D formats), checked
against the oracle through the C ABI on ragged shapes, at every thread-block
cluster size, with rows of the second half past the batch, on the decoder
projections at full size, and for 4-D vectors (two launches of at most 8
rows)."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

FORMATS = [(2, 4, 64), (3, 4, 8192), (3, 3, 8192), (2, 2, 256), (2, 3, 64)]
FIDS = ["W2", "W3", "W3V3", "8-8-2", "8-6-3"]


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
@pytest.mark.parametrize("batch", [9, 12, 16])
def test_ragged_shapes(fmt, batch):
    bits, v, K = fmt
    # 63 row tiles with a ragged last tile, 6 radius groups
    codes, x = inp.random_codes(bits, 1001, 768, seed=2200 + batch + v + bits, B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    p = m.plan(batch)
    assert p["grid"] > 0 and p["ctas_per_sm"] == 1 and not p["staged_x"]
    G.check_gemv(m, codes, x)
    m.check()
    m.close()


@pytest.mark.parametrize("bits,rows,cols", [(2, 80, 1024), (3, 1000, 1024), (3, 112, 2048),
                                            (2, 1, 1024), (3, 17, 1024)])
@pytest.mark.parametrize("batch", [10, 16])
def test_every_cluster_size(bits, rows, cols, batch):
    codes, x = inp.random_codes(bits, rows, cols, seed=2300 + rows + bits + batch, B=batch)
    m = G.make_matrix(codes)
    auto = m.plan(batch)
    for cs in (1, 2, 4, 8):
        m.set_cluster_size(batch, cs)
        assert m.plan(batch)["cluster_size"] == cs
        G.check_gemv(m, codes, x)
        y1 = m.gemv(G.x_dev(x))
        y2 = m.gemv(G.x_dev(x))
        torch.cuda.synchronize()
        assert torch.equal(y1, y2)  # fixed summation order
    m.set_cluster_size(batch, 0)
    assert m.plan(batch) == auto
    m.check()
    m.close()


def test_second_half_rows_past_the_batch_and_first_rows_match_batch_8():
    # batch 9: one row in the second half; the first 8 rows must equal a
    # batch-8 call at the same cluster size (the same products in the same
    # order; only the second half's accumulators are added)
    codes, x = inp.random_codes(3, 512, 1024, seed=2400, B=9)
    m = G.make_matrix(codes)
    for cs in (1, 2):
        m.set_cluster_size(9, cs)
        m.set_cluster_size(8, cs)
        y9 = m.gemv(G.x_dev(x))
        y8 = m.gemv(G.x_dev(x[:8]))
        torch.cuda.synchronize()
        assert torch.equal(y9[:8].view(torch.int16), y8.view(torch.int16))
    G.check_gemv(m, codes, x)
    m.close()


@pytest.mark.parametrize("bits", [2, 3])
@pytest.mark.parametrize("name,rows,cols", [("q", 3584, 3584), ("k", 512, 3584),
                                            ("down", 3584, 18944)])
def test_decoder_projections_batch_16(bits, name, rows, cols):
    codes, x = inp.random_codes(bits, rows, cols, seed=2500 + bits + rows % 97, B=16)
    m = G.make_matrix(codes)
    G.check_gemv(m, codes, x, G.sample_rows(rows, 160, seed=rows))
    m.check()
    m.close()


@pytest.mark.parametrize("batch", [9, 12, 16])
def test_dim4_two_launches(batch):
    # 4-D vectors have no 16-row build: 8 rows, then the rest
    from paper_2609_24875_gb300 import SphqMatrix
    rows, cols = 200, 512
    codes, x = inp.random_codes_dim(4, 2, rows, cols, seed=2600 + batch, B=batch)
    m = SphqMatrix(rows, cols, 2, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset), radius_bits=4, K=4, dim=4)
    m.pack(G.to_dev(codes.sign.astype(np.uint8)), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    assert m.plan(batch)["grid"] == 0  # no 16-row plan for 4-D vectors
    y = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    got = y.float().cpu().numpy().astype(np.float64)
    w = oracle.decode_dim(codes.codebook, codes.scale, codes.offset, codes.sign, codes.idx,
                          codes.rcode)
    ref, absdot = oracle.gemv(w, x)
    assert np.all(np.abs(got - ref) <= oracle.gemv_tolerance(absdot))
    m.check()
    m.close()


@pytest.mark.parametrize("bits", [2, 3])
@pytest.mark.parametrize("batch", [9, 16])
def test_one_row_one_group(bits, batch):
    codes, x = inp.random_codes(bits, 1, 128, seed=2700 + bits + batch, B=batch)
    m = G.make_matrix(codes)
    G.check_gemv(m, codes, x)
    m.check()
    m.close()


@pytest.mark.parametrize("batch", [1, 2, 4, 8])
def test_w2_long_rows_one_cta_four_tile_strips(batch):
    # 3584 x 18944 (the down projection): more two-per-SM CTAs than SMs would
    # put two on some SMs, so the plan takes the one-CTA build with four-tile
    # strips; every row checked against the oracle
    codes, x = inp.random_codes(2, 3584, 18944, seed=2800 + batch, B=batch)
    m = G.make_matrix(codes)
    p = m.plan(batch)
    assert p["ctas_per_sm"] == 1 and p["tiles_per_cluster"] >= 3
    G.check_gemv(m, codes, x)
    m.check()
    m.close()


@pytest.mark.parametrize("batch", [4, 8])
def test_w2_square_one_cta_four_tile_strips_at_3_to_8_rows(batch):
    # 8192 x 8192 at 3-8 rows: the strips of four share each activation read,
    # so the plan takes the one-CTA build; sampled rows against the oracle
    codes, x = inp.random_codes(2, 8192, 8192, seed=2900 + batch, B=batch)
    m = G.make_matrix(codes)
    p = m.plan(batch)
    assert p["ctas_per_sm"] == 1 and p["tiles_per_cluster"] >= 3
    G.check_gemv(m, codes, x, G.sample_rows(8192, 256, seed=batch))
    m.check()
    m.close()
