"""W3 work items of four row tiles: the launch plan takes four-tile strips
when a cluster holds three or more tiles, and the last strip of a cluster
then holds T mod 4 = 1, 2 or 3 tiles.  Shapes with 3..7 tiles per cluster at
cluster sizes 1 and 2 drive every strip and tail size; every row is checked
against the oracle (batch 1, 2 and 5: both radius modes)."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


# row tiles 152 k + r: clusters of one CTA hold k or k + 1 tiles
@pytest.mark.parametrize("nrt", [152 * 3 + 50, 152 * 5 + 70, 152 * 6 + 100])
@pytest.mark.parametrize("csize", [1, 2])
@pytest.mark.parametrize("vbits", [4, 3])
def test_w3_four_tile_strips_every_tail(nrt, csize, vbits):
    rows, cols = 16 * nrt - 5, 512  # a ragged last tile as well
    codes, x = inp.random_codes(3, rows, cols, seed=7000 + nrt + csize + vbits, B=5,
                                radius_bits=vbits)
    m = G.make_matrix(codes)
    for batch in (1, 2, 5):
        m.set_cluster_size(batch, csize)
        p = m.plan(batch)
        assert p["cluster_size"] == csize
        y = m.gemv(G.x_dev(x[:batch]))
        torch.cuda.synchronize()
        got = y.float().cpu().numpy().astype(np.float64)
        ref, absdot = oracle.decode_gemv(codes.codebook, codes.scale, codes.offset, codes.sign,
                                         codes.idx, codes.rcode, x[:batch])
        err = np.abs(got - ref)
        assert np.all(err <= oracle.gemv_tolerance(absdot)), (batch, p)
    m.close()
