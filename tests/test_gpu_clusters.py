"""The GEMV at every thread-block cluster size (sphq_set_cluster_size), on
shapes whose row-tile counts leave partial strips and uneven clusters, checked
against the oracle through the C ABI.  Every cluster size exercises another
reduction path: CTAs of a cluster split the radius groups and send their
partial sums to each tile's owner CTA through distributed shared memory."""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

# (bits, rows, cols): 5 and 63 row tiles (a ragged last tile), 8 and 16 groups
SHAPES = [(2, 80, 1024), (2, 1000, 2048), (3, 112, 2048), (3, 1000, 1024)]


def _check(m, codes, x, batch):
    y = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    got = y.float().cpu().numpy().astype(np.float64)
    w = G.oracle_decode(codes)
    ref, absdot = oracle.gemv(w, x)
    tol = oracle.gemv_tolerance(absdot)
    assert got.shape == (batch, codes.rows)
    assert np.all(np.isfinite(got))
    assert np.all(np.abs(got - ref) <= tol), float(np.max(np.abs(got - ref) / tol))
    return y


@pytest.mark.parametrize("bits,rows,cols", SHAPES)
@pytest.mark.parametrize("batch", [1, 2, 5])
def test_every_cluster_size_matches_oracle(bits, rows, cols, batch):
    codes, x = inp.random_codes(bits, rows, cols, seed=900 + rows + bits + batch, B=batch)
    m = G.make_matrix(codes)
    auto = m.plan(batch)
    assert auto["cluster_size"] in (1, 2, 4, 8)
    assert auto["grid"] == auto["clusters"] * auto["cluster_size"]
    for cs in (1, 2, 4, 8):
        m.set_cluster_size(batch, cs)
        p = m.plan(batch)
        assert p["cluster_size"] == cs
        assert p["clusters"] * p["tiles_per_cluster"] >= (rows + 15) // 16
        y1 = _check(m, codes, x, batch)
        y2 = m.gemv(G.x_dev(x))
        torch.cuda.synchronize()
        assert torch.equal(y1, y2)  # fixed summation order
    m.set_cluster_size(batch, 0)
    assert m.plan(batch) == auto
    m.close()


def test_cluster_size_larger_than_groups_is_rejected():
    codes, x = inp.random_codes(2, 64, 256, seed=77)  # 2 groups
    m = G.make_matrix(codes)
    before = m.plan(1)
    from paper_2609_24875_gb300.sphq import SphqError
    with pytest.raises(SphqError):
        m.set_cluster_size(1, 4)
    assert m.plan(1) == before
    _check(m, codes, x, 1)
    m.close()


# Extreme aspect ratios: one row tile split over a whole cluster of CTAs
# (long rows), and 16384 row tiles of one group each (tall and thin), plus a
# W3 row so wide that its staged activations do not fit in shared memory at
# batch 2 (the plan falls back to reading them through L1).
@pytest.mark.parametrize("bits,rows,cols,batch", [(2, 16, 262144, 1), (2, 262144, 128, 1),
                                                  (3, 32, 196608, 2)])
def test_extreme_shapes(bits, rows, cols, batch):
    codes, x = inp.random_codes(bits, rows, cols, seed=4100 + bits + batch, B=batch)
    m = G.make_matrix(codes)
    p = m.plan(batch)
    if cols >= 196608 and bits == 3:
        assert p["staged_x"] == 0
    rows_chk = G.sample_rows(rows, 512, seed=5) if rows > 4096 else None
    y = m.gemv(G.x_dev(x))
    torch.cuda.synchronize()
    got = y.float().cpu().numpy().astype(np.float64)
    sel = np.arange(rows) if rows_chk is None else rows_chk
    w = G.oracle_decode(codes, sel)
    ref, absdot = oracle.gemv(w, x)
    err = np.abs(got[:, sel] - ref)
    assert np.all(np.isfinite(got[:, sel]))
    assert np.all(err <= oracle.gemv_tolerance(absdot)), float(np.max(err / oracle.gemv_tolerance(absdot)))
    m.close()


# W2 has two builds of the kernel: two CTAs per SM (at most 128 registers per
# thread) and one CTA per SM with the whole register file, which the plan
# takes when the row tiles bound the cluster count (no second CTA would share
# an SM).  W3 always runs one CTA per SM.  Every row, every batch mode.
@pytest.mark.parametrize("bits,rows,cols,ctas", [(2, 512, 3584, 1), (2, 4096, 1024, 2),
                                                 (2, 509, 3584, 1), (3, 512, 3584, 1)])
def test_kernel_build_per_plan(bits, rows, cols, ctas):
    codes, x = inp.random_codes(bits, rows, cols, seed=8800 + rows + bits, B=5)
    m = G.make_matrix(codes)
    for batch in (1, 2, 5):
        p = m.plan(batch)
        assert p["ctas_per_sm"] == ctas, (batch, p)
        _check(m, codes, x[:batch], batch)
    m.close()


# Batch 2 reads its activations through L1 (the full mode) for the 8192-entry
# tables and for matrices of up to 16384 units; larger small-codebook
# matrices stage them in shared memory (the factored mode).
@pytest.mark.parametrize("bits,rows,cols,staged", [(3, 512, 3584, False), (3, 18944, 3584, False),
                                                   (2, 512, 3584, False), (2, 3584, 18944, True)])
def test_batch2_mode_choice(bits, rows, cols, staged):
    codes, x = inp.random_codes(bits, rows, cols, seed=4200 + rows + bits, B=2)
    m = G.make_matrix(codes)
    assert bool(m.plan(2)["staged_x"]) == staged
    assert bool(m.plan(1)["staged_x"])  # batch 1 always stages
    G.check_gemv(m, codes, x, G.sample_rows(rows, 160, seed=rows))
    G.check_gemv(m, codes, x[:1], G.sample_rows(rows, 160, seed=rows + 1))
    m.check()
    m.close()
