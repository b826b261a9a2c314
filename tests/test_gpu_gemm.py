"""sphq_gemm, the tensor-core product for large batches (prefill), against the
float64 oracle through the C ABI: Y = X W_hat^T with W_hat of Eq. (7) and
Eq. (4), within 1e-3 * sum_j |w_hat_j||x_j| + 2^-24 per output.

Shapes cover every tile edge: rows below, at and past the 256-row tile
(ragged 16-row tiles and rows not a multiple of 16), batches below, at and
past the 128-row activation tile, columns from one radius group up, and every
bit split (W2, W3, W3 with 3-bit radius codes, a Tab. 4 split).
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402

# (bits, radius bits, K) of the formats checked
FORMATS = [(2, 4, 64), (3, 4, 8192), (3, 3, 8192), (2, 2, 256), (2, 3, 64)]
FIDS = ["W2", "W3", "W3V3", "8-8-2", "8-6-3"]


def check_gemm(m, codes, x, rows=None, stream=None):
    y = m.gemm(G.x_dev(x), stream=stream)
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().astype(np.float64)
    if rows is None:
        rows = np.arange(codes.rows)
    y_ref, absdot = oracle.gemv(G.oracle_decode(codes, rows), x)
    err = np.abs(y[:, rows] - y_ref)
    tol = oracle.gemv_tolerance(absdot)
    assert np.all(np.isfinite(y[:, rows]))
    assert np.all(err <= tol), f"max err/tol = {float(np.max(err / tol)):.3g}"
    return float(np.max(err / tol))


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
@pytest.mark.parametrize("rows,cols,batch", [(1, 128, 1), (33, 384, 9), (256, 256, 128),
                                             (257, 640, 130), (1000, 2048, 300)])
def test_small_shapes(fmt, rows, cols, batch):
    bits, v, K = fmt
    codes, x = inp.random_codes(bits, rows, cols, seed=900 + rows + cols + batch + v, B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    check_gemm(m, codes, x)
    m.check()
    m.close()


# every launch shape (activation tiles, weight rows per CTA) the library has,
# forced with sphq_set_gemm_shape, on shapes with ragged edges in every dimension
SHAPES = [(1, 128), (1, 256), (2, 256)]


@pytest.mark.parametrize("fmt", FORMATS, ids=FIDS)
@pytest.mark.parametrize("shape", SHAPES, ids=[f"mt{m}-bn{n}" for m, n in SHAPES])
def test_every_launch_shape(fmt, shape):
    bits, v, K = fmt
    rows, cols, batch = 1000, 1024, 300
    codes, x = inp.random_codes(bits, rows, cols, seed=55 + bits + v + shape[1], B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    m.set_gemm_shape(*shape)
    info = m.gemm_shape(batch)
    assert (info["act_tiles"], info["weight_rows"]) == shape
    assert info["stages"] >= 2 and info["stage_cols"] in (32, 64)
    assert info["grid_x"] == -(-((rows + 15) // 16) // (shape[1] // 16))
    assert info["grid_y"] == -(-batch // (128 * shape[0]))
    check_gemm(m, codes, x)
    m.check()
    m.set_gemm_shape(0, 0)
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:4], ids=FIDS[:4])
@pytest.mark.parametrize("batch,ntok,split", [(1250, 5, 16), (2600, 11, 96)])
def test_split_final_wave(fmt, batch, ntok, split):
    # 8000 rows (32 weight tiles, the last of 4 row tiles) x ntok tiles of 256
    # activation rows on 152 SMs: whole waves, and the output tiles of the
    # final partial wave split into two CTAs of one activation tile each (at
    # batch 2600 the second half of the last row of tiles is wholly past the
    # batch and does no work).  The split plan equals the whole-wave plan bit
    # for bit (the same products in the same order), the two-pass form equals
    # both, all against the oracle.
    bits, v, K = fmt
    rows, cols = 8000, 512
    codes, x = inp.random_codes(bits, rows, cols, seed=3100 + batch + v + bits, B=batch,
                                radius_bits=v, K=K)
    m = G.make_matrix(codes)
    info = m.gemm_shape(batch)
    assert (info["act_tiles"], info["grid_x"], info["grid_y"]) == (2, 32, ntok)
    if torch.cuda.get_device_properties(0).multi_processor_count == 152:
        assert info["split_ctas"] == split
    xd = G.x_dev(x)
    y_split = m.gemm(xd)
    ws = torch.empty(rows * cols, dtype=torch.float16, device="cuda")
    y_two = m.gemm_ws(xd, ws)
    m.set_gemm_shape(2, 256)
    assert m.gemm_shape(batch)["split_ctas"] == 0
    y_whole = m.gemm(xd)
    torch.cuda.synchronize()
    assert torch.equal(y_split.view(torch.int16), y_whole.view(torch.int16))
    assert torch.equal(y_two.view(torch.int16), y_whole.view(torch.int16))
    m.set_gemm_shape(0, 0)
    check_gemm(m, codes, x, G.sample_rows(rows, 400, seed=batch))
    m.check()
    m.close()


def test_shape_choice_and_invalid_shapes():
    codes, _ = inp.random_codes(2, 8192, 1024, seed=6)
    m = G.make_matrix(codes)
    assert m.gemm_shape(4096)["act_tiles"] == 2          # many tiles: two per CTA
    small = m.gemm_shape(64)
    assert small["act_tiles"] == 1
    for bad in ((3, 0), (2, 128), (0, 64), (-1, 0)):
        with pytest.raises(SphqError):
            m.set_gemm_shape(*bad)
    m.close()


def test_matches_gemv_within_tolerance_for_small_batches():
    codes, x = inp.random_codes(2, 3584, 3584, seed=41, B=8)
    m = G.make_matrix(codes)
    rs = G.sample_rows(3584, 128, seed=1)
    for B in (1, 3, 8):
        check_gemm(m, codes, x[:B], rs)
        G.check_gemv(m, codes, x[:B], rs)
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:3], ids=FIDS[:3])
def test_prefill_projection(fmt):
    # a 7B-class q projection at a 512-token prefill chunk, sampled rows checked
    bits, v, K = fmt
    rows, cols, batch = 3584, 3584, 512
    codes, x = inp.random_codes(bits, rows, cols, seed=77 + bits + v, B=batch, radius_bits=v,
                                K=K)
    m = G.make_matrix(codes)
    check_gemm(m, codes, x, G.sample_rows(rows, 96, seed=rows))
    m.check()
    m.close()


def test_encoded_square_4096_batch_256():
    n, batch = 4096, 256
    seed = inp.seed_for(1, 2)
    rs = G.sample_rows(n, 64, seed=n)
    w = inp.gaussian_weights(n, n, seed=seed)[rs]
    cb, x = inp.encoded_inputs_rng(2, n, seed=seed, B=batch)
    e = oracle.encode(w, cb, chunk=4096)
    codes, _ = inp.random_codes(2, n, n, seed=seed + 1, codebook=cb)
    for key in ("sign", "idx", "rcode", "scale", "offset"):
        getattr(codes, key)[rs] = e[key]
    m = G.make_matrix(codes)
    check_gemm(m, codes, x, rs)
    m.close()


def test_deterministic_unaligned_output_and_streams():
    # odd row count: every output row of a token starts at an odd fp16 offset
    codes, x = inp.random_codes(3, 1001, 1024, seed=5, B=200)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y1 = m.gemm(xd).clone()
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        y2 = m.gemm(xd, stream=s)
    s.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
    check_gemm(m, codes, x)
    m.close()


def test_argument_errors():
    codes, x = inp.random_codes(2, 64, 256, seed=3, B=4)
    m = G.make_matrix(codes)
    xb = torch.zeros(4 * 256 + 8, dtype=torch.float16, device=G.DEV)
    y = torch.empty((4, 64), dtype=torch.float16, device=G.DEV)
    with pytest.raises(SphqError) as e:
        m.gemm_ptr(xb.data_ptr() + 2, y.data_ptr(), 4, 0)   # x not 16-byte aligned
    assert e.value.status == 1
    with pytest.raises(SphqError) as e:
        m.gemm_ptr(xb.data_ptr(), y.data_ptr(), 0, 0)
    assert e.value.status == 2
    m.close()


@pytest.mark.parametrize("fmt", FORMATS[:3], ids=FIDS[:3])
@pytest.mark.parametrize("rows,cols,batch", [(8192, 8192, 4096), (18944, 3584, 2048)])
def test_report_sizes_sampled(fmt, rows, cols, batch):
    # the sizes `bench.py --report` times (prefill_gemm), in the launch shape
    # the library chooses for them, checked on sampled rows
    bits, v, K = fmt
    codes, _ = inp.random_codes(bits, rows, cols, seed=31 + rows + v, radius_bits=v, K=K)
    rng = np.random.default_rng(rows + bits)
    x = inp.to_f16_bits(rng.standard_normal((batch, cols)))
    m = G.make_matrix(codes)
    assert m.gemm_shape(batch)["act_tiles"] == 2
    check_gemm(m, codes, x, G.sample_rows(rows, 24, seed=rows))
    m.check()
    m.close()
    torch.cuda.empty_cache()


@pytest.mark.parametrize("fmt", FORMATS[:4], ids=FIDS[:4])
@pytest.mark.parametrize("batch", [9, 12, 13, 16, 19, 34, 64])
def test_batches_9_to_64(fmt, batch):
    # GEMV launches of 8 (or 6 before a last part of 3-4) rows where they are
    # estimated faster, with an odd row count, and the tensor-core kernel when
    # the shape is fixed: both against the oracle
    bits, v, K = fmt
    codes, x = inp.random_codes(bits, 1001, 768, seed=2100 + batch + v, B=batch, radius_bits=v,
                                K=K)
    m = G.make_matrix(codes)
    check_gemm(m, codes, x)
    m.set_gemm_shape(1, 256)
    check_gemm(m, codes, x)
    m.set_gemm_shape(0, 0)
    m.check()
    m.close()
