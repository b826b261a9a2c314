"""GPU parity: the CUDA path (through the C ABI) against the float64 oracle.

Decode must be bit-exact (including -0); the GEMV must satisfy
|y - W_hat x| <= 1e-3 * sum_j |w_hat_j||x_j| + 2^-24 per output.
Small cases are checked in full; the workload shapes (the 1024^2 case, the
4096^2 / 8192^2 encoded sweep, the 7B-class projections at W2 and W3 with
batch 1..8) run at full size in the launch configuration the benchmark uses,
with outputs checked on sampled rows plus the row-block edges.
"""
import numpy as np
import pytest
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqError, SphqMatrix

pytestmark = pytest.mark.gpu

import _gpu as G  # noqa: E402


# ---------------------------------------------------------------------------
# small shapes: every tile boundary, ragged row blocks, every batch size
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("bits", [2, 3])
@pytest.mark.parametrize("rows,cols", [(1, 128), (31, 256), (33, 384), (100, 1024), (257, 640)])
def test_small_shapes_decode_and_gemv(bits, rows, cols):
    codes, x = inp.random_codes(bits, rows, cols, seed=1000 + rows + cols + bits, B=8)
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    for B in (1, 2, 3, 5, 8):
        G.check_gemv(m, codes, x[:B])
    m.close()


def test_config0_w2_1024():
    codes, x = inp.random_codes(2, 1024, 1024, seed=inp.seed_for(0))
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    G.check_gemv(m, codes, x)
    m.close()


# ---------------------------------------------------------------------------
# edge cases of the code space and of the parameters
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("bits", [2, 3])
def test_edge_codes(bits):
    rows, cols = 64, 512
    codes, x = inp.random_codes(bits, rows, cols, seed=77 + bits, B=4)
    K = codes.K
    codes.codebook[: K // 2, 5] = 0          # zero coordinates -> +-0 weights
    codes.sign[:8] = 0xFF                    # all negative (gives -0 on zero coordinates)
    codes.sign[8:16] = 0
    codes.idx[16:24] = K - 1                 # largest index (W3: index bit 12 set)
    codes.rcode[24:32] = 15                  # largest radius code
    codes.rcode[32:40] = 0
    codes.scale[40:48] = 0                   # Delta = 0 -> r_hat = r_min
    codes.offset[48:56] = 0                  # r_min = 0
    codes.scale[56:64] = 0x0001              # subnormal Delta
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    G.check_gemv(m, codes, x)
    m.close()


def test_radius_single_rounding_case():
    """r_hat = RN16(3 * 0x3556 + 2^-24) = 0x3C01: one fp16 rounding of the exact
    fused multiply-add (tests/golden/decode_examples.txt)."""
    codes, x = inp.random_codes(2, 32, 128, seed=5)
    codes.rcode[:] = 3
    codes.scale[:] = 0x3556
    codes.offset[:] = 0x0001
    codes.codebook[:] = 0x3C00               # c = (1, ..., 1): w_hat = +-r_hat
    m = G.make_matrix(codes)
    w = G.decoded_bits(m)
    assert np.all((w & 0x7FFF) == 0x3C01)
    assert np.array_equal(w, G.oracle_decode(codes))
    m.close()


def test_wide_parameter_ranges():
    rng = np.random.default_rng(8)
    codes, x = inp.random_codes(3, 96, 768, seed=12, B=2)
    codes.scale = inp.to_f16_bits(np.exp2(rng.uniform(-24, 6, size=codes.scale.shape)))
    codes.offset = inp.to_f16_bits(np.exp2(rng.uniform(-24, 6, size=codes.offset.shape)))
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m), G.oracle_decode(codes))
    G.check_gemv(m, codes, x)
    m.close()


# ---------------------------------------------------------------------------
# error handling through the C ABI (host-detected, no device fault)
# ---------------------------------------------------------------------------

def test_invalid_codes_rejected_and_unpacked_handle_refuses():
    codes, x = inp.random_codes(2, 32, 256, seed=3)
    m = SphqMatrix(32, 256, 2, G.to_dev(codes.codebook), G.to_dev(codes.scale),
                   G.to_dev(codes.offset))
    with pytest.raises(SphqError) as e:
        m.gemv(G.x_dev(x))
    assert e.value.status == 3  # not packed
    bad = codes.idx.copy()
    bad[3, 7] = 64
    with pytest.raises(SphqError) as e:
        m.pack(G.to_dev(codes.sign), G.to_dev(bad), G.to_dev(codes.rcode))
    assert e.value.status == 1
    badr = codes.rcode.copy()
    badr[0, 0] = 16
    with pytest.raises(SphqError):
        m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(badr))
    with pytest.raises(SphqError):
        m.gemv(G.x_dev(x))
    m.pack(G.to_dev(codes.sign), G.to_dev(codes.idx), G.to_dev(codes.rcode))
    G.check_gemv(m, codes, x)
    # misaligned activations are refused
    xb = torch.zeros(2 * 256 + 8, dtype=torch.float16, device=G.DEV)
    with pytest.raises(SphqError):
        m.gemv_ptr(xb.data_ptr() + 2, xb.data_ptr(), 1, 0)
    with pytest.raises(SphqError):
        m.gemv(G.x_dev(np.zeros((17, 256), np.uint16)))
    m.close()


def test_gemv_is_deterministic():
    codes, x = inp.random_codes(3, 3584, 3584, seed=21, B=4)
    m = G.make_matrix(codes)
    xd = G.x_dev(x)
    y1 = m.gemv(xd).clone()
    y2 = m.gemv(xd).clone()
    torch.cuda.synchronize()
    assert torch.equal(y1.view(torch.int16), y2.view(torch.int16))
    m.close()


# ---------------------------------------------------------------------------
# workload shapes at full size
# ---------------------------------------------------------------------------

@pytest.mark.parametrize("name,rows,cols", inp.DECODER_PROJ)
def test_decoder_projections_w2_batch1(name, rows, cols):
    codes, x = inp.random_codes(2, rows, cols, seed=inp.seed_for(2, rows % 97), B=1)
    m = G.make_matrix(codes)
    rs = G.sample_rows(rows, 192, seed=rows)
    assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
    G.check_gemv(m, codes, x, rs)
    m.close()


@pytest.mark.parametrize("name,rows,cols", inp.DECODER_PROJ)
def test_decoder_projections_w3_small_batch(name, rows, cols):
    codes, x = inp.random_codes(3, rows, cols, seed=inp.seed_for(3, rows % 97), B=8)
    m = G.make_matrix(codes)
    rs = G.sample_rows(rows, 128, seed=rows + 1)
    assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
    for B in (1, 2, 4, 8):
        G.check_gemv(m, codes, x[:B], rs)
    m.close()


@pytest.mark.parametrize("shape_id,bits,n", [(i, b, n) for i, (b, n) in enumerate(inp.SQUARE_SWEEP)])
def test_encoded_square_sweep(shape_id, bits, n):
    # Output row r depends only on row r's codes, so the sampled rows carry codes
    # from the oracle's encoder (Gaussian weights with outliers) and the other rows
    # seeded random codes; the GEMV still runs on the full n x n matrix.
    seed = inp.seed_for(1, shape_id)
    rs = G.sample_rows(n, 128, seed=n + bits)
    w = inp.gaussian_weights(n, n, seed=seed)[rs]
    cb, x = inp.encoded_inputs_rng(bits, n, seed=seed)
    e = oracle.encode(w, cb, chunk=4096)
    codes, _ = inp.random_codes(bits, n, n, seed=seed + 1, codebook=cb)
    for key in ("sign", "idx", "rcode", "scale", "offset"):
        getattr(codes, key)[rs] = e[key]
    m = G.make_matrix(codes)
    assert np.array_equal(G.decoded_bits(m, rs), G.oracle_decode(codes, rs))
    G.check_gemv(m, codes, x, rs)
    m.close()


def test_chained_stack_in_a_cuda_graph():
    """One decoder layer's seven projections chained on one stream and replayed
    from a CUDA graph, as the stack benchmark runs them."""
    mats, xs, ys, cs = [], [], [], []
    for bits in (2, 3):
        for i, (name, rows, cols) in enumerate(inp.DECODER_PROJ):
            codes, x = inp.random_codes(bits, rows, cols, seed=inp.seed_for(4, 10 * bits + i))
            mats.append(G.make_matrix(codes))
            cs.append((codes, x))
            xs.append(G.x_dev(x))
            ys.append(torch.empty((1, rows), dtype=torch.float16, device=G.DEV))
    s = torch.cuda.Stream()
    s.wait_stream(torch.cuda.current_stream())
    with torch.cuda.stream(s):
        for m, xd, yd in zip(mats, xs, ys):       # warm up outside capture
            m.gemv(xd, yd, stream=s)
    torch.cuda.synchronize()
    g = torch.cuda.CUDAGraph()
    with torch.cuda.graph(g, stream=s):
        for m, xd, yd in zip(mats, xs, ys):
            m.gemv(xd, yd, stream=s)
    for yd in ys:
        yd.zero_()
    g.replay()
    torch.cuda.synchronize()
    for (codes, x), yd in zip(cs, ys):
        rs = G.sample_rows(codes.rows, 64, seed=codes.rows)
        y = yd.float().cpu().numpy().astype(np.float64)
        y_ref, absdot = oracle.gemv(G.oracle_decode(codes, rs), x)
        assert np.all(np.abs(y[:, rs] - y_ref) <= oracle.gemv_tolerance(absdot))
    for m in mats:
        m.close()
