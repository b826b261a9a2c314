"""Pins of the oracle's float64 matvec: brute force with Python loops on tiny
matrices, one-hot activations returning columns of W_hat, and linearity."""
import numpy as np
import pytest

import oracle
import sphq_inputs as inp


def _brute(w16, x16):
    w = w16.view(np.float16)
    x = x16.view(np.float16)
    rows, cols = w.shape
    y = [[0.0] * rows for _ in range(x.shape[0])]
    for b in range(x.shape[0]):
        for i in range(rows):
            acc = 0.0
            for j in range(cols):
                acc += float(w[i, j]) * float(x[b, j])
            y[b][i] = acc
    return np.array(y)


@pytest.mark.parametrize("rows,cols,B", [(8, 128, 1), (13, 256, 3), (3, 128, 8)])
def test_gemv_brute_force(rows, cols, B):
    codes, x = inp.random_codes(2, rows, cols, seed=rows * 7 + cols, B=B)
    w = oracle.decode(codes.codebook, codes.scale, codes.offset, codes.sign, codes.idx,
                      codes.rcode)
    y, a = oracle.gemv(w, x)
    yb = _brute(w, x)
    assert np.allclose(y, yb, rtol=1e-12, atol=1e-12)
    assert np.all(a >= np.abs(y) - 1e-9)
    # the fused row-by-row path computes the same values
    y2, a2 = oracle.decode_gemv(codes.codebook, codes.scale, codes.offset, codes.sign,
                                codes.idx, codes.rcode, x)
    assert np.array_equal(y2, y) and np.array_equal(a2, a)


def test_one_hot_returns_columns_and_is_linear():
    codes, _ = inp.random_codes(3, 9, 256, seed=4)
    w = oracle.decode(codes.codebook, codes.scale, codes.offset, codes.sign, codes.idx,
                      codes.rcode)
    wd = oracle.half_to_double(w)
    for j in (0, 7, 100, 255):
        e = np.zeros((1, 256), np.uint16)
        e[0, j] = 0x3C00  # 1.0
        y, _ = oracle.gemv(w, e)
        assert np.array_equal(y[0], wd[:, j])
    rng = np.random.default_rng(0)
    x1 = inp.make_x(rng, 1, 256)
    x2 = inp.make_x(rng, 1, 256)
    y1, _ = oracle.gemv(w, x1)
    y2, _ = oracle.gemv(w, x2)
    y12, _ = oracle.gemv(w, np.concatenate([x1, x2]))
    assert np.array_equal(y12, np.concatenate([y1, y2]))
    # against numpy's float64 matmul (a library routine, not the oracle's loop)
    ref = wd @ oracle.half_to_double(x1)[0]
    assert np.allclose(y1[0], ref, rtol=1e-12, atol=1e-12)


def test_tolerance_formula():
    a = np.array([0.0, 1.0, 1000.0])
    t = oracle.gemv_tolerance(a)
    assert np.array_equal(t, 1e-3 * a + 2.0 ** -24)
