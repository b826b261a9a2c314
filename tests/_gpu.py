"""Helpers for the GPU parity tests (CUDA path through the C ABI vs oracle)."""
import numpy as np
import torch

import oracle
import sphq_inputs as inp
from paper_2609_24875_gb300 import SphqMatrix

DEV = torch.device("cuda", 0)


def to_dev(a):
    a = np.ascontiguousarray(a)
    if a.dtype == np.uint16:
        a = a.view(np.int16)
    return torch.from_numpy(a).to(DEV)


def make_matrix(codes: inp.Codes) -> SphqMatrix:
    m = SphqMatrix(codes.rows, codes.cols, codes.bits, to_dev(codes.codebook),
                   to_dev(codes.scale), to_dev(codes.offset), radius_bits=codes.vbits,
                   K=codes.K)
    m.pack(to_dev(codes.sign), to_dev(codes.idx), to_dev(codes.rcode))
    return m


def x_dev(x):
    return to_dev(x).view(torch.float16)


def decoded_bits(m: SphqMatrix, rows=None) -> np.ndarray:
    w = m.decode()
    torch.cuda.synchronize()
    if rows is not None:
        w = w[torch.as_tensor(rows, device=DEV)]
    return w.cpu().view(torch.int16).numpy().view(np.uint16)


def oracle_decode(codes: inp.Codes, rows=None) -> np.ndarray:
    c = codes if rows is None else inp.Codes(codes.bits, codes.codebook, codes.scale[rows],
                                             codes.offset[rows], codes.sign[rows],
                                             codes.idx[rows], codes.rcode[rows], codes.vbits)
    return oracle.decode(c.codebook, c.scale, c.offset, c.sign, c.idx, c.rcode)


def check_gemv(m: SphqMatrix, codes: inp.Codes, x: np.ndarray, rows=None):
    """Runs the GEMV on the device and checks the given rows (all if None)
    against the oracle within the stated tolerance.  Returns max err/tol."""
    y = m.gemv(x_dev(x))
    torch.cuda.synchronize()
    y = y.float().cpu().numpy().astype(np.float64)
    if rows is None:
        rows = np.arange(codes.rows)
    w_ref = oracle_decode(codes, rows)
    y_ref, absdot = oracle.gemv(w_ref, x)
    err = np.abs(y[:, rows] - y_ref)
    tol = oracle.gemv_tolerance(absdot)
    ratio = float(np.max(err / tol))
    assert np.all(err <= tol), f"max err/tol = {ratio:.3g}"
    assert np.all(np.isfinite(y[:, rows]))
    return ratio


def sample_rows(n_rows: int, k: int, seed: int = 0) -> np.ndarray:
    rng = np.random.default_rng(seed)
    pick = rng.choice(n_rows, size=min(k, n_rows), replace=False)
    edge = np.array([0, 31, 32, n_rows - 1])
    return np.unique(np.concatenate([pick, edge[edge < n_rows]]))
