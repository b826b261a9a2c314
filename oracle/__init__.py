"""SPHQuant CPU oracle -- TEST INFRASTRUCTURE ONLY.

A plain float64 restatement of what the fused spherical dequantize-GEMV
computes, written from the SPHQuant paper (§3.1 Eqs. (3)-(7), §3.4 and App. D).
Only ``tests/``, ``__graft_entry__.smoke()`` and the ``cpu_baseline`` /
``--impl reference`` legs of ``bench.py`` may import it.  The product package
(``paper_2609_24875_gb300``) never imports it and shares no code with it.

Layers:
  * ``sphq_oracle.c`` (loaded through ctypes): IEEE binary16 rounding written
    from its definition, the decode of Eq. (7) + Eq. (4), the float64 matvec,
    and the paper's W2 word format (§3.4, Fig. 3(b)).
  * this module: numpy wrappers, the reference encoder of Eqs. (3), (5), (6),
    (7) used to produce codes from Gaussian weights, and the bit-budget
    formulas of §3.1, §4.3 (Tab. 4, Tab. 7) and App. B.

Array conventions (all host numpy arrays, row-major):
  codebook  (K, 8)          uint16  binary16 bit patterns, entries c_k >= 0
  sign      (rows, cols/8)  uint8   bit j set <=> coordinate j negative
  idx       (rows, cols/8)  uint16  direction index z < K
  rcode     (rows, cols/8)  uint8   radius code q in [0, 16)
  scale     (rows, cols/128) uint16 binary16 Delta_G
  offset    (rows, cols/128) uint16 binary16 r_min_G
  x         (B, cols)       uint16  binary16 activations
"""
from __future__ import annotations

import ctypes
import os
import subprocess
import threading

import numpy as np

_HERE = os.path.dirname(os.path.abspath(__file__))
_SRC = os.path.join(_HERE, "sphq_oracle.c")
_LIB_PATH = os.path.join(_HERE, "libsphq_oracle.so")
_lib = None
_lock = threading.Lock()

VEC = 8          # vector dimension k (§3.1)
GROUP_VECS = 16  # vectors per radius group (128 scalars, §3.1)
GROUP = VEC * GROUP_VECS


def build(force: bool = False) -> str:
    """Compile the C oracle with gcc (no GPU involved). Returns the .so path."""
    if force or not os.path.exists(_LIB_PATH) or (
        os.path.getmtime(_LIB_PATH) < os.path.getmtime(_SRC)
    ):
        tmp = _LIB_PATH + f".tmp{os.getpid()}"
        cmd = ["gcc", "-O2", "-fopenmp", "-ffp-contract=off", "-shared", "-fPIC",
               _SRC, "-o", tmp, "-lm"]
        subprocess.run(cmd, check=True)
        os.replace(tmp, _LIB_PATH)
    return _LIB_PATH


def lib() -> ctypes.CDLL:
    global _lib
    with _lock:
        if _lib is None:
            build()
            L = ctypes.CDLL(_LIB_PATH)
            u16, u8, u32, f64 = (ctypes.POINTER(ctypes.c_uint16), ctypes.POINTER(ctypes.c_uint8),
                                 ctypes.POINTER(ctypes.c_uint32), ctypes.POINTER(ctypes.c_double))
            i32, i64 = ctypes.c_int, ctypes.c_int64
            L.sphqo_half_to_double.argtypes = [ctypes.c_uint16]
            L.sphqo_half_to_double.restype = ctypes.c_double
            L.sphqo_round_half.argtypes = [ctypes.c_double]
            L.sphqo_round_half.restype = ctypes.c_uint16
            L.sphqo_round_half_array.argtypes = [f64, u16, i64]
            L.sphqo_half_to_double_array.argtypes = [u16, f64, i64]
            L.sphqo_radius.argtypes = [i32, ctypes.c_uint16, ctypes.c_uint16]
            L.sphqo_radius.restype = ctypes.c_uint16
            L.sphqo_decode.argtypes = [i32, i32, i32, u16, u16, u16, u8, u16, u8, u16]
            L.sphqo_decode.restype = i32
            L.sphqo_gemv.argtypes = [i32, i32, i32, u16, u16, f64, f64]
            L.sphqo_gemv.restype = i32
            L.sphqo_decode_gemv.argtypes = [i32, i32, i32, i32, u16, u16, u16, u8, u16, u8,
                                            u16, f64, f64]
            L.sphqo_decode_gemv.restype = i32
            L.sphqo_pack_w2_words.argtypes = [i32, i32, u8, u16, u8, u16, u32]
            L.sphqo_pack_w2_words.restype = i32
            L.sphqo_unpack_w2_words.argtypes = [i32, i32, u16, u32, u8, u16, u8]
            L.sphqo_unpack_w2_words.restype = i32
            L.sphqo_decode_dim.argtypes = [i32, i32, i32, i32, i32, u16, u16, u16, u16, u16, u8,
                                           u16]
            L.sphqo_decode_dim.restype = i32
            L.sphqo_encode_f32.argtypes = [i32, i32, i32, i32, u16, ctypes.POINTER(ctypes.c_float),
                                           u8, u16, u8, u16, u16]
            L.sphqo_encode_f32.restype = i32
            L.sphqo_set_threads.argtypes = [i32]
            L.sphqo_get_threads.restype = i32
            L.sphqo_max_threads.restype = i32
            _lib = L
    return _lib


def _p(a: np.ndarray, ctype):
    assert a.flags["C_CONTIGUOUS"]
    return a.ctypes.data_as(ctypes.POINTER(ctype))


def _c(a, dtype) -> np.ndarray:
    return np.ascontiguousarray(a, dtype=dtype)


def set_threads(n: int) -> None:
    lib().sphqo_set_threads(int(n))


def max_threads() -> int:
    return int(lib().sphqo_max_threads())


# --------------------------------------------------------------------------
# binary16
# --------------------------------------------------------------------------

def round_half(v) -> np.ndarray:
    """Nearest binary16 (ties to even) of float64 values, as uint16 bits."""
    v = _c(v, np.float64)
    out = np.empty(v.shape, np.uint16)
    lib().sphqo_round_half_array(_p(v, ctypes.c_double), _p(out, ctypes.c_uint16), v.size)
    return out


def half_to_double(h) -> np.ndarray:
    h = _c(h, np.uint16)
    out = np.empty(h.shape, np.float64)
    lib().sphqo_half_to_double_array(_p(h, ctypes.c_uint16), _p(out, ctypes.c_double), h.size)
    return out


def radius(q: int, scale: int, offset: int) -> int:
    """r_hat of Eq. (7) as binary16 bits: RN16(q * Delta + r_min)."""
    return int(lib().sphqo_radius(int(q), int(scale), int(offset)))


# --------------------------------------------------------------------------
# decode + matvec
# --------------------------------------------------------------------------

def decode(codebook, scale, offset, sign, idx, rcode) -> np.ndarray:
    """Decoded weights W_hat (rows, cols) as binary16 bits (Eq. (7), Eq. (4))."""
    codebook = _c(codebook, np.uint16)
    sign, idx, rcode = _c(sign, np.uint8), _c(idx, np.uint16), _c(rcode, np.uint8)
    scale, offset = _c(scale, np.uint16), _c(offset, np.uint16)
    rows, nv = sign.shape
    cols = nv * VEC
    assert idx.shape == rcode.shape == sign.shape
    assert scale.shape == offset.shape == (rows, cols // GROUP)
    K = codebook.shape[0]
    out = np.empty((rows, cols), np.uint16)
    rc = lib().sphqo_decode(rows, cols, K, _p(codebook, ctypes.c_uint16),
                            _p(scale, ctypes.c_uint16), _p(offset, ctypes.c_uint16),
                            _p(sign, ctypes.c_uint8), _p(idx, ctypes.c_uint16),
                            _p(rcode, ctypes.c_uint8), _p(out, ctypes.c_uint16))
    if rc != 0:
        raise ValueError("oracle decode: bad shape or out-of-range code")
    return out


def decode_dim(codebook, scale, offset, sign, idx, rcode, V: int = 4) -> np.ndarray:
    """W_hat for vectors of dim = 4, 8 or 16 coordinates (Tab. 7; Eq. (7),
    Eq. (4)); radius groups of 128 scalars.  codebook (K, dim) binary16 bits;
    sign (rows, cols/dim) u16; idx u16; rcode u8."""
    codebook = _c(codebook, np.uint16)
    sign, idx, rcode = _c(sign, np.uint16), _c(idx, np.uint16), _c(rcode, np.uint8)
    scale, offset = _c(scale, np.uint16), _c(offset, np.uint16)
    K, dim = codebook.shape
    rows, nv = sign.shape
    cols = nv * dim
    assert idx.shape == rcode.shape == sign.shape
    assert scale.shape == offset.shape == (rows, cols // GROUP)
    out = np.empty((rows, cols), np.uint16)
    rc = lib().sphqo_decode_dim(rows, cols, dim, K, V, _p(codebook, ctypes.c_uint16),
                                _p(scale, ctypes.c_uint16), _p(offset, ctypes.c_uint16),
                                _p(sign, ctypes.c_uint16), _p(idx, ctypes.c_uint16),
                                _p(rcode, ctypes.c_uint8), _p(out, ctypes.c_uint16))
    if rc != 0:
        raise ValueError("oracle decode_dim: bad shape or out-of-range code")
    return out


def gemv(w16, x16):
    """y = W x in float64 and sum_j |w||x| per output, for binary16 W (rows, cols)
    and x (B, cols).  Returns (y, absdot), both (B, rows) float64."""
    w16, x16 = _c(w16, np.uint16), _c(x16, np.uint16)
    if x16.ndim == 1:
        x16 = x16[None, :]
    rows, cols = w16.shape
    B = x16.shape[0]
    assert x16.shape[1] == cols
    y = np.empty((B, rows), np.float64)
    a = np.empty((B, rows), np.float64)
    rc = lib().sphqo_gemv(rows, cols, B, _p(w16, ctypes.c_uint16), _p(x16, ctypes.c_uint16),
                          _p(y, ctypes.c_double), _p(a, ctypes.c_double))
    if rc != 0:
        raise ValueError("oracle gemv: bad arguments")
    return y, a


def decode_gemv(codebook, scale, offset, sign, idx, rcode, x16):
    """Row-by-row decode + float64 matvec without materialising W_hat."""
    codebook = _c(codebook, np.uint16)
    sign, idx, rcode = _c(sign, np.uint8), _c(idx, np.uint16), _c(rcode, np.uint8)
    scale, offset = _c(scale, np.uint16), _c(offset, np.uint16)
    x16 = _c(x16, np.uint16)
    if x16.ndim == 1:
        x16 = x16[None, :]
    rows, nv = sign.shape
    cols = nv * VEC
    B = x16.shape[0]
    y = np.empty((B, rows), np.float64)
    a = np.empty((B, rows), np.float64)
    rc = lib().sphqo_decode_gemv(rows, cols, codebook.shape[0], B,
                                 _p(codebook, ctypes.c_uint16), _p(scale, ctypes.c_uint16),
                                 _p(offset, ctypes.c_uint16), _p(sign, ctypes.c_uint8),
                                 _p(idx, ctypes.c_uint16), _p(rcode, ctypes.c_uint8),
                                 _p(x16, ctypes.c_uint16), _p(y, ctypes.c_double),
                                 _p(a, ctypes.c_double))
    if rc != 0:
        raise ValueError("oracle decode_gemv: bad arguments")
    return y, a


def gemv_tolerance(absdot) -> np.ndarray:
    """Per-output bound on |y_gpu - y_ref|: 1e-3 * sum_j |w_hat_j||x_j| plus one
    binary16 subnormal spacing (2^-24), the resolution of the fp16 output."""
    return 1e-3 * np.asarray(absdot) + 2.0 ** -24


# --------------------------------------------------------------------------
# the paper's W2 word format (§3.4, Fig. 3(b), App. A step 10)
# --------------------------------------------------------------------------

def pack_w2_words(sign, idx, rcode):
    sign, idx, rcode = _c(sign, np.uint8), _c(idx, np.uint16), _c(rcode, np.uint8)
    rows, nv = sign.shape
    base = np.empty((rows, nv), np.uint16)
    extra = np.empty((rows, nv // GROUP_VECS), np.uint32)
    rc = lib().sphqo_pack_w2_words(rows, nv * VEC, _p(sign, ctypes.c_uint8),
                                   _p(idx, ctypes.c_uint16), _p(rcode, ctypes.c_uint8),
                                   _p(base, ctypes.c_uint16), _p(extra, ctypes.c_uint32))
    if rc != 0:
        raise ValueError("W2 words need idx < 64 and rcode < 16")
    return base, extra


def unpack_w2_words(base, extra):
    base, extra = _c(base, np.uint16), _c(extra, np.uint32)
    rows, nv = base.shape
    sign = np.empty((rows, nv), np.uint8)
    idx = np.empty((rows, nv), np.uint16)
    rcode = np.empty((rows, nv), np.uint8)
    rc = lib().sphqo_unpack_w2_words(rows, nv * VEC, _p(base, ctypes.c_uint16),
                                     _p(extra, ctypes.c_uint32), _p(sign, ctypes.c_uint8),
                                     _p(idx, ctypes.c_uint16), _p(rcode, ctypes.c_uint8))
    if rc != 0:
        raise ValueError("bad W2 word arrays")
    return sign, idx, rcode


# --------------------------------------------------------------------------
# bit budget (§3.1, §3.2, Tab. 4, Tab. 7, App. B)
# --------------------------------------------------------------------------

def direction_index_bits(bits: int, dim: int = VEC) -> int:
    """K_dir: (dim-1)*B bits for direction information minus dim sign bits
    (§3.1: 7B - 8 for 8-D vectors)."""
    return (dim - 1) * bits - dim


def codebook_entries(bits: int, dim: int = VEC) -> int:
    """|C| = 2^K_dir (§3.1)."""
    return 1 << direction_index_bits(bits, dim)


def codebook_bytes(bits: int, dim: int = VEC, signed: bool = False) -> int:
    """fp16 storage of the direction codebook; a signed-direction codebook needs
    2^dim times more entries (§3.1)."""
    n = codebook_entries(bits, dim) * (1 << dim if signed else 1)
    return n * dim * 2


def split_bits_per_weight(dir_bits: int, V: int, dim: int = VEC) -> float:
    """Encoded payload per weight of a sign / direction-index / radius split
    (Tab. 4): (dim sign bits + dir_bits + V) / dim."""
    return (dim + dir_bits + V) / dim


def payload_bits_per_weight(bits: int, V: int, dim: int = VEC) -> float:
    """Encoded payload (7B + V)/8 per weight for 8-D vectors (App. B): sign bits,
    direction index and radius code, excluding group parameters and codebook."""
    return (dim + direction_index_bits(bits, dim) + V) / dim


# --------------------------------------------------------------------------
# reference encoder (Eqs. (3), (5), (6), (7)) -- produces codes from weights
# --------------------------------------------------------------------------

def decompose(w) -> tuple:
    """Eq. (3) for one or many 8-D vectors (last axis): signs s (as bits),
    w_+ = |w|, r = ||w_+||_2 and d = w_+ / max(r, eps)."""
    w = np.asarray(w, np.float64)
    neg = (w < 0)
    sign_bits = np.zeros(w.shape[:-1], np.uint8)
    for j in range(VEC):
        sign_bits |= (neg[..., j].astype(np.uint8) << j)
    wp = np.abs(w)
    r = np.sqrt(np.sum(wp * wp, axis=-1))
    d = wp / np.maximum(r, 1e-12)[..., None]
    return sign_bits, wp, r, d


def encode(w, codebook, V: int = 4, chunk: int = 1 << 14):
    """Encode a float64 weight matrix (rows, cols) against a binary16 codebook.

    Steps, in the paper's order:
      Eq. (3)  s = sign(w), w_+ = |w|, r = ||w_+||, d = w_+ / max(r, eps)
      Eq. (5)  z = argmax_k d . c_k   (ties -> lowest k)
      Eq. (6)  r_tilde = <w_+, c_z>
      Eq. (7)  per group of 16 vectors: r_min, r_max, Delta = (r_max - r_min)/(2^V - 1);
               stored as binary16 Delta16 = RN16(Delta), m16 = RN16(r_min);
               q = clip(floor((r_tilde - m16)/Delta16 + 1/2), 0, 2^V - 1)  (q = 0 if Delta16 = 0)
    Returns dict(sign, idx, rcode, scale, offset, r_tilde).
    """
    w = np.asarray(w, np.float64)
    rows, cols = w.shape
    assert cols % GROUP == 0
    C = half_to_double(codebook)                      # (K, 8)
    vecs = w.reshape(rows, cols // VEC, VEC)
    sign, wp, r, d = decompose(vecs)
    flat_d = d.reshape(-1, VEC)
    z = np.empty(flat_d.shape[0], np.int64)
    for s in range(0, flat_d.shape[0], chunk):
        scores = flat_d[s:s + chunk] @ C.T
        z[s:s + chunk] = np.argmax(scores, axis=1)
    z = z.reshape(rows, cols // VEC)
    r_tilde = np.sum(wp * C[z], axis=-1)
    g = r_tilde.reshape(rows, cols // GROUP, GROUP_VECS)
    rmin = g.min(axis=-1)
    rmax = g.max(axis=-1)
    levels = (1 << V) - 1
    delta = (rmax - rmin) / levels
    scale16 = round_half(delta)
    offset16 = round_half(rmin)
    D = half_to_double(scale16)[..., None]
    M = half_to_double(offset16)[..., None]
    with np.errstate(divide="ignore", invalid="ignore"):
        qf = np.floor((g - M) / D + 0.5)
    qf = np.where(D == 0, 0.0, qf)
    q = np.clip(qf, 0, levels).astype(np.uint8).reshape(rows, cols // VEC)
    return dict(sign=sign, idx=z.astype(np.uint16), rcode=q, scale=scale16,
                offset=offset16, r_tilde=r_tilde)


def encode_fp32(w, codebook, V: int = 4):
    """The encoder of `encode` (Eqs. (3), (5), (6), (7)) with every decision in
    IEEE single precision and a fixed operation order (fused multiply-adds in
    coordinate order, correctly rounded sqrt and division; see the C source),
    so that a single-precision implementation elsewhere can match it bit for
    bit.  w: float32 (rows, cols).  Returns dict(sign, idx, rcode, scale, offset)."""
    w = np.ascontiguousarray(np.asarray(w, np.float32))
    rows, cols = w.shape
    cb = _c(codebook, np.uint16)
    K = cb.shape[0]
    nv = cols // VEC
    sign = np.empty((rows, nv), np.uint8)
    idx = np.empty((rows, nv), np.uint16)
    rcode = np.empty((rows, nv), np.uint8)
    scale = np.empty((rows, cols // GROUP), np.uint16)
    offset = np.empty((rows, cols // GROUP), np.uint16)
    rc = lib().sphqo_encode_f32(rows, cols, K, V, _p(cb, ctypes.c_uint16),
                                _p(w, ctypes.c_float), _p(sign, ctypes.c_uint8),
                                _p(idx, ctypes.c_uint16), _p(rcode, ctypes.c_uint8),
                                _p(scale, ctypes.c_uint16), _p(offset, ctypes.c_uint16))
    if rc != 0:
        raise ValueError("oracle encode_fp32: bad arguments")
    return dict(sign=sign, idx=idx, rcode=rcode, scale=scale, offset=offset)


# ---------------------------------------------------------------------------
# Quantize side of the path: codebook construction (§3.1, §3.3)
# ---------------------------------------------------------------------------

def angle_codebook(phi, eps: float = 1e-4) -> np.ndarray:
    """Positive unit directions from angle logits (§3.3).

    Eq. (sph-angle-logits): theta_j = eps + (pi/2 - 2 eps) * sigmoid(phi_j),
    so every angle lies in (0, pi/2).  Eq. (sph-angle-codebook): hyperspherical
    coordinates c_1 = cos th_1, c_i = (prod_{j<i} sin th_j) cos th_i for
    2 <= i <= 7, c_8 = prod_{j<=7} sin th_j.  phi has shape (..., 7); the result
    (..., 8) float64 is non-negative with unit norm by construction."""
    phi = np.asarray(phi, np.float64)
    assert phi.shape[-1] == VEC - 1
    theta = eps + (np.pi / 2 - 2 * eps) / (1.0 + np.exp(-phi))
    c = np.empty(phi.shape[:-1] + (VEC,), np.float64)
    run = np.ones(phi.shape[:-1], np.float64)  # prod of sines so far
    for i in range(VEC - 1):
        c[..., i] = run * np.cos(theta[..., i])
        run = run * np.sin(theta[..., i])
    c[..., VEC - 1] = run
    return c


def codebook_angles(c) -> np.ndarray:
    """Inverse of the coordinates map of Eq. (sph-angle-codebook) for unit
    vectors with non-negative coordinates: theta_i = atan2(||c_{i+1..8}||, c_i)."""
    c = np.asarray(c, np.float64)
    theta = np.empty(c.shape[:-1] + (VEC - 1,), np.float64)
    for i in range(VEC - 1):
        tail = np.sqrt(np.sum(c[..., i + 1:] ** 2, axis=-1))
        theta[..., i] = np.arctan2(tail, c[..., i])
    return theta


def sample_directions(w, u):
    """Radius-weighted sampling of directions (§3.1): 8-D vector i of w is
    drawn with probability r_i^2 / sum_j r_j^2 by inverse transform of the
    uniforms u in [0, 1): P = cumsum(r^2) in vector order, the pick for u is
    the first i with P_i > u * P_last (so vectors of zero radius are never
    drawn; u = 1, whose product is P_last itself, takes the last vector of
    nonzero radius).  r_i^2 = w_0^2 + ... + w_7^2 summed in coordinate order, r_i its
    square root and the direction d_i = |w_i| / r_i, all in float64 from the
    float32 weights.  Returns (directions (len(u), 8) float64, indices)."""
    w = np.asarray(w, np.float32).astype(np.float64).reshape(-1, VEC)
    r2 = w[:, 0] * w[:, 0]
    for j in range(1, VEC):
        r2 = r2 + w[:, j] * w[:, j]
    P = np.cumsum(r2)
    if P[-1] <= 0:
        raise ValueError("all vectors are zero")
    u = np.asarray(u, np.float64)
    idx = np.searchsorted(P, u * P[-1], side="right")
    # fl(u * total) < total for every double u < 1; u = 1 reaches the total,
    # which no P_i exceeds: the pick is the first i with P_i = total
    idx = np.where(idx >= P.shape[0], np.searchsorted(P, P[-1], side="left"), idx)
    r = np.sqrt(r2[idx])
    return np.abs(w[idx]) / r[:, None], idx


def kmeans_scores(D, C):
    """d_i . c_k for every sample and centre in float64, each dot taken in
    coordinate order (products rounded, then added left to right)."""
    s = D[:, None, 0] * C[None, :, 0]
    for j in range(1, VEC):
        s = s + D[:, None, j] * C[None, :, j]
    return s


def kmeans_step(D, C, chunk: int = 1024):
    """One iteration of the radius-weighted spherical k-means of §3.1 on
    sampled unit directions D (S, 8) from centres C (K, 8), float64:
    every sample goes to the centre of largest cosine (Eq. (5); the scores of
    kmeans_scores, ties to the lowest index); every centre becomes the
    normalised sum of its members (an empty cluster keeps its centre).
    Returns (new centres, assignment z, objective = mean of the assigned
    scores, taken before the update)."""
    D = np.asarray(D, np.float64)
    C = np.asarray(C, np.float64)
    S = D.shape[0]
    z = np.empty(S, np.int64)
    best = np.empty(S, np.float64)
    for s0 in range(0, S, chunk):
        sc = kmeans_scores(D[s0:s0 + chunk], C)
        z[s0:s0 + chunk] = np.argmax(sc, axis=1)
        best[s0:s0 + chunk] = sc[np.arange(sc.shape[0]), z[s0:s0 + chunk]]
    sums = np.zeros_like(C)
    np.add.at(sums, z, D)
    norms = np.sqrt(np.sum(sums * sums, axis=1))
    out = C.copy()
    keep = norms > 0
    out[keep] = sums[keep] / norms[keep, None]
    return out, z, float(np.mean(best))


def kmeans_codebook(w, K: int, samples: int = 65536, iters: int = 20, seed: int = 0):
    """Radius-weighted spherical k-means initialisation of the positive
    direction codebook (§3.1, App. A step 6; 65,536 samples and 20 iterations
    in the paper's runs).

    The 8-D vectors of w (rows, cols) are decomposed by Eq. (3); `samples`
    directions are drawn with probability proportional to r_i^2
    (sample_directions, uniforms from a seeded generator); K of them, chosen
    without replacement, seed the centres; then `iters` steps of kmeans_step.
    Directions are non-negative, so the centres stay in the positive orthant.
    Returns (centres (K, 8) float64, objective per iteration: the mean of
    max_k d_i . c_k over the samples, taken before each update)."""
    rng = np.random.default_rng(seed)
    D, _ = sample_directions(w, rng.random(samples))
    centres = D[rng.choice(samples, size=K, replace=False)].copy()
    history = []
    for _ in range(iters):
        centres, _, obj = kmeans_step(D, centres)
        history.append(obj)
    return centres, history
