"""Seeded synthetic inputs for the SPHQuant decode GEMV.

This module only draws random numbers and lays them out; it holds none of the
method's arithmetic (no decode, no radius dequantisation, no matvec).  Both the
CUDA path (tests, bench.py, smoke()) and the oracle consume what it returns.

Recipe (every draw from numpy's PCG64, seed = 20260 + 100*config + shape):
  draw order  codebook, scale, offset, sign, idx, rcode, x
  codebook    K rows of |N(0, I_8)|, each scaled to unit length, rounded to fp16
  scale       Delta_G ~ U(0.5, 2)  -> fp16, one per 128-column group
  offset      r_min_G ~ U(0, 1)    -> fp16
  sign        U{0..255} per 8-D vector
  idx         U{0..K-1}
  rcode       U{0..2^V - 1}, V = 4 (or 3 for the 3-bit-radius W3 split)
  x           N(0, 1) -> fp16, shape (B, cols)
Gaussian weight matrices (the encoded configuration) are N(0, 0.02^2) with
0.1% of the scalars, chosen uniformly, multiplied by 20.

fp16 values are carried as uint16 bit patterns (numpy float16 views).
"""
from __future__ import annotations

from dataclasses import dataclass

import numpy as np

VEC = 8
GROUP_COLS = 128
RADIUS_BITS = 4


def bits_to_K(bits: int) -> int:
    """Codebook size for the W2 / W3 settings: 2^(7B-8) entries."""
    return 1 << (7 * bits - 8)


@dataclass
class Codes:
    """Canonical codes of one quantised rows x cols matrix (host numpy)."""
    bits: int
    codebook: np.ndarray  # (K, 8) uint16 fp16 bits
    scale: np.ndarray     # (rows, cols/128) uint16 fp16 bits
    offset: np.ndarray    # (rows, cols/128) uint16 fp16 bits
    sign: np.ndarray      # (rows, cols/8) uint8
    idx: np.ndarray       # (rows, cols/8) uint16
    rcode: np.ndarray     # (rows, cols/8) uint8
    vbits: int = RADIUS_BITS  # radius code width V (codes < 2^V)

    @property
    def rows(self) -> int:
        return self.sign.shape[0]

    @property
    def cols(self) -> int:
        return self.sign.shape[1] * VEC

    @property
    def K(self) -> int:
        return self.codebook.shape[0]

    def row_slice(self, r0: int, r1: int) -> "Codes":
        return Codes(self.bits, self.codebook, self.scale[r0:r1], self.offset[r0:r1],
                     self.sign[r0:r1], self.idx[r0:r1], self.rcode[r0:r1], self.vbits)


def seed_for(config: int, shape: int = 0) -> int:
    return 20260 + 100 * config + shape


def to_f16_bits(a) -> np.ndarray:
    return np.asarray(a, np.float64).astype(np.float16).view(np.uint16)


def make_codebook(rng: np.random.Generator, K: int, dim: int = VEC) -> np.ndarray:
    c = np.abs(rng.standard_normal((K, dim)))
    c /= np.linalg.norm(c, axis=1, keepdims=True)
    return to_f16_bits(c)


def make_params(rng: np.random.Generator, rows: int, cols: int):
    ng = cols // GROUP_COLS
    scale = to_f16_bits(rng.uniform(0.5, 2.0, size=(rows, ng)))
    offset = to_f16_bits(rng.uniform(0.0, 1.0, size=(rows, ng)))
    return scale, offset


def make_x(rng: np.random.Generator, B: int, cols: int) -> np.ndarray:
    return to_f16_bits(rng.standard_normal((B, cols)))


def random_codes(bits: int, rows: int, cols: int, seed: int, B: int = 1,
                 codebook: np.ndarray | None = None, radius_bits: int = RADIUS_BITS,
                 K: int | None = None):
    """Uniformly random codes (configurations 0, 2, 3, 4), radius codes drawn
    from U{0..2^radius_bits - 1}, direction indices from U{0..K-1} (K defaults
    to the codebook size of `bits`).  Returns (Codes, x)."""
    if cols % GROUP_COLS:
        raise ValueError("cols must be a multiple of 128")
    rng = np.random.Generator(np.random.PCG64(seed))
    K = bits_to_K(bits) if K is None else K
    cb = make_codebook(rng, K)
    if codebook is not None:
        cb = codebook
    scale, offset = make_params(rng, rows, cols)
    nv = cols // VEC
    sign = rng.integers(0, 256, size=(rows, nv), dtype=np.uint8)
    idx = rng.integers(0, K, size=(rows, nv), dtype=np.uint16)
    rcode = rng.integers(0, 1 << radius_bits, size=(rows, nv), dtype=np.uint8)
    x = make_x(rng, B, cols)
    return Codes(bits, cb, scale, offset, sign, idx, rcode, radius_bits), x


@dataclass
class CodesDim:
    """Canonical codes of a matrix of dim-D vectors (Tab. 7: dim 4, 8, 16)."""
    dim: int
    bits: int
    codebook: np.ndarray  # (K, dim) uint16 fp16 bits
    scale: np.ndarray     # (rows, cols/128) uint16 fp16 bits
    offset: np.ndarray
    sign: np.ndarray      # (rows, cols/dim) uint16, bit j = coordinate j negative
    idx: np.ndarray       # (rows, cols/dim) uint16
    rcode: np.ndarray     # (rows, cols/dim) uint8
    vbits: int = RADIUS_BITS

    @property
    def rows(self) -> int:
        return self.sign.shape[0]

    @property
    def cols(self) -> int:
        return self.sign.shape[1] * self.dim

    @property
    def K(self) -> int:
        return self.codebook.shape[0]


def random_codes_dim(dim: int, bits: int, rows: int, cols: int, seed: int, B: int = 1,
                     radius_bits: int = RADIUS_BITS):
    """Uniformly random codes of dim-D vectors: K = 2^((dim-1) bits - dim) entries
    of |N(0, I_dim)| normalised, same draw order as random_codes.  Returns
    (CodesDim, x)."""
    if cols % GROUP_COLS:
        raise ValueError("cols must be a multiple of 128")
    rng = np.random.Generator(np.random.PCG64(seed))
    K = 1 << ((dim - 1) * bits - dim)
    cb = make_codebook(rng, K, dim)
    scale, offset = make_params(rng, rows, cols)
    nv = cols // dim
    sign = rng.integers(0, 1 << dim, size=(rows, nv), dtype=np.uint32).astype(np.uint16)
    idx = rng.integers(0, K, size=(rows, nv), dtype=np.uint16)
    rcode = rng.integers(0, 1 << radius_bits, size=(rows, nv), dtype=np.uint8)
    x = make_x(rng, B, cols)
    return CodesDim(dim, bits, cb, scale, offset, sign, idx, rcode, radius_bits), x


def gaussian_weights(rows: int, cols: int, seed: int, std: float = 0.02,
                     outlier_frac: float = 1e-3, outlier_mult: float = 20.0):
    """W ~ N(0, std^2) with a uniformly chosen fraction of scalars scaled up."""
    rng = np.random.Generator(np.random.PCG64(seed + 7))
    w = rng.standard_normal((rows, cols)) * std
    n_out = int(round(outlier_frac * rows * cols))
    pos = rng.choice(rows * cols, size=n_out, replace=False)
    w.reshape(-1)[pos] *= outlier_mult
    return w


def encoded_inputs_rng(bits: int, cols: int, seed: int, B: int = 1):
    """Codebook and activations for the encoded configuration (the codes themselves
    come from an encoder run on gaussian_weights)."""
    rng = np.random.Generator(np.random.PCG64(seed))
    cb = make_codebook(rng, bits_to_K(bits))
    x = make_x(rng, B, cols)
    return cb, x


# ---------------------------------------------------------------------------
# workload shapes
# ---------------------------------------------------------------------------

# 7B-class decoder projections (hidden 3584, 28 q heads / 4 kv heads of 128, FFN 18944):
# (name, rows = d_out, cols = d_in)
DECODER_PROJ = [
    ("q", 3584, 3584),
    ("k", 512, 3584),
    ("v", 512, 3584),
    ("o", 3584, 3584),
    ("gate", 18944, 3584),
    ("up", 18944, 3584),
    ("down", 3584, 18944),
]
DECODER_LAYERS = 28
# The same linears with the projections that read the same activations fused
# by row concatenation (q|k|v and gate|up), as serving engines store them.
DECODER_PROJ_FUSED = [("qkv", 3584 + 512 + 512, 3584), ("o", 3584, 3584),
                      ("gate_up", 2 * 18944, 3584), ("down", 3584, 18944)]

# square sweep at batch 1: (bits, n)
SQUARE_SWEEP = [(2, 4096), (2, 8192), (3, 4096), (3, 8192)]
