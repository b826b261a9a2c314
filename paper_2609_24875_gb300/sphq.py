"""Thin Python binding of libsphq.so (include/sphq.h): argument marshalling only.

Every step of the decode-GEMV runs in the library's CUDA kernels; PyTorch is
used here only to own device memory and to name the current CUDA stream.
If the library has not been built this module raises on import of the
library -- there is no CPU fallback.
"""
from __future__ import annotations

import ctypes
import os
import re

HERE = os.path.dirname(os.path.abspath(__file__))
LIB_PATH = os.path.join(HERE, "libsphq.so")
HEADER = os.path.join(os.path.dirname(HERE), "include", "sphq.h")

SPHQ_OK = 0
STATUS = {0: "SPHQ_OK", 1: "SPHQ_ERR_INVALID_ARG", 2: "SPHQ_ERR_UNSUPPORTED",
          3: "SPHQ_ERR_NOT_PACKED", 4: "SPHQ_ERR_CUDA", 5: "SPHQ_ERR_OOM",
          6: "SPHQ_ERR_DEVICE", 7: "SPHQ_ERR_TIMEOUT"}
MAX_BATCH = 16

_lib = None


class SphqError(RuntimeError):
    def __init__(self, status: int, msg: str):
        super().__init__(f"{STATUS.get(status, status)}: {msg}")
        self.status = status


class PlanInfo(ctypes.Structure):
    """sphq_plan_info: the GEMV launch shape for one batch size."""
    _fields_ = [("grid", ctypes.c_int), ("cluster_size", ctypes.c_int),
                ("clusters", ctypes.c_int), ("tiles_per_cluster", ctypes.c_int),
                ("warps_per_cta", ctypes.c_int), ("smem_bytes", ctypes.c_int),
                ("staged_x", ctypes.c_int), ("ctas_per_sm", ctypes.c_int)]


class GemmInfo(ctypes.Structure):
    """sphq_gemm_info: the prefill GEMM launch shape for one batch size."""
    _fields_ = [("act_tiles", ctypes.c_int), ("weight_rows", ctypes.c_int),
                ("stage_cols", ctypes.c_int), ("stages", ctypes.c_int),
                ("grid_x", ctypes.c_int), ("grid_y", ctypes.c_int),
                ("smem_bytes", ctypes.c_longlong), ("split_ctas", ctypes.c_int),
                ("ksplit", ctypes.c_int)]


def load() -> ctypes.CDLL:
    """Load libsphq.so (built by __graft_entry__.build()); raises if missing."""
    global _lib
    if _lib is None:
        if not os.path.exists(LIB_PATH):
            raise RuntimeError(
                f"{LIB_PATH} is missing: build the CUDA library first "
                "(python -c 'import __graft_entry__ as g; g.build()')")
        L = ctypes.CDLL(LIB_PATH)
        vp, i32, sz = ctypes.c_void_p, ctypes.c_int, ctypes.c_size_t
        L.sphq_create.argtypes = [i32, i32, i32, i32, vp, vp, vp, ctypes.POINTER(vp)]
        L.sphq_create.restype = i32
        L.sphq_create_v.argtypes = [i32, i32, i32, i32, i32, vp, vp, vp, ctypes.POINTER(vp)]
        L.sphq_create_v.restype = i32
        L.sphq_create_dim.argtypes = [i32, i32, i32, i32, i32, i32, vp, vp, vp,
                                      ctypes.POINTER(vp)]
        L.sphq_create_dim.restype = i32
        L.sphq_pack.argtypes = [vp, vp, vp, vp, vp]
        L.sphq_pack.restype = i32
        L.sphq_gemv.argtypes = [vp, vp, vp, i32, vp]
        L.sphq_gemv.restype = i32
        L.sphq_gemv_noalloc.argtypes = [vp, vp, vp, i32, vp]
        L.sphq_gemv_noalloc.restype = i32
        L.sphq_sample_directions.argtypes = [vp, ctypes.c_longlong, vp, i32, vp, vp, vp]
        L.sphq_sample_directions.restype = i32
        L.sphq_kmeans_step.argtypes = [vp, i32, vp, i32, vp, vp, vp, vp]
        L.sphq_kmeans_step.restype = i32
        L.sphq_kmeans.argtypes = [vp, i32, vp, i32, i32, vp, vp]
        L.sphq_kmeans.restype = i32
        L.sphq_angle_codebook.argtypes = [vp, i32, ctypes.c_double, vp, vp, vp]
        L.sphq_angle_codebook.restype = i32
        L.sphq_gemm.argtypes = [vp, vp, vp, i32, vp]
        L.sphq_gemm.restype = i32
        L.sphq_gemm_workspace.argtypes = [vp, i32, ctypes.POINTER(sz)]
        L.sphq_gemm_workspace.restype = i32
        L.sphq_gemm_ws.argtypes = [vp, vp, vp, i32, vp, sz, vp]
        L.sphq_gemm_ws.restype = i32
        L.sphq_check.argtypes = [vp, vp]
        L.sphq_check.restype = i32
        L.sphq_export.argtypes = [vp, vp, sz, ctypes.POINTER(sz)]
        L.sphq_export.restype = i32
        L.sphq_import.argtypes = [vp, sz, ctypes.POINTER(vp)]
        L.sphq_import.restype = i32
        L.sphq_selftest_wait_timeout.argtypes = [vp, vp]
        L.sphq_selftest_wait_timeout.restype = i32
        L.sphq_encode.argtypes = [vp, vp, vp, vp, vp, vp, vp, vp]
        L.sphq_encode.restype = i32
        L.sphq_get_gemm_shape.argtypes = [vp, i32, ctypes.POINTER(GemmInfo)]
        L.sphq_get_gemm_shape.restype = i32
        L.sphq_set_gemm_shape.argtypes = [vp, i32, i32]
        L.sphq_set_gemm_shape.restype = i32
        L.sphq_gemv_host.argtypes = [vp, vp, vp, i32, vp]
        L.sphq_gemv_host.restype = i32
        L.sphq_decode.argtypes = [vp, vp, vp]
        L.sphq_decode.restype = i32
        L.sphq_bytes.argtypes = [vp, i32]
        L.sphq_bytes.restype = sz
        L.sphq_destroy.argtypes = [vp]
        L.sphq_destroy.restype = i32
        L.sphq_last_error.argtypes = []
        L.sphq_last_error.restype = ctypes.c_char_p
        L.sphq_version.argtypes = []
        L.sphq_version.restype = i32
        L.sphq_get_plan.argtypes = [vp, i32, ctypes.POINTER(PlanInfo)]
        L.sphq_get_plan.restype = i32
        L.sphq_set_cluster_size.argtypes = [vp, i32, i32]
        L.sphq_set_cluster_size.restype = i32
        L.sphq_set_pdl.argtypes = [vp, i32]
        L.sphq_set_pdl.restype = i32
        _lib = L
    return _lib


def header_functions() -> list[str]:
    """Names of the functions include/sphq.h declares."""
    text = open(HEADER).read()
    text = re.sub(r"/\*.*?\*/", "", text, flags=re.S)
    return sorted(set(re.findall(r"\b(sphq_[a-z_0-9]+)\s*\(", text)))


def _check(status: int) -> None:
    if status != SPHQ_OK:
        raise SphqError(status, load().sphq_last_error().decode())


def _stream_ptr(stream) -> int:
    import torch
    if stream is None:
        stream = torch.cuda.current_stream()
    return int(stream.cuda_stream)


class SphqMatrix:
    """One quantised weight matrix resident on the current CUDA device.

    codebook: (K, 8) float16/uint16 tensor; scale, offset: (rows, cols/128).
    Host or device tensors are accepted for these three (they are copied).
    """

    def __init__(self, rows: int, cols: int, bits: int, codebook, scale, offset,
                 radius_bits: int = 4, K: int | None = None, dim: int = 8):
        """bits 2 or 3; K defaults to 2^((dim-1)*bits - dim) (64 / 8192 for 8-D);
        the Tab. 4 splits take K = 128 or 256 at bits = 2 and radius_bits 2 or 3
        (sphq_create_v); dim = 4 takes bits 2, K 4 and dim = 16 bits 2, K 16384
        (sphq_create_dim)."""
        import torch
        L = load()
        if K is None:
            K = 1 << ((dim - 1) * bits - dim)
        cb = codebook.contiguous()
        sc = scale.contiguous()
        of = offset.contiguous()
        for t, shape in ((cb, (K, dim)), (sc, (rows, cols // 128)), (of, (rows, cols // 128))):
            if tuple(t.shape) != shape or t.element_size() != 2:
                raise ValueError(f"expected a 2-byte tensor of shape {shape}, got "
                                 f"{tuple(t.shape)} {t.dtype}")
        h = ctypes.c_void_p()
        _check(L.sphq_create_dim(rows, cols, dim, bits, radius_bits, K, cb.data_ptr(),
                                 sc.data_ptr(), of.data_ptr(), ctypes.byref(h)))
        self._h = h
        self.rows, self.cols, self.bits, self.K = rows, cols, bits, K
        self.radius_bits, self.dim = radius_bits, dim
        self.device = torch.device("cuda", torch.cuda.current_device())

    @property
    def handle(self) -> int:
        return self._h.value

    def pack(self, sign, idx, rcode, stream=None) -> None:
        """sign/idx/rcode: (rows, cols/dim) uint8 (16-D: 2-byte) / uint16(int16) / uint8
        device tensors."""
        nv = self.cols // self.dim
        for t in (sign, idx, rcode):
            if tuple(t.shape) != (self.rows, nv) or not t.is_cuda or not t.is_contiguous():
                raise ValueError("codes must be contiguous CUDA tensors of shape (rows, cols/8)")
        if (sign.element_size() != (2 if self.dim == 16 else 1) or rcode.element_size() != 1
                or idx.element_size() != 2):
            raise ValueError("sign (2 bytes for 16-D vectors, else 1) / rcode 1-byte and idx "
                             "2-byte tensors expected")
        _check(load().sphq_pack(self._h, sign.data_ptr(), idx.data_ptr(), rcode.data_ptr(),
                                _stream_ptr(stream)))

    def gemv(self, x, y=None, stream=None):
        """y = W_hat x.  x: (batch, cols) fp16 on the device; returns (batch, rows) fp16."""
        import torch
        if x.dim() == 1:
            x = x.unsqueeze(0)
        B = x.shape[0]
        if x.shape[1] != self.cols or x.element_size() != 2 or not x.is_cuda:
            raise ValueError("x must be a (batch, cols) 2-byte CUDA tensor")
        x = x.contiguous()
        if y is None:
            y = torch.empty((B, self.rows), dtype=torch.float16, device=x.device)
        _check(load().sphq_gemv(self._h, x.data_ptr(), y.data_ptr(), B, _stream_ptr(stream)))
        return y

    def export(self) -> bytes:
        """sphq_export: the packed device image as a host blob."""
        L = load()
        size = ctypes.c_size_t()
        _check(L.sphq_export(self._h, None, 0, ctypes.byref(size)))
        buf = ctypes.create_string_buffer(size.value)
        _check(L.sphq_export(self._h, buf, size.value, ctypes.byref(size)))
        return buf.raw

    @classmethod
    def from_blob(cls, blob: bytes) -> "SphqMatrix":
        """sphq_import: a packed matrix on the current device from a blob."""
        import struct

        import torch
        L = load()
        h = ctypes.c_void_p()
        _check(L.sphq_import(blob, len(blob), ctypes.byref(h)))
        _, _, rows, cols, bits, vbits, K, dim = struct.unpack_from("<4sIiiiiii", blob, 0)
        m = cls.__new__(cls)
        m._h = h
        m.rows, m.cols, m.bits, m.K, m.radius_bits = rows, cols, bits, K, vbits
        m.dim = dim or 8
        m.device = torch.device("cuda", torch.cuda.current_device())
        return m

    def selftest_wait_timeout(self, stream=None) -> None:
        """sphq_selftest_wait_timeout: a kernel whose one wait never completes
        (it gives up after ~2 s and sets the error word; see check())."""
        _check(load().sphq_selftest_wait_timeout(self._h, _stream_ptr(stream)))

    def encode(self, w, stream=None):
        """sphq_encode: quantise w ((rows, cols) float32 CUDA tensor) with this
        matrix's codebook and pack it.  Returns the canonical codes and group
        parameters as CUDA tensors: sign, idx, rcode (rows, cols/8) and scale,
        offset (rows, cols/128, fp16 bits as int16)."""
        import torch
        if (tuple(w.shape) != (self.rows, self.cols) or w.dtype != torch.float32
                or not w.is_cuda or not w.is_contiguous()):
            raise ValueError("w must be a contiguous (rows, cols) float32 CUDA tensor")
        nv, ng = self.cols // 8, self.cols // 128
        dev = w.device
        sign = torch.empty((self.rows, nv), dtype=torch.uint8, device=dev)
        idx = torch.empty((self.rows, nv), dtype=torch.int16, device=dev)
        rcode = torch.empty((self.rows, nv), dtype=torch.uint8, device=dev)
        scale = torch.empty((self.rows, ng), dtype=torch.int16, device=dev)
        offset = torch.empty((self.rows, ng), dtype=torch.int16, device=dev)
        _check(load().sphq_encode(self._h, w.data_ptr(), sign.data_ptr(), idx.data_ptr(),
                                  rcode.data_ptr(), scale.data_ptr(), offset.data_ptr(),
                                  _stream_ptr(stream)))
        return sign, idx, rcode, scale, offset

    def gemm(self, x, y=None, stream=None):
        """Y = X W_hat^T on the tensor cores for any batch (prefill).
        x: (batch, cols) fp16 on the device; returns (batch, rows) fp16."""
        import torch
        if x.dim() == 1:
            x = x.unsqueeze(0)
        B = x.shape[0]
        if x.shape[1] != self.cols or x.element_size() != 2 or not x.is_cuda:
            raise ValueError("x must be a (batch, cols) 2-byte CUDA tensor")
        x = x.contiguous()
        if y is None:
            y = torch.empty((B, self.rows), dtype=torch.float16, device=x.device)
        _check(load().sphq_gemm(self._h, x.data_ptr(), y.data_ptr(), B, _stream_ptr(stream)))
        return y

    def gemm_workspace(self, batch: int) -> int:
        """Workspace bytes for sphq_gemm_ws at `batch` when the two-pass form
        is estimated faster, else 0 (sphq_gemm_workspace)."""
        n = ctypes.c_size_t(0)
        _check(load().sphq_gemm_workspace(self._h, batch, ctypes.byref(n)))
        return n.value

    def gemm_ws(self, x, workspace, y=None, stream=None):
        """sphq_gemm_ws: the product with a caller-provided device workspace
        (W_hat decoded into it, then a dense tensor-core pass); workspace None
        runs the fused kernel.  x: (batch, cols) fp16; returns (batch, rows)."""
        import torch
        if x.dim() == 1:
            x = x.unsqueeze(0)
        B = x.shape[0]
        if x.shape[1] != self.cols or x.element_size() != 2 or not x.is_cuda:
            raise ValueError("x must be a (batch, cols) 2-byte CUDA tensor")
        x = x.contiguous()
        if y is None:
            y = torch.empty((B, self.rows), dtype=torch.float16, device=x.device)
        elif y.dtype != torch.float16 or y.numel() < B * self.rows or not y.is_contiguous():
            raise ValueError("y must be a contiguous fp16 tensor of batch x rows elements")
        if workspace is None:
            wp, wn = None, 0
        else:
            if not workspace.is_cuda or not workspace.is_contiguous():
                raise ValueError("workspace must be a contiguous CUDA tensor")
            wp, wn = workspace.data_ptr(), workspace.numel() * workspace.element_size()
        _check(load().sphq_gemm_ws(self._h, x.data_ptr(), y.data_ptr(), B, wp, wn,
                                   _stream_ptr(stream)))
        return y

    def gemm_ptr(self, x_ptr: int, y_ptr: int, batch: int, stream_ptr: int) -> None:
        """Raw-pointer sphq_gemm (no tensor checks)."""
        _check(load().sphq_gemm(self._h, x_ptr, y_ptr, batch, stream_ptr))

    def gemm_shape(self, batch: int) -> dict:
        """The launch shape sphq_gemm uses for `batch` (sphq_get_gemm_shape)."""
        info = GemmInfo()
        _check(load().sphq_get_gemm_shape(self._h, batch, ctypes.byref(info)))
        return {name: getattr(info, name) for name, _ in GemmInfo._fields_}

    def set_gemm_shape(self, act_tiles: int = 0, weight_rows: int = 0) -> None:
        """Fix sphq_gemm's activation tiles per CTA (1, 2) and weight rows per
        CTA (128, 256); 0 = automatic."""
        _check(load().sphq_set_gemm_shape(self._h, act_tiles, weight_rows))

    def check(self, stream=None) -> None:
        """sphq_check: synchronise the stream and raise if a kernel on this
        handle gave up an on-chip wait since the last check."""
        _check(load().sphq_check(self._h, _stream_ptr(stream)))

    def gemv_ptr(self, x_ptr: int, y_ptr: int, batch: int, stream_ptr: int) -> None:
        """Raw-pointer call (no tensor checks), for graph capture and benchmarks."""
        _check(load().sphq_gemv(self._h, x_ptr, y_ptr, batch, stream_ptr))

    def gemv_noalloc(self, x, y, stream=None):
        """sphq_gemv_noalloc: the GEMV through the entry point that guarantees
        no allocation on any call, the first included.
        x: (batch, cols) and y: (batch, rows) fp16 CUDA tensors."""
        import torch
        if x.dim() == 1:
            x = x.unsqueeze(0)
        B = x.shape[0]
        if (x.shape[1] != self.cols or not x.is_cuda or not y.is_cuda
                or not x.is_contiguous() or not y.is_contiguous() or y.numel() != B * self.rows):
            raise ValueError("x must be (batch, cols) and y (batch, rows), contiguous CUDA tensors")
        if x.element_size() != 2 or y.dtype != torch.float16:
            raise ValueError("x must hold 2-byte (fp16) elements and y must be float16")
        _check(load().sphq_gemv_noalloc(self._h, x.data_ptr(), y.data_ptr(), B,
                                        _stream_ptr(stream)))
        return y

    def gemv_host(self, x_host, y_host, stream=None) -> None:
        """Host-buffer GEMV: x_host (batch, cols) and y_host (batch, rows) are
        2-byte CPU tensors (pinned for asynchrony); the copies and the GEMV are
        enqueued on the stream, so synchronise it before reading y_host."""
        xs, ys = x_host.shape, y_host.shape
        if len(xs) == 1:
            xs = (1, xs[0])
        B = xs[0]
        if (xs[1] != self.cols or len(ys) == 0 or ys[-1] != self.rows or x_host.is_cuda
                or y_host.is_cuda or not x_host.is_contiguous() or not y_host.is_contiguous()
                or y_host.numel() != B * self.rows):
            raise ValueError("gemv_host takes contiguous host tensors x_host (batch, cols) and "
                             "y_host (batch, rows)")
        _check(load().sphq_gemv_host(self._h, x_host.data_ptr(), y_host.data_ptr(), B,
                                     _stream_ptr(stream)))

    def decode(self, stream=None):
        """W_hat as a (rows, cols) fp16 tensor (verification path)."""
        import torch
        w = torch.empty((self.rows, self.cols), dtype=torch.float16, device=self.device)
        _check(load().sphq_decode(self._h, w.data_ptr(), _stream_ptr(stream)))
        return w

    def bytes(self, batch: int = 1) -> int:
        return int(load().sphq_bytes(self._h, batch))

    def plan(self, batch: int = 1) -> dict:
        """The launch shape sphq_gemv uses for `batch` (sphq_get_plan)."""
        info = PlanInfo()
        _check(load().sphq_get_plan(self._h, batch, ctypes.byref(info)))
        return {name: getattr(info, name) for name, _ in PlanInfo._fields_}

    def set_cluster_size(self, batch: int, cluster_size: int) -> None:
        """Fix the cluster size of the launch shape for `batch` (0: automatic)."""
        _check(load().sphq_set_cluster_size(self._h, batch, cluster_size))

    def set_pdl(self, enabled: bool) -> None:
        """GEMVs as programmatic dependent launches (default) or plain ones."""
        _check(load().sphq_set_pdl(self._h, 1 if enabled else 0))

    def close(self) -> None:
        if getattr(self, "_h", None) is not None and self._h.value:
            load().sphq_destroy(self._h)
            self._h = ctypes.c_void_p()

    def __del__(self):
        try:
            self.close()
        except Exception:
            pass


# ---------------------------------------------------------------------------
# codebook construction (§3.1 sampling and spherical k-means, §3.3 angles)
# ---------------------------------------------------------------------------

def _dev_f64(t, shape, what):
    import torch
    if not t.is_cuda or t.dtype != torch.float64 or not t.is_contiguous() or tuple(t.shape) != shape:
        raise ValueError(f"{what} must be a contiguous {shape} float64 CUDA tensor")


def sample_directions(w, u, stream=None):
    """sphq_sample_directions: directions of the 8-D vectors of w (float32
    CUDA tensor, any shape with a multiple of 8 elements) drawn with
    probability proportional to r^2 by inverse transform of u (float64 CUDA
    tensor of uniforms in [0, 1)).  Returns (directions (S, 8) float64,
    indices (S,) int32)."""
    import torch
    if not w.is_cuda or w.dtype != torch.float32 or not w.is_contiguous() or w.numel() % 8:
        raise ValueError("w must be a contiguous float32 CUDA tensor of 8-D vectors")
    S = u.numel()
    _dev_f64(u, (S,), "u")
    dirs = torch.empty((S, 8), dtype=torch.float64, device=w.device)
    idx = torch.empty((S,), dtype=torch.int32, device=w.device)
    _check(load().sphq_sample_directions(w.data_ptr(), w.numel() // 8, u.data_ptr(), S,
                                         dirs.data_ptr(), idx.data_ptr(), _stream_ptr(stream)))
    return dirs, idx


def kmeans_step(dirs, centres, stream=None):
    """sphq_kmeans_step: one spherical k-means iteration.  Returns (new
    centres (K, 8) float64, assignment (S,) int32, objective (1,) float64),
    all CUDA tensors."""
    import torch
    S, K = dirs.shape[0], centres.shape[0]
    _dev_f64(dirs, (S, 8), "dirs")
    _dev_f64(centres, (K, 8), "centres")
    out = torch.empty_like(centres)
    z = torch.empty((S,), dtype=torch.int32, device=dirs.device)
    obj = torch.empty((1,), dtype=torch.float64, device=dirs.device)
    _check(load().sphq_kmeans_step(dirs.data_ptr(), S, centres.data_ptr(), K, out.data_ptr(),
                                   z.data_ptr(), obj.data_ptr(), _stream_ptr(stream)))
    return out, z, obj


def kmeans(dirs, centres, iters: int = 20, stream=None):
    """sphq_kmeans: `iters` k-means steps from `centres` (copied).  Returns
    (final centres (K, 8) float64, objective per step (iters,) float64)."""
    import torch
    S, K = dirs.shape[0], centres.shape[0]
    _dev_f64(dirs, (S, 8), "dirs")
    _dev_f64(centres, (K, 8), "centres")
    c = centres.clone()
    hist = torch.empty((max(1, iters),), dtype=torch.float64, device=dirs.device)
    _check(load().sphq_kmeans(dirs.data_ptr(), S, c.data_ptr(), K, iters, hist.data_ptr(),
                              _stream_ptr(stream)))
    return c, hist[:iters]


def angle_codebook(phi, eps: float = 1e-4, stream=None):
    """sphq_angle_codebook: (K, 7) float32 CUDA logits -> (codebook (K, 8)
    float64, codebook (K, 8) fp16) CUDA tensors."""
    import torch
    if not phi.is_cuda or phi.dtype != torch.float32 or not phi.is_contiguous() or \
            phi.dim() != 2 or phi.shape[1] != 7:
        raise ValueError("phi must be a contiguous (K, 7) float32 CUDA tensor")
    K = phi.shape[0]
    c64 = torch.empty((K, 8), dtype=torch.float64, device=phi.device)
    c16 = torch.empty((K, 8), dtype=torch.float16, device=phi.device)
    _check(load().sphq_angle_codebook(phi.data_ptr(), K, float(eps), c64.data_ptr(),
                                      c16.data_ptr(), _stream_ptr(stream)))
    return c64, c16
