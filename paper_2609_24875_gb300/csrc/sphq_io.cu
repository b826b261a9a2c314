// Export / import of a packed handle (the device image as one host blob) and
// the self-test of the bounded on-chip waits.  Neither has a counterpart in
// the paper; they are interface choices of this library.
#include <cuda_runtime.h>

#include <cstring>

#include "sphq_gemv_kernel.cuh"

namespace sphq {

// Blob layout (little-endian host memory):
//   header  48 B: "SPHQ", format 1 (u32), rows, cols, bits, radius_bits, K,
//           vector dimension (i32; 0 reads as 8), unit bytes (u64),
//           packed-units bytes (u64)
//   codebook K x dim fp16 | scale rows x ng fp16 | offset rows x ng fp16 | units
struct BlobHeader {
  char magic[4];
  uint32_t format;
  int32_t rows, cols, bits, radius_bits, K, dim;
  uint64_t unit_bytes, units_bytes;
};
static_assert(sizeof(BlobHeader) == 48, "blob header");
constexpr uint32_t kBlobFormat = 1;

static size_t blob_size(const sphq_handle_s* h, size_t* units_bytes) {
  const size_t ub = (size_t)h->nrt * h->ng * h->unit_bytes;
  if (units_bytes) *units_bytes = ub;
  return sizeof(BlobHeader) + (size_t)h->K * h->dim * 2 + 2 * (size_t)h->rows * h->ng * 2 + ub;
}

// The one wait of this kernel can never complete (nothing arrives on the
// mbarrier): it gives up after ~2 s like every other on-chip wait of the
// library, records bit 1 in the error word and returns.
__global__ void wait_timeout_kernel(int* flag) {
  __shared__ __align__(8) uint64_t bar;
  if (threadIdx.x == 0) {
    mbar_init(smem_u32(&bar), 1);
    fence_mbar_init();
    if (!mbar_wait(smem_u32(&bar), 0)) atomicOr(flag, 2);
  }
}

}  // namespace sphq

using namespace sphq;

extern "C" {

sphq_status sphq_export(sphq_handle h, void* buf, size_t capacity, size_t* size) {
  clear_error();
  if (!h || !size) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_export: NULL argument");
  size_t ub = 0;
  const size_t need = blob_size(h, &ub);
  *size = need;
  if (!buf) return SPHQ_OK;
  if (capacity < need) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_export: buffer too small");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_export: handle not packed");
  BlobHeader hd;
  std::memset(&hd, 0, sizeof(hd));
  std::memcpy(hd.magic, "SPHQ", 4);
  hd.format = kBlobFormat;
  hd.rows = h->rows;
  hd.cols = h->cols;
  hd.bits = h->bits;
  hd.radius_bits = h->vbits;
  hd.K = h->K;
  hd.dim = h->dim;
  hd.unit_bytes = h->unit_bytes;
  hd.units_bytes = ub;
  uint8_t* p = static_cast<uint8_t*>(buf);
  std::memcpy(p, &hd, sizeof(hd));
  p += sizeof(hd);
  const size_t np = (size_t)h->rows * h->ng;
  const size_t cbb = (size_t)h->K * h->dim * 2;
  cudaError_t e = cudaMemcpy(p, h->codebook, cbb, cudaMemcpyDeviceToHost);
  p += cbb;
  if (e == cudaSuccess) e = cudaMemcpy(p, h->params, 2 * np * 2, cudaMemcpyDeviceToHost);
  p += 2 * np * 2;
  if (e == cudaSuccess) e = cudaMemcpy(p, h->units, ub, cudaMemcpyDeviceToHost);
  if (e != cudaSuccess) return cuda_error(e, "sphq_export: copy");
  return SPHQ_OK;
}

sphq_status sphq_import(const void* buf, size_t size, sphq_handle* out) {
  clear_error();
  if (!out) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: out is NULL");
  *out = nullptr;
  if (!buf || size < sizeof(BlobHeader))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: blob too small");
  BlobHeader hd;
  std::memcpy(&hd, buf, sizeof(hd));
  if (std::memcmp(hd.magic, "SPHQ", 4) != 0 || hd.format != kBlobFormat)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: not an sphq blob of this format");
  if (hd.rows < 1 || hd.cols < 128 || hd.cols % 128 != 0 || hd.K < 1 ||
      (long long)hd.rows * hd.cols > (1LL << 40))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: bad shape in header");
  const uint8_t* p = static_cast<const uint8_t*>(buf) + sizeof(BlobHeader);
  const int dim = hd.dim == 0 ? 8 : hd.dim;
  if (dim != 4 && dim != 8 && dim != 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: bad dimension");
  const size_t np = (size_t)hd.rows * (hd.cols / 128);
  const size_t cbb = (size_t)hd.K * dim * 2;
  const size_t fixed = sizeof(BlobHeader) + cbb + 2 * np * 2;
  if (size < fixed) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: blob truncated");
  sphq_handle h = nullptr;
  sphq_status st = sphq_create_dim(hd.rows, hd.cols, dim, hd.bits, hd.radius_bits, hd.K, p,
                                   p + cbb, p + cbb + np * 2, &h);
  if (st != SPHQ_OK) return st;
  size_t ub = 0;
  const size_t need = blob_size(h, &ub);
  if (size != need || hd.units_bytes != ub || hd.unit_bytes != h->unit_bytes) {
    sphq_destroy(h);
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_import: blob size does not match its header");
  }
  cudaError_t e = cudaMemcpy(h->units, p + cbb + 2 * np * 2, ub,
                             cudaMemcpyHostToDevice);
  if (e != cudaSuccess) {
    sphq_destroy(h);
    return cuda_error(e, "sphq_import: copy");
  }
  h->packed = true;
  *out = h;
  return SPHQ_OK;
}

sphq_status sphq_selftest_wait_timeout(sphq_handle h, sphq_stream stream) {
  clear_error();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_selftest_wait_timeout: NULL handle");
  wait_timeout_kernel<<<1, 32, 0, reinterpret_cast<cudaStream_t>(stream)>>>(h->flag + 1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "sphq_selftest_wait_timeout launch");
  return SPHQ_OK;
}

}  // extern "C"
