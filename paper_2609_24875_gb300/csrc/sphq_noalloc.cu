// sphq_gemv_noalloc: the GEMV with any split-K scratch in a fixed, file-scope
// device array instead of memory allocated for it (the current kernel reduces
// on chip and uses none).
//
// The scratch is one `static __device__` array of kScratchBytes on every GPU
// that loads this library; it lives until the process exits.  Host code may
// not pass the array's name to a kernel (on the host that name is only a
// stand-in for the symbol), so the first call on each device looks up the
// array's device address with cudaGetSymbolAddress, with that device current,
// and caches it.  Every call shares the array: calls that run concurrently on
// the GPU (on different streams, or from different threads) race on it.
#include <cuda_runtime.h>

#include <mutex>

#include "sphq_internal.h"

namespace sphq {

constexpr size_t kScratchBytes = 4u << 20;       // 4 MiB in all
constexpr size_t kTicketBytes = 64u << 10;       // counters for up to 16384 row tiles
constexpr size_t kPartialBytes = kScratchBytes - kTicketBytes;

static __device__ __align__(256) unsigned char g_scratch[kScratchBytes];

static std::mutex g_scratch_mu;
static void* g_scratch_addr[64] = {};

// Device address of g_scratch on the current device (looked up once per device).
static sphq_status scratch_address(int device, void** out) {
  std::lock_guard<std::mutex> lock(g_scratch_mu);
  if (device < 0 || device >= 64)
    return set_error(SPHQ_ERR_DEVICE, "sphq_gemv_noalloc: device index out of range");
  if (!g_scratch_addr[device]) {
    void* p = nullptr;
    cudaError_t e = cudaGetSymbolAddress(&p, g_scratch);
    if (e != cudaSuccess) return cuda_error(e, "sphq_gemv_noalloc: cudaGetSymbolAddress");
    g_scratch_addr[device] = p;
  }
  *out = g_scratch_addr[device];
  return SPHQ_OK;
}

}  // namespace sphq

using namespace sphq;

extern "C" sphq_status sphq_gemv_noalloc(sphq_handle h, const void* x, void* y, int batch,
                                         sphq_stream stream) {
  set_error(SPHQ_OK, "");
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_noalloc: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv_noalloc: batch must be 1..16");
  if (!x || reinterpret_cast<uintptr_t>(x) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG,
                     "sphq_gemv_noalloc: x must be a 16-byte aligned pointer");
  if (!y || reinterpret_cast<uintptr_t>(y) % 4)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_noalloc: y must be a 4-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemv_noalloc: handle not packed");
  // The limit binds only a plan that reduces through global scratch; the
  // current plans reduce on chip and take any shape sphq_gemv takes.
  if (h->ws_floats > 0 && ((size_t)h->nrt * sizeof(unsigned) > kTicketBytes ||
                           h->ws_floats * sizeof(float) > kPartialBytes))
    return set_error(SPHQ_ERR_UNSUPPORTED,
                     "sphq_gemv_noalloc: the matrix needs more split-K scratch than the fixed "
                     "4 MiB device array holds (at most 16384 row tiles of 16 rows and "
                     "4128768 bytes of partial sums); use sphq_gemv");
  int dev = -1;
  cudaError_t e = cudaGetDevice(&dev);
  if (e != cudaSuccess) return cuda_error(e, "sphq_gemv_noalloc: cudaGetDevice");
  if (dev != h->device)
    return set_error(SPHQ_ERR_DEVICE,
                     "sphq_gemv_noalloc: the current device is not the handle's device");
  void* base = nullptr;
  sphq_status st = scratch_address(dev, &base);
  if (st != SPHQ_OK) return st;
  unsigned char* b = static_cast<unsigned char*>(base);
  unsigned* tickets = reinterpret_cast<unsigned*>(b);
  float* ws = reinterpret_cast<float*>(b + kTicketBytes);
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  if (h->ws_floats > 0) {
    // a plan with split-K partials needs its row-tile counters at zero; the
    // array keeps whatever the previous call left, so clear the part it uses
    e = cudaMemsetAsync(tickets, 0, (size_t)h->nrt * sizeof(unsigned), s);
    if (e != cudaSuccess) return cuda_error(e, "sphq_gemv_noalloc: clear counters");
  }
  return launch_gemv_scratch(h, x, y, batch, s, ws, tickets);
}
