// Host-side internals of the sphq library (not part of the C ABI).
#pragma once
#include <cuda_runtime.h>

#include <cstddef>
#include <cstdint>
#include <string>

#include "../../include/sphq.h"

namespace sphq {

// Launch plan of the GEMV kernel for one batch size.
struct GemvPlan {
  int warps_per_cta = 0;   // threads / 32
  int grid = 0;            // CTAs (persistent: at most SMs x resident CTAs)
  int units_per_warp = 0;  // contiguous (row block, group) units per warp
  int max_slots = 0;       // most warps that share one row block
  size_t smem = 0;         // dynamic shared memory per CTA
  int mode = 0;            // radius application: 1, 2 (factored) or 8 (full)
};

}  // namespace sphq

struct sphq_handle_s {
  int rows = 0, cols = 0, bits = 0, K = 0;
  int nrt = 0;             // row tiles of 16 rows
  int ng = 0;              // radius groups per row (cols / 128)
  int device = 0;
  int sm_count = 0;
  size_t unit_bytes = 0;
  void* units = nullptr;       // packed units, nrt * ng * unit_bytes
  void* codebook = nullptr;    // K * 8 fp16
  uint32_t* params = nullptr;  // rows * ng words: Delta | r_min << 16
  float* ws = nullptr;         // split-K partial sums
  size_t ws_floats = 0;
  unsigned* tickets = nullptr; // one arrival counter per row tile
  int* flag = nullptr;         // pack validation flag
  void* xstage = nullptr;      // SPHQ_MAX_BATCH x cols fp16 (sphq_gemv_host)
  void* ystage = nullptr;      // SPHQ_MAX_BATCH x rows fp16
  void* zeros = nullptr;       // 256 B of zeros (activations of non-supplying lanes)
  bool packed = false;
  sphq::GemvPlan plan[SPHQ_MAX_BATCH + 1];
};

namespace sphq {

sphq_status set_error(sphq_status s, const std::string& msg);
sphq_status cuda_error(cudaError_t e, const char* what);

// Builds the GEMV launch plans of a handle (sizes its workspace needs).
sphq_status make_gemv_plans(sphq_handle h);
// Enqueues the GEMV (validated arguments).
sphq_status launch_gemv(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s);
// Enqueues the GEMV with caller-provided split-K scratch: `ws` holds at least
// h->ws_floats floats and `tickets` h->nrt zeroed counters.
sphq_status launch_gemv_scratch(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s,
                                float* ws, unsigned* tickets);

}  // namespace sphq
