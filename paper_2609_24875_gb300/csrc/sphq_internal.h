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
  int grid = 0;            // CTAs = nclusters x csize
  int csize = 1;           // CTAs per thread-block cluster (split of the groups)
  int nclusters = 0;       // clusters, each with a contiguous range of row tiles
  int tmax = 0;            // most row tiles of one cluster
  size_t smem = 0;         // dynamic shared memory per CTA
  int mode = 0;            // radius application: 1, 2 (factored) or 8 (full)
  int strip = 2;           // row tiles per work item (2, or 4 for W3 with >= 3 tiles per cluster)
  bool solo = false;       // W2: the kernel built for one CTA per SM (whole register file)
  int ctas_per_sm = 0;     // CTAs per SM the kernel is built for (its register budget)
  uint32_t cb_bytes = 0;   // staged codebook image
  uint32_t x_pitch = 0;    // bytes between staged activation rows
  uint32_t off_x = 0, off_zero = 0, off_recv = 0, off_bar = 0;
};

}  // namespace sphq

struct sphq_handle_s {
  int rows = 0, cols = 0, bits = 0, K = 0;
  int vbits = 4;           // radius code bits V
  int dbits = 6;           // direction index bits D = log2 K
  int dim = 8;             // vector dimension (8, 4 or 16)
  int fmt = 0;             // device format id (sphq_layout.cuh), one per bit split
  int nrt = 0;             // row tiles of 16 rows
  int ng = 0;              // radius groups per row (cols / 128)
  int device = 0;
  int sm_count = 0;
  size_t unit_bytes = 0;
  void* units = nullptr;       // packed units, nrt * ng * unit_bytes
  void* codebook = nullptr;    // K * 8 fp16
  void* cbimage = nullptr;     // W2: eight interleaved codebook copies (8 KiB); 16-D: lane-ordered entries
  uint32_t* params = nullptr;  // rows * ng words: Delta | r_min << 16
  float* ws = nullptr;         // split-K partial sums of plans that need them (none today)
  size_t ws_floats = 0;
  int* flag = nullptr;         // [0] pack validation, [1] kernel wait timeouts (gemv, gemm)
  void* xstage = nullptr;      // SPHQ_MAX_BATCH x cols fp16 (sphq_gemv_host)
  void* ystage = nullptr;      // SPHQ_MAX_BATCH x rows fp16
  void* zeros = nullptr;       // 256 B of zeros (activations of non-supplying lanes)
  bool pdl = true;             // sphq_set_pdl: GEMV launched as a programmatic dependent
  int gemm_mt = 0;             // sphq_set_gemm_shape: activation tiles (0 = automatic)
  int gemm_bn = 0;             //   weight rows per CTA tile (0 = automatic)
  bool packed = false;
  sphq::GemvPlan plan[SPHQ_MAX_BATCH + 1];
};

namespace sphq {

void clear_error();
bool log_enabled();  // SPHQ_LOG set: host logging to stderr
sphq_status set_error(sphq_status s, const std::string& msg);
sphq_status cuda_error(cudaError_t e, const char* what);

// Builds the GEMV launch plans of a handle (sizes its workspace needs).
sphq_status make_gemv_plans(sphq_handle h);
// Re-plans one batch size at a fixed cluster size (0: automatic choice).
sphq_status set_gemv_cluster_size(sphq_handle h, int batch, int csize);
// Enqueues the GEMV (validated arguments).
sphq_status launch_gemv(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s);
// Enqueues the encoder: codes and per-vector radii, then the group
// parameters into the handle's parameter planes.
sphq_status launch_encode(sphq_handle h, const float* w, uint8_t* sign, uint16_t* idx,
                          uint8_t* rcode, float* rtilde, cudaStream_t s);
// Launch shape sphq_gemm would use for `batch`.
sphq_status gemm_shape_info(sphq_handle h, int batch, sphq_gemm_info* out);
// Enqueues the tensor-core product for any batch (validated arguments).
sphq_status launch_gemm(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s);
// Whether a batch of 9..64 rows is estimated faster as GEMV launches of 3..8
// rows than on the tensor-core kernel.
bool gemm_prefers_gemv(sphq_handle h, int batch);
// Workspace bytes of the two-pass product for `batch` when it is estimated
// faster than the fused kernel, else 0.
sphq_status gemm_workspace_bytes(sphq_handle h, int batch, size_t* bytes);
// Enqueues the two-pass product: W_hat decoded into `ws`, then the dense
// tensor-core product reading it (validated x, y, batch).
sphq_status launch_gemm_two_pass(sphq_handle h, const void* x, void* y, int batch, void* ws,
                                 size_t ws_bytes, cudaStream_t s);
// sphq_gemm_ws with a workspace: the split-K form of the fused kernel where it
// applies (mid-size batches, few output tiles), else the two-pass form.
sphq_status launch_gemm_ws(sphq_handle h, const void* x, void* y, int batch, void* ws,
                           size_t ws_bytes, cudaStream_t s);
// 16-D vectors (sphq_dim16.cu): the lane-ordered codebook image (synchronous),
// pack and decode launches, the GEMV plan of one batch size (csize 0:
// automatic) and its launch (batch 1..8).
sphq_status build_cbimage16(sphq_handle h);
sphq_status pack16(sphq_handle h, const uint16_t* sign, const uint16_t* idx, const uint8_t* rcode,
                   const uint16_t* scale, const uint16_t* offset, cudaStream_t s);
sphq_status decode16(sphq_handle h, void* w, cudaStream_t s);
sphq_status make_gemv16_plan(sphq_handle h, int batch, int csize, GemvPlan& out);
sphq_status launch_gemv16(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s);
// Enqueues the GEMV with caller-provided split-K scratch: `ws` holds at least
// h->ws_floats floats and `tickets` h->nrt zeroed counters.
sphq_status launch_gemv_scratch(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s,
                                float* ws, unsigned* tickets);

}  // namespace sphq
