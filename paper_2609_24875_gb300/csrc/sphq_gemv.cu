// Fused spherical dequantize-GEMV for decode (SPHQuant §3.4, App. D), sm_103a.
//
// y[b][r] = sum_j w_hat[r][j] x[b][j], with w_hat rebuilt in registers from
// the packed codes (Eq. (7) radius, Eq. (4) reconstruction) and never stored.
//
// Work decomposition (stream-K over group tiles).  The (row block, group)
// units of the matrix are laid out in memory order and cut into equal
// contiguous spans, one span per warp of a persistent grid.  Lane l of a warp
// owns row 32*rb + l of the current row block and walks the span's groups,
// so every warp-wide code load is a contiguous 512-byte burst and the fp32
// accumulators never leave registers until the span crosses into the next
// row block.  A row block covered by one warp is written directly; otherwise
// each covering warp stores its fp32 partial into the handle's workspace and
// the last one to arrive (an atomic ticket per row block, no waiting) sums
// the partials in a fixed order and writes y, so results are deterministic.
//
// Codebook: staged once per CTA in shared memory.  W2 keeps 8 interleaved
// copies of its 1 KiB codebook (entry k of copy c at 16*(8k + c)); lane l
// reads copy l % 8, so the 8 lanes of each quarter-warp hit 8 different
// 16-byte bank groups whatever their indices are.  W3's 128 KiB codebook is
// a single copy (one CTA per SM).
//
// Arithmetic per 8-D vector: r_hat by one fp16 FMA (Eq. (7)), w_hat by four
// fp16x2 multiplies and a sign XOR (Eq. (4)), then eight fp16 x fp16 -> fp32
// fused multiply-adds per batch row (exact products, fp32 sums).
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <string>

#include "sphq_internal.h"
#include "sphq_layout.cuh"

namespace sphq {

struct GemvArgs {
  const uint8_t* tiles;
  const uint4* codebook;
  const uint16_t* x;
  uint16_t* y;
  float* ws;
  unsigned* tickets;
  int rows, cols, ng, nrb;
  int units_per_warp;
  int max_slots;
  long long total_units;
};

template <int BITS>
__device__ __forceinline__ uint4 lookup(const uint4* cb, uint32_t k, int copy) {
  if (BITS == 2) return cb[k * 8 + copy];
  return cb[k];
}

__device__ __forceinline__ uint4 ldg_x16(const uint16_t* p) {
  return __ldg(reinterpret_cast<const uint4*>(p));
}

template <int BITS, int BATCH>
__device__ __forceinline__ void process_group(const GroupData<BITS>& d, const uint4* cb, int copy,
                                              const uint16_t* xg, int cols, float (&acc)[BATCH]) {
#pragma unroll
  for (int j = 0; j < kGroupVecs; ++j) {
    const Fields f = unpack(d, j);
    const uint16_t r = radius16(f.q, d.params);
    const uint4 c = lookup<BITS>(cb, f.k, copy);
    const uint4 w = reconstruct(f.sign, r, c);
#pragma unroll
    for (int b = 0; b < BATCH; ++b) {
      const uint4 xv = ldg_x16(xg + (size_t)b * cols + j * kVec);
      float a = acc[b];
      a = fma_h2_f32(w.x, xv.x, a);
      a = fma_h2_f32(w.y, xv.y, a);
      a = fma_h2_f32(w.z, xv.z, a);
      a = fma_h2_f32(w.w, xv.w, a);
      acc[b] = a;
    }
  }
}

// Writes the warp's fp32 partial of row block rb; the last contributor
// reduces all partials in slot order and stores fp16 y.
template <int BATCH>
__device__ __forceinline__ void flush_row_block(const GemvArgs& a, int rb, long long gw, int lane,
                                                float (&acc)[BATCH]) {
  const long long L = a.units_per_warp;
  const long long first = ((long long)rb * a.ng) / L;
  const long long last = ((long long)(rb + 1) * a.ng - 1) / L;
  const int count = (int)(last - first + 1);
  const int row = rb * kRowsPerBlock + lane;
  if (count == 1) {
    if (row < a.rows) {
#pragma unroll
      for (int b = 0; b < BATCH; ++b) a.y[(size_t)b * a.rows + row] = f32_to_h_rn(acc[b]);
    }
    return;
  }
  const int slot = (int)(gw - first);
  float* base = a.ws + (size_t)rb * a.max_slots * BATCH * kRowsPerBlock;
#pragma unroll
  for (int b = 0; b < BATCH; ++b) base[((size_t)slot * BATCH + b) * kRowsPerBlock + lane] = acc[b];
  __threadfence();
  __syncwarp();
  unsigned ticket = 0;
  if (lane == 0) ticket = atomicAdd(&a.tickets[rb], 1u);
  ticket = __shfl_sync(0xFFFFFFFFu, ticket, 0);
  if (ticket != (unsigned)(count - 1)) return;
  __threadfence();
  float sum[BATCH];
#pragma unroll
  for (int b = 0; b < BATCH; ++b) sum[b] = 0.f;
  for (int s = 0; s < count; ++s) {
#pragma unroll
    for (int b = 0; b < BATCH; ++b)
      sum[b] += __ldcg(base + ((size_t)s * BATCH + b) * kRowsPerBlock + lane);
  }
  if (row < a.rows) {
#pragma unroll
    for (int b = 0; b < BATCH; ++b) a.y[(size_t)b * a.rows + row] = f32_to_h_rn(sum[b]);
  }
  if (lane == 0) a.tickets[rb] = 0u;  // ready for the next call
}

template <int BITS, int BATCH, int WARPS>
__global__ void __launch_bounds__(WARPS * 32) gemv_kernel(const GemvArgs a) {
  extern __shared__ uint4 smem_cb[];
  // stage the codebook (W2: 8 interleaved copies)
  if (BITS == 2) {
    for (int i = threadIdx.x; i < Layout<2>::K * 8; i += WARPS * 32)
      smem_cb[i] = __ldg(a.codebook + (i >> 3));
  } else {
    for (int i = threadIdx.x; i < Layout<3>::K; i += WARPS * 32) smem_cb[i] = __ldg(a.codebook + i);
  }
  __syncthreads();

  const int lane = threadIdx.x & 31;
  const int copy = lane & 7;
  const long long gw = (long long)blockIdx.x * WARPS + (threadIdx.x >> 5);
  long long u = gw * a.units_per_warp;
  const long long u_end = min(u + (long long)a.units_per_warp, a.total_units);
  if (u >= u_end) return;

  float acc[BATCH];
#pragma unroll
  for (int b = 0; b < BATCH; ++b) acc[b] = 0.f;

  const uint8_t* tiles = a.tiles;
  constexpr int TB = Layout<BITS>::kTileBytes;
  GroupData<BITS> cur = load_group<BITS>(tiles + (size_t)u * TB, lane);
  int rb = (int)(u / a.ng);
  int g = (int)(u % a.ng);
  for (; u < u_end; ++u) {
    GroupData<BITS> nxt = cur;
    if (u + 1 < u_end) nxt = load_group<BITS>(tiles + (size_t)(u + 1) * TB, lane);
    process_group<BITS, BATCH>(cur, smem_cb, copy, a.x + (size_t)g * kGroupCols, a.cols, acc);
    if (++g == a.ng || u + 1 == u_end) {
      flush_row_block<BATCH>(a, rb, gw, lane, acc);
#pragma unroll
      for (int b = 0; b < BATCH; ++b) acc[b] = 0.f;
      if (g == a.ng) {
        g = 0;
        ++rb;
      }
    }
    cur = nxt;
  }
}

template <int BITS> struct KernelShape;
template <> struct KernelShape<2> {
  static constexpr int kWarps = 8;
  static constexpr size_t kSmem = (size_t)Layout<2>::K * 8 * 16;
};
template <> struct KernelShape<3> {
  static constexpr int kWarps = 16;
  static constexpr size_t kSmem = (size_t)Layout<3>::K * 16;
};

template <int BITS, int BATCH>
static const void* kernel_ptr() {
  return reinterpret_cast<const void*>(&gemv_kernel<BITS, BATCH, KernelShape<BITS>::kWarps>);
}

static const void* select_kernel(int bits, int batch) {
#define SPHQ_K(B)                                                      \
  case B:                                                              \
    return bits == 2 ? kernel_ptr<2, B>() : kernel_ptr<3, B>();
  switch (batch) {
    SPHQ_K(1) SPHQ_K(2) SPHQ_K(3) SPHQ_K(4) SPHQ_K(5) SPHQ_K(6) SPHQ_K(7) SPHQ_K(8)
  }
#undef SPHQ_K
  return nullptr;
}

sphq_status make_gemv_plans(sphq_handle h) {
  const long long units = (long long)h->nrb * h->ng;
  size_t ws = 0;
  for (int batch = 1; batch <= SPHQ_MAX_BATCH; ++batch) {
    GemvPlan& p = h->plan[batch];
    const void* k = select_kernel(h->bits, batch);
    p.warps_per_cta = h->bits == 2 ? KernelShape<2>::kWarps : KernelShape<3>::kWarps;
    p.smem = h->bits == 2 ? KernelShape<2>::kSmem : KernelShape<3>::kSmem;
    cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)p.smem);
    if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute");
    int occ = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, p.warps_per_cta * 32, p.smem);
    if (e != cudaSuccess) return cuda_error(e, "occupancy query");
    if (occ < 1) return set_error(SPHQ_ERR_CUDA, "gemv kernel cannot be resident");
    const long long max_warps = (long long)h->sm_count * occ * p.warps_per_cta;
    // at least two groups per warp so each warp can prefetch one tile ahead
    long long L = std::max<long long>(2, (units + max_warps - 1) / max_warps);
    L = std::min<long long>(L, units);
    const long long warps = (units + L - 1) / L;
    p.units_per_warp = (int)L;
    p.grid = (int)((warps + p.warps_per_cta - 1) / p.warps_per_cta);
    p.max_slots = (int)((h->ng + L - 1) / L + 1);
    ws = std::max(ws, (size_t)h->nrb * p.max_slots * batch * kRowsPerBlock);
  }
  h->ws_floats = ws;
  return SPHQ_OK;
}

sphq_status launch_gemv(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s) {
  const GemvPlan& p = h->plan[batch];
  GemvArgs a;
  a.tiles = (const uint8_t*)h->tiles;
  a.codebook = (const uint4*)h->codebook;
  a.x = (const uint16_t*)x;
  a.y = (uint16_t*)y;
  a.ws = h->ws;
  a.tickets = h->tickets;
  a.rows = h->rows;
  a.cols = h->cols;
  a.ng = h->ng;
  a.nrb = h->nrb;
  a.units_per_warp = p.units_per_warp;
  a.max_slots = p.max_slots;
  a.total_units = (long long)h->nrb * h->ng;
  const void* k = select_kernel(h->bits, batch);
  void* args[] = {&a};
  cudaError_t e = cudaLaunchKernel(k, dim3(p.grid), dim3(p.warps_per_cta * 32), args, p.smem, s);
  if (e != cudaSuccess) return cuda_error(e, "gemv launch");
  return SPHQ_OK;
}

}  // namespace sphq
