// Codebook construction on the GPU (the quantise side of the path, §3.1 and
// §3.3): radius-weighted sampling of directions, spherical k-means, and the
// angle-parameterised codebook.  Offline steps, run once per layer before
// encoding; the decode GEMV never calls them.
//
// Numerics.  Directions and centres are float64 (the weights are float32 and
// every value derived from them is exact or correctly rounded in float64).
//  * r_i^2 = w_0^2 + ... + w_7^2 added in coordinate order; r_i = sqrt; the
//    direction d_i = |w_i| / r_i.
//  * Sampling: prefix sums P of r^2 over the vectors (block-wise, then the
//    block totals), and the pick for a uniform u in [0, 1) is the first i with
//    P_i > u * P_last -- the inverse transform of the r^2 distribution;
//    zero-radius vectors are never drawn.
//  * k-means assignment (Eq. (5)): every score d_i . c_k is first bounded in
//    single precision (a pass over all centres finds the largest); the
//    centres within 1e-5 of it -- the single-precision error of an 8-term dot
//    of unit vectors is below 1e-6 -- are re-scored exactly as
//    ((d_0 c_0 + d_1 c_1) + d_2 c_2) + ... in float64 with each product and
//    sum rounded once, and the largest wins (lowest index on ties).  The
//    decision is therefore the float64 argmax of those fixed-order dots.
//  * k-means update: each centre becomes the normalised sum of its members
//    (float64, summed in a fixed order: lane-strided over the samples, then a
//    fixed shuffle tree); an empty cluster keeps its centre.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "sphq_internal.h"

namespace sphq {

constexpr int kCbThreads = 256;
constexpr int kScanPer = 8;                           // elements per thread in a scan block
constexpr int kScanBlock = kCbThreads * kScanPer;     // 2048 elements per block
constexpr int kCentreChunk = 1024;                    // centres staged per pass (32 KiB fp32)
constexpr double kMargin = 1e-5;

__device__ __forceinline__ double r2_of(const float* w) {
  double s = __dmul_rn((double)w[0], (double)w[0]);
#pragma unroll
  for (int j = 1; j < 8; ++j) s = __dadd_rn(s, __dmul_rn((double)w[j], (double)w[j]));
  return s;
}

// Block-wise inclusive scan of r^2 (each thread 8 consecutive vectors in
// order, thread totals combined in thread order); block totals to `tot`.
__global__ void __launch_bounds__(kCbThreads) r2_scan_kernel(const float* __restrict__ w,
                                                             long long n, double* __restrict__ P,
                                                             double* __restrict__ tot) {
  __shared__ double part[kCbThreads];
  const long long base = (long long)blockIdx.x * kScanBlock + (long long)threadIdx.x * kScanPer;
  double v[kScanPer];
  double run = 0.0;
#pragma unroll
  for (int k = 0; k < kScanPer; ++k) {
    const long long i = base + k;
    const double r2 = i < n ? r2_of(w + 8 * i) : 0.0;
    run = k ? __dadd_rn(run, r2) : r2;
    v[k] = run;
  }
  part[threadIdx.x] = run;
  __syncthreads();
  if (threadIdx.x == 0) {
    double acc = 0.0;
    for (int t = 0; t < kCbThreads; ++t) {
      const double p = part[t];
      part[t] = acc;  // exclusive offset of thread t
      acc = t ? __dadd_rn(acc, p) : p;
    }
    tot[blockIdx.x] = acc;
  }
  __syncthreads();
  const double off = part[threadIdx.x];
#pragma unroll
  for (int k = 0; k < kScanPer; ++k) {
    const long long i = base + k;
    if (i < n) P[i] = threadIdx.x ? __dadd_rn(off, v[k]) : v[k];
  }
}

// Exclusive offsets of the block totals, in block order (one thread).
__global__ void block_offsets_kernel(double* tot, int nb) {
  if (threadIdx.x != 0 || blockIdx.x != 0) return;
  double acc = 0.0;
  for (int b = 0; b < nb; ++b) {
    const double t = tot[b];
    tot[b] = acc;
    acc = b ? __dadd_rn(acc, t) : t;
  }
  tot[nb] = acc;  // total
}

__global__ void __launch_bounds__(kCbThreads) add_offsets_kernel(double* __restrict__ P, long long n,
                                                                 const double* __restrict__ off) {
  const long long i = (long long)blockIdx.x * kCbThreads + threadIdx.x;
  if (i < n) {
    const long long b = i / kScanBlock;
    if (b > 0) P[i] = __dadd_rn(off[b], P[i]);
  }
}

// One sample per thread: the first i with P_i > u * total, then d = |w_i| / r_i.
__global__ void __launch_bounds__(kCbThreads) sample_kernel(
    const float* __restrict__ w, long long n, const double* __restrict__ P,
    const double* __restrict__ total_p, const double* __restrict__ u, int S,
    double* __restrict__ dirs, int* __restrict__ idx_out) {
  const int s = blockIdx.x * kCbThreads + threadIdx.x;
  if (s >= S) return;
  const double total = *total_p;
  double target = __dmul_rn(u[s], total);
  // For u < 1 the rounded product stays below the total (total * 2^-53 is
  // more than half a unit in the last place below a total that is not a
  // power of two, and the product is exact when it is one); u = 1 reaches
  // the total, which no P_i exceeds: the pick is then the last vector of
  // nonzero radius (the first i with P_i = total)
  const bool top = !(target < total);
  long long lo = 0, hi = n - 1;
  while (lo < hi) {
    const long long mid = (lo + hi) >> 1;
    if (top ? P[mid] >= total : P[mid] > target) hi = mid;
    else lo = mid + 1;
  }
  const float* v = w + 8 * lo;
  const double r = __dsqrt_rn(r2_of(v));
#pragma unroll
  for (int j = 0; j < 8; ++j) dirs[8 * (size_t)s + j] = __ddiv_rn(fabs((double)v[j]), r);
  if (idx_out) idx_out[s] = (int)lo;
}

// Exact score in coordinate order: products and sums rounded once each.
__device__ __forceinline__ double dot8_exact(const double* d, const double* c) {
  double s = __dmul_rn(d[0], c[0]);
#pragma unroll
  for (int j = 1; j < 8; ++j) s = __dadd_rn(s, __dmul_rn(d[j], c[j]));
  return s;
}

// Assignment, one sample per thread; centres staged in chunks as float32.
__global__ void __launch_bounds__(kCbThreads) kmeans_assign_kernel(
    const double* __restrict__ D, int S, const double* __restrict__ C, int K,
    int* __restrict__ z, double* __restrict__ best) {
  __shared__ float4 cs[kCentreChunk * 2];  // centre k: cs[2k], cs[2k+1]
  const int s = blockIdx.x * kCbThreads + threadIdx.x;
  const bool live = s < S;
  double d[8];
  float df[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    d[j] = live ? D[8 * (size_t)s + j] : 0.0;
    df[j] = (float)d[j];
  }
  auto stage = [&](int k0, int cnt) {
    __syncthreads();
    for (int e = threadIdx.x; e < 8 * cnt; e += kCbThreads) {
      const int k = e >> 3, j = e & 7;
      reinterpret_cast<float*>(cs)[8 * k + j] = (float)C[8 * (size_t)(k0 + k) + j];
    }
    __syncthreads();
  };
  auto score32 = [&](int k) {
    const float4 a = cs[2 * k], b = cs[2 * k + 1];
    float v = df[0] * a.x;
    v = fmaf(df[1], a.y, v);
    v = fmaf(df[2], a.z, v);
    v = fmaf(df[3], a.w, v);
    v = fmaf(df[4], b.x, v);
    v = fmaf(df[5], b.y, v);
    v = fmaf(df[6], b.z, v);
    v = fmaf(df[7], b.w, v);
    return v;
  };
  // pass 1: the largest single-precision score
  float mx = -3.0e38f;
  for (int k0 = 0; k0 < K; k0 += kCentreChunk) {
    const int cnt = min(kCentreChunk, K - k0);
    stage(k0, cnt);
    for (int k = 0; k < cnt; ++k) mx = fmaxf(mx, score32(k));
  }
  // pass 2: exact scores of the candidates, in increasing k (the margin
  // assumes directions and centres of norm at most about 1)
  const float thr = mx - (float)kMargin * (1.0f + fabsf(mx));
  int bk = -1;
  double bs = 0.0;
  for (int k0 = 0; k0 < K; k0 += kCentreChunk) {
    const int cnt = min(kCentreChunk, K - k0);
    stage(k0, cnt);
    for (int k = 0; k < cnt; ++k) {
      if (score32(k) >= thr) {
        const double e = dot8_exact(d, C + 8 * (size_t)(k0 + k));
        if (bk < 0 || e > bs) {
          bk = k0 + k;
          bs = e;
        }
      }
    }
  }
  if (live) {
    z[s] = bk;
    best[s] = bs;
  }
}

// Update, one warp per centre: lane l sums the members i = l (mod 32) in
// increasing i; a fixed shuffle tree adds the lanes.
__global__ void __launch_bounds__(kCbThreads) kmeans_update_kernel(
    const double* __restrict__ D, int S, const int* __restrict__ z,
    const double* __restrict__ Cin, int K, double* __restrict__ Cout) {
  const int warp = (blockIdx.x * kCbThreads + threadIdx.x) >> 5;
  const int lane = threadIdx.x & 31;
  if (warp >= K) return;
  double acc[8];
#pragma unroll
  for (int j = 0; j < 8; ++j) acc[j] = 0.0;
  for (int i = lane; i < S; i += 32) {
    if (z[i] == warp) {
#pragma unroll
      for (int j = 0; j < 8; ++j) acc[j] = __dadd_rn(acc[j], D[8 * (size_t)i + j]);
    }
  }
#pragma unroll
  for (int off = 16; off > 0; off >>= 1)
#pragma unroll
    for (int j = 0; j < 8; ++j) acc[j] = __dadd_rn(acc[j], __shfl_down_sync(0xFFFFFFFFu, acc[j], off));
  if (lane == 0) {
    double n2 = __dmul_rn(acc[0], acc[0]);
#pragma unroll
    for (int j = 1; j < 8; ++j) n2 = __dadd_rn(n2, __dmul_rn(acc[j], acc[j]));
    const double nr = __dsqrt_rn(n2);
#pragma unroll
    for (int j = 0; j < 8; ++j)
      Cout[8 * (size_t)warp + j] = nr > 0.0 ? __ddiv_rn(acc[j], nr) : Cin[8 * (size_t)warp + j];
  }
}

// Mean of the assigned scores: one block, thread-strided sums combined in
// thread order.
__global__ void __launch_bounds__(kCbThreads) mean_kernel(const double* __restrict__ v, int n,
                                                          double* __restrict__ out) {
  __shared__ double part[kCbThreads];
  double a = 0.0;
  for (int i = threadIdx.x; i < n; i += kCbThreads) a = __dadd_rn(a, v[i]);
  part[threadIdx.x] = a;
  __syncthreads();
  if (threadIdx.x == 0) {
    double s = 0.0;
    for (int t = 0; t < kCbThreads; ++t) s = __dadd_rn(s, part[t]);
    *out = __ddiv_rn(s, (double)n);
  }
}

// Eq. (sph-angle-logits) then Eq. (sph-angle-codebook), one entry per thread.
__global__ void __launch_bounds__(kCbThreads) angle_codebook_kernel(
    const float* __restrict__ phi, int K, double eps, double* __restrict__ c64,
    __half* __restrict__ c16) {
  const int k = blockIdx.x * kCbThreads + threadIdx.x;
  if (k >= K) return;
  const double span = 1.5707963267948966 - 2.0 * eps;  // pi/2 - 2 eps
  double run = 1.0;  // product of the sines so far
  double c[8];
#pragma unroll
  for (int i = 0; i < 7; ++i) {
    const double p = (double)phi[7 * (size_t)k + i];
    const double th = eps + span / (1.0 + exp(-p));
    c[i] = run * cos(th);
    run = run * sin(th);
  }
  c[7] = run;
#pragma unroll
  for (int j = 0; j < 8; ++j) {
    if (c64) c64[8 * (size_t)k + j] = c[j];
    if (c16) c16[8 * (size_t)k + j] = __double2half(c[j]);
  }
}

static int blocks_for(long long n, int per) { return (int)((n + per - 1) / per); }

}  // namespace sphq

using namespace sphq;

extern "C" {

sphq_status sphq_sample_directions(const float* w, long long nvec, const double* u, int samples,
                                   double* dirs, int* idx, sphq_stream stream) {
  clear_error();
  if (!w || !u || !dirs || nvec < 1 || samples < 1 || nvec > (1ll << 40))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_sample_directions: bad argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const int nb = blocks_for(nvec, kScanBlock);
  double* P = nullptr;
  cudaError_t e = cudaMallocAsync(reinterpret_cast<void**>(&P),
                                  sizeof(double) * ((size_t)nvec + (size_t)nb + 1), s);
  if (e != cudaSuccess) return cuda_error(e, "sphq_sample_directions: cudaMallocAsync");
  double* tot = P + nvec;
  r2_scan_kernel<<<nb, kCbThreads, 0, s>>>(w, nvec, P, tot);
  block_offsets_kernel<<<1, 32, 0, s>>>(tot, nb);
  add_offsets_kernel<<<blocks_for(nvec, kCbThreads), kCbThreads, 0, s>>>(P, nvec, tot);
  sample_kernel<<<blocks_for(samples, kCbThreads), kCbThreads, 0, s>>>(w, nvec, P, tot + nb, u,
                                                                       samples, dirs, idx);
  e = cudaGetLastError();
  cudaFreeAsync(P, s);
  if (e != cudaSuccess) return cuda_error(e, "sphq_sample_directions: launch");
  return SPHQ_OK;
}

static sphq_status kmeans_step_impl(const double* dirs, int S, const double* C, int K,
                                    double* Cout, int* z, double* best, double* objective,
                                    cudaStream_t s) {
  kmeans_assign_kernel<<<blocks_for(S, kCbThreads), kCbThreads, 0, s>>>(dirs, S, C, K, z, best);
  if (objective) mean_kernel<<<1, kCbThreads, 0, s>>>(best, S, objective);
  kmeans_update_kernel<<<blocks_for((long long)K * 32, kCbThreads), kCbThreads, 0, s>>>(
      dirs, S, z, C, K, Cout);
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "sphq_kmeans: launch");
  return SPHQ_OK;
}

sphq_status sphq_kmeans_step(const double* dirs, int samples, const double* centres, int K,
                             double* centres_out, int* assign, double* objective,
                             sphq_stream stream) {
  clear_error();
  if (!dirs || !centres || !centres_out || samples < 1 || K < 1 || K > (1 << 20))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_kmeans_step: bad argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  void* tmp = nullptr;
  const size_t bytes = sizeof(double) * (size_t)samples + (assign ? 0 : sizeof(int) * (size_t)samples);
  cudaError_t e = cudaMallocAsync(&tmp, bytes, s);
  if (e != cudaSuccess) return cuda_error(e, "sphq_kmeans_step: cudaMallocAsync");
  double* best = static_cast<double*>(tmp);
  int* z = assign ? assign : reinterpret_cast<int*>(best + samples);
  const sphq_status st = kmeans_step_impl(dirs, samples, centres, K, centres_out, z, best,
                                          objective, s);
  cudaFreeAsync(tmp, s);
  return st;
}

sphq_status sphq_kmeans(const double* dirs, int samples, double* centres, int K, int iters,
                        double* objective_history, sphq_stream stream) {
  clear_error();
  if (!dirs || !centres || samples < 1 || K < 1 || K > (1 << 20) || iters < 0)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_kmeans: bad argument");
  if (iters == 0) return SPHQ_OK;
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  void* tmp = nullptr;
  cudaError_t e = cudaMallocAsync(&tmp, (sizeof(double) + sizeof(int)) * (size_t)samples, s);
  if (e != cudaSuccess) return cuda_error(e, "sphq_kmeans: cudaMallocAsync");
  double* best = static_cast<double*>(tmp);
  int* z = reinterpret_cast<int*>(best + samples);
  sphq_status st = SPHQ_OK;
  // in place: the assignment reads every centre before the update, and the
  // update of centre k reads and writes centre k only
  for (int it = 0; it < iters && st == SPHQ_OK; ++it)
    st = kmeans_step_impl(dirs, samples, centres, K, centres, z, best,
                          objective_history ? objective_history + it : nullptr, s);
  cudaFreeAsync(tmp, s);
  return st;
}

sphq_status sphq_angle_codebook(const float* phi, int K, double eps, double* codebook_f64,
                                void* codebook_f16, sphq_stream stream) {
  clear_error();
  if (!phi || K < 1 || !(eps >= 0.0 && eps < 0.7853981633974483) ||
      (!codebook_f64 && !codebook_f16))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_angle_codebook: bad argument");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  angle_codebook_kernel<<<blocks_for(K, kCbThreads), kCbThreads, 0, s>>>(
      phi, K, eps, codebook_f64, static_cast<__half*>(codebook_f16));
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "sphq_angle_codebook: launch");
  return SPHQ_OK;
}

}  // extern "C"
