// Gather-rate study for 16-D vectors (Tab. 7): at the W2 allocation a 16-D
// codebook holds 2^14 entries of 32 bytes (512 KiB), beyond one SM's shared
// memory, so a 16-D GEMV would gather each vector's entry from L2 or from the
// shared memory of a thread-block cluster.  These kernels measure the rate of
// random 32-byte entry reads each way, next to the local shared-memory gather
// the 8-D kernels use, on a table of that size.  No counterpart in the paper.
//
// A profiling tool of the benchmark (`bench.py --report`), built as its own
// library (libsphq_study.so); it is not part of the sphq C ABI.
#include <cuda_runtime.h>

#include <cstdint>

namespace sphq_study {

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(addr), "r"(rank));
  return d;
}

constexpr int kStudyThreads = 256;
constexpr uint32_t kStudyEntries = 1u << 14;   // 16-D W2 codebook: 2^14 x 32 B
constexpr uint32_t kStudyEntryBytes = 32;

__device__ __forceinline__ uint32_t study_hash(uint32_t x) {
  x ^= x >> 16;
  x *= 0x7feb352du;
  x ^= x >> 15;
  x *= 0x846ca68bu;
  x ^= x >> 16;
  return x;
}

// mode 0: entries read from global memory (L2-resident 512 KiB table).
__global__ void __launch_bounds__(kStudyThreads) study_l2_kernel(const uint4* __restrict__ table,
                                                                 int iters, uint32_t* out) {
  const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t acc = 0, s = tid;
  for (int i = 0; i < iters; ++i) {
    s = study_hash(s + (uint32_t)i);
    const uint32_t e = s & (kStudyEntries - 1);
    const uint4 a = __ldg(table + 2 * e), b = __ldg(table + 2 * e + 1);
    acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w;
  }
  if (acc == 0x12345678u) out[tid] = acc;  // keeps the loads live
}

// mode 1: the table split over a cluster of 4 CTAs (128 KiB each) and read
// through distributed shared memory; mode 2: each CTA reads only its own
// 128 KiB quarter (the local shared-memory reference of the 8-D kernels).
template <bool REMOTE>
__global__ void __launch_bounds__(kStudyThreads) study_dsmem_kernel(const uint4* __restrict__ table,
                                                                    int iters, uint32_t* out) {
  extern __shared__ __align__(16) uint8_t sm[];
  constexpr uint32_t kQuarter = kStudyEntries / 4 * kStudyEntryBytes;  // 128 KiB
  const uint32_t rank = cluster_rank();
  const uint4* src = table + (size_t)rank * (kQuarter / 16);
  for (uint32_t i = threadIdx.x; i < kQuarter / 16; i += blockDim.x)
    reinterpret_cast<uint4*>(sm)[i] = src[i];
  __syncthreads();
  // release: the table quarters are written before any CTA of the cluster reads
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
  cluster_wait();
  const uint32_t base = smem_u32(sm);
  const uint32_t tid = blockIdx.x * blockDim.x + threadIdx.x;
  uint32_t acc = 0, s = tid;
  for (int i = 0; i < iters; ++i) {
    s = study_hash(s + (uint32_t)i);
    const uint32_t e = s & (kStudyEntries - 1);
    const uint32_t owner = REMOTE ? e >> 12 : rank;
    const uint32_t off = (e & (kStudyEntries / 4 - 1)) * kStudyEntryBytes;
    const uint32_t addr = REMOTE ? mapa(base + off, owner) : base + off;
    uint4 a, b;
    if (REMOTE) {
      asm volatile("ld.shared::cluster.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w) : "r"(addr));
      asm volatile("ld.shared::cluster.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w) : "r"(addr + 16));
    } else {
      asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(a.x), "=r"(a.y), "=r"(a.z), "=r"(a.w) : "r"(addr));
      asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
                   : "=r"(b.x), "=r"(b.y), "=r"(b.z), "=r"(b.w) : "r"(addr + 16));
    }
    acc ^= a.x ^ a.y ^ a.z ^ a.w ^ b.x ^ b.y ^ b.z ^ b.w;
  }
  // no CTA leaves while others may still read its shared memory
  cluster_arrive_relaxed();
  cluster_wait();
  if (acc == 0x12345678u) out[tid] = acc;
}

}  // namespace sphq_study

using namespace sphq_study;

extern "C" {

// Runs study `mode` (0: L2, 1: cluster shared memory, 2: local shared memory)
// with `iters` reads per thread on every SM and stores the rate in entries
// read per second (events around one launch after a warm-up launch).
// Returns 0 on success, 1 for a bad argument, else the CUDA error code.
int sphq_study_gather16(int mode, int iters, double* entries_per_s) {
  if (!entries_per_s || iters < 1 || mode < 0 || mode > 2) return 1;
  int dev = 0, sms = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&sms, cudaDevAttrMultiProcessorCount, dev);
  if (e != cudaSuccess) return (int)e;
  uint4* table = nullptr;
  uint32_t* out = nullptr;
  const size_t tbytes = (size_t)kStudyEntries * kStudyEntryBytes;
  const int ctas = (sms / 4) * 4 * 2;  // two CTAs per SM, whole clusters of 4
  if ((e = cudaMalloc(&table, tbytes)) != cudaSuccess) return (int)e;
  if ((e = cudaMalloc(&out, (size_t)ctas * kStudyThreads * 4)) != cudaSuccess) {
    cudaFree(table);
    return (int)e;
  }
  cudaMemset(table, 0x5A, tbytes);
  const uint32_t smem = kStudyEntries / 4 * kStudyEntryBytes;
  auto launch = [&]() -> cudaError_t {
    if (mode == 0) {
      study_l2_kernel<<<ctas, kStudyThreads>>>(table, iters, out);
      return cudaGetLastError();
    }
    const void* k = mode == 1 ? (const void*)&study_dsmem_kernel<true>
                              : (const void*)&study_dsmem_kernel<false>;
    cudaError_t r = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, smem);
    if (r != cudaSuccess) return r;
    cudaLaunchConfig_t cfg = {};
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeClusterDimension;
    attr[0].val.clusterDim.x = 4;
    attr[0].val.clusterDim.y = 1;
    attr[0].val.clusterDim.z = 1;
    cfg.gridDim = dim3(ctas / 2);  // one 128 KiB CTA per SM
    cfg.blockDim = dim3(kStudyThreads);
    cfg.dynamicSmemBytes = smem;
    cfg.attrs = attr;
    cfg.numAttrs = 1;
    void* args[] = {&table, &iters, &out};
    return cudaLaunchKernelExC(&cfg, k, args);
  };
  cudaEvent_t e0, e1;
  cudaEventCreate(&e0);
  cudaEventCreate(&e1);
  e = launch();
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e == cudaSuccess) {
    cudaEventRecord(e0);
    e = launch();
    cudaEventRecord(e1);
    if (e == cudaSuccess) e = cudaEventSynchronize(e1);
  }
  float ms = 0.f;
  if (e == cudaSuccess) cudaEventElapsedTime(&ms, e0, e1);
  cudaEventDestroy(e0);
  cudaEventDestroy(e1);
  cudaFree(table);
  cudaFree(out);
  if (e != cudaSuccess) return (int)e;
  const double threads = (double)(mode == 0 ? ctas : ctas / 2) * kStudyThreads;
  *entries_per_s = threads * iters / (ms * 1e-3);
  return 0;
}

}  // extern "C"
