// 16-D vectors at the W2 allocation (Tab. 7): pack, decode and the fused
// dequantize-GEMV.
//
// A 16-D vector carries 16 sign bits, a 14-bit index into K = 16384 unit
// directions ((dim - 1) B - dim = 15 * 2 - 16, §3.1) and a 4-bit radius code:
// 34 bits per 16 weights (2.125 bits per weight), radius groups of 128
// scalars (8 vectors) as for 8-D.  The fp16 codebook is 512 KiB, beyond an
// SM's shared memory (227 KiB), so the GEMV gathers each vector's 32-byte
// entry from global memory (L2-resident, partly caught by L1).  Those random
// reads, not HBM, bound it: random 32-byte reads from an L2-resident 512 KiB
// table run at ~199 G entries/s on this GB300 (`sphq_study_gather16`), about
// 14% of the rate at which the HBM could stream the codes.  This is the
// paper's reason for preferring 8-D vectors (the 16-D table does not fit in
// shared memory).
//
// Unit (16 rows x 128 columns, indexed like the 8-D units: group-major):
//   bytes   0..511  lane l = 4 gid + q holds four words: the vectors of
//                   (row gid, k-step 2q), (row gid, 2q+1), (row gid+8, 2q),
//                   (row gid+8, 2q+1); k-step t covers columns 16t..16t+15
//                   of the group (one vector per row: the K = 16 of an
//                   m16n8k16 product).
//   bytes 512..543  8 words H(row gid) | H(row gid+8) << 16; H(row) holds
//                   radius-code bits 2-3 of k-step t at bits 2t, 2t+1.
//   bytes 544..607  8 pairs {P(row gid), P(row gid+8)}, P = Delta | r_min << 16.
// Word of a vector: the sign of element e at bit q (e = 2q), 16 + q (2q+1),
// 4 + q (2q+8) or 20 + q (2q+9), q = 0..3 -- the elements that lane q of
// a quad holds in the mma.sync A fragment, so that its two sign masks are
// the word shifted left by 15 - q and by 11 - q; direction index bits 0-7 at
// bits 8-15 and bits 8-13 at bits 24-29; radius-code bits 0-1 at bits 30-31.
// Codebook image: entry k at byte 32 k with its elements in the order
// (0,1,8,9, 2,3,10,11, 4,5,12,13, 6,7,14,15): lane q reads bytes 8q..8q+7.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>

#include "sphq_gemv_kernel.cuh"

namespace sphq {

constexpr int kUB16 = Layout<kFmt16D>::kUnitBytes;
constexpr int kWarps16 = 8;

// bit position of the sign of element e (0..15) in a 16-D word
__host__ __device__ constexpr int sign_pos16(int e) {
  return e < 8 ? ((e & 1) ? 16 : 0) + (e >> 1) : ((e & 1) ? 20 : 4) + ((e - 8) >> 1);
}
// element stored at slot j (0..15) of an entry of the codebook image
__host__ __device__ constexpr int image_elem16(int j) {
  return 2 * (j >> 2) + ((j & 2) ? 8 : 0) + (j & 1);
}

__global__ void cbimage16_kernel(const uint16_t* __restrict__ cb, uint16_t* __restrict__ img,
                                 int K) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= (long long)K * 16) return;
  const long long k = i >> 4;
  img[i] = cb[k * 16 + image_elem16((int)(i & 15))];
}

// One warp per unit; lane (gid, q) packs its four vectors (App. A step 10).
// Codes of rows past the matrix are zero; an index >= K or a radius code >= 16
// sets flag[0].
__global__ void pack16_kernel(const uint16_t* __restrict__ sign, const uint16_t* __restrict__ idx,
                              const uint8_t* __restrict__ rcode, const uint16_t* __restrict__ scale,
                              const uint16_t* __restrict__ offset, uint8_t* __restrict__ units,
                              int rows, int ng, int nrt, int* flag) {
  const long long unit = ((long long)blockIdx.x * blockDim.x + threadIdx.x) >> 5;
  if (unit >= (long long)nrt * ng) return;  // whole warps: blockDim is a multiple of 32
  const int lane = threadIdx.x & 31, gid = lane >> 2, q = lane & 3;
  const int rt = (int)(unit % nrt), g = (int)(unit / nrt);
  const size_t nv = (size_t)ng * 8;  // vectors per row
  uint32_t wv[4];
  uint32_t H[2] = {0u, 0u};
  bool bad = false;
#pragma unroll
  for (int half = 0; half < 2; ++half) {
    const int row = rt * kRowsPerTile + gid + 8 * half;
#pragma unroll
    for (int j = 0; j < 2; ++j) {
      const int t = 2 * q + j;
      uint32_t word = 0u;
      if (row < rows) {
        const size_t v = (size_t)row * nv + (size_t)g * 8 + t;
        const uint32_t s = sign[v], k = idx[v], rq = rcode[v];
        bad |= k >= (uint32_t)Layout<kFmt16D>::K || rq >= 16u;
#pragma unroll
        for (int e = 0; e < 16; ++e) word |= ((s >> e) & 1u) << sign_pos16(e);
        word |= (k & 0xFFu) << 8 | ((k >> 8) & 0x3Fu) << 24 | (rq & 3u) << 30;
        H[half] |= ((rq >> 2) & 3u) << (2 * t);
      }
      wv[2 * half + j] = word;
    }
  }
  if (bad) atomicOr(flag, 1);
#pragma unroll
  for (int m = 1; m <= 2; m <<= 1) {
    H[0] |= __shfl_xor_sync(0xFFFFFFFFu, H[0], m);
    H[1] |= __shfl_xor_sync(0xFFFFFFFFu, H[1], m);
  }
  uint8_t* base = units + (size_t)unit * kUB16;
  *reinterpret_cast<uint4*>(base + lane * 16) = make_uint4(wv[0], wv[1], wv[2], wv[3]);
  if (q == 0) {
    *reinterpret_cast<uint32_t*>(base + Layout<kFmt16D>::kHiOff + gid * 4) =
        (H[0] & 0xFFFFu) | (H[1] << 16);
    const int ra = rt * kRowsPerTile + gid, rb = ra + 8;
    uint32_t pa = 0u, pb = 0u;
    if (ra < rows) pa = (uint32_t)scale[(size_t)ra * ng + g] | ((uint32_t)offset[(size_t)ra * ng + g] << 16);
    if (rb < rows) pb = (uint32_t)scale[(size_t)rb * ng + g] | ((uint32_t)offset[(size_t)rb * ng + g] << 16);
    *reinterpret_cast<uint2*>(base + Layout<kFmt16D>::kParamOff + gid * 8) = make_uint2(pa, pb);
  }
}

// W_hat from the packed units and the plain (K x 16) codebook: one thread per
// vector, Eq. (7) then Eq. (4), 32 bytes written.
__global__ void decode16_kernel(const uint8_t* __restrict__ units, const uint16_t* __restrict__ cb,
                                uint16_t* __restrict__ w, int rows, int cols, int nrt) {
  const long long i = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int nv = cols / 16;
  if (i >= (long long)rows * nv) return;
  const int row = (int)(i / nv), v = (int)(i % nv);
  const int g = v >> 3, t = v & 7;
  const int rt = row / kRowsPerTile, r16 = row % kRowsPerTile, gid = r16 & 7, half = r16 >> 3;
  const uint8_t* u = units + ((size_t)g * nrt + rt) * kUB16;
  const int lane = 4 * gid + (t >> 1);
  const uint32_t word = *reinterpret_cast<const uint32_t*>(u + lane * 16 + 4 * ((t & 1) + 2 * half));
  const uint32_t H =
      (*reinterpret_cast<const uint32_t*>(u + Layout<kFmt16D>::kHiOff + 4 * gid) >> (16 * half)) & 0xFFFFu;
  const uint32_t P = *reinterpret_cast<const uint32_t*>(u + Layout<kFmt16D>::kParamOff + 8 * gid + 4 * half);
  const uint32_t k = ((word >> 8) & 0xFFu) | ((word >> 16) & 0x3F00u);
  const uint32_t rq = (word >> 30) | (((H >> (2 * t)) & 3u) << 2);
  const uint32_t r2 = bcast_lo(radius_pair<4>(rq, P & 0xFFFFu, P >> 16));
  const uint32_t* c = reinterpret_cast<const uint32_t*>(cb + (size_t)k * 16);
  uint32_t out[8];
#pragma unroll
  for (int p = 0; p < 8; ++p) {
    const uint32_t m = ((word >> sign_pos16(2 * p)) & 1u) << 15 | ((word >> sign_pos16(2 * p + 1)) & 1u) << 31;
    out[p] = hmul2_rn(r2, c[p] ^ m);
  }
  uint4* dst = reinterpret_cast<uint4*>(w + (size_t)row * cols + (size_t)v * 16);
  dst[0] = make_uint4(out[0], out[1], out[2], out[3]);
  dst[1] = make_uint4(out[4], out[5], out[6], out[7]);
}

struct Gemv16Args {
  const uint8_t* units;
  const uint8_t* cbimage;  // K x 32 B, lane-ordered entries
  const uint16_t* x;       // batch x cols fp16
  const uint16_t* zeros;   // 256 zero bytes (activations of lanes past the batch)
  uint16_t* y;             // batch x rows fp16
  int rows, cols, ng, nrt, batch;
  int csize;               // CTAs per cluster, each a share of the groups of one row tile
};

__device__ __forceinline__ void st_cluster_f32(uint32_t raddr, float v) {
  asm volatile("st.shared::cluster.f32 [%0], %1;" ::"r"(raddr), "f"(v) : "memory");
}
__device__ __forceinline__ void cluster_arrive_release() {
  asm volatile("barrier.cluster.arrive.release.aligned;" ::: "memory");
}

// One cluster per row tile; its CTAs split the radius groups, the warps of a
// CTA take the CTA's groups round robin (one unit each).  Per unit and
// k-step a lane rebuilds its four elements of rows gid and gid+8 exactly
// (w_hat = RN16(r_hat * (s (.) c)), Eq. (7) and Eq. (4)) and one m16n8k16
// accumulates them against activation rows 0..7 in fp32 (batch = the N
// dimension; rows past the batch read zeros).  Partial sums: warps in order
// through shared memory, then the cluster's CTAs in rank order through
// distributed shared memory into rank 0, which rounds to fp16 and writes y.
// The two cluster barriers are hardware barriers that every thread of every
// CTA of the cluster reaches (no early exit before them).  MINB: CTAs per SM
// the build's registers allow (2: 115 registers, 4: 64, neither spills).
template <int MINB>
__global__ void __launch_bounds__(kWarps16 * 32, MINB) gemv16_kernel(const Gemv16Args a) {
  __shared__ float red[kWarps16][kRowsPerTile][8];
  __shared__ float recv[8][kRowsPerTile][8];
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, q = lane & 3;
  const int cs = a.csize;
  const int rank = cs > 1 ? (int)cluster_rank() : 0;
  const int rt = (int)blockIdx.x / cs;
  if (cs > 1) cluster_arrive_relaxed();  // waited on before the first remote store

  const int gq = a.ng / cs, gr = a.ng % cs;
  const int g0 = rank * gq + min(rank, gr);
  const int gn = gq + (rank < gr ? 1 : 0);
  const size_t gstride = (size_t)a.nrt * kUB16;
  const uint8_t* ub = a.units + ((size_t)g0 * a.nrt + rt) * kUB16;
  const uint8_t* cbq = a.cbimage + q * 8;
  const bool provider = gid < a.batch;
  const uint8_t* xrow = provider ? reinterpret_cast<const uint8_t*>(a.x + (size_t)gid * a.cols)
                                 : reinterpret_cast<const uint8_t*>(a.zeros);
  const int xgstep = provider ? kGroupCols * 2 : 0;
  const int sl = 15 - q, sh = 11 - q;

  float d[4] = {0.f, 0.f, 0.f, 0.f};
  uint4 w = {};
  uint32_t hi = 0u;
  uint2 par = {};
  int i = warp;
  if (i < gn) {  // codes are immutable: loaded before the dependency wait
    const uint8_t* u = ub + (size_t)i * gstride;
    w = ldg_stream16(u + lane * 16);
    hi = ldg_stream4(u + Layout<kFmt16D>::kHiOff + gid * 4);
    par = ldg_stream8(u + Layout<kFmt16D>::kParamOff + gid * 8);
  }
  pdl_wait();  // the previous kernel's outputs (our activations) are complete
  for (; i < gn; i += kWarps16) {
    const uint4 cw = w;
    const uint32_t chi = hi;
    const uint2 cpar = par;
    if (i + kWarps16 < gn) {
      const uint8_t* u = ub + (size_t)(i + kWarps16) * gstride;
      w = ldg_stream16(u + lane * 16);
      hi = ldg_stream4(u + Layout<kFmt16D>::kHiOff + gid * 4);
      par = ldg_stream8(u + Layout<kFmt16D>::kParamOff + gid * 8);
    }
    const uint32_t d2 = prmt<0x5410u>(cpar.x, cpar.y);  // (Delta, Delta) of rows gid, gid+8
    const uint32_t m2 = prmt<0x7632u>(cpar.x, cpar.y);  // (r_min, r_min)
    const uint8_t* xg = xrow + (size_t)(g0 + i) * xgstep + 4 * q;
#pragma unroll
    for (int t = 0; t < 8; ++t) {
      const int src = 4 * gid + (t >> 1);
      const uint32_t wa = __shfl_sync(0xFFFFFFFFu, (t & 1) ? cw.y : cw.x, src);  // row gid
      const uint32_t wb = __shfl_sync(0xFFFFFFFFu, (t & 1) ? cw.w : cw.z, src);  // row gid+8
      const uint32_t ka = ((wa >> 8) & 0xFFu) | ((wa >> 16) & 0x3F00u);
      const uint32_t kb = ((wb >> 8) & 0xFFu) | ((wb >> 16) & 0x3F00u);
      const uint2 ca = __ldg(reinterpret_cast<const uint2*>(cbq + ((size_t)ka << 5)));
      const uint2 cb = __ldg(reinterpret_cast<const uint2*>(cbq + ((size_t)kb << 5)));
      const uint32_t qp = ((wa >> 30) | ((wb >> 30) << 16)) | (((chi >> (2 * t)) & 0x00030003u) << 2);
      const uint32_t r = radius_pair<4>(qp, d2, m2);
      const uint32_t ra = bcast_lo(r), rb = bcast_hi(r);
      const uint32_t a0 = hmul2_rn(ra, ca.x ^ ((wa << sl) & kSignMask));
      const uint32_t a2 = hmul2_rn(ra, ca.y ^ ((wa << sh) & kSignMask));
      const uint32_t a1 = hmul2_rn(rb, cb.x ^ ((wb << sl) & kSignMask));
      const uint32_t a3 = hmul2_rn(rb, cb.y ^ ((wb << sh) & kSignMask));
      const uint32_t b0 = __ldg(reinterpret_cast<const unsigned*>(xg + 32 * t));
      const uint32_t b1 = __ldg(reinterpret_cast<const unsigned*>(xg + 32 * t + 16));
      mma16816(d, a0, a1, a2, a3, b0, b1);
    }
  }

  red[warp][gid][2 * q] = d[0];
  red[warp][gid][2 * q + 1] = d[1];
  red[warp][gid + 8][2 * q] = d[2];
  red[warp][gid + 8][2 * q + 1] = d[3];
  __syncthreads();
  const int row = (threadIdx.x >> 3) & 15, n = threadIdx.x & 7;
  float s = 0.f;
  if (threadIdx.x < 128) {
#pragma unroll
    for (int v = 0; v < kWarps16; ++v) s += red[v][row][n];
  }
  if (cs > 1) {
    cluster_wait();  // every CTA of the cluster is running
    if (threadIdx.x < 128) st_cluster_f32(mapa(smem_u32(&recv[rank][row][n]), 0u), s);
    cluster_arrive_release();
    cluster_wait();
    if (rank != 0) return;
    if (threadIdx.x < 128) {
      s = 0.f;
      for (int k = 0; k < cs; ++k) s += recv[k][row][n];
    }
  }
  if (threadIdx.x < 128) {
    const int r = rt * kRowsPerTile + row;
    if (n < a.batch && r < a.rows) a.y[(size_t)n * a.rows + r] = f32_to_h_rn(s);
  }
}

// ---------------------------------------------------------------------------
// Host side
// ---------------------------------------------------------------------------

sphq_status build_cbimage16(sphq_handle h) {
  cudaError_t e = cudaMalloc(&h->cbimage, (size_t)h->K * 32);
  if (e != cudaSuccess) return cuda_error(e, "cudaMalloc(codebook image)");
  const long long n = (long long)h->K * 16;
  cbimage16_kernel<<<(unsigned)((n + 255) / 256), 256>>>((const uint16_t*)h->codebook,
                                                         (uint16_t*)h->cbimage, h->K);
  e = cudaGetLastError();
  if (e == cudaSuccess) e = cudaDeviceSynchronize();
  if (e != cudaSuccess) return cuda_error(e, "codebook image");
  return SPHQ_OK;
}

sphq_status pack16(sphq_handle h, const uint16_t* sign, const uint16_t* idx, const uint8_t* rcode,
                   const uint16_t* scale, const uint16_t* offset, cudaStream_t s) {
  const long long threads = (long long)h->nrt * h->ng * 32;
  pack16_kernel<<<(unsigned)((threads + 255) / 256), 256, 0, s>>>(
      sign, idx, rcode, scale, offset, (uint8_t*)h->units, h->rows, h->ng, h->nrt, h->flag);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SPHQ_OK : cuda_error(e, "pack16 kernel launch");
}

sphq_status decode16(sphq_handle h, void* w, cudaStream_t s) {
  const long long n = (long long)h->rows * (h->cols / 16);
  decode16_kernel<<<(unsigned)((n + 255) / 256), 256, 0, s>>>(
      (const uint8_t*)h->units, (const uint16_t*)h->codebook, (uint16_t*)w, h->rows, h->cols,
      h->nrt);
  const cudaError_t e = cudaGetLastError();
  return e == cudaSuccess ? SPHQ_OK : cuda_error(e, "decode16 kernel launch");
}

// Plan for batch 1..8: one cluster per row tile, of csize CTAs (0: the
// smallest of 1, 2, 4, 8 that puts a CTA on every SM, at most the largest
// power of two <= the group count).  Measured on this GB300 (steady state,
// batch 1 and 8): a CTA per SM beats more CTAs -- 4096^2 7.7 / 10.2 / 13.1 us
// at clusters of 1 / 2 / 4, 8192^2 25.9 / 31.1 / 34.1 -- while 512 x 3584
// (32 row tiles) needs clusters of 8 to fill the SMs (3.0 us against 4.9 for
// single CTAs).  Grids of three CTAs per SM or more take the 4-per-SM build
// (more warps hide the L2 gathers: 8192^2 26.0 -> 24.7 us, 18944 x 3584
// 26.0 -> 23.8); smaller grids the 2-per-SM one (the 4-per-SM build put
// 4096^2's 256 CTAs on fewer SMs: 7.8 -> 12.9 us).
sphq_status make_gemv16_plan(sphq_handle h, int batch, int csize, GemvPlan& out) {
  (void)batch;
  int cs = csize;
  if (cs == 0) {
    const int sms = std::max(h->sm_count, 1);
    cs = 1;
    while (cs < 8 && 2 * cs <= h->ng && (long long)h->nrt * cs < sms) cs *= 2;
  }
  if ((long long)h->nrt * cs > 0x7FFFFFFFLL)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv: too many row tiles for one 16-D launch");
  GemvPlan p;
  p.warps_per_cta = kWarps16;
  p.csize = cs;
  p.nclusters = h->nrt;
  p.grid = h->nrt * cs;
  p.tmax = 1;
  p.smem = 0;
  p.mode = kFull;
  p.strip = 1;
  p.ctas_per_sm = (long long)p.grid >= 3LL * std::max(h->sm_count, 1) ? 4 : 2;
  out = p;
  return SPHQ_OK;
}

sphq_status launch_gemv16(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s) {
  const GemvPlan& p = h->plan[batch];
  if (p.grid <= 0 || batch > kMaxBatch)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv: no 16-D plan for this batch");
  Gemv16Args a;
  a.units = (const uint8_t*)h->units;
  a.cbimage = (const uint8_t*)h->cbimage;
  a.x = (const uint16_t*)x;
  a.zeros = (const uint16_t*)h->zeros;
  a.y = (uint16_t*)y;
  a.rows = h->rows;
  a.cols = h->cols;
  a.ng = h->ng;
  a.nrt = h->nrt;
  a.batch = batch;
  a.csize = p.csize;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3((unsigned)p.grid);
  cfg.blockDim = dim3(kWarps16 * 32);
  cfg.dynamicSmemBytes = 0;
  cfg.stream = s;
  cudaLaunchAttribute attr[2];
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)p.csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = h->pdl ? 2 : 1;
  void* args[] = {&a};
  const void* k = p.ctas_per_sm == 4 ? (const void*)gemv16_kernel<4> : (const void*)gemv16_kernel<2>;
  cudaError_t e = cudaLaunchKernelExC(&cfg, k, args);
  if (e != cudaSuccess) return cuda_error(e, "gemv16 launch");
  return SPHQ_OK;
}

}  // namespace sphq
