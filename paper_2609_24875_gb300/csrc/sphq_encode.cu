// Encoder (§3.1: Eq. (3) decomposition, Eq. (5) nearest direction, Eq. (6)
// radius projection, Eq. (7) group quantisation) on the GPU, sm_103a.
//
// Every decision is taken in IEEE single precision with a fixed operation
// order (fused multiply-adds in coordinate order, correctly rounded square
// root and division):
//   p_j = |w_j|, sign bit j = (w_j < 0), r = sqrt(sum p_j^2), d = p / max(r, 1e-12)
//   z = argmax_k d . c_k (ties -> lowest k), r~ = p . c_z
//   per group of 16 vectors: Delta = (max r~ - min r~) / (2^V - 1),
//   Delta16 = RN16(Delta), m16 = RN16(min r~),
//   q = 0 if Delta16 = 0 else clip(floor((r~ - m16) / Delta16 + 1/2), 0, 2^V - 1).
//
// The search of Eq. (5) is a dense contraction (every direction against every
// codebook entry) and runs on the tensor cores in two passes:
//  1. coarse scores: d is split into fp16 parts d = d_hi + d_lo (+ 2^-22 |d|),
//     and one tcgen05.mma of K = 16 forms d_hi . c_k + d_lo . c_k for 128
//     vectors (M) x 256 entries (N) in fp32 tensor memory.  The codebook is a
//     plain table in shared memory (entry k at 16 k bytes); the MMA's B
//     operand reads each entry twice (the K-major no-swizzle layout with a
//     zero leading-dimension offset), so no [c | c] copy is needed.  The
//     coarse score is within 3e-6 of the single-precision score.
//  2. exact choice: a first pass over the coarse scores takes their maximum,
//     a second (the MMAs repeated) keeps, in increasing k, the entries within
//     kDelta (1e-5, relative above 1) of it; they are re-scored with the
//     single-precision fused multiply-add chain and the largest is taken,
//     lowest k on ties.  The single-precision argmax is
//     always among them (its coarse score is within 2 x 3e-6 of the coarse
//     maximum).  If more than kCand entries qualify (degenerate codebooks,
//     zero vectors) the thread re-scores all K entries the same way.
// So the result equals a single-precision CPU encoder bit for bit.
//
// Kernel 1 (persistent, one CTA per SM): 4 primary vector warps (one vector
// per thread, 128 per tile) decompose, write the split directions as the A
// operand and take the final choice; they and 4 partner warps (one per
// tensor-memory lane quarter) scan the scores, each warp half of every chunk;
// one MMA warp issues one MMA per chunk of 256 entries into a double-buffered
// 2 x 256-column tensor-memory ring.  Kernel 2 quantises the radii per group.
// Every mbarrier wait is bounded (2 s; error word bit 1).
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>

#include "sphq_gemv_kernel.cuh"
#include "sphq_umma.cuh"

namespace sphq {

constexpr int kEncPrimWarps = 4;                // 128 vectors per tile = MMA M
constexpr int kEncVecWarps = 2 * kEncPrimWarps;  // + a partner per lane quarter for the scan
constexpr int kEncThreads = (kEncVecWarps + 1) * 32;
constexpr int kEncTile = 32 * kEncPrimWarps;
constexpr int kEncChunk = 256;                  // entries per MMA (N), at most
constexpr int kCand = 4;                        // candidates kept per vector
constexpr float kDelta = 1e-5f;                 // candidate window (relative to max(1, |best|))
constexpr uint32_t kEncPlane = kEncTile * 16;   // bytes of one A plane (d_hi or d_lo)

struct EncodeArgs {
  const float* w;          // vectors x 8 fp32
  const uint8_t* codebook; // K x 16 B (fp16 entries)
  uint8_t* sign;
  uint16_t* idx;
  float* rtilde;
  int* flag;
  long long nvec;
  int K;
  int chunk;               // entries per MMA: min(K, 256)
  uint32_t off_a, off_bar; // from the 1024-aligned base; codebook at 0
};

__device__ __forceinline__ void enc_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}

// K-major operand without swizzle: 8-row core matrices of 16-byte rows
// (row r at (r % 8) * 16 + (r / 8) * 128), K-adjacent core matrices `lbo`
// bytes apart (0: both K halves read the same 16 bytes).
__device__ __forceinline__ uint64_t desc_noswizzle(uint32_t saddr, uint32_t lbo) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)((lbo >> 4) & 0x3FFFu) << 16) |
         ((uint64_t)(128u >> 4) << 32) | ((uint64_t)1u << 46);
}

// d . c_k (or p . c_k) in single precision: fused multiply-adds in order.
__device__ __forceinline__ float dot8(const float (&d)[8], const uint8_t* cb, int k) {
  const uint4 c = *reinterpret_cast<const uint4*>(cb + 16 * k);
  const uint32_t cw[4] = {c.x, c.y, c.z, c.w};
  float s = 0.f;
#pragma unroll
  for (int j = 0; j < 4; ++j) {
    s = fmaf(d[2 * j], h_lo_to_f32(cw[j]), s);
    s = fmaf(d[2 * j + 1], h_hi_to_f32(cw[j]), s);
  }
  return s;
}

__global__ void __launch_bounds__(kEncThreads, 1) encode_vectors_kernel(const EncodeArgs a) {
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const uint32_t cb_bar = sbase + a.off_bar, a_full = cb_bar + 8;
  const uint32_t t_full0 = a_full + 8, t_free0 = t_full0 + 16;  // [2] each
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + a.off_bar + 48);
  const uint32_t abase = sbase + a.off_a;
  const long long ntiles = (a.nvec + kEncTile - 1) / kEncTile;
  const int nchunks = a.K / a.chunk;

  if (threadIdx.x == 0) {
    mbar_init(cb_bar, 1);
    mbar_init(a_full, kEncPrimWarps);
    for (int b = 0; b < 2; ++b) {
      mbar_init(t_full0 + 8u * b, 1);
      mbar_init(t_free0 + 8u * b, kEncVecWarps);
    }
    fence_mbar_init();
    const uint32_t bytes = (uint32_t)a.K * 16u;
    mbar_arrive_expect_tx(cb_bar, bytes);
    for (uint32_t o = 0; o < bytes; o += 32768u)
      bulk_g2s(sbase + o, a.codebook + o, min(32768u, bytes - o), cb_bar);
  }
  if (warp == kEncVecWarps) {
    umma::tmem_alloc(smem_u32(tslot), 2 * kEncChunk);
    umma::tmem_relinquish();
  }
  umma::fence_before_sync();
  __syncthreads();
  umma::fence_after_sync();
  const uint32_t taddr = *tslot;
  if (!mbar_wait(cb_bar, 0) && lane == 0) atomicOr(a.flag, 2);

  if (warp == kEncVecWarps) {
    // ---- MMA warp: one MMA per chunk of entries ----
    if (lane == 0) {
      const uint32_t idesc = umma::idesc_f16_f32(kEncTile, a.chunk);
      long long u = 0;  // chunk uses so far (ring position)
      int it = 0;
      for (long long tile = blockIdx.x; tile < ntiles; tile += gridDim.x, ++it) {
        if (!mbar_wait(a_full, it & 1)) atomicOr(a.flag, 2);
        umma::fence_after_sync();
        for (int c = 0; c < 2 * nchunks; ++c, ++u) {  // two passes over the entries
          const int b = (int)(u & 1);
          const int ch = c < nchunks ? c : c - nchunks;
          if (u >= 2 && !mbar_wait(t_free0 + 8u * b, (uint32_t)((u / 2 - 1) & 1)))
            atomicOr(a.flag, 2);
          umma::fence_after_sync();
          umma::mma_f16(taddr + (uint32_t)(b * kEncChunk), desc_noswizzle(abase, kEncPlane),
                        desc_noswizzle(sbase + (uint32_t)(ch * a.chunk) * 16u, 0u), idesc, 0u);
          umma::commit(t_full0 + 8u * b);
        }
      }
    }
    __syncwarp();
  } else {
    // ---- vector warps ----
    // Warps w and w + 4 read the same tensor-memory lanes (the same 32
    // vectors): the first ("primary") decomposes its vectors, writes the A
    // operand and takes the final choice; both scan the coarse scores, the
    // primary the first half of every chunk of entries and its partner the
    // second half, and they exchange their maxima and candidates through
    // shared memory at a barrier of the pair.
    __shared__ float x_max[kEncPrimWarps][32];
    __shared__ int x_nc[kEncPrimWarps][32];
    __shared__ int x_ck[kEncPrimWarps][kCand][32];
    const bool prim = warp < kEncPrimWarps;
    const int quarter = warp & (kEncPrimWarps - 1);
    const int half = prim ? 0 : 1;
    const int hcols = a.chunk / 2;  // columns of a chunk one warp scans
    const int pair_bar = 1 + quarter;
    auto pair_sync = [&]() { asm volatile("bar.sync %0, 64;" ::"r"(pair_bar) : "memory"); };
    long long u = 0;
    for (long long tile = blockIdx.x; tile < ntiles; tile += gridDim.x) {
      const long long v = tile * kEncTile + quarter * 32 + lane;
      const bool valid = v < a.nvec;
      float p[8], d[8];
      uint32_t sbits = 0;
      if (prim) {
        {
          float x[8] = {0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f, 0.f};
          if (valid) {
            const float4 x0 = reinterpret_cast<const float4*>(a.w + v * 8)[0];
            const float4 x1 = reinterpret_cast<const float4*>(a.w + v * 8)[1];
            x[0] = x0.x, x[1] = x0.y, x[2] = x0.z, x[3] = x0.w;
            x[4] = x1.x, x[5] = x1.y, x[6] = x1.z, x[7] = x1.w;
          }
          float acc = 0.f;
#pragma unroll
          for (int j = 0; j < 8; ++j) {
            p[j] = fabsf(x[j]);
            if (x[j] < 0.f) sbits |= 1u << j;
            acc = fmaf(p[j], p[j], acc);
          }
          const float r = __fsqrt_rn(acc);
          const float den = r > 1e-12f ? r : 1e-12f;
#pragma unroll
          for (int j = 0; j < 8; ++j) d[j] = __fdiv_rn(p[j], den);
        }
        // A operand: d_hi and d_lo planes, row = vector of the tile
        {
          uint32_t hi[4], lo[4];
#pragma unroll
          for (int j = 0; j < 4; ++j) {
            const __half h0 = __float2half_rn(d[2 * j]), h1 = __float2half_rn(d[2 * j + 1]);
            const __half l0 = __float2half_rn(__fsub_rn(d[2 * j], __half2float(h0)));
            const __half l1 = __float2half_rn(__fsub_rn(d[2 * j + 1], __half2float(h1)));
            hi[j] = (uint32_t)__half_as_ushort(h0) | ((uint32_t)__half_as_ushort(h1) << 16);
            lo[j] = (uint32_t)__half_as_ushort(l0) | ((uint32_t)__half_as_ushort(l1) << 16);
          }
          const int t = quarter * 32 + lane;
          const uint32_t off = (uint32_t)((t & 7) * 16 + (t >> 3) * 128);
          *reinterpret_cast<uint4*>(smem + a.off_a + off) = make_uint4(hi[0], hi[1], hi[2], hi[3]);
          *reinterpret_cast<uint4*>(smem + a.off_a + kEncPlane + off) =
              make_uint4(lo[0], lo[1], lo[2], lo[3]);
        }
        umma::fence_proxy_async_smem();
        __syncwarp();
        if (lane == 0) enc_arrive(a_full);
      }

      // Two passes over the coarse scores (the MMAs are repeated, which is
      // cheap): the first takes the maximum, the second collects, in
      // increasing k, the entries within the window below it.  Each block of
      // 32 scores is reduced to its maximum first, so a score costs about one
      // instruction per pass and only the block holding the maximum (or a
      // near tie) is inspected element by element.
      float cmax = -INFINITY, thr = -INFINITY;
      int ck[kCand];
      int nc = 0;
      bool overflow = false;
      for (int c = 0; c < 2 * nchunks; ++c, ++u) {
        const bool collect = c >= nchunks;
        if (c == nchunks) {  // the pair's maximum, then the window
          x_max[quarter][lane] = cmax;
          pair_sync();
          cmax = fmaxf(cmax, x_max[quarter][lane]);
          pair_sync();  // both read before either writes again
          thr = cmax - kDelta * fmaxf(1.f, fabsf(cmax));
        }
        const int b = (int)(u & 1);
        if (!mbar_wait(t_full0 + 8u * b, (uint32_t)((u / 2) & 1)) && lane == 0)
          atomicOr(a.flag, 2);
        umma::fence_after_sync();
        const int kc = (collect ? c - nchunks : c) * a.chunk + half * hcols;
        for (int cc = 0; cc < hcols / 32; ++cc) {
          uint32_t sv[32];
          umma::ld_32x32b_x32(taddr + ((uint32_t)(32 * quarter) << 16) +
                                  (uint32_t)(b * kEncChunk + half * hcols + 32 * cc),
                              sv);
          umma::wait_ld();
          float m8[8];
#pragma unroll
          for (int i = 0; i < 8; ++i)
            m8[i] = fmaxf(fmaxf(__uint_as_float(sv[4 * i]), __uint_as_float(sv[4 * i + 1])),
                          fmaxf(__uint_as_float(sv[4 * i + 2]), __uint_as_float(sv[4 * i + 3])));
          const float bm = fmaxf(fmaxf(fmaxf(m8[0], m8[1]), fmaxf(m8[2], m8[3])),
                                 fmaxf(fmaxf(m8[4], m8[5]), fmaxf(m8[6], m8[7])));
          if (!collect) {
            cmax = fmaxf(cmax, bm);
          } else if (bm >= thr) {
            const int k0 = kc + 32 * cc;
#pragma unroll
            for (int jj = 0; jj < 32; ++jj)
              if (__uint_as_float(sv[jj]) >= thr) {
                if (nc < kCand)
                  ck[nc++] = k0 + jj;
                else
                  overflow = true;
              }
          }
        }
        umma::fence_before_sync();
        __syncwarp();
        if (lane == 0) enc_arrive(t_free0 + 8u * b);
      }

      // the partner's candidates (the second halves of the chunks) to the
      // primary; more than kCand in all is an overflow
      if (!prim) {
        x_nc[quarter][lane] = overflow ? -1 : nc;
#pragma unroll
        for (int i = 0; i < kCand; ++i) x_ck[quarter][i][lane] = i < nc ? ck[i] : 0;
      }
      pair_sync();
      if (prim) {
        const int nq = x_nc[quarter][lane];
        int cq[kCand];
#pragma unroll
        for (int i = 0; i < kCand; ++i) cq[i] = x_ck[quarter][i][lane];
        if (nq < 0 || nc + nq > kCand) overflow = true;
        // exact choice among the candidates of both halves (all entries after
        // an overflow): the largest single-precision score, lowest k on ties
        int z = 0;
        float zs = 0.f;
        if (overflow) {
          for (int k = 0; k < a.K; ++k) {
            const float s2 = dot8(d, smem, k);
            if (k == 0 || s2 > zs) zs = s2, z = k;
          }
        } else {
          bool any = false;
#pragma unroll
          for (int i = 0; i < 2 * kCand; ++i) {
            const bool have = i < kCand ? i < nc : i - kCand < nq;
            if (have) {
              const int k = i < kCand ? ck[i] : cq[i - kCand];
              const float s2 = dot8(d, smem, k);
              if (!any || s2 > zs || (s2 == zs && k < z)) zs = s2, z = k;
              any = true;
            }
          }
        }
        if (valid) {
          a.sign[v] = (uint8_t)sbits;
          a.idx[v] = (uint16_t)z;
          a.rtilde[v] = dot8(p, smem, z);
        }
      }
      pair_sync();  // the partner's lists are read before it writes the next tile's
    }
  }
  umma::fence_before_sync();
  __syncthreads();
  if (warp == kEncVecWarps) {
    umma::fence_after_sync();
    umma::tmem_dealloc(taddr, 2 * kEncChunk);
  }
}

// Eq. (7) per group of 16 vectors: thread per (row, group).
__global__ void encode_groups_kernel(const float* __restrict__ rtilde, uint8_t* __restrict__ rcode,
                                     uint16_t* __restrict__ scale, uint16_t* __restrict__ offset,
                                     long long ngroups, int V) {
  const long long gi = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (gi >= ngroups) return;
  const float* rt = rtilde + gi * kGroupVecs;
  float r[kGroupVecs];
#pragma unroll
  for (int i = 0; i < kGroupVecs; ++i) r[i] = rt[i];
  float mn = r[0], mx = r[0];
#pragma unroll
  for (int i = 1; i < kGroupVecs; ++i) mn = fminf(mn, r[i]), mx = fmaxf(mx, r[i]);
  const int qmax = (1 << V) - 1;
  const float delta = __fdiv_rn(__fsub_rn(mx, mn), (float)qmax);
  const __half d16 = __float2half_rn(delta), m16 = __float2half_rn(mn);
  const float df = __half2float(d16), mf = __half2float(m16);
  scale[gi] = __half_as_ushort(d16);
  offset[gi] = __half_as_ushort(m16);
#pragma unroll
  for (int i = 0; i < kGroupVecs; ++i) {
    int q = 0;
    if (df != 0.f) {
      const float t = floorf(__fadd_rn(__fdiv_rn(__fsub_rn(r[i], mf), df), 0.5f));
      q = t < 0.f ? 0 : (t > (float)qmax ? qmax : (int)t);
    }
    rcode[gi * kGroupVecs + i] = (uint8_t)q;
  }
}

sphq_status launch_encode(sphq_handle h, const float* w, uint8_t* sign, uint16_t* idx,
                          uint8_t* rcode, float* rtilde, cudaStream_t s) {
  int optin = 0;
  cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
  EncodeArgs a;
  a.w = w;
  a.codebook = (const uint8_t*)h->codebook;
  a.sign = sign;
  a.idx = idx;
  a.rtilde = rtilde;
  a.flag = h->flag + 1;
  a.nvec = (long long)h->rows * (h->cols / kVec);
  a.K = h->K;
  a.chunk = std::min(h->K, kEncChunk);
  a.off_a = (uint32_t)(((size_t)h->K * 16 + 1023) / 1024 * 1024);
  a.off_bar = a.off_a + 2 * kEncPlane;
  // at least ~120 KiB so that one CTA (which holds all 512 tensor-memory
  // columns) runs per SM
  const size_t need = 1024 + (size_t)a.off_bar + 64;
  const size_t smem = std::max(need, (size_t)120 * 1024);
  // the kernel's static shared memory (the scan partners' exchange) counts
  // against the same per-block limit as the dynamic part
  cudaFuncAttributes fa;
  e = cudaFuncGetAttributes(&fa, encode_vectors_kernel);
  if (e != cudaSuccess) return cuda_error(e, "cudaFuncGetAttributes(encode)");
  const size_t dyn_max = (size_t)optin > fa.sharedSizeBytes ? (size_t)optin - fa.sharedSizeBytes : 0;
  if (smem > dyn_max) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_encode: shared memory");
  {
    // once per device (the attribute belongs to the kernel on the current device)
    static std::mutex mu;
    static bool done[64] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (h->device < 0 || h->device >= 64) return set_error(SPHQ_ERR_DEVICE, "device index out of range");
    if (!done[h->device]) {
      e = cudaFuncSetAttribute(encode_vectors_kernel, cudaFuncAttributeMaxDynamicSharedMemorySize,
                               (int)dyn_max);
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(encode)");
      done[h->device] = true;
    }
  }
  const long long ntiles = (a.nvec + kEncTile - 1) / kEncTile;
  const unsigned grid = (unsigned)std::max(1LL, std::min<long long>(ntiles, h->sm_count));
  encode_vectors_kernel<<<grid, kEncThreads, smem, s>>>(a);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "encode launch");
  const long long ngroups = (long long)h->rows * h->ng;
  uint16_t* p16 = reinterpret_cast<uint16_t*>(h->params);
  encode_groups_kernel<<<(unsigned)((ngroups + 255) / 256), 256, 0, s>>>(
      rtilde, rcode, p16, p16 + ngroups, ngroups, h->vbits);
  e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_error(e, "encode groups launch");
  return SPHQ_OK;
}

}  // namespace sphq
