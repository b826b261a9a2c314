// Prefill / large-batch product Y = X W_hat^T on the fifth-generation tensor
// cores (tcgen05), sm_103a.
//
// For batches above the decode GEMV's eight rows the product is a dense
// contraction (2 * batch * rows * cols flops against rows * cols decoded
// weights), so it runs as a tensor-core GEMM whose B operand is decoded on
// the fly: W_hat is rebuilt exactly as Eq. (7) and Eq. (4) define it (the
// decode of the GEMV's batch 3-8 mode) straight into shared memory, never to
// HBM.
//
// Tiles: an output tile is 128 or 256 activation rows (one or two MMAs of
// M = 128; tokens) x 256 or 128 weight rows (the MMA's N; 16 or 8 row tiles
// of the unit layout; 128 only with one activation tile, for grids that
// would otherwise leave SMs idle), accumulated in fp32 in tensor memory (256 or all 512 columns) over
// the columns in steps of 64 (128-byte swizzled operand rows) or 32 (64-byte
// swizzle).  Two activation tiles per decoded weight tile halve the decode
// and shared-memory traffic per flop; they are used when the batch exceeds
// 128.  With two, a final partial wave of CTAs (e.g. 512 output tiles on 152
// SMs: three full waves and 56 tiles, which would take as long as a fourth
// full wave) can be split: each of its output tiles goes to two CTAs of one
// activation tile, so it spreads over twice the SMs (8192^2 x 4096: the
// two-pass product 3.6-3.8% faster, the fused one 1.6% (W2) to 3.8% (W3)).
// Next to the 128 KiB W3 codebook only
// 32-column steps leave room for a ring of three stages with two activation
// tiles.  Per step:
//  * one TMA warp loads the 128 (256) x BK activation tile (A operand,
//    K-major, swizzled; rows past the batch read zeros);
//  * one decode warp per 16-row tile (16 or 8 warps) rebuilds its 16 x BK
//    slice of W_hat (half or a quarter of a unit) into the B operand tile in
//    the same swizzled K-major layout, fence them to the async proxy and arrive on the stage's
//    mbarrier;
//  * one MMA warp issues BK / 16 (times the activation tiles) 128 x BN x 16
//    tcgen05.mma (fp16 x fp16 -> fp32) when both halves of the stage are in, and commits their completion
//    to the stage's "empty" mbarrier, which releases the buffers.
// Stages rotate through a ring of buffers (two to four, as shared memory
// allows next to the codebook).  After the last step the decode warps read
// the accumulators from tensor memory (warp w: lanes 32 (w % 4).., the warps
// of one lane quarter splitting the columns), round to fp16 and store Y.
//
// Every mbarrier wait gives up after about two seconds and records bit 1 in
// the handle's device error word, so a fault cannot hang the GPU.  The ring's
// waits (one polling thread per warp) poll without a suspend hint, so a stage
// is picked up as soon as it completes (fused W3 product 5-6% faster).
#include <cuda.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <cstdio>
#include <mutex>

#include "sphq_gemv_kernel.cuh"
#include "sphq_umma.cuh"

namespace sphq {

constexpr int kGemmBM = 128;                    // activation rows per tile (MMA M)
// Pseudo format of the two-pass product: the B operand is a decoded W_hat
// (rows x cols fp16 in global memory, written by decode_units_kernel) that
// the TMA warp loads beside the activations; no codebook, no decode warps.
constexpr int kFmtDense = 0;
// Batches taking the split-K form (with a workspace, the shape automatic).
constexpr int kSplitMinBatch = 41, kSplitMaxBatch = 256, kSplitMinGroups = 16;
// One decode warp per 16-row tile of the weight tile (16 or 8), then the MMA
// warp and the TMA warp.
constexpr int gemm_threads(int bn) { return (bn / kRowsPerTile + 2) * 32; }
// operand tile bytes for a stage of BK columns
constexpr uint32_t tile_a_bytes(int bk) { return (uint32_t)kGemmBM * bk * 2; }  // per 128 rows
constexpr uint32_t tile_b_bytes(int bk, int bn) { return (uint32_t)bn * bk * 2; }

struct GemmArgs {
  const uint8_t* units;
  const uint8_t* cbimage;  // codebook as laid out in shared memory
  uint16_t* y;             // batch x rows fp16
  int* flag;               // device error word: bit 1 = an mbarrier wait gave up
  int rows, cols, nrt, batch;
  int nwt;                 // weight tiles (of BN rows) across the rows
  int n_big;               // CTAs with MT activation tiles; the rest take one
  int ksplit;              // CTAs per output tile, each a share of the radius groups (split-K)
  float* part;             // split-K: fp32 partial tiles, [tile][ksplit][MT x 128][BN]
  unsigned* tickets;       // split-K: per output tile, CTAs done (zeroed before the launch)
  int stages;              // ring depth
  uint32_t cb_bytes;
  uint32_t off_b, off_cb, off_bar;  // from the 1024-byte aligned base; A tiles at 0
};

__device__ __forceinline__ void mbar_arrive(uint32_t bar) {
  asm volatile("mbarrier.arrive.shared::cta.b64 _, [%0];" ::"r"(bar) : "memory");
}
__device__ __forceinline__ void sts16(uint32_t addr, uint4 v) {
  asm volatile("st.shared.v4.u32 [%0], {%1, %2, %3, %4};" ::"r"(addr), "r"(v.x), "r"(v.y),
               "r"(v.z), "r"(v.w)
               : "memory");
}

__device__ __forceinline__ uint4 sel4(bool p, uint4 a, uint4 b) {
  return make_uint4(p ? a.x : b.x, p ? a.y : b.y, p ? a.z : b.z, p ? a.w : b.w);
}

// Element (activation row t, weight row n) of a split-K partial tile sits at
// t * BN + n; a thread stores / sums 32 consecutive weight rows of one
// activation row (one tcgen05.ld of 32 columns).
__device__ __forceinline__ void store_part32(float* p, const uint32_t (&v)[32]) {
#pragma unroll
  for (int t = 0; t < 8; ++t)
    reinterpret_cast<float4*>(p)[t] =
        make_float4(__uint_as_float(v[4 * t]), __uint_as_float(v[4 * t + 1]),
                    __uint_as_float(v[4 * t + 2]), __uint_as_float(v[4 * t + 3]));
}
__device__ __forceinline__ void named_sync(int id, int threads) {
  asm volatile("bar.sync %0, %1;" ::"r"(id), "r"(threads) : "memory");
}

// Decodes words M and M+1 (the stage's 64 columns) of the lane's unit and
// stores its four 16-byte blocks into the B tile: vector (row, slot) goes to
// tile row n and 16-byte chunk c = slot % 8, at chunk position c ^ (n % 8).
// Lanes of odd gid store word M+1 first: the two gids of a quarter warp then
// write disjoint chunk positions ({q ^ gid} and {(4 + q) ^ (gid + 1)}), so
// each 16-byte store is free of bank conflicts.
template <int FMT, int M>
__device__ __forceinline__ void decode_half(const Unit<FMT>& u, const UnitConst<FMT>& kc, int q,
                                            int gid, int jt, const SmemCodebook& cb,
                                            uint32_t btile) {
  uint4 wa[2], wb[2];
#pragma unroll
  for (int mm = 0; mm < 2; ++mm) {
    uint4 sa, sb;
    uint32_t qp;
    word_directions<FMT>(u, kc, M + mm, q, cb, sa, sb, qp);
    const uint32_t r = radius_pair<fmt_radius_bits(FMT)>(qp, kc.d2, kc.m2);
    wa[mm] = scale_block(sa, bcast_lo(r));
    wb[mm] = scale_block(sb, bcast_hi(r));
  }
  const bool odd = gid & 1;
  const int nA = kRowsPerTile * jt + gid, nB = nA + 8;
  const uint32_t rowA = btile + nA * 128, rowB = btile + nB * 128;
  const int c0 = (odd ? 4 : 0) + q, c1 = c0 ^ 4;  // first / second chunk stored
  sts16(rowA + ((c0 ^ (nA & 7)) << 4), sel4(odd, wa[1], wa[0]));
  sts16(rowB + ((c0 ^ (nB & 7)) << 4), sel4(odd, wb[1], wb[0]));
  sts16(rowA + ((c1 ^ (nA & 7)) << 4), sel4(odd, wa[0], wa[1]));
  sts16(rowB + ((c1 ^ (nB & 7)) << 4), sel4(odd, wb[0], wb[1]));
}

// Decodes word M (a stage of 32 columns) of the lane's unit into a B tile of
// 64-byte rows in the 64-byte swizzle: chunk q of row n at q ^ ((n / 2) % 4).
// Rows gid and gid + 1 of a quarter warp are 64 bytes apart, so the eight
// lanes hit distinct 16-byte bank groups.
template <int FMT, int M>
__device__ __forceinline__ void decode_word(const Unit<FMT>& u, const UnitConst<FMT>& kc, int q,
                                            int gid, int jt, const SmemCodebook& cb,
                                            uint32_t btile) {
  uint4 sa, sb;
  uint32_t qp;
  word_directions<FMT>(u, kc, M, q, cb, sa, sb, qp);
  const uint32_t r = radius_pair<fmt_radius_bits(FMT)>(qp, kc.d2, kc.m2);
  const int nA = kRowsPerTile * jt + gid, nB = nA + 8;
  sts16(btile + nA * 64 + ((q ^ ((nA >> 1) & 3)) << 4), scale_block(sa, bcast_lo(r)));
  sts16(btile + nB * 64 + ((q ^ ((nB >> 1) & 3)) << 4), scale_block(sb, bcast_hi(r)));
}

// MT activation tiles of 128 rows share each decoded B tile (MT accumulators
// of 256 tensor-memory columns); BK columns per stage: 64 (128-byte swizzle)
// or 32 (64-byte swizzle, half the ring memory, for the 128 KiB W3 codebook).
template <int FMT, int MT, int BK, int BN>
__global__ void __launch_bounds__(gemm_threads(BN), 1)
    gemm_kernel(const GemmArgs a, const __grid_constant__ CUtensorMap tmap,
                const __grid_constant__ CUtensorMap tmap_w) {
  constexpr bool kDense = FMT == kFmtDense;   // B tiles by TMA from a decoded W_hat
  constexpr int kTilesN = BN / kRowsPerTile;  // row tiles per weight tile
  constexpr int kDecodeWarps = kTilesN;       // one row tile each
  constexpr int kMmaWarp = kDecodeWarps, kTmaWarp = kDecodeWarps + 1;
  constexpr uint32_t kTileA = tile_a_bytes(BK), kTileB = tile_b_bytes(BK, BN);
  constexpr uint32_t kStageA = MT * kTileA;
  constexpr uint32_t kCols = MT * BN;  // tensor-memory columns
  constexpr int kStepsPerGroup = kGroupCols / BK;
  extern __shared__ uint8_t smem_raw[];
  uint8_t* smem = reinterpret_cast<uint8_t*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) &
                                             ~static_cast<uintptr_t>(1023));
  const uint32_t sbase = smem_u32(smem);
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int S = a.stages;
  const int ng = a.cols / kGroupCols;
  const uint32_t full0 = sbase + a.off_bar;  // full[S], empty[S], acc, cb, tmem slot
  const uint32_t empty0 = full0 + 8u * S;
  const uint32_t acc_bar = empty0 + 8u * S;
  const uint32_t cb_bar = acc_bar + 8u;
  uint32_t* tslot = reinterpret_cast<uint32_t*>(smem + a.off_bar + 16u * S + 16u);
  // Split-K: the ksplit consecutive CTAs of an output tile take consecutive
  // shares of the radius groups (columns) and sum their fp32 partials through
  // global memory in share order.
  int bid = (int)blockIdx.x, kidx = 0;
  if (a.ksplit > 1) {
    kidx = bid % a.ksplit;
    bid /= a.ksplit;
  }
  const int g_lo = kidx * (ng / a.ksplit) + min(kidx, ng % a.ksplit);
  const int g_hi = g_lo + ng / a.ksplit + (kidx < ng % a.ksplit ? 1 : 0);
  const int i_lo = g_lo * kStepsPerGroup, i_hi = g_hi * kStepsPerGroup;
  // This CTA's output tile.  The first n_big CTAs take MT activation tiles
  // (weight tile fastest); the rest split the remaining MT-tile outputs into
  // one activation tile each (two CTAs per output tile, a final wave that
  // spreads over twice the SMs).
  int wt, tok0, mt;
  if (bid < a.n_big) {
    wt = bid % a.nwt;
    tok0 = bid / a.nwt * (kGemmBM * MT);
    mt = MT;
  } else {
    const int j = bid - a.n_big, L = a.n_big + (j >> 1);
    wt = L % a.nwt;
    tok0 = L / a.nwt * (kGemmBM * MT) + (j & 1) * kGemmBM;
    mt = 1;
  }
  if (tok0 >= a.batch) return;  // a half tile wholly past the batch: no work
  // activation tiles wholly past the batch are neither loaded nor multiplied
  mt = min(mt, (a.batch - tok0 + kGemmBM - 1) / kGemmBM);
  const int rt0 = wt * kTilesN;

  if (threadIdx.x == 0) {
    for (int s = 0; s < S; ++s) {
      mbar_init(full0 + 8u * s, kDense ? 1 : kDecodeWarps + 1);
      mbar_init(empty0 + 8u * s, 1);
    }
    mbar_init(acc_bar, 1);
    mbar_init(cb_bar, 1);
    fence_mbar_init();
    if constexpr (!kDense) {
      mbar_arrive_expect_tx(cb_bar, a.cb_bytes);
      for (uint32_t o = 0; o < a.cb_bytes; o += 32768u)
        bulk_g2s(sbase + a.off_cb + o, a.cbimage + o, min(32768u, a.cb_bytes - o), cb_bar);
    }
  }
  if (warp == kMmaWarp) {
    umma::tmem_alloc(smem_u32(tslot), kCols);
    umma::tmem_relinquish();
  }
  umma::fence_before_sync();
  __syncthreads();
  umma::fence_after_sync();
  const uint32_t taddr = *tslot;

  if (warp == kTmaWarp) {
    if (lane == 0) {
      umma::prefetch_tmap(&tmap);
      if constexpr (kDense) umma::prefetch_tmap(&tmap_w);
      for (int i = i_lo, s = 0, r = 0; i < i_hi; ++i) {
        if (r > 0 && !mbar_wait_poll(empty0 + 8u * s, (r - 1) & 1)) atomicOr(a.flag, 2);
        mbar_arrive_expect_tx(full0 + 8u * s, (uint32_t)mt * kTileA + (kDense ? kTileB : 0u));
#pragma unroll
        for (int t = 0; t < MT; ++t)
          if (t < mt)
            umma::tma_load_2d(sbase + s * kStageA + t * kTileA, &tmap, i * BK, tok0 + t * kGemmBM,
                              full0 + 8u * s);
        if constexpr (kDense)  // the W_hat tile: BN weight rows x BK columns
          umma::tma_load_2d(sbase + a.off_b + s * kTileB, &tmap_w, i * BK, rt0 * kRowsPerTile,
                            full0 + 8u * s);
        if (++s == S) s = 0, ++r;
      }
    }
    __syncwarp();
  } else if (warp == kMmaWarp) {
    if (lane == 0) {
      constexpr uint32_t idesc = umma::idesc_f16_f32(kGemmBM, BN);
      for (int i = i_lo, s = 0, r = 0; i < i_hi; ++i) {
        if (!mbar_wait_poll(full0 + 8u * s, r & 1)) atomicOr(a.flag, 2);
        umma::fence_after_sync();
        const uint32_t at = sbase + s * kStageA, bt = sbase + a.off_b + s * kTileB;
#pragma unroll
        for (int t = 0; t < MT; ++t) {
          if (t >= mt) break;
#pragma unroll
          for (int kk = 0; kk < BK / 16; ++kk) {
            const uint32_t ad = at + t * kTileA + 32u * kk, bd = bt + 32u * kk;
            umma::mma_f16(taddr + t * BN,
                          BK == 64 ? umma::smem_desc_sw128(ad) : umma::smem_desc_sw64(ad),
                          BK == 64 ? umma::smem_desc_sw128(bd) : umma::smem_desc_sw64(bd), idesc,
                          (i != i_lo || kk != 0));
          }
        }
        umma::commit(empty0 + 8u * s);
        if (++s == S) s = 0, ++r;
      }
      umma::commit(acc_bar);
    }
    __syncwarp();
  } else {
    if constexpr (!kDense) {
    // ---- decode warps: W_hat slices into the B tiles ----
    const int q = lane & 3, gid = lane >> 2;
    constexpr int UB = Layout<FMT>::kUnitBytes;
    SmemCodebook cb;
    cb.base = smem + a.off_cb;
    cb.copyoff = fmt_small(FMT) ? (uint32_t)(lane & 7) * 16u : 0u;
    const int jt = warp;  // this warp's row tile within the weight tile
    const bool ok = rt0 + jt < a.nrt;
    const uint8_t* ub0 = a.units + (size_t)(rt0 + jt) * UB;  // group 0; + g * nrt * UB
    const size_t gstride = (size_t)a.nrt * UB;
    Unit<FMT> cur = {}, nxt = {};
    if (ok) nxt = load_unit<FMT>(ub0 + (size_t)g_lo * gstride, lane);
    if (!mbar_wait(cb_bar, 0) && lane == 0) atomicOr(a.flag, 2);
    for (int i = i_lo, s = 0, r = 0; i < i_hi; ++i) {
      const int g = i / kStepsPerGroup;
      const int step = i % kStepsPerGroup;
      if (step == 0) {
        cur = nxt;
        if (ok && g + 1 < g_hi) nxt = load_unit<FMT>(ub0 + (size_t)(g + 1) * gstride, lane);
      }
      // one lane polls the stage's release (the MMAs that read it are
      // complete); the warp's stores follow it through __syncwarp
      if (r > 0 && lane == 0 && !mbar_wait_poll(empty0 + 8u * s, (r - 1) & 1)) atomicOr(a.flag, 2);
      __syncwarp();
      const uint32_t bt = sbase + a.off_b + s * kTileB;
      if (ok) {
        const UnitConst<FMT> kc = unit_const<FMT>(cur, q);
        if constexpr (BK == 64) {
          if (step)
            decode_half<FMT, 2>(cur, kc, q, gid, jt, cb, bt);
          else
            decode_half<FMT, 0>(cur, kc, q, gid, jt, cb, bt);
        } else {
          if (step == 0)
            decode_word<FMT, 0>(cur, kc, q, gid, jt, cb, bt);
          else if (step == 1)
            decode_word<FMT, 1>(cur, kc, q, gid, jt, cb, bt);
          else if (step == 2)
            decode_word<FMT, 2>(cur, kc, q, gid, jt, cb, bt);
          else
            decode_word<FMT, 3>(cur, kc, q, gid, jt, cb, bt);
        }
      }
      umma::fence_proxy_async_smem();
      __syncwarp();
      if (lane == 0) mbar_arrive(full0 + 8u * s);
      if (++s == S) s = 0, ++r;
    }
    }  // decode warps (the two-pass form has none in the main loop)

    // ---- epilogue: accumulators -> fp16 Y ----
    if (!mbar_wait(acc_bar, 0) && lane == 0) atomicOr(a.flag, 2);
    umma::fence_after_sync();
    // warp w reads lanes 32 (w % 4).. (its quarter of tensor memory); the
    // kDecodeWarps / 4 warps of a quarter split the MT x BN columns evenly
    constexpr int kParts = kDecodeWarps / 4;
    constexpr int kColsPerWarp = MT * BN / kParts;
    static_assert(kColsPerWarp <= BN && kColsPerWarp % 32 == 0, "epilogue split");
    const int quarter = warp & 3, part = warp >> 2;
    const int start = part * kColsPerWarp;
    const int acc = start / BN;
    const int token = tok0 + kGemmBM * acc + 32 * quarter + lane;
    const int ncc = acc < mt ? kColsPerWarp / 32 : 0;
    // 32 results of this thread's activation row, weight rows row0.. -> fp16 Y
    auto store_y = [&](int row0, const uint32_t (&v)[32]) {
      if (token >= a.batch || row0 >= a.rows) return;
      uint16_t* dst = a.y + (size_t)token * a.rows + row0;
      if (row0 + 32 <= a.rows && (reinterpret_cast<uintptr_t>(dst) & 15u) == 0) {
        uint32_t hv[16];
#pragma unroll
        for (int t = 0; t < 16; ++t) {
          const __half2 p = __floats2half2_rn(__uint_as_float(v[2 * t]),
                                              __uint_as_float(v[2 * t + 1]));
          hv[t] = *reinterpret_cast<const uint32_t*>(&p);
        }
#pragma unroll
        for (int t = 0; t < 4; ++t)
          reinterpret_cast<uint4*>(dst)[t] =
              make_uint4(hv[4 * t], hv[4 * t + 1], hv[4 * t + 2], hv[4 * t + 3]);
      } else {
#pragma unroll
        for (int t = 0; t < 32; ++t)
          if (row0 + t < a.rows) dst[t] = f32_to_h_rn(__uint_as_float(v[t]));
      }
    };
    // split-K partial rows of this thread: activation row (token - tok0)
    constexpr size_t kPartFloats = (size_t)kGemmBM * MT * BN;
    const size_t prow = (size_t)(kGemmBM * acc + 32 * quarter + lane) * BN;
#pragma unroll 1
    for (int cc = 0; cc < ncc; ++cc) {
      const int col = start % BN + 32 * cc;  // within the accumulator
      const uint32_t tcol = (uint32_t)(acc * BN + col);
      uint32_t v[32];
      umma::ld_32x32b_x32(taddr + ((uint32_t)(32 * quarter) << 16) + tcol, v);
      umma::wait_ld();
      if (a.ksplit > 1)
        store_part32(a.part + ((size_t)bid * a.ksplit + kidx) * kPartFloats + prow + col, v);
      else
        store_y(rt0 * kRowsPerTile + col, v);
    }
    if (a.ksplit > 1) {
      // The last of the tile's CTAs to finish sums the partials in share
      // order (a fixed order: deterministic) and writes Y.  No CTA waits for
      // another: the others just leave.
      int* last = reinterpret_cast<int*>(tslot + 1);
      __threadfence();
      named_sync(1, kDecodeWarps * 32);
      if (warp == 0 && lane == 0)
        *last = atomicAdd(a.tickets + bid, 1u) == (unsigned)(a.ksplit - 1);
      named_sync(1, kDecodeWarps * 32);
      if (*last) {
        __threadfence();
#pragma unroll 1
        for (int cc = 0; cc < ncc; ++cc) {
          const int col = start % BN + 32 * cc;
          float sum[32];
#pragma unroll
          for (int t = 0; t < 32; ++t) sum[t] = 0.f;
          for (int k = 0; k < a.ksplit; ++k) {  // shares in order
            const float4* pp = reinterpret_cast<const float4*>(
                a.part + ((size_t)bid * a.ksplit + k) * kPartFloats + prow + col);
#pragma unroll
            for (int t = 0; t < 8; ++t) {
              const float4 q4 = __ldcg(pp + t);
              sum[4 * t] += q4.x;
              sum[4 * t + 1] += q4.y;
              sum[4 * t + 2] += q4.z;
              sum[4 * t + 3] += q4.w;
            }
          }
          uint32_t v[32];
#pragma unroll
          for (int t = 0; t < 32; ++t) v[t] = __float_as_uint(sum[t]);
          store_y(rt0 * kRowsPerTile + col, v);
        }
      }
    }
  }
  umma::fence_before_sync();
  __syncthreads();
  if (warp == kMmaWarp) {
    umma::fence_after_sync();
    umma::tmem_dealloc(taddr, kCols);
  }
}

// First pass of the two-pass product: W_hat (rows x cols fp16, row-major)
// from the packed units, exactly as Eq. (7) and Eq. (4) define it (the
// GEMV's batch 3-8 decode, bit for bit the output of sphq_decode).  CTAs are
// persistent (a grid of the resident count) and stage the codebook image once;
// each of the 16 warps takes whole units, with the next unit's load in flight
// while it decodes the current one; a lane rebuilds its eight vectors and
// stores each as 16 bytes (a row's four lanes write 64 contiguous bytes per
// word).
constexpr int kDecodeUnitsWarps = 16;
template <int FMT>
__global__ void __launch_bounds__(kDecodeUnitsWarps * 32) decode_units_kernel(const uint8_t* __restrict__ units,
                                                           const uint8_t* __restrict__ cbimage,
                                                           uint32_t cb_bytes, uint16_t* __restrict__ w,
                                                           int rows, int cols, int nrt, int ng,
                                                           int* flag) {
  extern __shared__ __align__(128) uint8_t smem[];
  __shared__ __align__(8) uint64_t bar;
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  const int q = lane & 3, gid = lane >> 2;
  const uint32_t b = smem_u32(&bar);
  if (threadIdx.x == 0) {
    mbar_init(b, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(b, cb_bytes);
    for (uint32_t o = 0; o < cb_bytes; o += 32768u)
      bulk_g2s(smem_u32(smem) + o, cbimage + o, min(32768u, cb_bytes - o), b);
  }
  __syncthreads();
  if (!mbar_wait(b, 0) && lane == 0) atomicOr(flag, 2);
  SmemCodebook cb;
  cb.base = smem;
  cb.copyoff = fmt_small(FMT) ? (uint32_t)(lane & 7) * 16u : 0u;
  constexpr int UB = Layout<FMT>::kUnitBytes;
  const int total = nrt * ng;
  const int nwarps = (int)gridDim.x * kDecodeUnitsWarps;
  int u = (int)blockIdx.x * kDecodeUnitsWarps + warp;
  Unit<FMT> nxt = {};
  if (u < total) nxt = load_unit<FMT>(units + (size_t)u * UB, lane);
  for (; u < total; u += nwarps) {
    const int g = u / nrt, rt = u - g * nrt;  // unit (rt, g) is number g * nrt + rt
    const Unit<FMT> un = nxt;
    if (u + nwarps < total) nxt = load_unit<FMT>(units + (size_t)(u + nwarps) * UB, lane);
    const UnitConst<FMT> kc = unit_const<FMT>(un, q);
    const int rA = rt * kRowsPerTile + gid, rB = rA + 8;
    uint16_t* pa = w + (size_t)rA * cols + (size_t)g * kGroupCols + 8 * q;
    uint16_t* pb = pa + (size_t)8 * cols;
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      uint4 sa, sb;
      uint32_t qp;
      word_directions<FMT>(un, kc, m, q, cb, sa, sb, qp);
      const uint32_t r = radius_pair<fmt_radius_bits(FMT)>(qp, kc.d2, kc.m2);
      if (rA < rows) *reinterpret_cast<uint4*>(pa + 32 * m) = scale_block(sa, bcast_lo(r));
      if (rB < rows) *reinterpret_cast<uint4*>(pb + 32 * m) = scale_block(sb, bcast_hi(r));
    }
  }
}

// ---------------------------------------------------------------------------
// host side
// ---------------------------------------------------------------------------

typedef CUresult (*EncodeTiledFn)(CUtensorMap*, CUtensorMapDataType, cuuint32_t, void*,
                                  const cuuint64_t*, const cuuint64_t*, const cuuint32_t*,
                                  const cuuint32_t*, CUtensorMapInterleave, CUtensorMapSwizzle,
                                  CUtensorMapL2promotion, CUtensorMapFloatOOBfill);

static EncodeTiledFn encode_fn() {
  static EncodeTiledFn fn = nullptr;
  static std::once_flag once;
  std::call_once(once, [] {
    void* p = nullptr;
    cudaDriverEntryPointQueryResult q;
    if (cudaGetDriverEntryPointByVersion("cuTensorMapEncodeTiled", &p, 12000, cudaEnableDefault,
                                         &q) == cudaSuccess &&
        q == cudaDriverEntryPointSuccess)
      fn = reinterpret_cast<EncodeTiledFn>(p);
    else
      (void)cudaGetLastError();
  });
  return fn;
}

// Instantiated shapes (MT, BK, BN): 128-row weight tiles only with one
// activation tile; 32-column stages only for the W3 tables.
template <int FMT>
static const void* gemm_ptr(int mt, int bk, int bn) {
  const void* p = nullptr;
  if (bn == 256) {
    if (bk == 64) p = mt == 2 ? (const void*)&gemm_kernel<FMT, 2, 64, 256>
                              : (const void*)&gemm_kernel<FMT, 1, 64, 256>;
    if constexpr (!fmt_small(FMT))
      if (bk == 32) p = mt == 2 ? (const void*)&gemm_kernel<FMT, 2, 32, 256>
                                : (const void*)&gemm_kernel<FMT, 1, 32, 256>;
  } else if (bn == 128 && mt == 1) {
    if (bk == 64) p = (const void*)&gemm_kernel<FMT, 1, 64, 128>;
    if constexpr (!fmt_small(FMT))
      if (bk == 32) p = (const void*)&gemm_kernel<FMT, 1, 32, 128>;
  }
  return p;
}

static const void* gemm_kernel_ptr(int fmt, int mt, int bk, int bn) {
  if (fmt == kFmtDense) {
    if (bk != 64) return nullptr;
    if (bn == 256) return mt == 2 ? (const void*)&gemm_kernel<kFmtDense, 2, 64, 256>
                                  : (const void*)&gemm_kernel<kFmtDense, 1, 64, 256>;
    return bn == 128 && mt == 1 ? (const void*)&gemm_kernel<kFmtDense, 1, 64, 128> : nullptr;
  }
  switch (fmt) {
#define SPHQ_GEMM_PTR(F) \
  case F:                \
    return gemm_ptr<F>(mt, bk, bn);
    SPHQ_GEMM_PTR(2)
    SPHQ_GEMM_PTR(3)
    SPHQ_GEMM_PTR(4)
    SPHQ_GEMM_PTR(5)
    SPHQ_GEMM_PTR(6)
    SPHQ_GEMM_PTR(7)
    SPHQ_GEMM_PTR(8)
    SPHQ_GEMM_PTR(9)
#undef SPHQ_GEMM_PTR
    default:
      return nullptr;
  }
}

static size_t align_to(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Shared-memory layout of the GEMM for a handle: ring depth and offsets.
struct GemmSmem {
  int stages = 0;
  uint32_t cb_bytes = 0, off_b = 0, off_cb = 0, off_bar = 0;
  size_t total = 0;
};

static GemmSmem gemm_smem(const sphq_handle_s* h, int optin, int mt, int bk, int bn,
                          bool dense = false) {
  GemmSmem L;
  L.cb_bytes = dense ? 0u : fmt_small(h->fmt) ? (uint32_t)h->K * 8u * 16u : (uint32_t)h->K * 16u;
  for (int S = 4; S >= 2; --S) {
    const size_t off_b = (size_t)S * mt * tile_a_bytes(bk);
    const size_t off_cb = off_b + (size_t)S * tile_b_bytes(bk, bn);
    const size_t off_bar = align_to(off_cb + L.cb_bytes, 16);
    const size_t total = 1024 + off_bar + 16u * S + 16u + 16u;  // alignment slack + barriers + slot
    if (total <= (size_t)optin) {
      L.stages = S;
      L.off_b = (uint32_t)off_b;
      L.off_cb = (uint32_t)off_cb;
      L.off_bar = (uint32_t)off_bar;
      L.total = total;
      return L;
    }
  }
  return L;
}

struct GemmShape {
  int mt = 0, bk = 0, bn = 0;
  GemmSmem L;
};

// Split-K plan of sphq_gemm_ws (gemm_splitk_plan below): CTAs per output
// tile, workspace bytes (partials, then one counter per tile).
struct SplitK {
  int ksplit = 1;
  size_t part_bytes = 0, bytes = 0;
  long long tiles = 0;
};
static SplitK gemm_splitk_plan(const sphq_handle_s* h, int batch);

// The grid of a launch shape: nwt x ntok output tiles of BN weight rows x MT
// activation tiles, in whole waves of SMs plus a final partial wave.  With
// MT = 2 (and MT automatic), a final wave of r tiles that fit twice over on
// the SMs goes to 2r CTAs of one activation tile each when that is estimated
// faster: a wave of one-tile CTAs takes c of a wave of two-tile CTAs
// (measured on this GB300 at 8192^2 x 4096, 56 output tiles in the final
// wave: the dense pass 0.8, the fused kernel 0.85 (W3) to 0.94 (W2)).
// `waves` is the estimated time in two-tile CTA times.
struct GemmGrid {
  int nwt = 0, ntok = 0, n_big = 0, n_small = 0;
  double waves = 0;
};

static GemmGrid gemm_grid(const sphq_handle_s* h, int batch, int mt, int bn, bool dense) {
  GemmGrid G;
  const long long sms = h->sm_count > 0 ? h->sm_count : 1;
  G.nwt = (h->nrt + bn / kRowsPerTile - 1) / (bn / kRowsPerTile);
  G.ntok = (batch + kGemmBM * mt - 1) / (kGemmBM * mt);
  const long long n = (long long)G.nwt * G.ntok;
  G.n_big = (int)n;
  G.waves = (double)((n + sms - 1) / sms);
  if (mt == 2 && !h->gemm_mt) {
    const long long full = n / sms, r = n - full * sms;
    const double c = dense ? 0.8 : 0.9;
    if (full >= 1 && r > 0 && 2 * r <= sms && full + c < G.waves - 1e-9) {
      G.n_big = (int)(full * sms);
      G.n_small = (int)(2 * r);
      G.waves = (double)full + c;
    }
  }
  return G;
}

// Shape (MT activation tiles, BN weight rows per CTA): the least estimated
// time = waves of CTAs x time per CTA, the latter relative to the work of one
// CTA (MT x BN) over its measured efficiency (two tiles of 256 rows: 1, one:
// 0.64, one of 128 rows: 0.5), unless sphq_set_gemm_shape fixed MT / BN; a
// candidate needs a ring of two stages next to the codebook, with 64-column
// stages if they fit, else 32-column ones (W3 with two activation tiles).
static GemmShape select_gemm_shape(const sphq_handle_s* h, int batch, int optin,
                                   bool dense = false) {
  const int sms = h->sm_count > 0 ? h->sm_count : 1;
  static const int kShapes[3][2] = {{2, 256}, {1, 256}, {1, 128}};
  static const double kEff[3] = {1.0, 0.64, 0.5};
  GemmShape best;
  double best_t = 0;
  for (int c = 0; c < 3; ++c) {
    const int m = kShapes[c][0], n = kShapes[c][1];
    if (h->gemm_mt ? m != h->gemm_mt : (m == 2 && batch <= kGemmBM)) continue;
    if (h->gemm_bn && n != h->gemm_bn) continue;
    for (int k : {64, 32}) {
      if (!gemm_kernel_ptr(dense ? kFmtDense : h->fmt, m, k, n)) continue;
      const GemmSmem T = gemm_smem(h, optin, m, k, n, dense);
      if (T.stages < 2) continue;
      const double t = gemm_grid(h, batch, m, n, dense).waves * (m * n) / kEff[c];
      if (!best.mt || t < best_t - 1e-9) {
        best.mt = m, best.bk = k, best.bn = n, best.L = T;
        best_t = t;
      }
      break;  // 64-column stages when they fit
    }
  }
  return best;
}

static sphq_status device_smem_optin(const sphq_handle_s* h, int* optin) {
  cudaError_t e = cudaDeviceGetAttribute(optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
  return SPHQ_OK;
}

sphq_status gemm_shape_info(sphq_handle h, int batch, sphq_gemm_info* out) {
  int optin = 0;
  sphq_status st = device_smem_optin(h, &optin);
  if (st != SPHQ_OK) return st;
  const GemmShape g = select_gemm_shape(h, batch, optin);
  if (!g.mt) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm: no shape fits this device");
  out->act_tiles = g.mt;
  out->weight_rows = g.bn;
  out->stage_cols = g.bk;
  out->stages = g.L.stages;
  const GemmGrid G = gemm_grid(h, batch, g.mt, g.bn, false);
  out->grid_x = G.nwt;
  out->grid_y = G.ntok;
  out->smem_bytes = (long long)g.L.total;
  out->split_ctas = G.n_small;
  out->ksplit = gemm_splitk_plan(h, batch).ksplit;
  return SPHQ_OK;
}

// One launch of the product kernel: the fused form (w_hat == nullptr), or the
// second pass of the two-pass form reading the decoded w_hat.
static sphq_status launch_gemm_kernel(sphq_handle h, const void* x, void* y, int batch,
                                      cudaStream_t s, const void* w_hat, int ksplit = 1,
                                      float* part = nullptr, unsigned* tickets = nullptr) {
  const bool dense = w_hat != nullptr;
  EncodeTiledFn enc = encode_fn();
  if (!enc) return set_error(SPHQ_ERR_CUDA, "sphq_gemm: cuTensorMapEncodeTiled unavailable");
  int optin = 0;
  sphq_status st = device_smem_optin(h, &optin);
  if (st != SPHQ_OK) return st;
  const GemmShape g = select_gemm_shape(h, batch, optin, dense);
  if (!g.mt) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm: no shape fits this device");
  const int mt = g.mt, bk = g.bk, bn = g.bn;
  const GemmSmem& L = g.L;
  const GemmGrid G = gemm_grid(h, batch, mt, bn, dense);
  if (log_enabled())
    std::fprintf(stderr,
                 "sphq: gemm %d x %d, batch %d%s: %d activation tile(s) x %d weight rows, "
                 "%d-column stages x %d, %zu B shared, %d + %d split CTAs\n",
                 h->rows, h->cols, batch, dense ? " (two-pass, decoded W_hat)" : "", mt, bn, bk,
                 L.stages, L.total, G.n_big, G.n_small);
  cudaError_t e;
  const int kfmt = dense ? kFmtDense : h->fmt;
  const void* kfn = gemm_kernel_ptr(kfmt, mt, bk, bn);
  {
    // the attribute belongs to the kernel on the current device: once per
    // (device, kernel)
    static std::mutex mu;
    static bool done[64][16][3][2][2] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (h->device < 0 || h->device >= 64) return set_error(SPHQ_ERR_DEVICE, "device index out of range");
    bool& d = done[h->device][kfmt][mt][bk == 64][bn == 256];
    if (!d) {
      e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(gemm)");
      d = true;
    }
  }
  // activations: a batch x cols fp16 tensor, boxes of 128 rows x BK columns
  // (one per activation tile)
  CUtensorMap tmap;
  const cuuint64_t gdim[2] = {(cuuint64_t)h->cols, (cuuint64_t)batch};
  const cuuint64_t gstride[1] = {(cuuint64_t)h->cols * 2};
  const cuuint32_t box[2] = {(cuuint32_t)bk, (cuuint32_t)kGemmBM};
  const cuuint32_t estride[2] = {1, 1};
  CUresult cr = enc(&tmap, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(x), gdim, gstride,
                    box, estride, CU_TENSOR_MAP_INTERLEAVE_NONE,
                    bk == 64 ? CU_TENSOR_MAP_SWIZZLE_128B : CU_TENSOR_MAP_SWIZZLE_64B,
                    CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
  if (cr != CUDA_SUCCESS)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm: cuTensorMapEncodeTiled rejected x");
  // decoded weights (two-pass form): rows x cols fp16, boxes of BN rows x 64
  // columns in the 128-byte swizzle, the layout the decode warps write
  CUtensorMap tmap_w = tmap;
  if (dense) {
    const cuuint64_t wdim[2] = {(cuuint64_t)h->cols, (cuuint64_t)h->rows};
    const cuuint64_t wstride[1] = {(cuuint64_t)h->cols * 2};
    const cuuint32_t wbox[2] = {(cuuint32_t)bk, (cuuint32_t)bn};
    cr = enc(&tmap_w, CU_TENSOR_MAP_DATA_TYPE_FLOAT16, 2, const_cast<void*>(w_hat), wdim, wstride,
             wbox, estride, CU_TENSOR_MAP_INTERLEAVE_NONE, CU_TENSOR_MAP_SWIZZLE_128B,
             CU_TENSOR_MAP_L2_PROMOTION_L2_256B, CU_TENSOR_MAP_FLOAT_OOB_FILL_NONE);
    if (cr != CUDA_SUCCESS)
      return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: cuTensorMapEncodeTiled rejected the workspace");
  }
  GemmArgs a;
  a.units = dense ? nullptr : (const uint8_t*)h->units;
  a.cbimage = dense ? nullptr : (const uint8_t*)(fmt_small(h->fmt) ? h->cbimage : h->codebook);
  a.y = (uint16_t*)y;
  a.flag = h->flag + 1;
  a.rows = h->rows;
  a.cols = h->cols;
  a.nrt = h->nrt;
  a.batch = batch;
  a.nwt = G.nwt;
  a.n_big = G.n_big;
  a.ksplit = ksplit;
  a.part = part;
  a.tickets = tickets;
  a.stages = L.stages;
  a.cb_bytes = L.cb_bytes;
  a.off_b = L.off_b;
  a.off_cb = L.off_cb;
  a.off_bar = L.off_bar;
  const dim3 grid((unsigned)((G.n_big + G.n_small) * ksplit));
  void* args[] = {&a, &tmap, &tmap_w};
  e = cudaLaunchKernel(kfn, grid, dim3(gemm_threads(bn)), args, L.total, s);
  if (e != cudaSuccess) return cuda_error(e, "gemm launch");
  return SPHQ_OK;
}

sphq_status launch_gemm(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s) {
  return launch_gemm_kernel(h, x, y, batch, s, nullptr);
}

static const void* decode_units_ptr(int fmt) {
  switch (fmt) {
#define SPHQ_DECODE_UNITS_PTR(F) \
  case F:                        \
    return (const void*)&decode_units_kernel<F>;
    SPHQ_DECODE_UNITS_PTR(2)
    SPHQ_DECODE_UNITS_PTR(3)
    SPHQ_DECODE_UNITS_PTR(4)
    SPHQ_DECODE_UNITS_PTR(5)
    SPHQ_DECODE_UNITS_PTR(6)
    SPHQ_DECODE_UNITS_PTR(7)
    SPHQ_DECODE_UNITS_PTR(8)
    SPHQ_DECODE_UNITS_PTR(9)
#undef SPHQ_DECODE_UNITS_PTR
    default:
      return nullptr;
  }
}

// Estimated times (us) of the two forms on this GB300: the fused kernel at its
// measured rate per format family at large shapes (small codebooks ~1.3
// PFLOP/s, the 8192-entry tables ~0.8, bound by their shared-memory
// codebook gathers), the two-pass form as the decode pass (bytes written and
// read at ~5 TB/s) plus the dense product at ~1.45 PFLOP/s.
static void gemm_form_times(const sphq_handle_s* h, int batch, double* fused, double* two_pass) {
  const double flops = 2.0 * batch * (double)h->rows * h->cols;
  const double fused_rate = fmt_small(h->fmt) ? 1.30e15 : 0.80e15;
  *fused = flops / fused_rate * 1e6;
  const double wbytes = 2.0 * (double)h->rows * h->cols + (double)h->unit_bytes * h->nrt * h->ng;
  *two_pass = wbytes / 5.0e12 * 1e6 + flops / 1.45e15 * 1e6;
}

// Batches of 9..64 rows: whether ceil(batch / 16) GEMV launches (each
// streaming the weights once with every SM busy) are estimated faster than
// the tensor-core kernel, whose CTAs each run the whole K and number only
// rows / BN per 128 activation rows.  Per-CTA time of that kernel measured on
// this GB300: ~5.2e-5 us per (column x weight row) for the small codebooks,
// ~7.3e-5 for the 8192-entry tables; a GEMV of up to 16 rows ~2 us plus its
// bytes at 25% of the HBM rate.
bool gemm_prefers_gemv(sphq_handle h, int batch) {
  if (batch <= 8 || batch > 64) return false;
  int optin = 0;
  if (device_smem_optin(h, &optin) != SPHQ_OK) return false;
  const GemmShape g = select_gemm_shape(h, batch, optin);
  if (!g.mt) return true;
  const int sms = h->sm_count > 0 ? h->sm_count : 1;
  const long long ctas = (long long)((h->nrt + g.bn / kRowsPerTile - 1) / (g.bn / kRowsPerTile)) *
                         ((batch + kGemmBM * g.mt - 1) / (kGemmBM * g.mt));
  const double waves = (double)((ctas + sms - 1) / sms);
  const double per_cta = (double)h->cols * g.bn * g.mt * (fmt_small(h->fmt) ? 5.2e-5 : 7.3e-5);
  const double bytes8 = (double)h->unit_bytes * h->nrt * h->ng + 32.0 * (h->rows + h->cols);
  const double t_gemv = (double)((batch + SPHQ_MAX_BATCH - 1) / SPHQ_MAX_BATCH) *
                        (2.0 + bytes8 / (0.25 * 6794e9) * 1e6);
  return t_gemv < waves * per_cta;
}

// Split-K form of the fused kernel for mid-size batches: with the shape
// automatic and fewer output tiles than half the SMs, each tile's columns
// (whole radius groups) are shared by ksplit CTAs, as many as fill the SMs
// in one wave with at least two groups each, and their fp32 partials are
// summed in share order by the tile's last CTA.  Workspace: the partial
// tiles, then one counter per tile.
static SplitK gemm_splitk_plan(const sphq_handle_s* h, int batch) {
  SplitK r;
  if (h->gemm_mt || h->gemm_bn || h->dim != 8 || batch < kSplitMinBatch || batch > kSplitMaxBatch)
    return r;
  int optin = 0;
  if (cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device) !=
      cudaSuccess) {
    (void)cudaGetLastError();
    return r;
  }
  const GemmShape g = select_gemm_shape(h, batch, optin);
  if (!g.mt) return r;
  const GemmGrid G = gemm_grid(h, batch, g.mt, g.bn, false);
  const long long sms = h->sm_count > 0 ? h->sm_count : 1;
  const long long tiles = G.n_big;
  if (G.n_small || 2 * tiles > sms) return r;
  // at least kSplitMinGroups radius groups per CTA: below that the shares'
  // partial tiles cost more to write and sum than their columns save
  // (measured: 3584^2 in 5 shares of 5-6 groups 28-31 us against 16-33 for
  // the unsplit kernel or GEMV launches; 8192^2 in 2 shares of 32 groups 45
  // against 62-65 at batch 48-128)
  const int ks = (int)std::min<long long>(std::min<long long>(sms / tiles, h->ng / kSplitMinGroups), 64);
  if (ks < 2) return r;
  r.ksplit = ks;
  r.tiles = tiles;
  r.part_bytes = align_to((size_t)tiles * ks * kGemmBM * g.mt * g.bn * sizeof(float), 256);
  r.bytes = r.part_bytes + align_to((size_t)tiles * sizeof(unsigned), 256);
  return r;
}

sphq_status gemm_workspace_bytes(sphq_handle h, int batch, size_t* bytes) {
  const SplitK sk = gemm_splitk_plan(h, batch);
  if (sk.ksplit > 1) {
    *bytes = sk.bytes;
    return SPHQ_OK;
  }
  double tf = 0, tt = 0;
  gemm_form_times(h, batch, &tf, &tt);
  *bytes = tt < tf ? (size_t)h->rows * h->cols * 2 : 0;
  return SPHQ_OK;
}

// sphq_gemm_ws with a workspace: the split-K form where it applies and the
// workspace holds its partials, else the two-pass form (validated x, y, batch).
sphq_status launch_gemm_ws(sphq_handle h, const void* x, void* y, int batch, void* ws,
                           size_t ws_bytes, cudaStream_t s) {
  const SplitK sk = gemm_splitk_plan(h, batch);
  if (sk.ksplit > 1 && ws_bytes >= sk.bytes) {
    if (reinterpret_cast<uintptr_t>(ws) % 16)
      return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: workspace must be 16-byte aligned");
    float* part = static_cast<float*>(ws);
    unsigned* tickets = reinterpret_cast<unsigned*>(static_cast<uint8_t*>(ws) + sk.part_bytes);
    cudaError_t e = cudaMemsetAsync(tickets, 0, (size_t)sk.tiles * sizeof(unsigned), s);
    if (e != cudaSuccess) return cuda_error(e, "sphq_gemm_ws: clear split-K counters");
    return launch_gemm_kernel(h, x, y, batch, s, nullptr, sk.ksplit, part, tickets);
  }
  return launch_gemm_two_pass(h, x, y, batch, ws, ws_bytes, s);
}

sphq_status launch_gemm_two_pass(sphq_handle h, const void* x, void* y, int batch, void* ws,
                                 size_t ws_bytes, cudaStream_t s) {
  const size_t need = (size_t)h->rows * h->cols * 2;
  if (ws_bytes < need)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: workspace smaller than rows x cols x 2 bytes");
  if (reinterpret_cast<uintptr_t>(ws) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: workspace must be 16-byte aligned");
  const void* kfn = decode_units_ptr(h->fmt);
  if (!kfn) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm_ws: unknown format");
  const uint32_t cb_bytes = fmt_small(h->fmt) ? (uint32_t)h->K * 8u * 16u : (uint32_t)h->K * 16u;
  cudaError_t e;
  const int threads = kDecodeUnitsWarps * 32;
  int per_sm = 0;
  {
    // the kernel's shared-memory attribute and its resident count, once per
    // (device, format), so that later calls (and stream captures) only launch
    static std::mutex mu;
    static int resident[64][16] = {};
    std::lock_guard<std::mutex> lock(mu);
    if (h->device < 0 || h->device >= 64) return set_error(SPHQ_ERR_DEVICE, "device index out of range");
    if (!resident[h->device][h->fmt]) {
      e = cudaFuncSetAttribute(kfn, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)cb_bytes);
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute(decode_units)");
      int n = 0;
      e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&n, kfn, threads, cb_bytes);
      if (e != cudaSuccess) return cuda_error(e, "decode_units occupancy");
      if (n < 1) return set_error(SPHQ_ERR_CUDA, "decode_units: no resident block");
      resident[h->device][h->fmt] = n;
    }
    per_sm = resident[h->device][h->fmt];
  }
  const long long units = (long long)h->nrt * h->ng;
  const long long want = (units + kDecodeUnitsWarps - 1) / kDecodeUnitsWarps;
  const int grid = (int)std::min<long long>(want, (long long)h->sm_count * per_sm);
  const uint8_t* cb = (const uint8_t*)(fmt_small(h->fmt) ? h->cbimage : h->codebook);
  const uint8_t* un = (const uint8_t*)h->units;
  uint16_t* w = (uint16_t*)ws;
  int rows = h->rows, cols = h->cols, nrt = h->nrt, ng = h->ng;
  int* flag = h->flag + 1;
  void* args[] = {&un, &cb, const_cast<uint32_t*>(&cb_bytes), &w, &rows, &cols, &nrt, &ng, &flag};
  e = cudaLaunchKernel(kfn, dim3(grid), dim3(threads), args, cb_bytes, s);
  if (e != cudaSuccess) return cuda_error(e, "decode_units launch");
  return launch_gemm_kernel(h, x, y, batch, s, ws);
}

}  // namespace sphq
