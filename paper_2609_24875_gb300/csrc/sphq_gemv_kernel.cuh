// Fused spherical dequantize-GEMV kernel for decode (SPHQuant §3.4, App. D), sm_103a.
//
// y[n][r] = sum_j w_hat[r][j] x[n][j] for a batch of n <= 16 activation rows.
//
// Decode stays on the CUDA cores: each thread rebuilds whole 8-D blocks in
// registers (codebook entry from shared memory, coordinate signs, radius of
// Eq. (7)) and never writes them to memory.  The multiply-accumulate with the
// activations runs on the tensor cores as m16n8k16 MMAs with fp32
// accumulation; the thread/fragment mapping of the unit layout
// (sphq_layout.cuh) puts the two blocks a thread decodes from word w_m
// directly into the A fragment -- coordinates 0-3 feed one MMA and 4-7 the
// next -- and the matching activations go in the B fragment.  Products of two
// fp16 values are exact in fp32.
//
// Two ways of applying the radius, chosen by batch size:
//  * batch 1-2 ("factored"; the planner takes it for batch 1, and for batch
//    2 on small-codebook matrices of more than 16384 units): the A fragment
//    holds the signed unit direction
//    s (.) c_z and the B fragment is block diagonal -- column 2c + b carries
//    batch row b of slot c only -- so every MMA pair returns, in the lane
//    that decoded them, the per-vector dots d = (s (.) c_z) . x_b.  The lane
//    then adds r_hat * d with one fp32 FMA (r_hat from the fp16 FMA of
//    Eq. (7)).  This skips the four half-rate fp16 products per block; the
//    result differs from the exact W_hat x by at most one fp16 rounding of
//    each product r_hat * c (2^-11 relative), inside the stated tolerance.
//  * batch 3-8 ("full"): the lane forms w_hat = RN16(r_hat * (s (.) c_z))
//    exactly as Eq. (4) defines it and the MMA's N dimension is the batch;
//    batch 9-16 feeds each such block to a second pair of MMAs for batch
//    rows 8-15.
//
// Work decomposition.  The row tiles (16 rows) are dealt to thread-block
// clusters in contiguous, near-equal ranges; every CTA of a cluster takes the
// same tiles and its own contiguous share of the radius groups (split-K
// inside the cluster).  Inside a CTA the tiles are cut into strips (of two
// tiles for the small-codebook formats, four for W3): a work item is (strip,
// group), i.e. the units of one group below each other, so the activations of
// a group are loaded once for all of them.  The
// items are dealt to the warps in contiguous ranges.  Sums are reduced on
// chip only and in a fixed order, so results do not depend on scheduling:
// when a warp leaves a strip it sends its quad-reduced sums of each of the
// strip's tiles to the tile's owner CTA (tile index mod cluster size) with
// st.async into the owner's shared memory, completing on the owner's
// mbarrier; the owner adds the blocks of all covering warps in (rank, warp)
// order and writes fp16 y.
//
// Staging.  The codebook image (W2 and the other small-codebook splits: eight
// interleaved copies, K x 128 B; W3: the 128 KiB table) and, for batch 1-2, the
// CTA's slice of the activations are
// copied into shared memory by bulk asynchronous copies completing on
// mbarriers.  Codes stream from HBM through registers (16-byte loads that
// bypass L1) one work item ahead of use, and a bulk L2 prefetch runs two
// items further ahead (an item's units are contiguous in memory).
//
// Programmatic dependent launch: the kernel lets the next kernel on the
// stream launch at once, prefetches its codes, issues its first unit loads
// and the codebook copy, and only then waits (griddepcontrol.wait) for the
// previous kernel -- before it touches activations or outputs.  Codes and
// codebook are immutable after sphq_pack, so this overlap is safe.
//
// Every wait on an mbarrier gives up after about two seconds, records an
// error bit in the handle's device flag word and carries on, so a fault in
// the exchange cannot hang the GPU.  On that failure path an owner CTA that
// gave up may exit while a peer's st.async into its shared memory is still in
// flight; a remote store to an exited CTA is undefined, so after a reported
// timeout the results are void and the context should be treated as suspect
// (the path is never taken when every covering warp sends, which the byte
// count of the receive barrier guarantees in a correct launch).  A cluster
// barrier before exit would close the gap but cannot be bounded in time.
//
// This header holds the device code; sphq_gemv.cu instantiates it for the W2
// and W3 formats and holds the launch plans, sphq_gemv_splits.cu instantiates
// the Tab. 4 splits.
#pragma once
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "sphq_internal.h"
#include "sphq_layout.cuh"

namespace sphq {

// Row tiles per work item (the units that share one load of a group's
// activations) is the kernel's template parameter S: 2, or 4 for the W3
// formats, whose 8 warps per SM have the registers for four units in flight
// (the launch plan takes 4 when a cluster holds at least three row tiles).
__host__ __device__ constexpr bool fmt_has_strip4(int fmt) { return fmt == 3 || fmt == 4; }

// Radius application modes.
constexpr int kFactored1 = 1;  // batch 1
constexpr int kFactored2 = 2;  // batch 2
constexpr int kFull = 8;       // batch 3..8
constexpr int kFull16 = 16;    // batch 9..16: two batch halves of 8 rows per decoded block
// Modes that form w_hat exactly and put the batch in the MMA's N dimension.
__host__ __device__ constexpr bool mode_full(int m) { return m == kFull || m == kFull16; }

struct GemvArgs {
  const uint8_t* units;
  const uint8_t* cbimage;  // codebook image as laid out in shared memory
  const uint16_t* x;
  uint16_t* y;
  int* flag;               // device error word: bit 1 = an mbarrier wait gave up
  int rows, cols, ng, nrt;
  int batch;
  int nclusters;           // clusters holding tiles (grid = nclusters x cluster size)
  uint32_t cb_bytes;       // codebook image bytes
  uint32_t x_pitch;        // bytes between staged activation rows (factored modes)
  uint32_t off_x, off_zero, off_recv, off_bar;  // dynamic smem offsets
  const uint16_t* zeros;   // 256 B of zeros in global memory (batch 3-8 non-suppliers)
  // Work split, precomputed on the host so that the prologue has no runtime
  // division: cluster c holds tiles [c*tq + min(c, tr), +tq + (c < tr));
  // rank r of a cluster holds groups [r*gq + min(r, gr), +gq + (r < gr));
  // clusters have 2^cshift CTAs; ngc_m[k] = ceil(2^32 / (gq + k)) divides
  // item indices by the group count.
  int tq, tr, gq, gr, cshift;
  unsigned long long ngc_m[2];
};

// ---------------------------------------------------------------------------
// PTX wrappers
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t smem_u32(const void* p) {
  return static_cast<uint32_t>(__cvta_generic_to_shared(p));
}
__device__ __forceinline__ void mbar_init(uint32_t bar, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(bar), "r"(count) : "memory");
}
// Makes mbarrier initialisation visible to the async proxy and the cluster.
__device__ __forceinline__ void fence_mbar_init() {
  asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
}
__device__ __forceinline__ void mbar_arrive_expect_tx(uint32_t bar, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(bar), "r"(bytes)
               : "memory");
}
// Tests phase `parity` of a local mbarrier; while it is incomplete the thread
// may sleep up to ~20 us (it wakes as soon as the phase completes), so a
// waiting warp does not spin on the issue slots.
__device__ __forceinline__ bool mbar_try_wait(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2, %3;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity), "r"(20000u)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}
// Waits for phase `parity` of a local mbarrier; gives up after ~2 s.
__device__ __forceinline__ bool mbar_wait(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (;;) {
    if (mbar_try_wait(bar, parity)) return true;
    if (globaltimer() - t0 > 2000000000ull) return false;
  }
}
// The same wait without the suspend hint: the thread polls, so it resumes as
// soon as the phase completes (the GEMV's few one-off waits sit on its
// critical path).  Gives up after ~2 s.
__device__ __forceinline__ bool mbar_try_wait_poll(uint32_t bar, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(bar), "r"(parity)
      : "memory");
  return ok != 0;
}
__device__ __forceinline__ bool mbar_wait_poll(uint32_t bar, uint32_t parity) {
  if (mbar_try_wait_poll(bar, parity)) return true;
  const uint64_t t0 = globaltimer();
  for (;;) {
    if (mbar_try_wait_poll(bar, parity)) return true;
    if (globaltimer() - t0 > 2000000000ull) return false;
  }
}
// Bulk copy global -> own shared memory, completing on a local mbarrier.
// dst, src and bytes must be multiples of 16.
__device__ __forceinline__ void bulk_g2s(uint32_t dst, const void* src, uint32_t bytes,
                                         uint32_t bar) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          dst),
      "l"(src), "r"(bytes), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}
__device__ __forceinline__ uint32_t cluster_rank() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%cluster_ctarank;" : "=r"(r));
  return r;
}
__device__ __forceinline__ uint32_t cluster_id() {
  uint32_t r;
  asm volatile("mov.u32 %0, %%clusterid.x;" : "=r"(r));
  return r;
}
// Relaxed arrive: it orders nothing (the mbarrier initialisation is published
// by fence.mbarrier_init), so it does not wait for this thread's loads in flight.
__device__ __forceinline__ void cluster_arrive_relaxed() {
  asm volatile("barrier.cluster.arrive.relaxed.aligned;" ::: "memory");
}
__device__ __forceinline__ void cluster_wait() {
  asm volatile("barrier.cluster.wait.acquire.aligned;" ::: "memory");
}
// Address of the same shared-memory location in cluster CTA `rank`.
__device__ __forceinline__ uint32_t mapa(uint32_t addr, uint32_t rank) {
  uint32_t d;
  asm volatile("mapa.shared::cluster.u32 %0, %1, %2;" : "=r"(d) : "r"(addr), "r"(rank));
  return d;
}
// 16-byte store into another CTA's shared memory, completing on its mbarrier.
__device__ __forceinline__ void st_async16(uint32_t raddr, float4 v, uint32_t rbar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.v4.f32 [%0], {%1, %2, %3, %4}, "
      "[%5];" ::"r"(raddr),
      "f"(v.x), "f"(v.y), "f"(v.z), "f"(v.w), "r"(rbar)
      : "memory");
}
__device__ __forceinline__ void st_async4(uint32_t raddr, float v, uint32_t rbar) {
  asm volatile(
      "st.async.shared::cluster.mbarrier::complete_tx::bytes.b32 [%0], %1, [%2];" ::"r"(raddr),
      "r"(__float_as_uint(v)), "r"(rbar)
      : "memory");
}
__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

// The MMAs are pure register computations (no volatile), so the compiler may
// interleave the words of a unit freely.
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}
// D = A B (C = 0)
__device__ __forceinline__ void mma16816_zero(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
  const float z = 0.f;
  asm("mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(z));
}

// Activations of batch 3-8 are re-read by every strip: keep them in L1.
__device__ __forceinline__ uint4 ldg_x16(const uint16_t* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::evict_last.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w)
               : "l"(p));
  return v;
}

__device__ __forceinline__ float h_lo_to_f32(uint32_t h2) {
  float f;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tcvt.f32.f16 %0, lo;\n\t}"
      : "=f"(f)
      : "r"(h2));
  return f;
}
__device__ __forceinline__ float h_hi_to_f32(uint32_t h2) {
  float f;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tcvt.f32.f16 %0, hi;\n\t}"
      : "=f"(f)
      : "r"(h2));
  return f;
}

// ---------------------------------------------------------------------------
// Decode + multiply of one unit
// ---------------------------------------------------------------------------

template <int BITS>
struct UnitConst {
  uint32_t d2, m2, e;
};

template <int BITS>
__device__ __forceinline__ UnitConst<BITS> unit_const(const Unit<BITS>& u, int q) {
  UnitConst<BITS> c;
  if constexpr (fmt_small(BITS)) {
    c.d2 = params_delta(u.par.x, u.par.y);
    c.m2 = params_rmin(u.par.x, u.par.y);
    c.e = sign_extra<BITS>(u, q);
  } else {
    c.d2 = params_delta(u.par.x, u.par.y);
    c.m2 = params_rmin(u.par.x, u.par.y);
    c.e = 0;
  }
  return c;
}

template <int BITS>
__device__ __forceinline__ void word_directions(const Unit<BITS>& u, const UnitConst<BITS>& k,
                                                int m, int q, const SmemCodebook& cb, uint4& sa,
                                                uint4& sb, uint32_t& qp) {
  if constexpr (fmt_small(BITS)) {
    const uint32_t W = word_of(u.w, m);
    directions_small<BITS>(W, k.e, m, cb, cb.copyoff, true, sa, sb);
    qp = W;
  } else if constexpr (BITS == kFmtW3V3) {
    directions_w3v3(u, m, cb, sa, sb);
    qp = qpair_w3v3(u, m);
  } else {
    directions_w3(u, m, q, cb, sa, sb);
    qp = qpair_w3(u, m);
  }
}

// Accumulators of one warp for one row tile.
template <int MODE>
struct Acc {
  static constexpr int NB = mode_full(MODE) ? 1 : MODE;
  float f[NB][2];  // factored: [batch row][row gid / gid+8]
  float d[4];      // full: MMA accumulator fragment (batch rows 0-7)
  float e[MODE == kFull16 ? 4 : 1];  // batch rows 8-15 (kFull16)
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int i = 0; i < NB; ++i) f[i][0] = f[i][1] = 0.f;
#pragma unroll
    for (int i = 0; i < 4; ++i) d[i] = 0.f;
    if constexpr (MODE == kFull16) {
#pragma unroll
      for (int i = 0; i < 4; ++i) e[i] = 0.f;
    }
  }
};

// The lane's B-fragment data of one group: 8-D, v[m] = its activation row
// at slot 4m+q (16 bytes), v2[m] the same for the second batch half (kFull16);
// 4-D, v[s] = at vector 4s+q (8 bytes); or zeros.
template <int BITS> struct XFrag { uint4 v[4]; uint4 v2[4]; };
template <> struct XFrag<kFmt4D> { uint2 v[8]; };

// 8-byte activation load kept in L1 (batch 3-8, 4-D vectors)
__device__ __forceinline__ uint2 ldg_x8(const uint8_t* p) {
  uint2 v;
  asm volatile("ld.global.nc.L1::evict_last.v2.u32 {%0,%1}, [%2];" : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}

// xp: this lane's first activation bytes of the group (8-D: slot q at 16 q,
// words 64 bytes apart; 4-D: vector q at 8 q, pairs 32 bytes apart); x2off:
// bytes from its row to its second-half row (kFull16).
template <int BITS, int MODE>
__device__ __forceinline__ void load_x(XFrag<BITS>& xv, const uint8_t* xp, int x2off = 0) {
  if constexpr (BITS == kFmt4D) {
#pragma unroll
    for (int s = 0; s < 8; ++s) {
      if constexpr (MODE == kFull)
        xv.v[s] = ldg_x8(xp + 32 * s);
      else
        xv.v[s] = *reinterpret_cast<const uint2*>(xp + 32 * s);
    }
  } else {
#pragma unroll
    for (int m = 0; m < 4; ++m) {
      if constexpr (mode_full(MODE))
        xv.v[m] = ldg_x16(reinterpret_cast<const uint16_t*>(xp) + 32 * m);
      else
        xv.v[m] = *reinterpret_cast<const uint4*>(xp + 64 * m);
      if constexpr (MODE == kFull16)
        xv.v2[m] = ldg_x16(reinterpret_cast<const uint16_t*>(xp + x2off) + 32 * m);
    }
  }
  (void)x2off;
}

// One pair s of a 4-D unit: one MMA for the two 4-D vectors of the lane.
template <int MODE, int S>
__device__ __forceinline__ void process_pair_4d(const Unit<kFmt4D>& cur,
                                                const UnitConst<kFmt4D>& kc,
                                                const XFrag<kFmt4D>& xv, const SmemCodebook& cb,
                                                Acc<MODE>& acc) {
  static_assert(MODE != kFull16, "4-D vectors take batches of at most 8 rows per launch");
  uint2 sa, sb;
  directions_4d<S>(cur.w, cur.s1, cb, cb.copyoff, true, sa, sb);
  const uint32_t r = radius_pair<4>(qpair_4d<S>(cur.w), kc.d2, kc.m2);
  if constexpr (MODE == kFull) {
    const uint32_t ra = bcast_lo(r), rb = bcast_hi(r);
    mma16816(acc.d, hmul2_rn(ra, sa.x), hmul2_rn(rb, sb.x), hmul2_rn(ra, sa.y),
             hmul2_rn(rb, sb.y), xv.v[S].x, xv.v[S].y);
  } else {
    float d[4];
    mma16816_zero(d, sa.x, sb.x, sa.y, sb.y, xv.v[S].x, xv.v[S].y);
    const float rA = h_lo_to_f32(r), rB = h_hi_to_f32(r);
    acc.f[0][0] = __fmaf_rn(rA, d[0], acc.f[0][0]);
    acc.f[0][1] = __fmaf_rn(rB, d[2], acc.f[0][1]);
    if constexpr (MODE == kFactored2) {
      acc.f[1][0] = __fmaf_rn(rA, d[1], acc.f[1][0]);
      acc.f[1][1] = __fmaf_rn(rB, d[3], acc.f[1][1]);
    }
  }
}

// Word m of one unit (the two vectors of slot 4m+q of rows gid and gid+8)
// against the activations xm of that slot (8-D formats); xm2: the second
// batch half's (kFull16).
template <int BITS, int MODE>
__device__ __forceinline__ void process_word(const Unit<BITS>& cur, const UnitConst<BITS>& kc,
                                             const uint4& xm, int m, int q,
                                             const SmemCodebook& cb, Acc<MODE>& acc,
                                             const uint4& xm2 = uint4{}) {
  uint4 sa, sb;
  uint32_t qp;
  word_directions<BITS>(cur, kc, m, q, cb, sa, sb, qp);
  const uint32_t r = radius_pair<fmt_radius_bits(BITS)>(qp, kc.d2, kc.m2);
  if constexpr (mode_full(MODE)) {
    const uint4 wa = scale_block(sa, bcast_lo(r));
    const uint4 wb = scale_block(sb, bcast_hi(r));
    mma16816(acc.d, wa.x, wb.x, wa.y, wb.y, xm.x, xm.y);
    mma16816(acc.d, wa.z, wb.z, wa.w, wb.w, xm.z, xm.w);
    if constexpr (MODE == kFull16) {
      mma16816(acc.e, wa.x, wb.x, wa.y, wb.y, xm2.x, xm2.y);
      mma16816(acc.e, wa.z, wb.z, wa.w, wb.w, xm2.z, xm2.w);
    }
  } else {
    float d[4];
    mma16816_zero(d, sa.x, sb.x, sa.y, sb.y, xm.x, xm.y);
    mma16816(d, sa.z, sb.z, sa.w, sb.w, xm.z, xm.w);
    const float rA = h_lo_to_f32(r), rB = h_hi_to_f32(r);
    acc.f[0][0] = __fmaf_rn(rA, d[0], acc.f[0][0]);
    acc.f[0][1] = __fmaf_rn(rB, d[2], acc.f[0][1]);
    if constexpr (MODE == kFactored2) {
      acc.f[1][0] = __fmaf_rn(rA, d[1], acc.f[1][0]);
      acc.f[1][1] = __fmaf_rn(rB, d[3], acc.f[1][1]);
    }
  }
}

// The activations of word m of a group for this lane (8-D formats).
template <int MODE>
__device__ __forceinline__ uint4 load_x_word(const uint8_t* xp, int m) {
  if constexpr (mode_full(MODE))
    return ldg_x16(reinterpret_cast<const uint16_t*>(xp) + 32 * m);
  else
    return *reinterpret_cast<const uint4*>(xp + 64 * m);
}

// One unit (16 rows x 128 columns).
template <int BITS, int MODE>
__device__ __forceinline__ void process_unit(const Unit<BITS>& cur, const XFrag<BITS>& xf, int q,
                                             const SmemCodebook& cb, Acc<MODE>& acc) {
  const UnitConst<BITS> kc = unit_const<BITS>(cur, q);
  if constexpr (BITS == kFmt4D) {
    process_pair_4d<MODE, 0>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 1>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 2>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 3>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 4>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 5>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 6>(cur, kc, xf, cb, acc);
    process_pair_4d<MODE, 7>(cur, kc, xf, cb, acc);
    return;
  } else {
  const auto& xv = xf.v;
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    uint4 sa, sb;
    uint32_t qp;
    word_directions<BITS>(cur, kc, m, q, cb, sa, sb, qp);
    const uint32_t r = radius_pair<fmt_radius_bits(BITS)>(qp, kc.d2, kc.m2);
    if constexpr (mode_full(MODE)) {
      const uint4 wa = scale_block(sa, bcast_lo(r));
      const uint4 wb = scale_block(sb, bcast_hi(r));
      mma16816(acc.d, wa.x, wb.x, wa.y, wb.y, xv[m].x, xv[m].y);
      mma16816(acc.d, wa.z, wb.z, wa.w, wb.w, xv[m].z, xv[m].w);
      if constexpr (MODE == kFull16) {
        mma16816(acc.e, wa.x, wb.x, wa.y, wb.y, xf.v2[m].x, xf.v2[m].y);
        mma16816(acc.e, wa.z, wb.z, wa.w, wb.w, xf.v2[m].z, xf.v2[m].w);
      }
    } else {
      float d[4];
      mma16816_zero(d, sa.x, sb.x, sa.y, sb.y, xv[m].x, xv[m].y);
      mma16816(d, sa.z, sb.z, sa.w, sb.w, xv[m].z, xv[m].w);
      const float rA = h_lo_to_f32(r), rB = h_hi_to_f32(r);
      acc.f[0][0] = __fmaf_rn(rA, d[0], acc.f[0][0]);
      acc.f[0][1] = __fmaf_rn(rB, d[2], acc.f[0][1]);
      if constexpr (MODE == kFactored2) {
        acc.f[1][0] = __fmaf_rn(rA, d[1], acc.f[1][0]);
        acc.f[1][1] = __fmaf_rn(rB, d[3], acc.f[1][1]);
      }
    }
  }
  }
}

// Sends a warp's accumulators of one row tile to the tile's owner CTA:
// 4-byte st.async stores into the owner's receive slot ([batch row][row]),
// completing on the owner's receive mbarrier (raddr / rbar are addresses in
// the owner's shared memory).
template <int MODE>
__device__ __forceinline__ void send_partial(uint32_t raddr, uint32_t rbar, Acc<MODE>& acc,
                                             int lane, int batch) {
  const int gid = lane >> 2, q = lane & 3;
  if constexpr (mode_full(MODE)) {
    // d[0..3] = D[gid][2q], D[gid][2q+1], D[gid+8][2q], D[gid+8][2q+1]
    if (2 * q < batch) {
      st_async4(raddr + 4u * ((2 * q) * kRowsPerTile + gid), acc.d[0], rbar);
      st_async4(raddr + 4u * ((2 * q) * kRowsPerTile + gid + 8), acc.d[2], rbar);
    }
    if (2 * q + 1 < batch) {
      st_async4(raddr + 4u * ((2 * q + 1) * kRowsPerTile + gid), acc.d[1], rbar);
      st_async4(raddr + 4u * ((2 * q + 1) * kRowsPerTile + gid + 8), acc.d[3], rbar);
    }
    if constexpr (MODE == kFull16) {  // e: batch rows 8 + 2q, 8 + 2q + 1
      if (8 + 2 * q < batch) {
        st_async4(raddr + 4u * ((8 + 2 * q) * kRowsPerTile + gid), acc.e[0], rbar);
        st_async4(raddr + 4u * ((8 + 2 * q) * kRowsPerTile + gid + 8), acc.e[2], rbar);
      }
      if (9 + 2 * q < batch) {
        st_async4(raddr + 4u * ((9 + 2 * q) * kRowsPerTile + gid), acc.e[1], rbar);
        st_async4(raddr + 4u * ((9 + 2 * q) * kRowsPerTile + gid + 8), acc.e[3], rbar);
      }
    }
  } else {
    // sum the lane's slots, then the quad's four lanes (slots q = 0..3)
#pragma unroll
    for (int i = 0; i < MODE; ++i) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float t = acc.f[i][h];
        t += __shfl_xor_sync(0xFFFFFFFFu, t, 1);
        t += __shfl_xor_sync(0xFFFFFFFFu, t, 2);
        if (q == 0) st_async4(raddr + 4u * (i * kRowsPerTile + gid + 8 * h), t, rbar);
      }
    }
  }
}

// First item of warp w when the items of a CTA are dealt to WARPS warps in
// contiguous ranges of near-equal unit counts: items are (strip, group) in
// strip-major order, ngc per strip, S units each except in the last strip
// when the tile count T is not a multiple of S (T mod S units).  The unit share of warp w starts
// at unit U*w/WARPS, rounded to an item boundary.
template <int WARPS, int S>
__device__ __forceinline__ int warp_item(int T, int ngc, int w) {
  const int full = (T / S) * ngc;  // items of S units
  const int rest = T - S * (T / S);
  const int units = T * ngc;
  const int u = (int)((unsigned)units * (unsigned)w / (unsigned)WARPS);
  if (u < S * full) return (u + S / 2) / S;
  // the tail strip's items of `rest` (1..S-1) units, without a runtime division
  const unsigned v = (unsigned)(u - S * full + rest / 2);
  return full + (rest == 1 ? (int)v
                 : rest == 2 ? (int)(v >> 1)
                 : rest == 3 ? (int)(((unsigned long long)v * 0xAAAAAAABull) >> 33)
                             : 0);
}

// ---------------------------------------------------------------------------
// The kernel
// ---------------------------------------------------------------------------

// Contiguous near-equal share [lo, hi) of n items for part i of p (32-bit
// arithmetic when n * p fits, which is every practical case).
__device__ __forceinline__ int share_lo(int n, int i, int p) {
  if ((unsigned)n < 65536u && (unsigned)p < 65536u) return (int)((unsigned)n * (unsigned)i / (unsigned)p);
  return (int)(((long long)n * i) / p);
}
// The same for a compile-time number of parts (a shift for powers of two).
template <int P>
__device__ __forceinline__ int share_lo_c(int n, int i) {
  return (int)((unsigned)n * (unsigned)i / (unsigned)P);
}

// One work item: the activations of one group (xp: this lane's 16 bytes of
// word 0; words 1-3 follow at 64-byte steps) and the units of the strip's
// SIZE row tiles below each other (u[j]).  Each unit's register slot is
// refilled with the next item's unit j as soon as it is consumed: unit j of
// the same strip at the next group (base nb), or, for the strip's LAST item,
// the units in nmask of the warp's next strip.
template <int BITS, int MODE, int SIZE, bool LAST, int S>
__device__ __forceinline__ void run_item(Unit<BITS> (&u)[S], Acc<MODE> (&acc)[S],
                                         const uint8_t* xp, const uint8_t* nb, unsigned nmask,
                                         int lane, int q, const SmemCodebook& cb, int x2off) {
  constexpr int UB = Layout<BITS>::kUnitBytes;
  auto reload = [&](int j) {
    if (LAST) {
      if (nmask >> j & 1u) u[j] = load_unit<BITS>(nb + j * UB, lane);
    } else if (j < SIZE) {
      u[j] = load_unit<BITS>(nb + j * UB, lane);
    }
  };
  if constexpr (BITS == kFmt4D || SIZE == 1) {
    XFrag<BITS> xv;
    load_x<BITS, MODE>(xv, xp, x2off);
#pragma unroll
    for (int j = 0; j < S; ++j) {
      if (j < SIZE) process_unit<BITS, MODE>(u[j], xv, q, cb, acc[j]);
      reload(j);
    }
  } else {
    // The units share each word's activations: words 0-1 of every unit
    // first, then words 2-3 unit by unit, each unit's slot refilled as soon
    // as its last word is done; at most two words of activations are live.
    UnitConst<BITS> kc[SIZE];
#pragma unroll
    for (int j = 0; j < SIZE; ++j) kc[j] = unit_const<BITS>(u[j], q);
    const uint4 x0 = load_x_word<MODE>(xp, 0), x1 = load_x_word<MODE>(xp, 1);
    uint4 y0{}, y1{}, y2{}, y3{};  // the second batch half's words (kFull16)
    if constexpr (MODE == kFull16) y0 = load_x_word<MODE>(xp + x2off, 0), y1 = load_x_word<MODE>(xp + x2off, 1);
#pragma unroll
    for (int j = 0; j < SIZE; ++j) process_word<BITS, MODE>(u[j], kc[j], x0, 0, q, cb, acc[j], y0);
#pragma unroll
    for (int j = 0; j < SIZE; ++j) process_word<BITS, MODE>(u[j], kc[j], x1, 1, q, cb, acc[j], y1);
    const uint4 x2 = load_x_word<MODE>(xp, 2), x3 = load_x_word<MODE>(xp, 3);
    if constexpr (MODE == kFull16) y2 = load_x_word<MODE>(xp + x2off, 2), y3 = load_x_word<MODE>(xp + x2off, 3);
#pragma unroll
    for (int j = 0; j < SIZE; ++j) {
      process_word<BITS, MODE>(u[j], kc[j], x2, 2, q, cb, acc[j], y2);
      process_word<BITS, MODE>(u[j], kc[j], x3, 3, q, cb, acc[j], y3);
      reload(j);
    }
    if constexpr (LAST) {
#pragma unroll
      for (int j = SIZE; j < S; ++j) reload(j);
    }
  }
}

// cnt >= 1 items of one strip of SIZE tiles at consecutive groups, starting
// at unit base ub and activations xp; the last item loads the next strip's
// first units (base nb, mask nmask).
template <int BITS, int MODE, int SIZE, int S>
__device__ __forceinline__ void run_segment(Unit<BITS> (&u)[S], Acc<MODE> (&acc)[S],
                                            int cnt, const uint8_t* ub, size_t gstride,
                                            const uint8_t* xp, int xstep, const uint8_t* nb,
                                            unsigned nmask, int lane, int q,
                                            const SmemCodebook& cb, int x2off) {
  constexpr uint32_t kBytes = SIZE * Layout<BITS>::kUnitBytes;
  if constexpr (SIZE == 1) {
    // One-tile strips use the two register slots as a two-item ring (slot
    // c % 2 holds item c), so two units stay in flight.  The strip is the
    // warp's last, so nothing is loaded past it (nmask is 0).
    (void)nb;
    (void)nmask;
    if (cnt > 1) u[1] = load_unit<BITS>(ub + gstride, lane);
    int c = 0;
    for (; c + 1 < cnt; c += 2) {
      // items c+2, c+3 go to registers below; c+4, c+5 toward L2
      if (lane == 0 && c + 4 < cnt) prefetch_l2(ub + 4 * gstride, kBytes);
      if (lane == 0 && c + 5 < cnt) prefetch_l2(ub + 5 * gstride, kBytes);
      XFrag<BITS> xv;
      load_x<BITS, MODE>(xv, xp, x2off);
      process_unit<BITS, MODE>(u[0], xv, q, cb, acc[0]);
      if (c + 2 < cnt) u[0] = load_unit<BITS>(ub + 2 * gstride, lane);
      load_x<BITS, MODE>(xv, xp + xstep, x2off);
      process_unit<BITS, MODE>(u[1], xv, q, cb, acc[0]);
      if (c + 3 < cnt) u[1] = load_unit<BITS>(ub + 3 * gstride, lane);
      ub += 2 * gstride;
      xp += 2 * xstep;
    }
    if (c < cnt) run_item<BITS, MODE, 1, true, S>(u, acc, xp, nb, 0u, lane, q, cb, x2off);
    return;
  }
  if (lane == 0 && cnt > 1) prefetch_l2(ub + gstride, kBytes);
  for (int c = 0; c + 1 < cnt; ++c) {
    if (lane == 0 && c + 2 < cnt) prefetch_l2(ub + 2 * gstride, kBytes);
    run_item<BITS, MODE, SIZE, false, S>(u, acc, xp, ub + gstride, 0u, lane, q, cb, x2off);
    ub += gstride;
    xp += xstep;
  }
  run_item<BITS, MODE, SIZE, true, S>(u, acc, xp, nb, nmask, lane, q, cb, x2off);
}

template <int BITS, int MODE, int WARPS, int MINB, int S>
__global__ void __launch_bounds__(WARPS * 32, MINB) gemv_kernel(const GemvArgs a) {
  extern __shared__ __align__(128) uint8_t smem[];
  pdl_launch_dependents();
  constexpr int NBP = MODE;  // floats per row in a partial block (batch rows of the mode)
  constexpr int kBlk = kRowsPerTile * NBP;                // floats per partial block
  constexpr int UB = Layout<BITS>::kUnitBytes;
  static_assert(S == 2 || S == 4, "strip sizes");
  constexpr unsigned kStripMask = (1u << S) - 1u;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int gid = lane >> 2, q = lane & 3;
  const int cshift = a.cshift, csize = 1 << cshift;
  const int crank = csize > 1 ? (int)cluster_rank() : 0;
  const int cid = csize > 1 ? (int)cluster_id() : (int)blockIdx.x;

  // this cluster's row tiles
  const int t0 = cid * a.tq + min(cid, a.tr);
  const int T = a.tq + (cid < a.tr ? 1 : 0);
  const int nown = crank < T ? (T - crank + csize - 1) >> cshift : 0;  // tiles this CTA owns
  uint64_t* bars = reinterpret_cast<uint64_t*>(smem + a.off_bar);
  const uint32_t bar_cb = smem_u32(&bars[0]), bar_x = smem_u32(&bars[1]),
                 bar_recv = smem_u32(&bars[2]);
  // The codebook copy goes first: it is the longest transfer of the
  // prologue.  Every warp of the cluster sends one block per tile of the
  // cluster (its partial sums, or -0.0, the additive identity, for tiles
  // outside its items), so the receive barrier expects a fixed byte count.
  if (threadIdx.x == 0) {
    mbar_init(bar_cb, 1);
    mbar_init(bar_x, 1);
    mbar_init(bar_recv, 1);
    fence_mbar_init();
    mbar_arrive_expect_tx(bar_cb, a.cb_bytes);
    for (uint32_t o = 0; o < a.cb_bytes; o += 32768u)
      bulk_g2s(smem_u32(smem) + o, a.cbimage + o, min(32768u, a.cb_bytes - o), bar_cb);
    mbar_arrive_expect_tx(bar_recv, (uint32_t)(nown * csize * WARPS) * 64u * (uint32_t)a.batch);
  }

  // this CTA's radius groups and this warp's items
  const int g0 = crank * a.gq + min(crank, a.gr);
  const int ngc = a.gq + (crank < a.gr ? 1 : 0);
  const unsigned long long ngc_m = a.ngc_m[crank < a.gr ? 1 : 0];
  // v / ngc for 0 <= v < T * ngc: a multiply by the rounded-up reciprocal,
  // corrected by one where it overshoots
  auto div_ngc = [&](int v) {
    int d = (int)(((unsigned long long)(unsigned)v * ngc_m) >> 32);
    return d * ngc > v ? d - 1 : d;
  };
  const int nfull = T / S;  // strips with all S tiles
  const int rest = T - S * nfull;
  const unsigned last_mask = (1u << rest) - 1u;
  const int i0 = warp_item<WARPS, S>(T, ngc, warp), i1 = warp_item<WARPS, S>(T, ngc, warp + 1);

  // units (t0 + S s + j, g), j < S, start at strip_base(s, g) + j * UB
  const size_t gstride = (size_t)a.nrt * UB;
  auto strip_base = [&](int s, int g) {
    return a.units + ((size_t)g * a.nrt + t0 + S * s) * UB;
  };
  auto strip_mask = [&](int s) { return s < nfull ? kStripMask : last_mask; };

  // first item's units (codes are immutable: no wait needed)
  Unit<BITS> u[S] = {};
  int s = i0 < i1 ? div_ngc(i0) : 0;
  int g = i0 < i1 ? g0 + (i0 - s * ngc) : g0;
  if (i0 < i1) {
    const unsigned m0 = strip_mask(s);
#pragma unroll
    for (int j = 0; j < S; ++j)
      if (m0 >> j & 1u) u[j] = load_unit<BITS>(strip_base(s, g) + j * UB, lane);
  }

  if (!mode_full(MODE) && threadIdx.x < 16)  // zero block read by lanes that supply no activations
    reinterpret_cast<uint4*>(smem + a.off_zero)[threadIdx.x] = make_uint4(0, 0, 0, 0);
  __syncthreads();                  // mbarrier initialisation visible to the CTA
  if (csize > 1) cluster_arrive_relaxed();  // ... and to the cluster (waited on below)

  pdl_wait();  // the previous kernel's outputs (our activations) are complete
  if (!mode_full(MODE) && threadIdx.x == 0) {
    const uint32_t row_bytes = (uint32_t)ngc * kGroupCols * 2;
    mbar_arrive_expect_tx(bar_x, row_bytes * MODE);
    for (int b = 0; b < MODE; ++b)
      bulk_g2s(smem_u32(smem + a.off_x) + b * a.x_pitch,
               a.x + (size_t)b * a.cols + (size_t)g0 * kGroupCols, row_bytes, bar_x);
  }
  if (csize > 1) cluster_wait();  // every CTA's receive mbarrier is initialised
  bool ok = mbar_wait_poll(bar_cb, 0);
  if (!mode_full(MODE)) ok &= mbar_wait_poll(bar_x, 0);
  if (!ok && lane == 0) atomicOr(a.flag, 2);

  SmemCodebook cb;
  cb.base = smem;
  cb.copyoff = fmt_small(BITS) ? (uint32_t)(lane & 7) * 16u
                : BITS == kFmt4D ? (uint32_t)(lane & 15) * 8u
                                 : 0u;

  // The activation row this lane supplies to the B fragment; the other lanes
  // read a zero block (stride 0), so the loop has no lane-dependent branch.
  int xb;
  bool provider;
  if (mode_full(MODE)) {
    xb = gid;
    provider = gid < a.batch;
  } else {
    xb = gid - 2 * q;
    provider = xb >= 0 && xb < MODE;
  }
  const uint8_t* x0;  // this lane's activation bytes of group g0
  if (mode_full(MODE))
    x0 = provider ? reinterpret_cast<const uint8_t*>(a.x + (size_t)xb * a.cols + (size_t)g0 * kGroupCols)
                  : reinterpret_cast<const uint8_t*>(a.zeros);
  else
    x0 = provider ? smem + a.off_x + xb * a.x_pitch : smem + a.off_zero;
  x0 += q * (BITS == kFmt4D ? 8 : 16);
  const int xstep = provider ? kGroupCols * 2 : 0;
  // kFull16: bytes from this lane's activation row to its second-half row
  // (batch row gid + 8), or 0 where that row is past the batch (the lane then
  // reads its own row again; those product columns are never sent)
  const int x2off = MODE == kFull16 && gid + 8 < a.batch ? 16 * a.cols : 0;

  // receive slot of (owned tile k, rank r, warp w): ((k * csize + r) * WARPS + w) * kBlk floats
  const uint32_t recv_base = smem_u32(smem + a.off_recv);

  Acc<MODE> acc[S];
#pragma unroll
  for (int j = 0; j < S; ++j) acc[j].zero();

  // Units of a strip at one group are contiguous: one bulk L2 prefetch per
  // item, two items ahead inside the strip (the next item's units are already
  // in flight to registers).
  int left = i1 - i0;
  while (left > 0) {
    // the warp's items of strip s: groups g .. g + cnt - 1
    const int cnt = min(left, g0 + ngc - g);
    left -= cnt;
    const uint8_t* ub = strip_base(s, g);
    const uint8_t* xp = x0 + (g - g0) * xstep;
    const uint8_t* nb = strip_base(s + 1, g0);
    const unsigned nmask = left > 0 ? strip_mask(s + 1) : 0u;
    if (s < nfull)
      run_segment<BITS, MODE, S, S>(u, acc, cnt, ub, gstride, xp, xstep, nb, nmask, lane, q, cb, x2off);
    else if (S > 1 && rest == 1)
      run_segment<BITS, MODE, 1, S>(u, acc, cnt, ub, gstride, xp, xstep, nb, nmask, lane, q, cb, x2off);
    else if (S > 2 && rest == 2)
      run_segment<BITS, MODE, (S > 2 ? 2 : 1), S>(u, acc, cnt, ub, gstride, xp, xstep, nb, nmask,
                                                  lane, q, cb, x2off);
    else if (S > 3)
      run_segment<BITS, MODE, (S > 3 ? 3 : 1), S>(u, acc, cnt, ub, gstride, xp, xstep, nb, nmask,
                                                  lane, q, cb, x2off);
#pragma unroll
    for (int j = 0; j < S; ++j) {
      const int tau = s * S + j;
      if (tau < T) {
        const int owner = tau & (csize - 1);
        const uint32_t slot =
            recv_base + 4u * (uint32_t)(((((tau >> cshift) << cshift) + crank) * WARPS + warp) * kBlk);
        send_partial<MODE>(mapa(slot, (uint32_t)owner), mapa(bar_recv, (uint32_t)owner), acc[j],
                           lane, a.batch);
      }
      acc[j].zero();
    }
    ++s;
    g = g0;
  }
  // -0.0 blocks for the cluster's tiles outside this warp's items (tiles
  // [tau_lo, tau_hi) got its partial sums): 16 bytes per lane, 64 bytes per
  // batch row
  {
    const int w0 = warp_item<WARPS, S>(T, ngc, warp), w1 = warp_item<WARPS, S>(T, ngc, warp + 1);
    const int tau_lo = w0 < w1 ? div_ngc(w0) * S : 0;
    const int tau_hi = w0 < w1 ? min(T, (div_ngc(w1 - 1) + 1) * S) : 0;
  for (int tau = 0; tau < T; ++tau) {
    if (tau >= tau_lo && tau < tau_hi) continue;
    const uint32_t slot =
        recv_base + 4u * (uint32_t)(((((tau >> cshift) << cshift) + crank) * WARPS + warp) * kBlk);
    const uint32_t owner = (uint32_t)(tau & (csize - 1));
    if constexpr (MODE == kFull16) {
      for (int i = lane; i < 4 * a.batch; i += 32)  // 64 bytes per batch row
        st_async16(mapa(slot, owner) + 16u * (uint32_t)i, make_float4(-0.f, -0.f, -0.f, -0.f),
                   mapa(bar_recv, owner));
    } else if (lane < 4 * a.batch) {
      st_async16(mapa(slot, owner) + 16u * (uint32_t)lane, make_float4(-0.f, -0.f, -0.f, -0.f),
                 mapa(bar_recv, owner));
    }
  }
  }
  // Owned tiles (tau = crank + k * csize): wait for every warp of the
  // cluster, then sum their blocks in (rank, warp) order and write y.
  if (nown == 0) return;
  if (!mbar_wait_poll(bar_recv, 0) && threadIdx.x == 0) atomicOr(a.flag, 2);
  const float* recv = reinterpret_cast<const float*>(smem + a.off_recv);
  for (int e = threadIdx.x; e < nown * kBlk; e += WARPS * 32) {
    const int k = e / kBlk, i = e % kBlk;
    const int b = i / kRowsPerTile, r = (t0 + crank + k * csize) * kRowsPerTile + i % kRowsPerTile;
    if (b >= a.batch || r >= a.rows) continue;
    float sum = 0.f;
    for (int rk = 0; rk < csize; ++rk) {
#pragma unroll
      for (int w = 0; w < WARPS; ++w) sum += recv[(((size_t)k * csize + rk) * WARPS + w) * kBlk + i];
    }
    a.y[(size_t)b * a.rows + r] = f32_to_h_rn(sum);
  }
}


// Launch shape per format.  Small-codebook splits (W2 and Tab. 4): eight
// interleaved codebook copies (K x 128 B) and two CTAs per SM.
template <int BITS> struct KernelShape {
  static constexpr int kWarps = 8;
  static constexpr int kMinBlocks = 2;
  static constexpr uint32_t kCbBytes = (uint32_t)Layout<BITS>::K * 8 * 16;
};
// W3: the 128 KiB codebook allows one CTA per SM; 8 warps with the whole
// register file (up to 255 registers each) hide the codebook's bank-conflict
// latency better than 16 warps at 128 (measured 9-15% faster).
template <> struct KernelShape<3> {
  static constexpr int kWarps = 8;
  static constexpr int kMinBlocks = 1;
  static constexpr uint32_t kCbBytes = (uint32_t)Layout<3>::K * 16;
};
template <> struct KernelShape<kFmtW3V3> : KernelShape<3> {};

constexpr int kModes[4] = {kFactored1, kFactored2, kFull, kFull16};

// Batches of 9-16 rows (8-D formats): one build per format with the whole
// register file (one CTA per SM) and strips of two tiles, which hold the
// second batch half's accumulators and activations; none for 4-D vectors.
template <int FMT>
inline const void* kptr_full16() {
  if constexpr (FMT == kFmt4D)
    return nullptr;
  else
    return reinterpret_cast<const void*>(
        &gemv_kernel<FMT, kFull16, KernelShape<FMT>::kWarps, 1, 2>);
}

template <int BITS, int MODE, int S>
inline const void* kptr() {
  return reinterpret_cast<const void*>(
      &gemv_kernel<BITS, MODE, KernelShape<BITS>::kWarps, KernelShape<BITS>::kMinBlocks, S>);
}
template <int FMT, int S = 2>
inline const void* kptr_mode(int mode) {
  return mode == kFactored1 ? kptr<FMT, kFactored1, S>()
         : mode == kFactored2 ? kptr<FMT, kFactored2, S>()
         : mode == kFull      ? kptr<FMT, kFull, S>()
                              : kptr_full16<FMT>();
}

// W2 built for one CTA per SM, with the whole register file instead of the
// 128 registers that two resident CTAs allow: the launch plan takes it when
// the row tiles bound the cluster count, so that no second CTA would share
// the SM (measured on 512 x 3584 at batch 1: 1.90 us against 2.23).
template <int FMT, int S = 2>
inline const void* kptr_mode_solo(int mode) {
  constexpr int W = KernelShape<FMT>::kWarps;
  return mode == kFactored1   ? reinterpret_cast<const void*>(&gemv_kernel<FMT, kFactored1, W, 1, S>)
         : mode == kFactored2 ? reinterpret_cast<const void*>(&gemv_kernel<FMT, kFactored2, W, 1, S>)
         : mode == kFull      ? reinterpret_cast<const void*>(&gemv_kernel<FMT, kFull, W, 1, S>)
                              : kptr_full16<FMT>();
}

// Kernels of the Tab. 4 splits (formats 5-9), instantiated in their own
// translation unit; nullptr for other formats.
const void* split_kernel(int fmt, int mode);

}  // namespace sphq
