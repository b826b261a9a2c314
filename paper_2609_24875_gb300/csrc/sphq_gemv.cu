// Fused spherical dequantize-GEMV for decode (SPHQuant §3.4, App. D), sm_103a.
//
// y[n][r] = sum_j w_hat[r][j] x[n][j] for a batch of n <= 8 activation rows.
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
//  * batch 1-2 ("factored"): the A fragment holds the signed unit direction
//    s (.) c_z and the B fragment is block diagonal -- column 2c + b carries
//    batch row b of slot c only -- so every MMA pair returns, in the lane
//    that decoded them, the per-vector dots d = (s (.) c_z) . x_b.  The lane
//    then adds r_hat * d with one fp32 FMA (r_hat from the fp16 FMA of
//    Eq. (7)).  This skips the four half-rate fp16 products per block; the
//    result differs from the exact W_hat x by at most one fp16 rounding of
//    each product r_hat * c (2^-11 relative), inside the stated tolerance.
//  * batch 3-8 ("full"): the lane forms w_hat = RN16(r_hat * (s (.) c_z))
//    exactly as Eq. (4) defines it and the MMA's N dimension is the batch.
//
// Work decomposition (stream-K).  The (row tile, group) units are cut into
// equal contiguous spans, one per warp of a grid no larger than the resident
// capacity.  A warp accumulates in registers while its span stays in one row
// tile.  A row tile covered by one warp is written directly; otherwise each
// covering warp stores its fp32 partial (16 rows x batch) into the handle's
// workspace and the last to arrive (an acq_rel atomic ticket per row tile;
// nobody waits) sums the partials in slot order and writes y, so results do
// not depend on scheduling.
//
// Programmatic dependent launch: the kernel lets the next kernel on the
// stream launch at once, asks L2 to prefetch its whole span of codes, loads
// its first unit and stages the codebook, and only then waits
// (griddepcontrol.wait) for the previous kernel -- before it touches
// activations, outputs, workspace or tickets.  Codes and codebook are
// immutable after sphq_pack, so this overlap is safe.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <string>

#include "sphq_internal.h"
#include "sphq_layout.cuh"

namespace sphq {

struct GemvArgs {
  const uint8_t* units;
  const uint4* codebook;
  const uint16_t* x;
  uint16_t* y;
  float* ws;
  unsigned* tickets;
  int rows, cols, ng, nrt;
  int batch;
  int units_per_warp;
  int max_slots;
  long long total_units;
  const uint16_t* zeros;  // 256 B zero block: activations of lanes that supply none
};

// Zero block read by lanes that supply no activations: 256 B used, placed
// 64 B into a 320 B region so its 16-byte chunks (4m + q) fall in the other
// half of the shared-memory bank groups from the activations' chunks.
constexpr int kZeroVec = 20;
constexpr int kZeroSkew = 4;  // uint4

// Radius application modes.
constexpr int kFactored1 = 1;  // batch 1
constexpr int kFactored2 = 2;  // batch 2
constexpr int kFull = 8;       // batch 3..8

// The MMAs are pure register computations (no volatile), so the compiler may
// interleave the words of a unit freely.
__device__ __forceinline__ void mma16816(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                         uint32_t a3, uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1));
}

// D = A B (C = 0)
__device__ __forceinline__ void mma16816_zero(float (&d)[4], uint32_t a0, uint32_t a1, uint32_t a2,
                                              uint32_t a3, uint32_t b0, uint32_t b1) {
  const float z = 0.f;
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 "
      "{%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, {%10,%10,%10,%10};"
      : "=f"(d[0]), "=f"(d[1]), "=f"(d[2]), "=f"(d[3])
      : "r"(a0), "r"(a1), "r"(a2), "r"(a3), "r"(b0), "r"(b1), "f"(z));
}

// Activations are re-read by every row tile: keep them in L1.
__device__ __forceinline__ uint4 ldg_x16(const uint16_t* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::evict_last.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}

__device__ __forceinline__ float h_lo_to_f32(uint32_t h2) {
  float f;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tcvt.f32.f16 %0, lo;\n\t}"
      : "=f"(f) : "r"(h2));
  return f;
}
__device__ __forceinline__ float h_hi_to_f32(uint32_t h2) {
  float f;
  asm("{\n\t.reg .f16 lo, hi;\n\tmov.b32 {lo, hi}, %1;\n\tcvt.f32.f16 %0, hi;\n\t}"
      : "=f"(f) : "r"(h2));
  return f;
}

__device__ __forceinline__ void pdl_launch_dependents() {
  asm volatile("griddepcontrol.launch_dependents;" ::: "memory");
}
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }

__device__ __forceinline__ void prefetch_l2(const void* p, uint32_t bytes) {
  asm volatile("cp.async.bulk.prefetch.L2.global [%0], %1;" ::"l"(p), "r"(bytes) : "memory");
}

__device__ __forceinline__ unsigned ticket_acq_rel(unsigned* p) {
  unsigned old;
  asm volatile("atom.acq_rel.gpu.global.add.u32 %0, [%1], 1;" : "=r"(old) : "l"(p) : "memory");
  return old;
}

// Writes a warp's partial of row tile rt; the last contributor sums all
// partials in slot order and stores fp16 y.  v[i][h] is this lane's value of
// batch row bidx[i] at row gid + 8h of the tile, valid where own[i] is set.
template <int NB>
__device__ __forceinline__ void flush_row_tile(const GemvArgs& a, int rt, long long gw, int lane,
                                               const float (&v)[NB][2], const bool (&own)[NB],
                                               const int (&bidx)[NB]) {
  const long long L = a.units_per_warp;
  const long long first = ((long long)rt * a.ng) / L;
  const long long last = ((long long)(rt + 1) * a.ng - 1) / L;
  const int count = (int)(last - first + 1);
  const int gid = lane >> 2;
  const int row0 = rt * kRowsPerTile;
  if (count == 1) {
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      if (!own[i]) continue;
      const int b = bidx[i];
      if (row0 + gid < a.rows) a.y[(size_t)b * a.rows + row0 + gid] = f32_to_h_rn(v[i][0]);
      if (row0 + gid + 8 < a.rows) a.y[(size_t)b * a.rows + row0 + gid + 8] = f32_to_h_rn(v[i][1]);
    }
    return;
  }
  const int per = kRowsPerTile * a.batch;  // floats per partial
  const int slot = (int)(gw - first);
  float* base = a.ws + (size_t)rt * a.max_slots * kRowsPerTile * kMaxBatch;
  float* mine = base + (size_t)slot * per;
#pragma unroll
  for (int i = 0; i < NB; ++i) {
    if (!own[i]) continue;
    const int b = bidx[i];
    mine[b * kRowsPerTile + gid] = v[i][0];
    mine[b * kRowsPerTile + gid + 8] = v[i][1];
  }
  __syncwarp();
  unsigned ticket = 0;
  if (lane == 0) ticket = ticket_acq_rel(&a.tickets[rt]);
  ticket = __shfl_sync(0xFFFFFFFFu, ticket, 0);
  if (ticket != (unsigned)(count - 1)) return;
  __syncwarp();  // order every lane's reads after lane 0's acquire
  for (int i = lane; i < per; i += 32) {
    float s = 0.f;
    for (int k = 0; k < count; ++k) s += __ldcg(base + (size_t)k * per + i);
    const int b = i / kRowsPerTile, r = row0 + i % kRowsPerTile;
    if (r < a.rows) a.y[(size_t)b * a.rows + r] = f32_to_h_rn(s);
  }
  __syncwarp();
  if (lane == 0) atomicExch(&a.tickets[rt], 0u);  // ready for the next call
}

template <int BITS>
struct UnitConst {
  uint32_t d2, m2, e;
};

template <int BITS>
__device__ __forceinline__ UnitConst<BITS> unit_const(const Unit<BITS>& u, int q) {
  UnitConst<BITS> c;
  if constexpr (BITS == 2) {
    c.d2 = params_delta(u.rec.z, u.rec.w);
    c.m2 = params_rmin(u.rec.z, u.rec.w);
    c.e = w2_sign3(u, q);
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
  if constexpr (BITS == 2) {
    const uint32_t W = word_of(u.w, m);
    directions_w2(W, k.e, m, cb, cb.copyoff, true, sa, sb);
    qp = qpair_w2(W);
  } else {
    directions_w3(u, m, q, cb, sa, sb);
    qp = qpair_w3(u, m);
  }
}

// Accumulators of one warp for the current row tile.
template <int MODE>
struct Acc {
  static constexpr int NB = MODE == kFull ? 2 : MODE;
  float f[2][NB][2];  // factored: [set][batch row][row gid / gid+8]
  float d[2][4];      // full: MMA accumulators [set][fragment]
  __device__ __forceinline__ void zero() {
#pragma unroll
    for (int s = 0; s < 2; ++s) {
#pragma unroll
      for (int i = 0; i < NB; ++i) f[s][i][0] = f[s][i][1] = 0.f;
#pragma unroll
      for (int i = 0; i < 4; ++i) d[s][i] = 0.f;
    }
  }
};

// One unit (16 rows x 16 slots).  For word m the lane supplies to the B
// fragment 16 B at xsrc + 32*m halves: its activation row at slot 4m+q, or the
// zero block.  Batch 1-2 reads x from shared memory (staged once per CTA),
// batch 3-8 from global memory through L1; the unit's four loads are issued
// together before any of its words is decoded.
template <int BITS, int MODE>
__device__ __forceinline__ void process_unit(const Unit<BITS>& cur, const uint16_t* xsrc, int q,
                                             const SmemCodebook& cb, Acc<MODE>& acc) {
  uint4 xv[4];
  if constexpr (MODE == kFull) {
#pragma unroll
    for (int m = 0; m < 4; ++m) xv[m] = ldg_x16(xsrc + 32 * m);
  }
  const UnitConst<BITS> kc = unit_const<BITS>(cur, q);
#pragma unroll
  for (int m = 0; m < 4; ++m) {
    if constexpr (MODE != kFull) xv[m] = *reinterpret_cast<const uint4*>(xsrc + 32 * m);
    const uint4& xm = xv[m];
    uint4 sa, sb;
    uint32_t qp;
    word_directions<BITS>(cur, kc, m, q, cb, sa, sb, qp);
    const uint32_t r = radius_pair(qp, kc.d2, kc.m2);
    if constexpr (MODE == kFull) {
      const uint4 wa = scale_block(sa, bcast_lo(r));
      const uint4 wb = scale_block(sb, bcast_hi(r));
      float(&d)[4] = acc.d[m & 1];
      mma16816(d, wa.x, wb.x, wa.y, wb.y, xm.x, xm.y);
      mma16816(d, wa.z, wb.z, wa.w, wb.w, xm.z, xm.w);
    } else {
      float d[4];
      mma16816_zero(d, sa.x, sb.x, sa.y, sb.y, xm.x, xm.y);
      mma16816(d, sa.z, sb.z, sa.w, sb.w, xm.z, xm.w);
      const float rA = h_lo_to_f32(r), rB = h_hi_to_f32(r);
      auto& ac = acc.f[m & 1];
      ac[0][0] = __fmaf_rn(rA, d[0], ac[0][0]);
      ac[0][1] = __fmaf_rn(rB, d[2], ac[0][1]);
      if constexpr (MODE == kFactored2) {
        ac[1][0] = __fmaf_rn(rA, d[1], ac[1][0]);
        ac[1][1] = __fmaf_rn(rB, d[3], ac[1][1]);
      }
    }
  }
}

template <int MODE>
__device__ __forceinline__ void flush_acc(const GemvArgs& a, int rt, long long gw, int lane,
                                          Acc<MODE>& acc) {
  const int q = lane & 3;
  if constexpr (MODE == kFull) {
    // d[0..3] = D[gid][2q], D[gid][2q+1], D[gid+8][2q], D[gid+8][2q+1]
    float v[2][2] = {{acc.d[0][0] + acc.d[1][0], acc.d[0][2] + acc.d[1][2]},
                     {acc.d[0][1] + acc.d[1][1], acc.d[0][3] + acc.d[1][3]}};
    const bool own[2] = {2 * q < a.batch, 2 * q + 1 < a.batch};
    const int bidx[2] = {2 * q, 2 * q + 1};
    flush_row_tile<2>(a, rt, gw, lane, v, own, bidx);
  } else {
    constexpr int NB = MODE;
    // sum the lane's slots, then the quad's four lanes (slots q = 0..3)
    float v[NB][2];
#pragma unroll
    for (int i = 0; i < NB; ++i) {
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        float t = acc.f[0][i][h] + acc.f[1][i][h];
        t += __shfl_xor_sync(0xFFFFFFFFu, t, 1);
        t += __shfl_xor_sync(0xFFFFFFFFu, t, 2);
        v[i][h] = t;
      }
    }
    bool own[NB];
    int bidx[NB];
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      own[i] = q == 0;
      bidx[i] = i;
    }
    flush_row_tile<NB>(a, rt, gw, lane, v, own, bidx);
  }
  acc.zero();
}

template <int BITS, int MODE, int WARPS, int MINB>
__global__ void __launch_bounds__(WARPS * 32, MINB) gemv_kernel(const GemvArgs a) {
  extern __shared__ uint4 smem_cb[];
  pdl_launch_dependents();
  const int lane = threadIdx.x & 31;
  const int gid = lane >> 2, q = lane & 3;
  const long long gw = (long long)blockIdx.x * WARPS + (threadIdx.x >> 5);
  long long u = gw * a.units_per_warp;
  const long long u_end = min(u + (long long)a.units_per_warp, a.total_units);
  constexpr int UB = Layout<BITS>::kUnitBytes;
  const uint8_t* const span = a.units + (size_t)u * UB;  // unit u of the span

  // Codes are immutable: stream the span toward L2 and start the first unit
  // while the codebook is staged and the previous kernel finishes.
  Unit<BITS> ua{}, ub{}, uc{};
  if (u < u_end) {
    if (lane == 0) prefetch_l2(span, (uint32_t)((u_end - u) * UB));
    ua = load_unit<BITS>(span, lane);
    ub = load_unit<BITS>(span + UB, lane);
  }
  if (BITS == 2) {
    for (int i = threadIdx.x; i < Layout<2>::K * 8; i += WARPS * 32)
      smem_cb[i] = __ldg(a.codebook + (i >> 3));
  } else {
    for (int i = threadIdx.x; i < Layout<3>::K; i += WARPS * 32) smem_cb[i] = __ldg(a.codebook + i);
  }
  // batch 1-2: a zero block and the activation rows follow the codebook
  constexpr int kCbVec = (BITS == 2 ? Layout<2>::K * 8 : Layout<3>::K);  // uint4 entries
  uint4* const smem_zero = smem_cb + kCbVec;
  uint16_t* const smem_x = reinterpret_cast<uint16_t*>(smem_zero + kZeroVec);
  if (MODE != kFull && threadIdx.x < kZeroVec) smem_zero[threadIdx.x] = make_uint4(0, 0, 0, 0);
  pdl_wait();
  if (MODE != kFull) {
    const int nx = a.batch * a.cols / 8;  // uint4 of activations (cols % 128 == 0)
    const uint4* xg = reinterpret_cast<const uint4*>(a.x);
    uint4* xs = reinterpret_cast<uint4*>(smem_x);
    for (int i = threadIdx.x; i < nx; i += WARPS * 32) xs[i] = ldg_x16(a.x + 8 * (size_t)i);
    (void)xg;
  }
  __syncthreads();
  if (u >= u_end) return;

  SmemCodebook cb;
  cb.base = reinterpret_cast<const uint8_t*>(smem_cb);
  cb.copyoff = BITS == 2 ? (uint32_t)(lane & 7) * 16u : 0u;

  // The activation row this lane supplies to the B fragment; lanes that
  // supply nothing read the handle's zero page (no predicates in the loop).
  bool provider;
  int xb;
  if (MODE == kFull) {
    xb = gid;
    provider = gid < a.batch;
  } else {
    xb = gid - 2 * q;
    provider = xb >= 0 && xb < MODE;
  }
  // providers walk their activation row group by group; the others keep
  // reading the same 256-byte zero block (stride 0), which stays in L1
  const uint16_t* xrow;
  if (MODE == kFull)
    xrow = (provider ? a.x + (size_t)xb * a.cols : a.zeros) + q * kVec;
  else
    xrow = (provider ? smem_x + (size_t)xb * a.cols
                     : reinterpret_cast<const uint16_t*>(smem_zero + kZeroSkew)) +
           q * kVec;
  const int xstride = provider ? kGroupCols : 0;

  // the unit buffer ends with two guard units, so prefetching up to two units
  // past the span stays in bounds (the data is never used)
  auto unit_ptr = [&](long long v) { return a.units + (size_t)v * UB; };

  int rt = (int)(u / a.ng);
  int g = (int)(u - (long long)rt * a.ng);
  Acc<MODE> acc;
  acc.zero();
  for (;;) {
    // one segment: the span's units inside row tile rt
    const long long seg_end = min(u_end, (long long)(rt + 1) * a.ng);
    long long n = seg_end - u;
    const uint16_t* xs = xrow + (size_t)g * xstride;
    // three units in registers: the one being decoded and two in flight
    for (; n >= 3; n -= 3) {
      uc = load_unit<BITS>(unit_ptr(u + 2), lane);
      process_unit<BITS, MODE>(ua, xs, q, cb, acc);
      ua = load_unit<BITS>(unit_ptr(u + 3), lane);
      process_unit<BITS, MODE>(ub, xs + xstride, q, cb, acc);
      ub = load_unit<BITS>(unit_ptr(u + 4), lane);
      process_unit<BITS, MODE>(uc, xs + 2 * xstride, q, cb, acc);
      xs += 3 * xstride;
      u += 3;
    }
    for (; n > 0; --n) {  // 1 or 2 left: rotate the ring
      uc = load_unit<BITS>(unit_ptr(u + 2), lane);
      process_unit<BITS, MODE>(ua, xs, q, cb, acc);
      ua = ub;
      ub = uc;
      xs += xstride;
      u += 1;
    }
    flush_acc<MODE>(a, rt, gw, lane, acc);
    if (u >= u_end) break;
    ++rt;  // the next segment starts at group 0 of the next row tile
    g = 0;
  }
}

template <int BITS> struct KernelShape;
template <> struct KernelShape<2> {
  static constexpr int kWarps = 8;
  static constexpr int kMinBlocks = 2;
  static constexpr size_t kSmem = (size_t)Layout<2>::K * 8 * 16;
};
template <> struct KernelShape<3> {
  static constexpr int kWarps = 16;
  static constexpr int kMinBlocks = 1;
  static constexpr size_t kSmem = (size_t)Layout<3>::K * 16;
};

template <int BITS, int MODE>
static const void* kptr() {
  return reinterpret_cast<const void*>(
      &gemv_kernel<BITS, MODE, KernelShape<BITS>::kWarps, KernelShape<BITS>::kMinBlocks>);
}

static int mode_for(int batch) { return batch == 1 ? kFactored1 : batch == 2 ? kFactored2 : kFull; }

static const void* select_kernel(int bits, int mode) {
  if (bits == 2)
    return mode == kFactored1 ? kptr<2, kFactored1>() : mode == kFactored2 ? kptr<2, kFactored2>()
                                                                           : kptr<2, kFull>();
  return mode == kFactored1 ? kptr<3, kFactored1>() : mode == kFactored2 ? kptr<3, kFactored2>()
                                                                         : kptr<3, kFull>();
}

// Dynamic shared memory is sized per handle (batch 1-2 stage their activation
// rows), while the attribute that permits it belongs to the kernel function and
// is process-wide: raise it once to the device's opt-in maximum.
static sphq_status allow_max_smem(int device, int optin) {
  static std::mutex mu;
  static bool done[64] = {};
  std::lock_guard<std::mutex> lock(mu);
  if (device < 0 || device >= 64) return set_error(SPHQ_ERR_DEVICE, "device index out of range");
  if (done[device]) return SPHQ_OK;
  const int modes[3] = {kFactored1, kFactored2, kFull};
  for (int bits = 2; bits <= 3; ++bits)
    for (int mode : modes) {
      cudaError_t e = cudaFuncSetAttribute(select_kernel(bits, mode),
                                           cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
      if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute");
    }
  done[device] = true;
  return SPHQ_OK;
}

sphq_status make_gemv_plans(sphq_handle h) {
  int optin = 0;
  cudaError_t e = cudaDeviceGetAttribute(&optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
  sphq_status st = allow_max_smem(h->device, optin);
  if (st != SPHQ_OK) return st;
  const long long units = (long long)h->nrt * h->ng;
  size_t ws = 0;
  for (int batch = 1; batch <= SPHQ_MAX_BATCH; ++batch) {
    GemvPlan& p = h->plan[batch];
    p.warps_per_cta = h->bits == 2 ? KernelShape<2>::kWarps : KernelShape<3>::kWarps;
    const size_t cb_smem = h->bits == 2 ? KernelShape<2>::kSmem : KernelShape<3>::kSmem;
    // batch 1-2 stage x in shared memory when it fits; otherwise read it through L1
    p.mode = mode_for(batch);
    p.smem = cb_smem;
    if (p.mode != kFull) {
      const size_t staged = cb_smem + kZeroVec * 16 + (size_t)batch * h->cols * 2;
      if (staged <= (size_t)optin * 7 / 8) p.smem = staged;
      else p.mode = kFull;
    }
    const void* k = select_kernel(h->bits, p.mode);
    int occ = 0;
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&occ, k, p.warps_per_cta * 32, p.smem);
    if (e != cudaSuccess) return cuda_error(e, "occupancy query");
    if (occ < 1) return set_error(SPHQ_ERR_CUDA, "gemv kernel cannot be resident");
    const long long max_warps = (long long)h->sm_count * occ * p.warps_per_cta;
    // at least two units per warp so each warp has one unit in flight while it
    // decodes the previous one
    long long L = std::max<long long>(2, (units + max_warps - 1) / max_warps);
    L = std::min<long long>(L, units);
    const long long warps = (units + L - 1) / L;
    p.units_per_warp = (int)L;
    p.grid = (int)((warps + p.warps_per_cta - 1) / p.warps_per_cta);
    p.max_slots = (int)((h->ng + L - 1) / L + 1);
    ws = std::max(ws, (size_t)h->nrt * p.max_slots * kRowsPerTile * kMaxBatch);
  }
  h->ws_floats = ws;
  return SPHQ_OK;
}

sphq_status launch_gemv(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s) {
  const GemvPlan& p = h->plan[batch];
  GemvArgs a;
  a.units = (const uint8_t*)h->units;
  a.codebook = (const uint4*)h->codebook;
  a.x = (const uint16_t*)x;
  a.y = (uint16_t*)y;
  a.ws = h->ws;
  a.tickets = h->tickets;
  a.rows = h->rows;
  a.cols = h->cols;
  a.ng = h->ng;
  a.nrt = h->nrt;
  a.batch = batch;
  a.units_per_warp = p.units_per_warp;
  a.max_slots = p.max_slots;
  a.total_units = (long long)h->nrt * h->ng;
  a.zeros = (const uint16_t*)h->zeros;

  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(p.warps_per_cta * 32);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {&a};
  cudaError_t e = cudaLaunchKernelExC(&cfg, select_kernel(h->bits, p.mode), args);
  if (e != cudaSuccess) return cuda_error(e, "gemv launch");
  return SPHQ_OK;
}

// Same launch as launch_gemv, with caller-provided split-K scratch (partials
// and per-row-tile tickets) instead of the handle's own workspace.
sphq_status launch_gemv_scratch(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s,
                                float* ws, unsigned* tickets) {
  const GemvPlan& p = h->plan[batch];
  GemvArgs a;
  a.units = (const uint8_t*)h->units;
  a.codebook = (const uint4*)h->codebook;
  a.x = (const uint16_t*)x;
  a.y = (uint16_t*)y;
  a.ws = ws;
  a.tickets = tickets;
  a.rows = h->rows;
  a.cols = h->cols;
  a.ng = h->ng;
  a.nrt = h->nrt;
  a.batch = batch;
  a.units_per_warp = p.units_per_warp;
  a.max_slots = p.max_slots;
  a.total_units = (long long)h->nrt * h->ng;
  a.zeros = (const uint16_t*)h->zeros;
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(p.warps_per_cta * 32);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  void* args[] = {&a};
  cudaError_t e = cudaLaunchKernelExC(&cfg, select_kernel(h->bits, p.mode), args);
  if (e != cudaSuccess) return cuda_error(e, "gemv launch");
  return SPHQ_OK;
}

}  // namespace sphq
