// Device layout of packed SPHQuant codes and the per-vector decode shared by
// the GEMV and decode kernels.  sm_103a only.
//
// Tiles.  Rows are padded to a multiple of 16 and cut into row tiles of 16
// rows (the M extent of one m16n8k16 MMA).  For row tile rt and radius group g
// (16 consecutive 8-D vectors = 128 columns, §3.1) one contiguous "unit" holds
// the 256 vectors (16 rows x 16 slots) in the order the GEMV's threads consume
// them: lane l = 4*gid + q (gid = l/4, q = l%4) owns rows gid and gid+8 at the
// group's slots q, 4+q, 8+q, 12+q.  Its 16-byte block holds four 32-bit words
// w_m (m = 0..3); word w_m holds vector A = (row gid, slot 4m+q) and vector
// B = (row gid+8, slot 4m+q).  Units are stored group-major: unit (rt, g) is
// number g * nrt + rt, so the units of consecutive row tiles at one group --
// the ones that share activations -- are adjacent in memory (their offsets
// from each other are compile-time constants in the GEMV), and every
// warp-wide 16-byte load is a 512-byte burst.
//
// W2 unit (640 B = 256 x 2.25 bits + 16 x 4 B of group parameters, §3.1, §3.4):
//   [0, 512)    lane l: words w_0..w_3 at 16*l, bits of w_m:
//                 0-3 radius code of A   4-9 direction index of A
//                 16-19 radius code of B 20-25 direction index of B
//                 15,31 / 14,30 / 13,29  sign bits (2p, 2p+1) of A, pairs p = 0,1,2
//                 12,28 / 11,27 / 10,26  sign bits of B, pairs p = 0,1,2
//   [512, 640)  quad gid (lanes 4gid..4gid+3): 16 B at 512 + 16*gid =
//                 { S01, S23, P_gid, P_gid+8 }
//                 S01: the sign bits 6, 7 of lane q=0's eight vectors in bits
//                      8-15 / 24-31 and of lane q=1's in bits 0-7 / 16-23
//                      (vector v = 2m + {0: A, 1: B}: bit 15-v = s6, bit 31-v = s7)
//                 S23: the same for lanes q = 2, 3
//                 P_r: Delta_G (low 16 bits) | r_min_G (high 16 bits) of row r
//   The bit positions make each sign mask one shift of a loaded word away
//   from bits 15/31 (the fp16 sign bits of a half2 register) and the two
//   radius codes of a word one AND away from two fp16 integers.
//
// W3 unit (864 B = 256 x 3.125 bits + 64 B of group parameters):
//   [0, 512)    lane l: words w_0..w_3, bits of w_m:
//                 0-7 direction index bits 0-7 of A, 16-23 of B
//                 15,31 / 14,30 / 13,29 / 12,28  sign bits of A, pairs 0..3
//                 11,27 / 10,26 /  9,25 /  8,24  sign bits of B, pairs 0..3
//   [512, 768)  lane l: 8 B at 512 + 8*l = { MID, QN }
//                 QN:  radius codes, word m: A at bits 4m..4m+3, B at 16+4m..
//                 MID: index bits 8-11, word m: A at bits 8-11 rotated right by
//                      4m (m=0: 8-11, 1: 12-15, 2: 0-3, 3: 4-7), B 16 bits higher
//   [768, 832)  quad gid: 8 B = { P_gid, P_gid+8 }
//   [832, 864)  quad gid: 4 B, bit (4q + m) = index bit 12 of A of lane q's
//                 word m, bit (16 + 4q + m) = that of B
//
// W3 unit with 3-bit radius codes (the 3.00-bit split of App. B,
// (7B + V)/8 with V = 3; format id 4 below), 832 B = 256 x 3 bits x 8 + 64 B:
//   [0, 512)    lane l: words w_0..w_3 exactly as in the W3 unit
//   [512, 768)  lane l: 8 B = { H0, H1 }; word m owns byte 2*(m%2) (A) and
//                 byte 2*(m%2)+1 (B) of H_{m/2}: index bits 8-12 in bits 0-4,
//                 radius code (0..7) in bits 5-7
//   [768, 832)  quad gid: 8 B = { P_gid, P_gid+8 }
//
// No byte beyond the algorithmic payload is stored; padded rows hold zero
// codes and parameters.
#pragma once
#include <cstdint>

namespace sphq {

constexpr int kVec = 8;                 // 8-D vectors (§3.1)
constexpr int kGroupVecs = 16;          // vectors per radius group
constexpr int kGroupCols = kVec * kGroupVecs;
constexpr int kRowsPerTile = 16;        // rows per unit (MMA M)
constexpr int kMaxBatch = 8;
constexpr uint32_t kSignMask = 0x80008000u;

// Index of unit (row tile rt, radius group g) in a matrix of nrt row tiles.
__host__ __device__ __forceinline__ long long unit_index(int rt, int g, int nrt) {
  return (long long)g * nrt + rt;
}

// Format ids used as template arguments: 2 = W2, 3 = W3, 4 = W3 with 3-bit
// radius codes.  The codebook size follows the weight bit-width B.
constexpr int kFmtW3V3 = 4;
__host__ __device__ constexpr int fmt_bits(int fmt) { return fmt == kFmtW3V3 ? 3 : fmt; }

template <int BITS> struct Layout;
template <> struct Layout<2> {
  static constexpr int K = 64;
  static constexpr int kUnitBytes = 640;
  static constexpr int kRecOff = 512;
};
template <> struct Layout<kFmtW3V3> {
  static constexpr int K = 8192;
  static constexpr int kUnitBytes = 832;
  static constexpr int kHiOff = 512;
  static constexpr int kParamOff = 768;
};
template <> struct Layout<3> {
  static constexpr int K = 8192;
  static constexpr int kUnitBytes = 864;
  static constexpr int kMidOff = 512;
  static constexpr int kParamOff = 768;
  static constexpr int kTopOff = 832;
};

// Per-lane data of one unit.
template <int BITS> struct Unit;
template <> struct Unit<2> {
  uint4 w;      // words w_0..w_3
  uint32_t s;   // the lane's sign word of the quad record: S01 (q < 2) or S23
  uint2 par;    // {P_gid, P_gid+8}
};
template <> struct Unit<kFmtW3V3> {
  uint4 w;
  uint2 hi;     // {H0, H1}
  uint2 par;    // {P_gid, P_gid+8}
};
template <> struct Unit<3> {
  uint4 w;
  uint2 mq;     // {MID, QN}
  uint2 par;    // {P_gid, P_gid+8}
  uint32_t top; // index bit 12 of the quad
};

// Code streams are read once: cache them in L2 only, never in L1.
__device__ __forceinline__ uint4 ldg_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.cg.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ uint2 ldg_stream8(const void* p) {
  uint2 v;
  asm volatile("ld.global.cg.v2.u32 {%0,%1}, [%2];"
               : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ldg_stream4(const void* p) {
  uint32_t v;
  asm volatile("ld.global.cg.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}

template <int BITS>
__device__ __forceinline__ Unit<BITS> load_unit(const uint8_t* unit, int lane);

template <>
__device__ __forceinline__ Unit<2> load_unit<2>(const uint8_t* unit, int lane) {
  Unit<2> u;
  u.w = ldg_stream16(unit + lane * 16);
  const uint8_t* rec = unit + Layout<2>::kRecOff + (lane >> 2) * 16;
  u.s = ldg_stream4(rec + 4 * ((lane >> 1) & 1));
  u.par = ldg_stream8(rec + 8);
  return u;
}

template <>
__device__ __forceinline__ Unit<3> load_unit<3>(const uint8_t* unit, int lane) {
  Unit<3> u;
  u.w = ldg_stream16(unit + lane * 16);
  u.mq = ldg_stream8(unit + Layout<3>::kMidOff + lane * 8);
  u.par = ldg_stream8(unit + Layout<3>::kParamOff + (lane >> 2) * 8);
  u.top = ldg_stream4(unit + Layout<3>::kTopOff + (lane >> 2) * 4);
  return u;
}

template <>
__device__ __forceinline__ Unit<kFmtW3V3> load_unit<kFmtW3V3>(const uint8_t* unit, int lane) {
  Unit<kFmtW3V3> u;
  u.w = ldg_stream16(unit + lane * 16);
  u.hi = ldg_stream8(unit + Layout<kFmtW3V3>::kHiOff + lane * 8);
  u.par = ldg_stream8(unit + Layout<kFmtW3V3>::kParamOff + (lane >> 2) * 8);
  return u;
}

__device__ __forceinline__ uint32_t word_of(const uint4& w, int m) {
  return m == 0 ? w.x : m == 1 ? w.y : m == 2 ? w.z : w.w;
}

// ---------------------------------------------------------------------------
// fp16 arithmetic with explicit round-to-nearest-even and no contraction
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t hmul2_rn(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
__device__ __forceinline__ uint32_t hfma2_rn(uint32_t a, uint32_t b, uint32_t c) {
  uint32_t d;
  asm("fma.rn.f16x2 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "r"(c));
  return d;
}
__device__ __forceinline__ uint32_t hsub2_rn(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("sub.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}
template <uint32_t SEL>
__device__ __forceinline__ uint32_t prmt(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("prmt.b32 %0, %1, %2, %3;" : "=r"(d) : "r"(a), "r"(b), "n"(SEL));
  return d;
}
// a << S as an integer multiply-add: it issues to the FMA pipe instead of the
// (half-rate, busier) integer ALU pipe that the masks and XORs use.
template <int S>
__device__ __forceinline__ uint32_t shl_fma(uint32_t a) {
  if constexpr (S == 0) {
    return a;
  } else {
    uint32_t d;
    asm("mad.lo.u32 %0, %1, %2, 0;" : "=r"(d) : "r"(a), "n"(1u << S));
    return d;
  }
}
__device__ __forceinline__ uint32_t shl_fma_rt(uint32_t a, int s) {
  uint32_t d;
  asm("mad.lo.u32 %0, %1, %2, 0;" : "=r"(d) : "r"(a), "r"(1u << s));
  return d;
}
__device__ __forceinline__ uint32_t rotl(uint32_t a, uint32_t n) {
  uint32_t d;
  asm("shf.l.wrap.b32 %0, %1, %1, %2;" : "=r"(d) : "r"(a), "r"(n));
  return d;
}
__device__ __forceinline__ uint16_t f32_to_h_rn(float v) {
  uint16_t d;
  asm("cvt.rn.f16.f32 %0, %1;" : "=h"(d) : "f"(v));
  return d;
}

// Radius pair of one word, Eq. (7): r_hat = RN16(q * Delta + r_min) with one
// fp16 fused multiply-add per vector.  qpair holds the codes of A (bits 0-3)
// and B (bits 16-19); 1024 + q is an exact fp16 value (bits 0x6400 | q), so
// subtracting 1024 gives q exactly.  d2 / m2: (Delta, r_min) of rows (A, B).
__device__ __forceinline__ uint32_t radius_pair(uint32_t qpair, uint32_t d2, uint32_t m2) {
  const uint32_t qh = (qpair & 0x000F000Fu) | 0x64006400u;
  return hfma2_rn(hsub2_rn(qh, 0x64006400u), d2, m2);
}

// Sign flip of one block: the signed unit direction s (.) c as four half2
// pairs.  masks m_p carry sign bits (2p, 2p+1) at bits 15 and 31 (the fp16
// sign bits of a half2 register); other bits are ignored.
__device__ __forceinline__ uint4 apply_signs(uint4 c, uint32_t m0, uint32_t m1, uint32_t m2,
                                             uint32_t m3) {
  return make_uint4(c.x ^ (m0 & kSignMask), c.y ^ (m1 & kSignMask), c.z ^ (m2 & kSignMask),
                    c.w ^ (m3 & kSignMask));
}

// Eq. (4) for one block: w_hat = RN16(r_hat * (s (.) c)).  Flipping the sign of
// c before the product equals flipping the rounded product (round-to-nearest
// is symmetric, and the sign of a product of zeros is the XOR of the signs).
__device__ __forceinline__ uint4 scale_block(uint4 a, uint32_t r2) {
  return make_uint4(hmul2_rn(r2, a.x), hmul2_rn(r2, a.y), hmul2_rn(r2, a.z), hmul2_rn(r2, a.w));
}

__device__ __forceinline__ uint32_t bcast_lo(uint32_t r) { return prmt<0x1010u>(r, 0u); }
__device__ __forceinline__ uint32_t bcast_hi(uint32_t r) { return prmt<0x3232u>(r, 0u); }

__device__ __forceinline__ uint4 lds16(uint32_t saddr) {
  uint4 v;
  asm volatile("ld.shared.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "r"(saddr));
  return v;
}

// Codebook access.  W2: eight interleaved copies in shared memory, entry k of
// copy c at byte 128*k + 16*c; lane l uses copy l % 8 (the eight lanes of a
// quarter-warp then touch eight distinct 16-byte bank groups).  W3: a single
// copy, entry k at byte 16*k.  `base` is a shared-memory address, or for the
// global-memory variant used by the decode kernel a generic pointer.
struct SmemCodebook {
  const uint8_t* base;  // the shared-memory table (a __shared__ array)
  uint32_t copyoff;     // W2: 16 * (lane % 8), W3: 0
  __device__ __forceinline__ uint4 at(uint32_t off) const {
    return *reinterpret_cast<const uint4*>(base + off);
  }
};
struct GlobalCodebook {
  const uint8_t* base;  // K x 16 B
  __device__ __forceinline__ uint4 at(uint32_t off) const {
    return *reinterpret_cast<const uint4*>(base + off);
  }
};

// Signed directions of the two vectors of word m of a W2 unit (A = row gid,
// B = row gid+8).  `e` is the lane's pair-3 sign word aligned to bits 8-15 /
// 24-31.  Codebook offsets: 128*k + copy offset (interleaved smem copies) or
// 16*k (a plain table).
template <class CB>
__device__ __forceinline__ void directions_w2(uint32_t W, uint32_t e, int m, const CB& cb,
                                              uint32_t copyoff, bool interleaved, uint4& sa,
                                              uint4& sb) {
  const uint32_t w3 = shl_fma<3>(W);
  uint32_t offA, offB;
  if (interleaved) {
    offA = (w3 & 0x1F80u) | copyoff;
    offB = ((W >> 13) & 0x1F80u) | copyoff;
  } else {
    offA = (W & 0x3F0u);
    offB = (W >> 16) & 0x3F0u;
  }
  const uint4 ca = cb.at(offA);
  const uint4 cbv = cb.at(offB);
  const uint32_t ea = shl_fma_rt(e, 2 * m);
  const uint32_t eb = shl_fma_rt(e, 2 * m + 1);
  sa = apply_signs(ca, W, shl_fma<1>(W), shl_fma<2>(W), ea);
  sb = apply_signs(cbv, w3, shl_fma<4>(W), shl_fma<5>(W), eb);
}

// The lane's pair-3 sign word of a W2 unit, aligned to bits 8-15 / 24-31.
__device__ __forceinline__ uint32_t w2_sign3(const Unit<2>& u, int q) {
  const uint32_t s = u.s;
  return (q & 1) ? (s << 8) : s;
}
__device__ __forceinline__ uint32_t params_delta(uint32_t pa, uint32_t pb) {
  return prmt<0x5410u>(pa, pb);
}
__device__ __forceinline__ uint32_t params_rmin(uint32_t pa, uint32_t pb) {
  return prmt<0x7632u>(pa, pb);
}

// Signed directions of word m of a W3 unit.  The index-bit-12 word is
// rotated by (12 - 4q - m) mod 32 to bring the lane's pair to bits 12 / 28.
template <class CB>
__device__ __forceinline__ void directions_w3(const Unit<3>& u, int m, int q, const CB& cb,
                                              uint4& sa, uint4& sb) {
  const uint32_t W = word_of(u.w, m);
  uint32_t mid;
  if (m == 0) mid = u.mq.x;
  else if (m == 1) mid = u.mq.x >> 4;
  else if (m == 2) mid = shl_fma<8>(u.mq.x);
  else mid = shl_fma<4>(u.mq.x);
  const uint32_t top = rotl(u.top, (uint32_t)(12 - 4 * q - m) & 31u);
  // bits 8-11 from mid, bit 12 from top (bits above 12 / 28 are don't-care)
  const uint32_t hi = (mid & 0x0F000F00u) | (top & ~0x0F000F00u);
  const uint32_t k2 = (W & 0x00FF00FFu) | (hi & ~0x00FF00FFu);
  const uint32_t offA = shl_fma<4>(k2) & 0x1FFF0u;
  const uint32_t offB = (k2 >> 12) & 0x1FFF0u;
  const uint4 ca = cb.at(offA);
  const uint4 cbv = cb.at(offB);
  sa = apply_signs(ca, W, shl_fma<1>(W), shl_fma<2>(W), shl_fma<3>(W));
  sb = apply_signs(cbv, shl_fma<4>(W), shl_fma<5>(W), shl_fma<6>(W), shl_fma<7>(W));
}

// The two bytes of word m of a 3-bit-radius W3 unit moved to bits 8-15 (A)
// and 24-31 (B) of a zeroed word: index bits 8-12 at 8-12 / 24-28, radius
// code at 13-15 / 29-31.
__device__ __forceinline__ uint32_t w3v3_hi(const Unit<kFmtW3V3>& u, int m) {
  const uint32_t h = (m < 2) ? u.hi.x : u.hi.y;
  return (m & 1) ? prmt<0x3424u>(h, 0u) : prmt<0x1404u>(h, 0u);
}

// Signed directions of word m of a 3-bit-radius W3 unit.
template <class CB>
__device__ __forceinline__ void directions_w3v3(const Unit<kFmtW3V3>& u, int m, const CB& cb,
                                                uint4& sa, uint4& sb) {
  const uint32_t W = word_of(u.w, m);
  const uint32_t k2 = (W & 0x00FF00FFu) | (w3v3_hi(u, m) & 0x1F001F00u);
  const uint32_t offA = shl_fma<4>(k2) & 0x1FFF0u;
  const uint32_t offB = (k2 >> 12) & 0x1FFF0u;
  const uint4 ca = cb.at(offA);
  const uint4 cbv = cb.at(offB);
  sa = apply_signs(ca, W, shl_fma<1>(W), shl_fma<2>(W), shl_fma<3>(W));
  sb = apply_signs(cbv, shl_fma<4>(W), shl_fma<5>(W), shl_fma<6>(W), shl_fma<7>(W));
}
// Radius codes of word m (A at bits 0-2, B at bits 16-18; bit 3 / 19 zero).
__device__ __forceinline__ uint32_t qpair_w3v3(const Unit<kFmtW3V3>& u, int m) {
  return w3v3_hi(u, m) >> 13;
}

// Radius codes of word m as a pair (A at bits 0-3, B at bits 16-19).
__device__ __forceinline__ uint32_t qpair_w2(uint32_t W) { return W; }
__device__ __forceinline__ uint32_t qpair_w3(const Unit<3>& u, int m) { return u.mq.y >> (4 * m); }

}  // namespace sphq
