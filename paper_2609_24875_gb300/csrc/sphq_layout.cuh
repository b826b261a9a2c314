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
// Small-codebook splits (Tab. 4: 8 sign bits, a D-bit direction index with
// K = 2^D entries, D = 6..8, and V-bit radius codes, D + V <= 10).  The W2
// unit above is the D = 6, V = 4 member; the others keep its word layout with
// their field widths:
//   word w_m, A in the low and B in the high 16 bits: radius code at bits
//   0..V-1 (16..), direction index at V..V+D-1 (16+V..); then sign pairs from
//   the top: A's pairs p at bits 15-p / 31-p, B's at (15-NA-p) / (31-NA-p),
//   where NA = 4 if D + V <= 9 else 3, NB = 4 if D + V = 8 else 3.  Pairs that
//   do not fit (D + V - 8 per vector) go to a record per quad:
//     D + V = 10: the W2 record, { S01, S23, P_gid, P_gid+8 } at 512 + 16*gid
//                 (640 B per unit)
//     D + V = 9:  B's pair 3 only, one word R at 512 + 4*gid: bit 15-4q-m
//                 = sign bit 6 and bit 31-4q-m = sign bit 7 of B of lane q's
//                 word m; then { P_gid, P_gid+8 } at 544 + 8*gid (608 B)
//     D + V = 8:  no record; { P_gid, P_gid+8 } at 512 + 8*gid (576 B)
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
// 4-D vectors (format id 10, Tab. 7 at the W2 allocation: 4 sign bits, a
// 2-bit index into K = 4 directions, a 4-bit radius code; 704 B = 512
// vectors x 10 bits + 64 B params).  Lane l = 4*gid + q owns rows gid (A) and
// gid+8 (B) at the group's vectors 4s+q, s = 0..7 ("pair s"); pair s fills
// the lane's K slots of the s-th MMA (one 4-D vector per lane and row):
//   [0, 512)    lane l: 16 B = { R0, R1, I, S0 }
//   [512, 640)  lane l: 4 B = S1
//   [640, 704)  quad gid: { P_gid, P_gid+8 }
//   R_{s/4}: radius code of A at bits 4(s%4)..+3, of B 16 bits higher
//   I: index of A at bits 2s..2s+1, of B at 16+2s..
//   S_{s/4}, j = s % 4: sign bits of A: coordinate 0 at 15-2j, 1 at 31-2j,
//     2 at 14-2j, 3 at 30-2j; of B: 0 at 7-2j, 1 at 23-2j, 2 at 6-2j, 3 at 22-2j
//     (each coordinate pair is one shift away from bits 15 / 31)
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

// Format ids used as template arguments, one per bit split (sign / direction
// index / radius bits): 2 = W2 (8/6/4), 3 = W3 (8/13/4), 4 = W3 with 3-bit
// radius codes (8/13/3), and the small-codebook splits of Tab. 4:
// 5 = 8/6/2, 6 = 8/6/3, 7 = 8/7/2, 8 = 8/7/3, 9 = 8/8/2.
constexpr int kFmtW3V3 = 4;
constexpr int kFmt862 = 5, kFmt863 = 6, kFmt872 = 7, kFmt873 = 8, kFmt882 = 9;
// 4-D vectors at the W2 allocation (Tab. 7): 4 sign bits, a 2-bit index into
// K = 4 directions, a 4-bit radius code (2.5 bits per weight).
constexpr int kFmt4D = 10;
// 16-D vectors at the W2 allocation (Tab. 7): 16 sign bits, a 14-bit index
// into K = 16384 directions (a 512 KiB codebook, gathered from global memory),
// a 4-bit radius code (2.125 bits per weight); kernels in sphq_dim16.cu.
constexpr int kFmt16D = 11;
__host__ __device__ constexpr int fmt_dir_bits(int fmt) {
  return fmt == 3 || fmt == 4 ? 13 : fmt == 7 || fmt == 8 ? 7 : fmt == 9 ? 8 : fmt == kFmt4D ? 2
         : fmt == kFmt16D ? 14 : 6;
}
__host__ __device__ constexpr int fmt_radius_bits(int fmt) {
  return fmt == 2 || fmt == 3 || fmt == kFmt4D || fmt == kFmt16D ? 4
         : fmt == 4 || fmt == 6 || fmt == 8 ? 3 : 2;
}
// vector dimension of a format
__host__ __device__ constexpr int fmt_dim(int fmt) {
  return fmt == kFmt4D ? 4 : fmt == kFmt16D ? 16 : 8;
}
// formats whose codebook (K <= 256) is kept as eight interleaved copies
__host__ __device__ constexpr bool fmt_small(int fmt) { return fmt == 2 || (fmt >= 5 && fmt <= 9); }
// format id of a split, or -1
__host__ __device__ constexpr int fmt_of_split(int dir_bits, int radius_bits) {
  return dir_bits == 13 ? (radius_bits == 4 ? 3 : radius_bits == 3 ? 4 : -1)
         : dir_bits == 6 ? (radius_bits == 4 ? 2 : radius_bits == 2 ? 5 : radius_bits == 3 ? 6 : -1)
         : dir_bits == 7 ? (radius_bits == 2 ? 7 : radius_bits == 3 ? 8 : -1)
         : dir_bits == 8 ? (radius_bits == 2 ? 9 : -1)
                         : -1;
}

// Small-codebook splits (W2 included).
template <int BITS> struct Layout {
  static_assert(fmt_small(BITS), "unknown format");
  static constexpr int D = fmt_dir_bits(BITS), V = fmt_radius_bits(BITS);
  static constexpr int K = 1 << D;
  static constexpr int kExtra = D + V - 8;    // sign bits per vector kept outside the words
  static constexpr int NA = kExtra <= 1 ? 4 : 3;  // sign pairs of A / B inside a word
  static constexpr int NB = kExtra == 0 ? 4 : 3;
  static constexpr int kRecOff = 512;
  static constexpr int kParamOff = kExtra == 2 ? 520 : kExtra == 1 ? 544 : 512;
  static constexpr int kParamStride = kExtra == 2 ? 16 : 8;  // bytes between quads' params
  static constexpr int kUnitBytes = kExtra == 2 ? 640 : kExtra == 1 ? 608 : 576;
  static_assert(kExtra >= 0 && kExtra <= 2, "split does not fit the word layout");
};
template <> struct Layout<kFmtW3V3> {
  static constexpr int K = 8192;
  static constexpr int kUnitBytes = 832;
  static constexpr int kHiOff = 512;
  static constexpr int kParamOff = 768;
};
// 4-D unit: 704 B = 512 vectors x 10 bits + 16 x 4 B params; see the
// format description at the top.
template <> struct Layout<kFmt4D> {
  static constexpr int K = 4;
  static constexpr int kUnitBytes = 704;
  static constexpr int kS1Off = 512;
  static constexpr int kParamOff = 640;
};
// 16-D unit (16 rows x 128 columns = 128 vectors): 608 B = 128 words of 32
// bits + 8 radius words + 8 parameter pairs; see sphq_dim16.cu.
template <> struct Layout<kFmt16D> {
  static constexpr int K = 16384;
  static constexpr int kUnitBytes = 608;
  static constexpr int kHiOff = 512;
  static constexpr int kParamOff = 544;
};
template <> struct Layout<3> {
  static constexpr int K = 8192;
  static constexpr int kUnitBytes = 864;
  static constexpr int kMidOff = 512;
  static constexpr int kParamOff = 768;
  static constexpr int kTopOff = 832;
};

// Unit bytes of a format (host-side mirror of Layout<F>::kUnitBytes).
__host__ __device__ constexpr int fmt_unit_bytes(int fmt) {
  return fmt == 3 ? Layout<3>::kUnitBytes
         : fmt == kFmtW3V3 ? Layout<kFmtW3V3>::kUnitBytes
         : fmt == kFmt4D ? Layout<kFmt4D>::kUnitBytes
         : fmt == kFmt16D ? Layout<kFmt16D>::kUnitBytes
         : fmt_dir_bits(fmt) + fmt_radius_bits(fmt) == 10 ? 640
         : fmt_dir_bits(fmt) + fmt_radius_bits(fmt) == 9 ? 608
                                                          : 576;
}
static_assert(fmt_unit_bytes(2) == Layout<2>::kUnitBytes && fmt_unit_bytes(5) == Layout<5>::kUnitBytes &&
                  fmt_unit_bytes(6) == Layout<6>::kUnitBytes && fmt_unit_bytes(7) == Layout<7>::kUnitBytes &&
                  fmt_unit_bytes(8) == Layout<8>::kUnitBytes && fmt_unit_bytes(9) == Layout<9>::kUnitBytes,
              "unit sizes");

// Per-lane data of one unit.
// Small-codebook splits: s is the lane's word of the quad's sign record (W2
// record: S01 for q < 2, S23 otherwise; one extra bit: R; none: 0).
template <int BITS> struct Unit {
  uint4 w;      // words w_0..w_3
  uint32_t s;
  uint2 par;    // {P_gid, P_gid+8}
};
template <> struct Unit<kFmtW3V3> {
  uint4 w;
  uint2 hi;     // {H0, H1}
  uint2 par;    // {P_gid, P_gid+8}
};
template <> struct Unit<kFmt4D> {
  uint4 w;      // {R0, R1, I, S0}
  uint32_t s1;  // S1
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

// Small-codebook splits (the W3 formats are specialised below).
template <int BITS>
__device__ __forceinline__ Unit<BITS> load_unit(const uint8_t* unit, int lane) {
  using L = Layout<BITS>;
  Unit<BITS> u;
  u.w = ldg_stream16(unit + lane * 16);
  if constexpr (L::kExtra == 2) {
    const uint8_t* rec = unit + L::kRecOff + (lane >> 2) * 16;
    u.s = ldg_stream4(rec + 4 * ((lane >> 1) & 1));
    u.par = ldg_stream8(rec + 8);
  } else if constexpr (L::kExtra == 1) {
    u.s = ldg_stream4(unit + L::kRecOff + (lane >> 2) * 4);
    u.par = ldg_stream8(unit + L::kParamOff + (lane >> 2) * 8);
  } else {
    u.s = 0;
    u.par = ldg_stream8(unit + L::kParamOff + (lane >> 2) * 8);
  }
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

template <>
__device__ __forceinline__ Unit<kFmt4D> load_unit<kFmt4D>(const uint8_t* unit, int lane) {
  Unit<kFmt4D> u;
  u.w = ldg_stream16(unit + lane * 16);
  u.s1 = ldg_stream4(unit + Layout<kFmt4D>::kS1Off + lane * 4);
  u.par = ldg_stream8(unit + Layout<kFmt4D>::kParamOff + (lane >> 2) * 8);
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
// fp16 fused multiply-add per vector.  qpair holds the V-bit codes of A (bits
// 0..V-1) and B (bits 16..16+V-1); 1024 + q is an exact fp16 value (bits 0x6400 | q), so
// subtracting 1024 gives q exactly.  d2 / m2: (Delta, r_min) of rows (A, B).
// V < 4: only bits 0..V-1 (16..16+V-1) are codes.
template <int V = 4>
__device__ __forceinline__ uint32_t radius_pair(uint32_t qpair, uint32_t d2, uint32_t m2) {
  constexpr uint32_t kMask = ((1u << V) - 1u) * 0x00010001u;
  const uint32_t qh = (qpair & kMask) | 0x64006400u;
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
// 4-D: sixteen interleaved copies of the 8-byte entries, entry k of copy c at
// 128*k + 8*c; lane l uses copy l % 16 (a half warp's 8-byte loads then touch
// sixteen distinct bank pairs).
struct SmemCodebook {
  const uint8_t* base;  // the shared-memory table (a __shared__ array)
  uint32_t copyoff;     // W2: 16 * (lane % 8), 4-D: 8 * (lane % 16), W3: 0
  __device__ __forceinline__ uint4 at(uint32_t off) const {
    return *reinterpret_cast<const uint4*>(base + off);
  }
  __device__ __forceinline__ uint2 at8(uint32_t off) const {
    return *reinterpret_cast<const uint2*>(base + off);
  }
};
struct GlobalCodebook {
  const uint8_t* base;  // K x 16 B (4-D: K x 8 B)
  __device__ __forceinline__ uint4 at(uint32_t off) const {
    return *reinterpret_cast<const uint4*>(base + off);
  }
  __device__ __forceinline__ uint2 at8(uint32_t off) const {
    return *reinterpret_cast<const uint2*>(base + off);
  }
};

// Signed directions of pair s of a 4-D unit (A = row gid, B = row gid+8):
// two half2 registers per vector (coordinates 0-1, 2-3).  Codebook offsets
// 128*k + copy offset, or 8*k for a plain table.
template <int S, class CB>
__device__ __forceinline__ void directions_4d(const uint4& w, uint32_t s1, const CB& cb,
                                              uint32_t copyoff, bool interleaved, uint2& sa,
                                              uint2& sb) {
  const uint32_t I = w.z;
  const uint32_t Sw = S < 4 ? w.w : s1;
  constexpr int j = S & 3;
  // index of A at bits 2S..2S+1, of B at 16+2S..
  uint32_t ia, ib;
  if constexpr (2 * S <= 7) ia = shl_fma<7 - 2 * S>(I) & 0x180u;
  else ia = (I >> (2 * S - 7)) & 0x180u;
  ib = (I >> (9 + 2 * S)) & 0x180u;
  uint32_t offA, offB;
  if (interleaved) {
    offA = ia | copyoff;
    offB = ib | copyoff;
  } else {
    offA = ia >> 4;
    offB = ib >> 4;
  }
  const uint2 ca = cb.at8(offA);
  const uint2 cbv = cb.at8(offB);
  sa = make_uint2(ca.x ^ (shl_fma<2 * j>(Sw) & kSignMask), ca.y ^ (shl_fma<2 * j + 1>(Sw) & kSignMask));
  sb = make_uint2(cbv.x ^ (shl_fma<8 + 2 * j>(Sw) & kSignMask),
                  cbv.y ^ (shl_fma<9 + 2 * j>(Sw) & kSignMask));
}
// Radius codes of pair s (A at bits 0-3, B at 16-19).
template <int S>
__device__ __forceinline__ uint32_t qpair_4d(const uint4& w) {
  return (S < 4 ? w.x : w.y) >> (4 * (S & 3));
}

// Signed directions of the two vectors of word m of a small-codebook unit
// (W2 and the other splits of Tab. 4; A = row gid, B = row gid+8).  `e` is
// the lane's sign_extra word.  Codebook offsets: 128*k + copy offset
// (interleaved shared-memory copies) or 16*k (a plain table).
template <int FMT, class CB>
__device__ __forceinline__ void directions_small(uint32_t W, uint32_t e, int m, const CB& cb,
                                                 uint32_t copyoff, bool interleaved, uint4& sa,
                                                 uint4& sb) {
  using L = Layout<FMT>;
  constexpr int V = L::V, NA = L::NA;
  constexpr uint32_t kIdx = (uint32_t)L::K - 1u;
  uint32_t offA, offB;
  if (interleaved) {
    offA = (shl_fma<7 - V>(W) & (kIdx << 7)) | copyoff;
    offB = ((W >> (9 + V)) & (kIdx << 7)) | copyoff;
  } else {
    offA = shl_fma<4 - V>(W) & (kIdx << 4);
    offB = (W >> (12 + V)) & (kIdx << 4);
  }
  const uint4 ca = cb.at(offA);
  const uint4 cbv = cb.at(offB);
  // pair 3 of A: in the word (NA = 4) or in the W2 record; pair 3 of B: in
  // the word (NB = 4), in R (one extra bit) or in the W2 record
  uint32_t a3, b3;
  if constexpr (L::kExtra == 2) {
    a3 = shl_fma_rt(e, 2 * m);
    b3 = shl_fma_rt(e, 2 * m + 1);
  } else if constexpr (L::kExtra == 1) {
    a3 = shl_fma<3>(W);
    b3 = shl_fma_rt(e, m);
  } else {
    a3 = shl_fma<3>(W);
    b3 = shl_fma<7>(W);
  }
  sa = apply_signs(ca, W, shl_fma<1>(W), shl_fma<2>(W), a3);
  sb = apply_signs(cbv, shl_fma<NA>(W), shl_fma<NA + 1>(W), shl_fma<NA + 2>(W), b3);
}

// The lane's sign word for the pairs kept outside the words: the W2 record
// word aligned to bits 8-15 / 24-31, or R shifted by 4q; zero without a record.
template <int FMT>
__device__ __forceinline__ uint32_t sign_extra(const Unit<FMT>& u, int q) {
  if constexpr (Layout<FMT>::kExtra == 2) {
    const uint32_t s = u.s;
    return (q & 1) ? (s << 8) : s;
  } else if constexpr (Layout<FMT>::kExtra == 1) {
    return shl_fma_rt(u.s, 4 * q);
  } else {
    return 0u;
  }
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

// Radius codes of word m as a pair (A at bits 0-3, B at bits 16-19); the
// small-codebook words carry their codes at bits 0 / 16 already.
__device__ __forceinline__ uint32_t qpair_w3(const Unit<3>& u, int m) { return u.mq.y >> (4 * m); }

}  // namespace sphq
