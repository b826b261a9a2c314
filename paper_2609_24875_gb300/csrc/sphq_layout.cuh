// Device layout of packed SPHQuant codes and the per-vector decode shared by
// the GEMV and decode kernels.  sm_103a only.
//
// Device layout ("group tiles").  Rows are padded to a multiple of 32 and cut
// into row blocks of 32 rows (one row per lane of a warp).  For row block rb
// and radius group g (16 consecutive 8-D vectors = 128 columns, §3.1) one
// contiguous tile holds, for each of the 32 rows, the group's 16 vectors:
//
//   W2 (1280 B = 32 rows x 40 B: 2.25 bits/weight + 4 B of group parameters)
//     [0, 1024)     codes: chunk c in {0,1} (vectors 8c..8c+7), lane l:
//                   16 B at c*512 + l*16 = eight 16-bit words in the paper's
//                   W2 format (§3.4): bits [0,8) signs, [8,14) direction
//                   index, [14,16) the low 2 bits of the radius code
//     [1024, 1280)  lane l: 8 B at 1024 + l*8 = { the paper's per-group 32-bit
//                   word of high radius bits (vector j at bits [2j, 2j+2)),
//                   params = Delta_G (low 16 bits) | r_min_G (high 16 bits) }
//
//   W3 (1728 B = 32 rows x 54 B: 3.125 bits/weight + 4 B of group parameters)
//     [0, 1024)     codes: as W2 but each 16-bit word = signs (bits 0-7) |
//                   index bits 0-7 (bits 8-15)
//     [1024, 1536)  lane l: 16 B = { radius codes of vectors 0-7 (nibble j),
//                   radius codes 8-15, index bits 8-11 of vectors 0-7
//                   (nibble j), index bits 8-11 of vectors 8-15 }
//     [1536, 1664)  lane l: 4 B params, as W2
//     [1664, 1728)  lane l: 2 B, bit j = index bit 12 of vector j
//
// Tiles are stored in (rb, g) order, so a warp that walks the groups of one
// row block streams contiguous memory, and each warp-wide 16-byte load is
// 512 contiguous bytes.  No byte beyond the algorithmic payload is stored.
#pragma once
#include <cstdint>

namespace sphq {

constexpr int kVec = 8;                 // 8-D vectors (§3.1)
constexpr int kGroupVecs = 16;          // vectors per radius group
constexpr int kGroupCols = kVec * kGroupVecs;
constexpr int kRowsPerBlock = 32;       // rows per tile (one per lane)
constexpr int kMaxBatch = 8;

template <int BITS> struct Layout;
template <> struct Layout<2> {
  static constexpr int K = 64;
  static constexpr int kTileBytes = 1280;
  static constexpr int kAuxOff = 1024;
};
template <> struct Layout<3> {
  static constexpr int K = 8192;
  static constexpr int kTileBytes = 1728;
  static constexpr int kAuxOff = 1024;
  static constexpr int kParamOff = 1536;
  static constexpr int kTopOff = 1664;
};

// Per-lane data of one group tile.
template <int BITS> struct GroupData;
template <> struct GroupData<2> {
  uint4 code[2];      // 16 x 16-bit words
  uint32_t extra;     // high radius bits
  uint32_t params;    // Delta | r_min << 16 (fp16 bits)
};
template <> struct GroupData<3> {
  uint4 code[2];      // 16 x (signs | index bits 0-7)
  uint4 aux;          // radius nibbles (x: 0-7, y: 8-15), index-hi nibbles (z: 0-7, w: 8-15)
  uint32_t params;
  uint32_t top;       // 16 bits: index bit 12
};

__device__ __forceinline__ uint4 ldg_stream16(const void* p) {
  uint4 v;
  asm volatile("ld.global.nc.L1::no_allocate.v4.u32 {%0,%1,%2,%3}, [%4];"
               : "=r"(v.x), "=r"(v.y), "=r"(v.z), "=r"(v.w) : "l"(p));
  return v;
}
__device__ __forceinline__ uint2 ldg_stream8(const void* p) {
  uint2 v;
  asm volatile("ld.global.nc.L1::no_allocate.v2.u32 {%0,%1}, [%2];"
               : "=r"(v.x), "=r"(v.y) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ldg_stream4(const void* p) {
  uint32_t v;
  asm volatile("ld.global.nc.L1::no_allocate.u32 %0, [%1];" : "=r"(v) : "l"(p));
  return v;
}
__device__ __forceinline__ uint32_t ldg_stream2(const void* p) {
  unsigned short v;
  asm volatile("ld.global.nc.L1::no_allocate.u16 %0, [%1];" : "=h"(v) : "l"(p));
  return v;
}

template <int BITS>
__device__ __forceinline__ GroupData<BITS> load_group(const uint8_t* tile, int lane);

template <>
__device__ __forceinline__ GroupData<2> load_group<2>(const uint8_t* tile, int lane) {
  GroupData<2> d;
  d.code[0] = ldg_stream16(tile + lane * 16);
  d.code[1] = ldg_stream16(tile + 512 + lane * 16);
  uint2 a = ldg_stream8(tile + Layout<2>::kAuxOff + lane * 8);
  d.extra = a.x;
  d.params = a.y;
  return d;
}

template <>
__device__ __forceinline__ GroupData<3> load_group<3>(const uint8_t* tile, int lane) {
  GroupData<3> d;
  d.code[0] = ldg_stream16(tile + lane * 16);
  d.code[1] = ldg_stream16(tile + 512 + lane * 16);
  d.aux = ldg_stream16(tile + Layout<3>::kAuxOff + lane * 16);
  d.params = ldg_stream4(tile + Layout<3>::kParamOff + lane * 4);
  d.top = ldg_stream2(tile + Layout<3>::kTopOff + lane * 2);
  return d;
}

__device__ __forceinline__ uint32_t word16(const GroupData<2>& d, int j) {
  const uint4& c = d.code[j >> 3];
  const int w = (j >> 1) & 3;
  uint32_t v = (w == 0) ? c.x : (w == 1) ? c.y : (w == 2) ? c.z : c.w;
  return (j & 1) ? (v >> 16) : (v & 0xFFFFu);
}
__device__ __forceinline__ uint32_t word16(const GroupData<3>& d, int j) {
  const uint4& c = d.code[j >> 3];
  const int w = (j >> 1) & 3;
  uint32_t v = (w == 0) ? c.x : (w == 1) ? c.y : (w == 2) ? c.z : c.w;
  return (j & 1) ? (v >> 16) : (v & 0xFFFFu);
}

// Unpacked fields of vector j (0..15) of a group: sign byte, direction index,
// radius code.  j must be a compile-time constant after unrolling.
struct Fields {
  uint32_t sign, k, q;
};

__device__ __forceinline__ Fields unpack(const GroupData<2>& d, int j) {
  const uint32_t w = word16(d, j);
  Fields f;
  f.sign = w & 0xFFu;
  f.k = (w >> 8) & 0x3Fu;
  f.q = (w >> 14) | (((d.extra >> (2 * j)) & 3u) << 2);
  return f;
}

__device__ __forceinline__ Fields unpack(const GroupData<3>& d, int j) {
  const uint32_t w = word16(d, j);
  const uint32_t qw = (j < 8) ? d.aux.x : d.aux.y;
  const uint32_t hw = (j < 8) ? d.aux.z : d.aux.w;
  const int n = 4 * (j & 7);
  Fields f;
  f.sign = w & 0xFFu;
  f.k = (w >> 8) | (((hw >> n) & 0xFu) << 8) | (((d.top >> j) & 1u) << 12);
  f.q = (qw >> n) & 0xFu;
  return f;
}

// ---------------------------------------------------------------------------
// fp16 arithmetic with explicit round-to-nearest-even and no contraction
// ---------------------------------------------------------------------------

__device__ __forceinline__ uint32_t hmul2_rn(uint32_t a, uint32_t b) {
  uint32_t d;
  asm("mul.rn.f16x2 %0, %1, %2;" : "=r"(d) : "r"(a), "r"(b));
  return d;
}

__device__ __forceinline__ uint16_t hfma_rn(uint16_t a, uint16_t b, uint16_t c) {
  uint16_t d;
  asm("fma.rn.f16 %0, %1, %2, %3;" : "=h"(d) : "h"(a), "h"(b), "h"(c));
  return d;
}

__device__ __forceinline__ uint16_t hsub_rn(uint16_t a, uint16_t b) {
  uint16_t d;
  asm("sub.rn.f16 %0, %1, %2;" : "=h"(d) : "h"(a), "h"(b));
  return d;
}

// r_hat = RN16(q * Delta + r_min): Eq. (7), one fp16 fused multiply-add.
// q (0..15) becomes an exact fp16 value through 1024 + q (bits 0x6400 | q) - 1024.
__device__ __forceinline__ uint16_t radius16(uint32_t q, uint32_t params) {
  const uint16_t qh = hsub_rn((uint16_t)(0x6400u | q), (uint16_t)0x6400u);
  return hfma_rn(qh, (uint16_t)(params & 0xFFFFu), (uint16_t)(params >> 16));
}

// Sign mask for coordinate pair p (coordinates 2p, 2p+1) of a half2 register.
__device__ __forceinline__ uint32_t sign_mask(uint32_t s, int p) {
  const uint32_t t = s >> (2 * p);
  return ((t << 15) & 0x8000u) | ((t << 30) & 0x80000000u);
}

// w_hat = s (.) RN16(r_hat * c): Eq. (4) on one block, as four half2 pairs.
__device__ __forceinline__ uint4 reconstruct(uint32_t sign, uint16_t r_hat, uint4 c) {
  const uint32_t r2 = (uint32_t)r_hat | ((uint32_t)r_hat << 16);
  uint4 w;
  w.x = hmul2_rn(r2, c.x) ^ sign_mask(sign, 0);
  w.y = hmul2_rn(r2, c.y) ^ sign_mask(sign, 1);
  w.z = hmul2_rn(r2, c.z) ^ sign_mask(sign, 2);
  w.w = hmul2_rn(r2, c.w) ^ sign_mask(sign, 3);
  return w;
}

// acc += w.lo * x.lo + w.hi * x.hi with fp16 inputs and fp32 accumulation:
// each product is exact in fp32 and added with one rounding.
__device__ __forceinline__ float fma_h2_f32(uint32_t w2, uint32_t x2, float acc) {
  asm("{\n\t.reg .f16 wl, wh, xl, xh;\n\t"
      "mov.b32 {wl, wh}, %1;\n\t"
      "mov.b32 {xl, xh}, %2;\n\t"
      "fma.rn.f32.f16 %0, wl, xl, %0;\n\t"
      "fma.rn.f32.f16 %0, wh, xh, %0;\n\t}"
      : "+f"(acc) : "r"(w2), "r"(x2));
  return acc;
}

__device__ __forceinline__ uint32_t f32x2_to_h2_rn(float lo, float hi) {
  uint32_t d;
  asm("cvt.rn.f16x2.f32 %0, %1, %2;" : "=r"(d) : "f"(hi), "f"(lo));
  return d;
}

__device__ __forceinline__ uint16_t f32_to_h_rn(float v) {
  uint16_t d;
  asm("cvt.rn.f16.f32 %0, %1;" : "=h"(d) : "f"(v));
  return d;
}

}  // namespace sphq
