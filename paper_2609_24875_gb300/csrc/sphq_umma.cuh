// Fifth-generation tensor core (tcgen05) and tensor-memory-accelerator (TMA)
// primitives for sm_103a, as inline PTX: tensor-memory allocation, the
// shared-memory matrix descriptor of a K-major operand in the 128-byte swizzle
// layout, the instruction descriptor of an fp16 x fp16 -> fp32 MMA, MMA issue
// and completion, tensor-memory loads, and 2-D tiled TMA loads.
//
// Operand layouts (both operands K-major): a tile of R rows x 64 fp16 (128
// bytes per row) at a 1024-byte aligned base; row r occupies bytes
// [128 r, 128 r + 128), and its 16-byte chunk c (fp16 columns 8c..8c+7) is
// stored at chunk position c ^ (r % 8).  Eight rows form one 1024-byte
// swizzle atom; atoms follow each other (stride 1024 bytes).  This is the
// layout a TMA load with CU_TENSOR_MAP_SWIZZLE_128B and a box of 64 fp16
// columns writes.  With 32 fp16 per row (64 bytes) the 64-byte swizzle puts
// chunk c of row r at c ^ ((r / 2) % 4), 512-byte atoms
// (CU_TENSOR_MAP_SWIZZLE_64B, a box of 32 columns).
#pragma once
#include <cstdint>

namespace sphq {
namespace umma {

// ---------------------------------------------------------------------------
// descriptors
// ---------------------------------------------------------------------------

// Shared-memory matrix descriptor (64 bits) of a K-major, 128-byte-swizzled
// operand tile whose first row starts at shared address `saddr` (for the k-th
// 16-column slice of a 64-column tile, saddr = tile base + 32 k):
//   bits  0-13  start address >> 4
//   bits 16-29  leading-dimension byte offset >> 4 (unused by this layout; 1)
//   bits 32-45  stride byte offset >> 4: 1024 bytes between 8-row atoms
//   bits 46-47  descriptor version: 1
//   bits 49-51  base offset: 0 (atoms 1024-byte aligned)
//   bits 61-63  layout: 2 = 128-byte swizzle
__host__ __device__ constexpr uint64_t smem_desc_sw128(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(1024u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)2u << 61);
}

// The same for rows of 64 bytes (32 fp16) in the 64-byte swizzle: chunk c
// (0..3) of row r at chunk position c ^ ((r / 2) % 4), 8-row atoms of 512
// bytes (stride byte offset 512), layout 4 = 64-byte swizzle.
__host__ __device__ constexpr uint64_t smem_desc_sw64(uint32_t saddr) {
  return (uint64_t)((saddr >> 4) & 0x3FFFu) | ((uint64_t)1u << 16) | ((uint64_t)(512u >> 4) << 32) |
         ((uint64_t)1u << 46) | ((uint64_t)4u << 61);
}

// Instruction descriptor (32 bits) of tcgen05.mma .kind::f16 with fp16 A and
// B, fp32 accumulation, both operands K-major, an M x N tile:
//   bits  4-5   D format: 1 = f32
//   bits  7-9   A format: 0 = f16       bits 10-12  B format: 0 = f16
//   bit  15/16  A / B major: 0 = K-major
//   bits 17-22  N >> 3                  bits 24-28  M >> 4
__host__ __device__ constexpr uint32_t idesc_f16_f32(int M, int N) {
  return (1u << 4) | ((uint32_t)(N >> 3) << 17) | ((uint32_t)(M >> 4) << 24);
}

// ---------------------------------------------------------------------------
// tensor memory
// ---------------------------------------------------------------------------

// Allocates `ncols` (a power of two >= 32) tensor-memory columns for this CTA
// and writes their address to shared memory at `slot`.  Whole warp.
__device__ __forceinline__ void tmem_alloc(uint32_t slot, uint32_t ncols) {
  asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(slot),
               "r"(ncols)
               : "memory");
}
// Lets other CTAs on the SM allocate (this CTA allocates once).  Whole warp.
__device__ __forceinline__ void tmem_relinquish() {
  asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
}
// Whole warp.
__device__ __forceinline__ void tmem_dealloc(uint32_t taddr, uint32_t ncols) {
  asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(taddr), "r"(ncols)
               : "memory");
}

// Ordering of tcgen05 operations around thread synchronisation.
__device__ __forceinline__ void fence_before_sync() {
  asm volatile("tcgen05.fence::before_thread_sync;" ::: "memory");
}
__device__ __forceinline__ void fence_after_sync() {
  asm volatile("tcgen05.fence::after_thread_sync;" ::: "memory");
}

// Makes this thread's ordinary shared-memory stores visible to the async
// proxy (the tensor core and TMA read shared memory through it).
__device__ __forceinline__ void fence_proxy_async_smem() {
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
}

// ---------------------------------------------------------------------------
// MMA
// ---------------------------------------------------------------------------

// D[tmem] (+)= A * B^T for one instruction (K = 16 fp16); issued by one thread.
__device__ __forceinline__ void mma_f16(uint32_t d_tmem, uint64_t adesc, uint64_t bdesc,
                                       uint32_t idesc, uint32_t accumulate) {
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "setp.ne.b32 p, %4, 0;\n\t"
      "tcgen05.mma.cta_group::1.kind::f16 [%0], %1, %2, %3, p;\n\t}" ::"r"(d_tmem),
      "l"(adesc), "l"(bdesc), "r"(idesc), "r"(accumulate)
      : "memory");
}

// Arrives (once) on the mbarrier at shared address `bar` when every MMA this
// thread issued before has completed.
__device__ __forceinline__ void commit(uint32_t bar) {
  asm volatile(
      "tcgen05.commit.cta_group::1.mbarrier::arrive::one.shared::cluster.b64 [%0];" ::"r"(bar)
      : "memory");
}

// ---------------------------------------------------------------------------
// tensor-memory loads: lane = thread's lane within the warp's 32-lane quarter
// ---------------------------------------------------------------------------

// 32 consecutive 32-bit columns of this thread's lane, starting at taddr
// (lane field bits 16-31, column bits 0-15).  Whole warp; complete after wait_ld.
__device__ __forceinline__ void ld_32x32b_x32(uint32_t taddr, uint32_t (&v)[32]) {
  asm volatile(
      "tcgen05.ld.sync.aligned.32x32b.x32.b32 "
      "{%0,%1,%2,%3,%4,%5,%6,%7,%8,%9,%10,%11,%12,%13,%14,%15,"
      "%16,%17,%18,%19,%20,%21,%22,%23,%24,%25,%26,%27,%28,%29,%30,%31}, [%32];"
      : "=r"(v[0]), "=r"(v[1]), "=r"(v[2]), "=r"(v[3]), "=r"(v[4]), "=r"(v[5]), "=r"(v[6]),
        "=r"(v[7]), "=r"(v[8]), "=r"(v[9]), "=r"(v[10]), "=r"(v[11]), "=r"(v[12]), "=r"(v[13]),
        "=r"(v[14]), "=r"(v[15]), "=r"(v[16]), "=r"(v[17]), "=r"(v[18]), "=r"(v[19]),
        "=r"(v[20]), "=r"(v[21]), "=r"(v[22]), "=r"(v[23]), "=r"(v[24]), "=r"(v[25]),
        "=r"(v[26]), "=r"(v[27]), "=r"(v[28]), "=r"(v[29]), "=r"(v[30]), "=r"(v[31])
      : "r"(taddr)
      : "memory");
}
__device__ __forceinline__ void wait_ld() {
  asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
}

// ---------------------------------------------------------------------------
// TMA
// ---------------------------------------------------------------------------

// 2-D tiled load of the box at (x, y) (x: innermost coordinate in elements; x
// times the element size must be a multiple of 16 bytes) of the tensor map at
// generic address `tmap` into shared address `dst`, completing on the
// mbarrier at `bar`.  Coordinates past the tensor's extent read zeros.
__device__ __forceinline__ void tma_load_2d(uint32_t dst, const void* tmap, int x, int y,
                                            uint32_t bar) {
  asm volatile(
      "cp.async.bulk.tensor.2d.shared::cluster.global.tile.mbarrier::complete_tx::bytes "
      "[%0], [%1, {%2, %3}], [%4];" ::"r"(dst),
      "l"(tmap), "r"(x), "r"(y), "r"(bar)
      : "memory");
}
__device__ __forceinline__ void prefetch_tmap(const void* tmap) {
  asm volatile("prefetch.tensormap [%0];" ::"l"(tmap) : "memory");
}

}  // namespace umma
}  // namespace sphq
