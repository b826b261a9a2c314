// GEMV kernels of the small-codebook bit splits of Tab. 4 (8/6/2, 8/6/3,
// 8/7/2, 8/7/3, 8/8/2) and of 4-D vectors (Tab. 7), in a translation unit of
// their own so that the library's sources compile in parallel.
#include "sphq_gemv_kernel.cuh"

namespace sphq {

const void* split_kernel(int fmt, int mode) {
  switch (fmt) {
    case kFmt862: return kptr_mode<kFmt862>(mode);
    case kFmt863: return kptr_mode<kFmt863>(mode);
    case kFmt872: return kptr_mode<kFmt872>(mode);
    case kFmt873: return kptr_mode<kFmt873>(mode);
    case kFmt882: return kptr_mode<kFmt882>(mode);
    case kFmt4D: return kptr_mode<kFmt4D>(mode);
    default: return nullptr;
  }
}

}  // namespace sphq
