// C ABI of the sphq library: handle lifetime, packing, decode, errors.
// The GEMV kernels live in sphq_gemv_kernel.cuh, their launch plans in sphq_gemv.cu.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <cstdlib>
#include <cstring>
#include <string>

#include "sphq_internal.h"
#include "sphq_layout.cuh"

namespace sphq {

// every format id (sphq_layout.cuh)
#define SPHQ_FOR_EACH_FMT(X) X(2) X(3) X(4) X(5) X(6) X(7) X(8) X(9)

static thread_local std::string g_last_error;
// zero block read by GEMV lanes that supply no activations (4 words x 4 lanes x 16 B)
constexpr size_t kZeroBytes = 256;

void clear_error() { g_last_error.clear(); }

// Host logging to stderr when the environment variable SPHQ_LOG is set
// (to anything but "0").
bool log_enabled() {
  static const bool on = [] {
    const char* v = std::getenv("SPHQ_LOG");
    return v && *v && std::strcmp(v, "0") != 0;
  }();
  return on;
}

sphq_status set_error(sphq_status s, const std::string& msg) {
  g_last_error = msg;
  return s;
}

sphq_status cuda_error(cudaError_t e, const char* what) {
  cudaGetLastError();  // clear sticky-free errors so the next call starts clean
  return set_error(e == cudaErrorMemoryAllocation ? SPHQ_ERR_OOM : SPHQ_ERR_CUDA,
                   std::string(what) + ": " + cudaGetErrorString(e));
}

#define SPHQ_CUDA(call, what)                      \
  do {                                             \
    cudaError_t e_ = (call);                       \
    if (e_ != cudaSuccess) return cuda_error(e_, what); \
  } while (0)

// ---------------------------------------------------------------------------
// pack: canonical codes -> units (the finalise-and-pack step, App. A step 10)
// ---------------------------------------------------------------------------

// One thread per (unit, lane): composes the lane's four words and its share of
// the quad records.  The unit buffer is zeroed before the launch, so padded
// rows keep zero codes and byte-wise record writes need no read-modify-write.
template <int BITS>
__global__ void pack_kernel(const uint8_t* __restrict__ sign, const uint16_t* __restrict__ idx,
                            const uint8_t* __restrict__ rcode,
                            const uint16_t* __restrict__ scale,
                            const uint16_t* __restrict__ offset, uint8_t* __restrict__ units,
                            int rows, int ng, int nrt, int* __restrict__ flag) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long total = (long long)nrt * ng * 32;
  if (tid >= total) return;
  const int lane = (int)(tid & 31);
  const long long unit = tid >> 5;  // unit_index(rt, g, nrt)
  const int rt = (int)(unit % nrt);
  const int g = (int)(unit / nrt);
  const int gid = lane >> 2, q = lane & 3;
  const int nv = ng * kGroupVecs;
  uint8_t* base = units + (size_t)unit * Layout<BITS>::kUnitBytes;

  constexpr bool kSmall = fmt_small(BITS);
  constexpr int kV = fmt_radius_bits(BITS);
  constexpr int kExtra = kSmall ? fmt_dir_bits(BITS) + kV - 8 : 0;
  uint32_t words[4] = {0, 0, 0, 0};
  uint32_t e_lo = 0, e_hi = 0;       // W2 record: pair-3 sign bytes of the lane
  uint32_t rword = 0;                // one extra bit per vector: the lane's bits of R
  uint32_t mid = 0, qn = 0, top = 0; // W3
  uint32_t hw[2] = {0, 0};            // W3, 3-bit radius: H0, H1
  bool bad = false;
  for (int m = 0; m < 4; ++m) {
    for (int half = 0; half < 2; ++half) {  // 0: A (row gid), 1: B (row gid + 8)
      const int row = rt * kRowsPerTile + gid + 8 * half;
      uint32_t s = 0, k = 0, rq = 0;
      if (row < rows) {
        const size_t v = (size_t)row * nv + (size_t)g * kGroupVecs + 4 * m + q;
        s = sign[v];
        k = idx[v];
        rq = rcode[v];
        if (k >= (uint32_t)Layout<BITS>::K || rq >= (1u << kV)) {
          bad = true;
          k = 0;
          rq = 0;
        }
      }
      const int v8 = 2 * m + half;   // vector number within the lane, 0..7
      const int hs = 16 * half;      // B's index/radius fields sit 16 bits higher
      // sign bits 2p / 2p+1 go to bits (top - p) / (top - p + 16), where top is
      // 15 for A and, below A's pairs, 15 - (A's pairs in the word) for B
      const int na = kSmall ? (kExtra <= 1 ? 4 : 3) : 4;
      const int nb = kSmall ? (kExtra == 0 ? 4 : 3) : 4;
      const int top_bit = half == 0 ? 15 : 15 - na;
      const int npairs = half == 0 ? na : nb;
      uint32_t w = 0;
      for (int p = 0; p < npairs; ++p) {
        w |= ((s >> (2 * p)) & 1u) << (top_bit - p);
        w |= ((s >> (2 * p + 1)) & 1u) << (top_bit - p + 16);
      }
      if (kSmall) {
        w |= (rq | (k << kV)) << hs;
        if (kExtra == 2) {
          e_lo |= ((s >> 6) & 1u) << (7 - v8);
          e_hi |= ((s >> 7) & 1u) << (7 - v8);
        } else if (kExtra == 1 && half == 1) {
          rword |= ((s >> 6) & 1u) << (15 - 4 * q - m);
          rword |= ((s >> 7) & 1u) << (31 - 4 * q - m);
        }
      } else if (BITS == kFmtW3V3) {
        w |= (k & 0xFFu) << hs;
        hw[m >> 1] |= (((k >> 8) & 0x1Fu) | (rq << 5)) << (8 * (2 * (m & 1) + half));
      } else {
        w |= (k & 0xFFu) << hs;
        qn |= rq << (4 * m + hs);
        mid |= ((k >> 8) & 0xFu) << (((8 + 4 * m) & 15) + hs);
        top |= ((k >> 12) & 1u) << (4 * q + m + hs);
      }
      words[m] |= w;
    }
  }
  if (bad) atomicOr(flag, 1);
  *reinterpret_cast<uint4*>(base + lane * 16) = make_uint4(words[0], words[1], words[2], words[3]);
  uint32_t pa = 0, pb = 0;
  const int ra = rt * kRowsPerTile + gid, rb = ra + 8;
  if (ra < rows) pa = (uint32_t)scale[(size_t)ra * ng + g] | ((uint32_t)offset[(size_t)ra * ng + g] << 16);
  if (rb < rows) pb = (uint32_t)scale[(size_t)rb * ng + g] | ((uint32_t)offset[(size_t)rb * ng + g] << 16);
  if constexpr (kSmall && kExtra == 2) {
    uint8_t* rec = base + Layout<BITS>::kRecOff + gid * 16;
    uint8_t* sw = rec + 4 * (q >> 1);          // S01 or S23
    const int b0 = (q & 1) ? 0 : 1;            // even lane: bytes 1, 3; odd lane: bytes 0, 2
    sw[b0] = (uint8_t)e_lo;
    sw[b0 + 2] = (uint8_t)e_hi;
    if (q == 0) {
      *reinterpret_cast<uint32_t*>(rec + 8) = pa;
      *reinterpret_cast<uint32_t*>(rec + 12) = pb;
    }
  } else if constexpr (kSmall) {
    if (kExtra == 1)
      atomicOr(reinterpret_cast<unsigned*>(base + Layout<BITS>::kRecOff + gid * 4), rword);
    if (q == 0)
      *reinterpret_cast<uint2*>(base + Layout<BITS>::kParamOff + gid * 8) = make_uint2(pa, pb);
  } else if constexpr (BITS == kFmtW3V3) {
    *reinterpret_cast<uint2*>(base + Layout<kFmtW3V3>::kHiOff + lane * 8) = make_uint2(hw[0], hw[1]);
    if (q == 0)
      *reinterpret_cast<uint2*>(base + Layout<kFmtW3V3>::kParamOff + gid * 8) = make_uint2(pa, pb);
  } else {
    *reinterpret_cast<uint2*>(base + Layout<3>::kMidOff + lane * 8) = make_uint2(mid, qn);
    if (q == 0)
      *reinterpret_cast<uint2*>(base + Layout<3>::kParamOff + gid * 8) = make_uint2(pa, pb);
    atomicOr(reinterpret_cast<unsigned*>(base + Layout<3>::kTopOff + gid * 4), top);
  }
}

// 4-D vectors: one thread per (unit, lane) composes the lane's five words
// (layout in sphq_layout.cuh).  sign: rows x cols/4 bytes (bits 0-3).
__global__ void pack4_kernel(const uint8_t* __restrict__ sign, const uint16_t* __restrict__ idx,
                             const uint8_t* __restrict__ rcode, const uint16_t* __restrict__ scale,
                             const uint16_t* __restrict__ offset, uint8_t* __restrict__ units,
                             int rows, int ng, int nrt, int* __restrict__ flag) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  if (tid >= (long long)nrt * ng * 32) return;
  const int lane = (int)(tid & 31);
  const long long unit = tid >> 5;
  const int rt = (int)(unit % nrt), g = (int)(unit / nrt);
  const int gid = lane >> 2, q = lane & 3;
  const int nv = ng * 32;
  uint8_t* base = units + (size_t)unit * Layout<kFmt4D>::kUnitBytes;
  uint32_t R[2] = {0, 0}, I = 0, S[2] = {0, 0};
  bool bad = false;
  for (int s = 0; s < 8; ++s) {
    for (int half = 0; half < 2; ++half) {
      const int row = rt * kRowsPerTile + gid + 8 * half;
      if (row >= rows) continue;
      const size_t v = (size_t)row * nv + (size_t)g * 32 + 4 * s + q;
      uint32_t sg = sign[v], k = idx[v], rq = rcode[v];
      if (k >= 4u || rq > 15u || sg > 15u) {
        bad = true;
        sg = k = rq = 0;
      }
      const int j = s & 3;
      const int top = (half ? 7 : 15) - 2 * j;  // coordinate 0's bit
      R[s >> 2] |= rq << (4 * j + 16 * half);
      I |= k << (2 * s + 16 * half);
      S[s >> 2] |= ((sg & 1u) << top) | (((sg >> 1) & 1u) << (top + 16)) |
                   (((sg >> 2) & 1u) << (top - 1)) | (((sg >> 3) & 1u) << (top + 15));
    }
  }
  if (bad) atomicOr(flag, 1);
  *reinterpret_cast<uint4*>(base + lane * 16) = make_uint4(R[0], R[1], I, S[0]);
  *reinterpret_cast<uint32_t*>(base + Layout<kFmt4D>::kS1Off + lane * 4) = S[1];
  if (q == 0) {
    uint32_t pa = 0, pb = 0;
    const int ra = rt * kRowsPerTile + gid, rb = ra + 8;
    if (ra < rows) pa = (uint32_t)scale[(size_t)ra * ng + g] | ((uint32_t)offset[(size_t)ra * ng + g] << 16);
    if (rb < rows) pb = (uint32_t)scale[(size_t)rb * ng + g] | ((uint32_t)offset[(size_t)rb * ng + g] << 16);
    *reinterpret_cast<uint2*>(base + Layout<kFmt4D>::kParamOff + gid * 8) = make_uint2(pa, pb);
  }
}

template <int S>
__device__ __forceinline__ void decode4_pair(const Unit<kFmt4D>& u, const GlobalCodebook& cb,
                                             uint2& wa, uint2& wb) {
  uint2 sa, sb;
  directions_4d<S>(u.w, u.s1, cb, 0u, false, sa, sb);
  const uint32_t r = radius_pair<4>(qpair_4d<S>(u.w), params_delta(u.par.x, u.par.y),
                                    params_rmin(u.par.x, u.par.y));
  const uint32_t ra = bcast_lo(r), rb = bcast_hi(r);
  wa = make_uint2(hmul2_rn(ra, sa.x), hmul2_rn(ra, sa.y));
  wb = make_uint2(hmul2_rn(rb, sb.x), hmul2_rn(rb, sb.y));
}

// W_hat of a 4-D matrix: one thread per vector.
__global__ void decode4_kernel(const uint8_t* __restrict__ units, const uint8_t* __restrict__ codebook,
                               uint16_t* __restrict__ w, int rows, int cols, int nrt) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int nv = cols / 4;
  if (tid >= (long long)rows * nv) return;
  const int row = (int)(tid / nv), t = (int)(tid % nv);
  const int rt = row / kRowsPerTile, r16 = row % kRowsPerTile;
  const int gid = r16 & 7, half = r16 >> 3;
  const int g = t / 32, s = (t % 32) / 4, q = t % 4;
  const Unit<kFmt4D> u = load_unit<kFmt4D>(
      units + (size_t)unit_index(rt, g, nrt) * Layout<kFmt4D>::kUnitBytes, 4 * gid + q);
  const GlobalCodebook cb{codebook};
  uint2 wa, wb;
  switch (s) {
    case 0: decode4_pair<0>(u, cb, wa, wb); break;
    case 1: decode4_pair<1>(u, cb, wa, wb); break;
    case 2: decode4_pair<2>(u, cb, wa, wb); break;
    case 3: decode4_pair<3>(u, cb, wa, wb); break;
    case 4: decode4_pair<4>(u, cb, wa, wb); break;
    case 5: decode4_pair<5>(u, cb, wa, wb); break;
    case 6: decode4_pair<6>(u, cb, wa, wb); break;
    default: decode4_pair<7>(u, cb, wa, wb); break;
  }
  *reinterpret_cast<uint2*>(w + (size_t)row * cols + (size_t)t * 4) = half ? wb : wa;
}

// ---------------------------------------------------------------------------
// decode: W_hat (rows x cols fp16), through the same unpack/reconstruct code
// ---------------------------------------------------------------------------

template <int BITS>
__global__ void decode_kernel(const uint8_t* __restrict__ units, const uint8_t* __restrict__ codebook,
                              uint16_t* __restrict__ w, int rows, int cols, int ng, int nrt) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int nv = cols / kVec;
  if (tid >= (long long)rows * nv) return;
  const int row = (int)(tid / nv);
  const int t = (int)(tid % nv);
  const int rt = row / kRowsPerTile, r16 = row % kRowsPerTile;
  const int gid = r16 & 7, half = r16 >> 3;
  const int g = t / kGroupVecs, s = t % kGroupVecs;
  const int m = s >> 2, q = s & 3;
  const int lane = 4 * gid + q;
  const uint8_t* unit = units + (size_t)unit_index(rt, g, nrt) * Layout<BITS>::kUnitBytes;
  const Unit<BITS> u = load_unit<BITS>(unit, lane);
  GlobalCodebook cb{codebook};
  uint4 sa, sb;
  uint32_t r;
  if constexpr (fmt_small(BITS)) {
    const uint32_t W = word_of(u.w, m);
    directions_small<BITS>(W, sign_extra<BITS>(u, q), m, cb, 0u, false, sa, sb);
    r = radius_pair<fmt_radius_bits(BITS)>(W, params_delta(u.par.x, u.par.y),
                                           params_rmin(u.par.x, u.par.y));
  } else if constexpr (BITS == kFmtW3V3) {
    directions_w3v3(u, m, cb, sa, sb);
    r = radius_pair<3>(qpair_w3v3(u, m), params_delta(u.par.x, u.par.y),
                       params_rmin(u.par.x, u.par.y));
  } else {
    directions_w3(u, m, q, cb, sa, sb);
    r = radius_pair(qpair_w3(u, m), params_delta(u.par.x, u.par.y),
                    params_rmin(u.par.x, u.par.y));
  }
  // Eq. (4): w_hat = RN16(r_hat * (s (.) c))
  const uint4 wa = scale_block(sa, bcast_lo(r));
  const uint4 wb = scale_block(sb, bcast_hi(r));
  *reinterpret_cast<uint4*>(w + (size_t)row * cols + (size_t)t * kVec) = half ? wb : wa;
}

}  // namespace sphq

using namespace sphq;

extern "C" {

int sphq_version(void) { return 10300; }

sphq_status sphq_get_plan(sphq_handle h, int batch, sphq_plan_info* out) {
  g_last_error.clear();
  if (!h || !out) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_get_plan: NULL handle or out");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_get_plan: batch must be 1..16");
  const GemvPlan& p = h->plan[batch];
  out->grid = p.grid;
  out->cluster_size = p.csize;
  out->clusters = p.nclusters;
  out->tiles_per_cluster = p.tmax;
  out->warps_per_cta = p.warps_per_cta;
  out->smem_bytes = (int)p.smem;
  out->staged_x = p.grid > 0 && p.mode <= 2;  // factored modes (1-2 rows) stage x
  out->ctas_per_sm = p.ctas_per_sm;
  return SPHQ_OK;
}

sphq_status sphq_set_cluster_size(sphq_handle h, int batch, int cluster_size) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_cluster_size: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_cluster_size: batch must be 1..16");
  if (cluster_size != 0 && cluster_size != 1 && cluster_size != 2 && cluster_size != 4 &&
      cluster_size != 8)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_cluster_size: size must be 0, 1, 2, 4 or 8");
  if (cluster_size > h->ng)
    return set_error(SPHQ_ERR_UNSUPPORTED,
                     "sphq_set_cluster_size: more CTAs per cluster than 128-column groups");
  int dev = -1;
  SPHQ_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  if (dev != h->device)
    return set_error(SPHQ_ERR_DEVICE, "sphq_set_cluster_size: current device is not the handle's");
  return set_gemv_cluster_size(h, batch, cluster_size);
}

sphq_status sphq_set_pdl(sphq_handle h, int enabled) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_pdl: NULL handle");
  if (enabled != 0 && enabled != 1)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_pdl: enabled must be 0 or 1");
  h->pdl = enabled != 0;
  return SPHQ_OK;
}

const char* sphq_last_error(void) { return g_last_error.c_str(); }

static void free_handle(sphq_handle h) {
  if (!h) return;
  cudaFree(h->units);
  cudaFree(h->codebook);
  cudaFree(h->params);
  cudaFree(h->ws);
  cudaFree(h->cbimage);
  cudaFree(h->flag);
  cudaFree(h->xstage);
  cudaFree(h->ystage);
  cudaFree(h->zeros);
  delete h;
}

sphq_status sphq_create(int rows, int cols, int bits, int K, const void* codebook,
                        const void* scale, const void* offset, sphq_handle* out) {
  return sphq_create_v(rows, cols, bits, 4, K, codebook, scale, offset, out);
}

static sphq_status create_impl(int rows, int cols, int dim, int bits, int radius_bits, int K,
                               const void* codebook, const void* scale, const void* offset,
                               sphq_handle* out) {
  g_last_error.clear();
  if (!out) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_create: out is NULL");
  *out = nullptr;
  if (rows < 1 || cols < kGroupCols || cols % kGroupCols != 0)
    return set_error(SPHQ_ERR_INVALID_ARG,
                     "sphq_create: need rows >= 1 and cols a positive multiple of 128");
  if (bits != 2 && bits != 3)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_create: bits must be 2 or 3");
  int dbits = -1;
  for (int d = 0; d < 31; ++d)
    if (K == (1 << d)) dbits = d;
  int fmt = -1;
  if (dim == 4) {
    // Tab. 7, W2 allocation: 3B - 4 = 2 index bits (K = 4), V = 4
    if (bits != 2 || K != 4 || radius_bits != 4)
      return set_error(SPHQ_ERR_UNSUPPORTED,
                       "sphq_create_dim: 4-D vectors take bits = 2, K = 4, radius_bits = 4");
    fmt = kFmt4D;
  } else if (dim == 16) {
    // Tab. 7, W2 allocation: 15 B - 16 = 14 index bits (K = 16384), V = 4
    if (bits != 2 || K != 16384 || radius_bits != 4)
      return set_error(SPHQ_ERR_UNSUPPORTED,
                       "sphq_create_dim: 16-D vectors take bits = 2, K = 16384, radius_bits = 4");
    fmt = kFmt16D;
  } else if (dim == 8) {
    // direction index bits D = log2 K: 13 for W3; 6 (the §3.1 rule), 7 or 8 (Tab. 4) for W2
    const bool k_ok = bits == 3 ? dbits == 13 : (dbits >= 6 && dbits <= 8);
    if (!k_ok)
      return set_error(SPHQ_ERR_UNSUPPORTED,
                       "sphq_create: K must be 8192 for bits = 3 and 64, 128 or 256 for bits = 2");
    fmt = fmt_of_split(dbits, radius_bits);
    if (fmt < 0)
      return set_error(SPHQ_ERR_UNSUPPORTED,
                       "sphq_create: unsupported split; sign/index/radius bits must be one of "
                       "8/6/4, 8/6/3, 8/6/2, 8/7/3, 8/7/2, 8/8/2, 8/13/4, 8/13/3");
  } else {
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_create_dim: dim must be 4, 8 or 16");
  }
  const size_t cb_bytes = (size_t)K * dim * 2;
  if (!codebook || !scale || !offset)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_create: NULL codebook/scale/offset");
  const long long nrt = (rows + kRowsPerTile - 1) / kRowsPerTile;
  const long long ng = cols / kGroupCols;
  if ((long long)rows * cols > (1LL << 40))
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_create: matrix too large");

  int dev = 0;
  SPHQ_CUDA(cudaGetDevice(&dev), "cudaGetDevice");
  cudaDeviceProp prop;
  SPHQ_CUDA(cudaGetDeviceProperties(&prop, dev), "cudaGetDeviceProperties");
  if (prop.major != 10 || prop.minor != 3)
    return set_error(SPHQ_ERR_DEVICE, "sphq_create: this library is built for sm_103 (GB300) only");

  sphq_handle h = new sphq_handle_s();
  h->rows = rows;
  h->cols = cols;
  h->bits = bits;
  h->K = K;
  h->nrt = (int)nrt;
  h->ng = (int)ng;
  h->device = dev;
  h->sm_count = prop.multiProcessorCount;
  h->vbits = radius_bits;
  h->dbits = dbits;
  h->dim = dim;
  h->fmt = fmt;
  h->unit_bytes = fmt_unit_bytes(fmt);

  auto fail = [&](sphq_status s) {
    free_handle(h);
    return s;
  };
  cudaError_t e;
  // two guard units after the last one: the GEMV prefetches up to two units
  // past a warp's span without bounds checks
  if ((e = cudaMalloc(&h->units, ((size_t)nrt * ng + 2) * h->unit_bytes)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(units)"));
  if ((e = cudaMalloc(&h->codebook, cb_bytes)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(codebook)"));
  if ((e = cudaMalloc(&h->params, (size_t)rows * ng * 4)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(params)"));
  if ((e = cudaMalloc(&h->flag, 2 * sizeof(int))) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(flag)"));
  if ((e = cudaMemset(h->flag, 0, 2 * sizeof(int))) != cudaSuccess)
    return fail(cuda_error(e, "memset flag"));
  if ((e = cudaMalloc(&h->xstage, (size_t)SPHQ_MAX_BATCH * cols * 2)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(x staging)"));
  if ((e = cudaMalloc(&h->ystage, (size_t)SPHQ_MAX_BATCH * rows * 2)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(y staging)"));
  if ((e = cudaMalloc(&h->zeros, kZeroBytes)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(zeros)"));
  if ((e = cudaMemset(h->zeros, 0, kZeroBytes)) != cudaSuccess)
    return fail(cuda_error(e, "memset zeros"));
  if ((e = cudaMemcpy(h->codebook, codebook, cb_bytes, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy codebook"));
  if (fmt == kFmt4D) {
    // shared-memory image of the 4-D GEMV: entry k, copy c (0..15) at 128 k + 8 c
    if ((e = cudaMalloc(&h->cbimage, (size_t)K * 128)) != cudaSuccess)
      return fail(cuda_error(e, "cudaMalloc(codebook image)"));
    for (int c = 0; c < 16; ++c)
      if ((e = cudaMemcpy2D(static_cast<uint8_t*>(h->cbimage) + 8 * c, 128, h->codebook, 8, 8,
                            (size_t)K, cudaMemcpyDeviceToDevice)) != cudaSuccess)
        return fail(cuda_error(e, "codebook image"));
  }
  if (fmt == kFmt16D) {
    sphq_status st = build_cbimage16(h);
    if (st != SPHQ_OK) return fail(st);
  }
  if (fmt_small(fmt)) {
    // shared-memory image of the small-codebook GEMV: entry k, copy c at 128 k + 16 c
    if ((e = cudaMalloc(&h->cbimage, (size_t)K * 8 * 16)) != cudaSuccess)
      return fail(cuda_error(e, "cudaMalloc(codebook image)"));
    for (int c = 0; c < 8; ++c)
      if ((e = cudaMemcpy2D(static_cast<uint8_t*>(h->cbimage) + 16 * c, 128, h->codebook, 16, 16,
                            (size_t)K, cudaMemcpyDeviceToDevice)) != cudaSuccess)
        return fail(cuda_error(e, "codebook image"));
  }
  // params are kept as two planes (scale, offset) until pack interleaves them
  uint16_t* p16 = reinterpret_cast<uint16_t*>(h->params);
  const size_t np = (size_t)rows * ng;
  if ((e = cudaMemcpy(p16, scale, np * 2, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy scale"));
  if ((e = cudaMemcpy(p16 + np, offset, np * 2, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy offset"));
  sphq_status st = make_gemv_plans(h);
  if (st != SPHQ_OK) return fail(st);
  if (log_enabled()) {
    std::fprintf(stderr, "sphq: matrix %d x %d, %d-D, split %d/%d/%d (format %d), unit %zu B\n",
                 rows, cols, dim, dim, dbits, radius_bits, fmt, h->unit_bytes);
    for (int b = 1; b <= SPHQ_MAX_BATCH; ++b) {
      const GemvPlan& p = h->plan[b];
      std::fprintf(stderr,
                   "sphq:   gemv batch %d: grid %d, cluster %d x %d, <= %d row tiles per cluster, "
                   "%d warps, %zu B shared, mode %d\n",
                   b, p.grid, p.nclusters, p.csize, p.tmax, p.warps_per_cta, p.smem, p.mode);
    }
  }
  if (h->ws_floats > 0 &&
      (e = cudaMalloc(&h->ws, h->ws_floats * sizeof(float))) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(workspace)"));
  *out = h;
  return SPHQ_OK;
}

sphq_status sphq_create_v(int rows, int cols, int bits, int radius_bits, int K,
                          const void* codebook, const void* scale, const void* offset,
                          sphq_handle* out) {
  return create_impl(rows, cols, 8, bits, radius_bits, K, codebook, scale, offset, out);
}

sphq_status sphq_create_dim(int rows, int cols, int dim, int bits, int radius_bits, int K,
                            const void* codebook, const void* scale, const void* offset,
                            sphq_handle* out) {
  return create_impl(rows, cols, dim, bits, radius_bits, K, codebook, scale, offset, out);
}

// Validates and packs canonical device codes into the handle (synchronous).
static sphq_status pack_codes(sphq_handle h, const uint8_t* sign, const uint16_t* idx,
                              const uint8_t* rcode, cudaStream_t s) {
  h->packed = false;
  const uint16_t* scale = reinterpret_cast<const uint16_t*>(h->params);
  const uint16_t* offset = scale + (size_t)h->rows * h->ng;
  SPHQ_CUDA(cudaMemsetAsync(h->flag, 0, sizeof(int), s), "memset flag");
  SPHQ_CUDA(cudaMemsetAsync(h->units, 0, ((size_t)h->nrt * h->ng + 2) * h->unit_bytes, s),
            "memset units");
  const long long threads = (long long)h->nrt * h->ng * 32;
  const int block = 256;
  const unsigned grid = (unsigned)((threads + block - 1) / block);
  if (h->fmt == kFmt16D) {
    if (reinterpret_cast<uintptr_t>(sign) % 2)
      return set_error(SPHQ_ERR_INVALID_ARG, "sphq_pack: 16-D signs must be 2-byte aligned");
    sphq_status st = pack16(h, reinterpret_cast<const uint16_t*>(sign), idx, rcode, scale, offset, s);
    if (st != SPHQ_OK) return st;
  } else if (h->fmt == kFmt4D) {
    pack4_kernel<<<grid, block, 0, s>>>(sign, idx, rcode, scale, offset, (uint8_t*)h->units,
                                        h->rows, h->ng, h->nrt, h->flag);
  } else switch (h->fmt) {
#define SPHQ_PACK_CASE(F)                                                                   \
  case F:                                                                                   \
    pack_kernel<F><<<grid, block, 0, s>>>(sign, idx, rcode, scale, offset,                  \
                                          (uint8_t*)h->units, h->rows, h->ng, h->nrt, h->flag); \
    break;
    SPHQ_FOR_EACH_FMT(SPHQ_PACK_CASE)
#undef SPHQ_PACK_CASE
    default:
      return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_pack: unknown format");
  }
  SPHQ_CUDA(cudaGetLastError(), "pack kernel launch");
  int flag = 0;
  SPHQ_CUDA(cudaMemcpyAsync(&flag, h->flag, sizeof(int), cudaMemcpyDeviceToHost, s), "read flag");
  SPHQ_CUDA(cudaStreamSynchronize(s), "pack");
  if (flag)
    return set_error(SPHQ_ERR_INVALID_ARG,
                     h->dim == 4 ? "sphq_pack: a direction index >= K, a radius code >= "
                                   "2^radius_bits or a sign above 15"
                                 : "sphq_pack: a direction index >= K or a radius code >= "
                                   "2^radius_bits");
  h->packed = true;
  return SPHQ_OK;
}

sphq_status sphq_pack(sphq_handle h, const uint8_t* sign, const uint16_t* idx,
                      const uint8_t* rcode, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_pack: NULL handle");
  if (!sign || !idx || !rcode)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_pack: NULL code pointer");
  if (reinterpret_cast<uintptr_t>(idx) % 2)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_pack: idx must be 2-byte aligned");
  return pack_codes(h, sign, idx, rcode, reinterpret_cast<cudaStream_t>(stream));
}

sphq_status sphq_encode(sphq_handle h, const float* w, uint8_t* sign, uint16_t* idx,
                        uint8_t* rcode, void* scale, void* offset, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_encode: NULL handle");
  if (!w || reinterpret_cast<uintptr_t>(w) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_encode: w must be a 16-byte aligned pointer");
  if (!sign || !idx || !rcode || reinterpret_cast<uintptr_t>(idx) % 2)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_encode: NULL or misaligned code pointer");
  if (h->dim != 8) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_encode: 8-D vectors only");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const size_t nvec = (size_t)h->rows * (h->cols / kVec);
  float* rtilde = nullptr;
  SPHQ_CUDA(cudaMalloc(&rtilde, nvec * sizeof(float)), "cudaMalloc(radii)");
  sphq_status st = launch_encode(h, w, sign, idx, rcode, rtilde, s);
  if (st == SPHQ_OK) {
    const size_t np = (size_t)h->rows * h->ng;
    const uint16_t* p16 = reinterpret_cast<const uint16_t*>(h->params);
    cudaError_t e = cudaSuccess;
    if (scale) e = cudaMemcpyAsync(scale, p16, np * 2, cudaMemcpyDefault, s);
    if (e == cudaSuccess && offset) e = cudaMemcpyAsync(offset, p16 + np, np * 2, cudaMemcpyDefault, s);
    if (e != cudaSuccess) st = cuda_error(e, "copy group parameters");
  }
  if (st == SPHQ_OK) st = pack_codes(h, sign, idx, rcode, s);  // synchronises s
  cudaError_t e = cudaStreamSynchronize(s);
  cudaFree(rtilde);
  if (st == SPHQ_OK && e != cudaSuccess) st = cuda_error(e, "sphq_encode");
  if (st == SPHQ_OK) {
    int word = 0;
    e = cudaMemcpy(&word, h->flag + 1, sizeof(int), cudaMemcpyDeviceToHost);
    if (e != cudaSuccess) return cuda_error(e, "read error word");
    if (word) {
      cudaMemset(h->flag + 1, 0, sizeof(int));
      h->packed = false;
      return set_error(SPHQ_ERR_TIMEOUT, "sphq_encode: a kernel gave up an on-chip wait");
    }
  }
  return st;
}

sphq_status sphq_decode(sphq_handle h, void* w, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_decode: NULL handle");
  if (!w || reinterpret_cast<uintptr_t>(w) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_decode: w must be a 16-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_decode: handle not packed");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  const long long n = (long long)h->rows * (h->cols / kVec);
  const int block = 256;
  const unsigned grid = (unsigned)((n + block - 1) / block);
  if (h->fmt == kFmt16D) {
    sphq_status st = decode16(h, w, s);
    if (st != SPHQ_OK) return st;
  } else if (h->fmt == kFmt4D) {
    const long long nv4 = (long long)h->rows * (h->cols / 4);
    decode4_kernel<<<(unsigned)((nv4 + 255) / 256), 256, 0, s>>>(
        (const uint8_t*)h->units, (const uint8_t*)h->codebook, (uint16_t*)w, h->rows, h->cols,
        h->nrt);
  } else switch (h->fmt) {
#define SPHQ_DECODE_CASE(F)                                                                    \
  case F:                                                                                      \
    decode_kernel<F><<<grid, block, 0, s>>>((const uint8_t*)h->units,                          \
                                            (const uint8_t*)h->codebook, (uint16_t*)w, h->rows, \
                                            h->cols, h->ng, h->nrt);                           \
    break;
    SPHQ_FOR_EACH_FMT(SPHQ_DECODE_CASE)
#undef SPHQ_DECODE_CASE
    default:
      return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_decode: unknown format");
  }
  SPHQ_CUDA(cudaGetLastError(), "decode kernel launch");
  return SPHQ_OK;
}

sphq_status sphq_gemv(sphq_handle h, const void* x, void* y, int batch, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv: batch must be 1..16");
  if (!x || reinterpret_cast<uintptr_t>(x) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: x must be a 16-byte aligned pointer");
  if (!y || reinterpret_cast<uintptr_t>(y) % 4)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: y must be a 4-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemv: handle not packed");
  return launch_gemv(h, x, y, batch, reinterpret_cast<cudaStream_t>(stream));
}

sphq_status sphq_gemm(sphq_handle h, const void* x, void* y, int batch, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm: NULL handle");
  if (batch < 1 || batch > SPHQ_GEMM_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm: batch must be 1..SPHQ_GEMM_MAX_BATCH");
  if (!x || reinterpret_cast<uintptr_t>(x) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm: x must be a 16-byte aligned pointer");
  if (!y || reinterpret_cast<uintptr_t>(y) % 2)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm: y must be a 2-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemm: handle not packed");
  if (h->dim != 8) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm: 8-D vectors only");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // 9..64 rows, when estimated faster: GEMV launches of 3..16 rows (their full
  // modes form every w_hat exactly and accumulate the exact products in
  // fp32, like the tensor-core kernel), which stream the weights once per
  // launch but keep every SM busy, where the tensor-core kernel has only
  // rows / BN CTAs per 128 rows.  Parts are 16 rows, or 14 before a last part
  // of 3 or 4, so every part starts at an even row and its y stays 4-byte
  // aligned; a y that is not 4-byte aligned, or a shape fixed with
  // sphq_set_gemm_shape, takes the tensor-core kernel.
  if (h->gemm_mt == 0 && h->gemm_bn == 0 && reinterpret_cast<uintptr_t>(y) % 4 == 0 &&
      gemm_prefers_gemv(h, batch)) {
    const uint16_t* xs = static_cast<const uint16_t*>(x);
    uint16_t* ys = static_cast<uint16_t*>(y);
    for (int done = 0; done < batch;) {
      const int left = batch - done;
      const int part = left > 18 ? 16 : left > 16 ? 14 : left;
      sphq_status st = launch_gemv(h, xs + (size_t)done * h->cols, ys + (size_t)done * h->rows,
                                   part, s);
      if (st != SPHQ_OK) return st;
      done += part;
    }
    return SPHQ_OK;
  }
  return launch_gemm(h, x, y, batch, s);
}

sphq_status sphq_gemm_workspace(sphq_handle h, int batch, size_t* bytes) {
  g_last_error.clear();
  if (!h || !bytes) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_workspace: NULL argument");
  *bytes = 0;
  if (batch < 1 || batch > SPHQ_GEMM_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm_workspace: batch out of range");
  if (h->dim != 8) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm_workspace: 8-D vectors only");
  return gemm_workspace_bytes(h, batch, bytes);
}

sphq_status sphq_gemm_ws(sphq_handle h, const void* x, void* y, int batch, void* workspace,
                         size_t workspace_bytes, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: NULL handle");
  if (batch < 1 || batch > SPHQ_GEMM_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm_ws: batch must be 1..SPHQ_GEMM_MAX_BATCH");
  if (!x || reinterpret_cast<uintptr_t>(x) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: x must be a 16-byte aligned pointer");
  if (!y || reinterpret_cast<uintptr_t>(y) % 2)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemm_ws: y must be a 2-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemm_ws: handle not packed");
  if (h->dim != 8) return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemm_ws: 8-D vectors only");
  if (!workspace) return launch_gemm(h, x, y, batch, reinterpret_cast<cudaStream_t>(stream));
  return launch_gemm_ws(h, x, y, batch, workspace, workspace_bytes,
                        reinterpret_cast<cudaStream_t>(stream));
}

sphq_status sphq_get_gemm_shape(sphq_handle h, int batch, sphq_gemm_info* out) {
  g_last_error.clear();
  if (!h || !out) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_get_gemm_shape: NULL argument");
  if (batch < 1 || batch > SPHQ_GEMM_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_get_gemm_shape: batch out of range");
  return gemm_shape_info(h, batch, out);
}

sphq_status sphq_set_gemm_shape(sphq_handle h, int act_tiles, int weight_rows) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_set_gemm_shape: NULL handle");
  if (act_tiles < 0 || act_tiles > 2 || (weight_rows != 0 && weight_rows != 128 && weight_rows != 256) ||
      (act_tiles == 2 && weight_rows == 128))
    return set_error(SPHQ_ERR_INVALID_ARG,
                     "sphq_set_gemm_shape: act_tiles 0..2, weight_rows 0/128/256, not 2 x 128");
  h->gemm_mt = act_tiles;
  h->gemm_bn = weight_rows;
  return SPHQ_OK;
}

sphq_status sphq_check(sphq_handle h, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_check: NULL handle");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  int word = 0;
  SPHQ_CUDA(cudaMemcpyAsync(&word, h->flag + 1, sizeof(int), cudaMemcpyDeviceToHost, s),
            "read error word");
  SPHQ_CUDA(cudaMemsetAsync(h->flag + 1, 0, sizeof(int), s), "clear error word");
  SPHQ_CUDA(cudaStreamSynchronize(s), "sphq_check");
  if (word)
    return set_error(SPHQ_ERR_TIMEOUT,
                     "sphq_check: a kernel gave up waiting on an mbarrier (results invalid)");
  return SPHQ_OK;
}

// Copies n16 16-byte words from host memory (a mapped pinned buffer read over
// the CPU-GPU link) into a device buffer.  Launched as a programmatic
// dependent: it lets the GEMV that follows launch at once (its prologue only
// reads the immutable codes and codebook), and waits for the previous kernel
// before it reads x (which that kernel may have written) or overwrites the
// staging buffer (which a previous GEMV of this handle may still read).
__global__ void stage_x_kernel(const uint4* __restrict__ src, uint4* __restrict__ dst, int n16) {
  asm volatile("griddepcontrol.launch_dependents;");
  asm volatile("griddepcontrol.wait;" ::: "memory");
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i < n16) dst[i] = src[i];
}

// Device address of a page-locked, mapped host buffer, or null for any other
// pointer (pageable memory, device memory, or an error from the query).
static const void* mapped_device_pointer(const void* p) {
  cudaPointerAttributes a;
  if (cudaPointerGetAttributes(&a, p) != cudaSuccess) {
    (void)cudaGetLastError();
    return nullptr;
  }
  if (a.type != cudaMemoryTypeHost || !a.devicePointer || !a.hostPointer) return nullptr;
  // the attributes describe the allocation's base; keep p's offset into it
  const ptrdiff_t off = static_cast<const char*>(p) - static_cast<const char*>(a.hostPointer);
  return static_cast<const char*>(a.devicePointer) + off;
}

sphq_status sphq_gemv_host(sphq_handle h, const void* x_host, void* y_host, int batch,
                           sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_host: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv_host: batch must be 1..16");
  if (!x_host || !y_host) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_host: NULL buffer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemv_host: handle not packed");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  // Page-locked host buffers mapped into the device address space: one small
  // kernel reads x over the CPU-GPU link (coherent on Grace-Blackwell) into
  // the handle's device staging buffer -- once, instead of every CTA of the
  // GEMV fetching its slice across the link -- and the GEMV writes y into
  // host memory directly.  No copy-engine operations on the stream.
  const void* xd = mapped_device_pointer(x_host);
  void* yd = const_cast<void*>(mapped_device_pointer(y_host));
  if (xd && yd && reinterpret_cast<uintptr_t>(xd) % 16 == 0 &&
      reinterpret_cast<uintptr_t>(yd) % 4 == 0) {
    int n16 = batch * h->cols * 2 / 16;
    cudaLaunchConfig_t cfg = {};
    cfg.gridDim = dim3((unsigned)((n16 + 255) / 256));
    cfg.blockDim = dim3(256);
    cfg.stream = s;
    cudaLaunchAttribute attr[1];
    attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
    attr[0].val.programmaticStreamSerializationAllowed = 1;
    cfg.attrs = attr;
    cfg.numAttrs = h->pdl ? 1 : 0;
    const uint4* src = static_cast<const uint4*>(xd);
    uint4* dst = static_cast<uint4*>(h->xstage);
    SPHQ_CUDA(cudaLaunchKernelEx(&cfg, stage_x_kernel, src, dst, n16), "stage x");
    return launch_gemv(h, h->xstage, yd, batch, s);
  }
  SPHQ_CUDA(cudaMemcpyAsync(h->xstage, x_host, (size_t)batch * h->cols * 2,
                            cudaMemcpyHostToDevice, s), "copy x to device");
  sphq_status st = launch_gemv(h, h->xstage, h->ystage, batch, s);
  if (st != SPHQ_OK) return st;
  SPHQ_CUDA(cudaMemcpyAsync(y_host, h->ystage, (size_t)batch * h->rows * 2,
                            cudaMemcpyDeviceToHost, s), "copy y to host");
  return SPHQ_OK;
}

size_t sphq_bytes(sphq_handle h, int batch) {
  if (!h || batch < 1 || batch > SPHQ_MAX_BATCH) return 0;
  const size_t weights = (size_t)h->rows * h->cols;
  // payload bits per dim-D vector: dim signs + D index bits + V radius bits
  const size_t vec_bits = (size_t)h->dim + h->dbits + h->vbits;
  const size_t payload = weights / h->dim * vec_bits / 8;
  const size_t params = (size_t)h->rows * h->ng * 4;
  const size_t codebook = (size_t)h->K * h->dim * 2;
  const size_t io = 2 * (size_t)batch * (h->cols + h->rows);
  return payload + params + codebook + io;
}

sphq_status sphq_destroy(sphq_handle h) {
  g_last_error.clear();
  free_handle(h);
  return SPHQ_OK;
}

}  // extern "C"
