// C ABI of the sphq library: handle lifetime, packing, decode, errors.
// The GEMV kernels and their launch plans live in sphq_gemv.cu.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <cstdio>
#include <cstring>
#include <string>

#include "sphq_internal.h"
#include "sphq_layout.cuh"

namespace sphq {

static thread_local std::string g_last_error;

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
// pack: canonical codes -> group tiles (the finalise-and-pack step, App. A step 10)
// ---------------------------------------------------------------------------

// One thread per (row block, group, lane): composes the lane's part of a tile.
template <int BITS>
__global__ void pack_kernel(const uint8_t* __restrict__ sign, const uint16_t* __restrict__ idx,
                            const uint8_t* __restrict__ rcode,
                            const uint16_t* __restrict__ scale,
                            const uint16_t* __restrict__ offset, uint8_t* __restrict__ tiles,
                            int rows, int ng, int nrb, int* __restrict__ flag) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const long long total = (long long)nrb * ng * kRowsPerBlock;
  if (tid >= total) return;
  const int lane = (int)(tid % kRowsPerBlock);
  const long long unit = tid / kRowsPerBlock;  // rb * ng + g
  const int g = (int)(unit % ng);
  const int rb = (int)(unit / ng);
  const int row = rb * kRowsPerBlock + lane;
  const int nv = ng * kGroupVecs;
  uint8_t* tile = tiles + (size_t)unit * Layout<BITS>::kTileBytes;

  uint32_t words[kGroupVecs];
  uint32_t aux0 = 0, aux1 = 0, aux2 = 0, aux3 = 0, top = 0, params = 0;
  bool bad = false;
  for (int j = 0; j < kGroupVecs; ++j) {
    uint32_t s = 0, k = 0, q = 0;
    if (row < rows) {
      const size_t v = (size_t)row * nv + (size_t)g * kGroupVecs + j;
      s = sign[v];
      k = idx[v];
      q = rcode[v];
      if (k >= (uint32_t)Layout<BITS>::K || q > 15u) {
        bad = true;
        k = 0;
        q = 0;
      }
    }
    if (BITS == 2) {
      words[j] = s | (k << 8) | ((q & 3u) << 14);
      aux0 |= ((q >> 2) & 3u) << (2 * j);
    } else {
      words[j] = s | ((k & 0xFFu) << 8);
      const int n = 4 * (j & 7);
      if (j < 8) {
        aux0 |= q << n;
        aux2 |= ((k >> 8) & 0xFu) << n;
      } else {
        aux1 |= q << n;
        aux3 |= ((k >> 8) & 0xFu) << n;
      }
      top |= ((k >> 12) & 1u) << j;
    }
  }
  if (row < rows) {
    const size_t gi = (size_t)row * ng + g;
    params = (uint32_t)scale[gi] | ((uint32_t)offset[gi] << 16);
  }
  if (bad) atomicOr(flag, 1);
  for (int c = 0; c < 2; ++c) {
    uint4 v;
    v.x = words[8 * c + 0] | (words[8 * c + 1] << 16);
    v.y = words[8 * c + 2] | (words[8 * c + 3] << 16);
    v.z = words[8 * c + 4] | (words[8 * c + 5] << 16);
    v.w = words[8 * c + 6] | (words[8 * c + 7] << 16);
    *reinterpret_cast<uint4*>(tile + c * 512 + lane * 16) = v;
  }
  if (BITS == 2) {
    *reinterpret_cast<uint2*>(tile + Layout<2>::kAuxOff + lane * 8) = make_uint2(aux0, params);
  } else {
    *reinterpret_cast<uint4*>(tile + Layout<3>::kAuxOff + lane * 16) =
        make_uint4(aux0, aux1, aux2, aux3);
    *reinterpret_cast<uint32_t*>(tile + Layout<3>::kParamOff + lane * 4) = params;
    *reinterpret_cast<uint16_t*>(tile + Layout<3>::kTopOff + lane * 2) = (uint16_t)top;
  }
}

// ---------------------------------------------------------------------------
// decode: W_hat (rows x cols fp16), through the same unpack/reconstruct code
// ---------------------------------------------------------------------------

template <int BITS>
__global__ void decode_kernel(const uint8_t* __restrict__ tiles, const uint4* __restrict__ codebook,
                              uint16_t* __restrict__ w, int rows, int cols, int ng) {
  const long long tid = (long long)blockIdx.x * blockDim.x + threadIdx.x;
  const int nv = cols / kVec;
  if (tid >= (long long)rows * nv) return;
  const int row = (int)(tid / nv);
  const int t = (int)(tid % nv);
  const int rb = row / kRowsPerBlock, lane = row % kRowsPerBlock;
  const int g = t / kGroupVecs, j = t % kGroupVecs;
  const uint8_t* tile = tiles + ((size_t)rb * ng + g) * Layout<BITS>::kTileBytes;
  const GroupData<BITS> d = load_group<BITS>(tile, lane);
  const Fields f = unpack(d, j);
  const uint16_t r = radius16(f.q, d.params);
  const uint4 c = codebook[f.k];
  *reinterpret_cast<uint4*>(w + (size_t)row * cols + (size_t)t * kVec) = reconstruct(f.sign, r, c);
}

}  // namespace sphq

using namespace sphq;

extern "C" {

int sphq_version(void) { return 10000; }

const char* sphq_last_error(void) { return g_last_error.c_str(); }

static void free_handle(sphq_handle h) {
  if (!h) return;
  cudaFree(h->tiles);
  cudaFree(h->codebook);
  cudaFree(h->params);
  cudaFree(h->ws);
  cudaFree(h->tickets);
  cudaFree(h->flag);
  cudaFree(h->xstage);
  cudaFree(h->ystage);
  delete h;
}

sphq_status sphq_create(int rows, int cols, int bits, int K, const void* codebook,
                        const void* scale, const void* offset, sphq_handle* out) {
  g_last_error.clear();
  if (!out) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_create: out is NULL");
  *out = nullptr;
  if (rows < 1 || cols < kGroupCols || cols % kGroupCols != 0)
    return set_error(SPHQ_ERR_INVALID_ARG,
                     "sphq_create: need rows >= 1 and cols a positive multiple of 128");
  if (bits != 2 && bits != 3)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_create: bits must be 2 or 3");
  if (K != (1 << (7 * bits - 8)))
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_create: K must be 2^(7*bits-8)");
  if (!codebook || !scale || !offset)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_create: NULL codebook/scale/offset");
  const long long nrb = (rows + kRowsPerBlock - 1) / kRowsPerBlock;
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
  h->nrb = (int)nrb;
  h->ng = (int)ng;
  h->device = dev;
  h->sm_count = prop.multiProcessorCount;
  h->tile_bytes = bits == 2 ? Layout<2>::kTileBytes : Layout<3>::kTileBytes;

  auto fail = [&](sphq_status s) {
    free_handle(h);
    return s;
  };
  cudaError_t e;
  if ((e = cudaMalloc(&h->tiles, (size_t)nrb * ng * h->tile_bytes)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(tiles)"));
  if ((e = cudaMalloc(&h->codebook, (size_t)K * 16)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(codebook)"));
  if ((e = cudaMalloc(&h->params, (size_t)rows * ng * 4)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(params)"));
  if ((e = cudaMalloc(&h->tickets, (size_t)nrb * sizeof(unsigned))) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(tickets)"));
  if ((e = cudaMalloc(&h->flag, sizeof(int))) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(flag)"));
  if ((e = cudaMalloc(&h->xstage, (size_t)SPHQ_MAX_BATCH * cols * 2)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(x staging)"));
  if ((e = cudaMalloc(&h->ystage, (size_t)SPHQ_MAX_BATCH * rows * 2)) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(y staging)"));
  if ((e = cudaMemcpy(h->codebook, codebook, (size_t)K * 16, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy codebook"));
  // params are kept as two planes (scale, offset) until pack interleaves them
  uint16_t* p16 = reinterpret_cast<uint16_t*>(h->params);
  const size_t np = (size_t)rows * ng;
  if ((e = cudaMemcpy(p16, scale, np * 2, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy scale"));
  if ((e = cudaMemcpy(p16 + np, offset, np * 2, cudaMemcpyDefault)) != cudaSuccess)
    return fail(cuda_error(e, "copy offset"));
  if ((e = cudaMemset(h->tickets, 0, (size_t)nrb * sizeof(unsigned))) != cudaSuccess)
    return fail(cuda_error(e, "memset tickets"));
  sphq_status st = make_gemv_plans(h);
  if (st != SPHQ_OK) return fail(st);
  if ((e = cudaMalloc(&h->ws, h->ws_floats * sizeof(float))) != cudaSuccess)
    return fail(cuda_error(e, "cudaMalloc(workspace)"));
  *out = h;
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
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
  h->packed = false;
  const uint16_t* scale = reinterpret_cast<const uint16_t*>(h->params);
  const uint16_t* offset = scale + (size_t)h->rows * h->ng;
  SPHQ_CUDA(cudaMemsetAsync(h->flag, 0, sizeof(int), s), "memset flag");
  SPHQ_CUDA(cudaMemsetAsync(h->tickets, 0, (size_t)h->nrb * sizeof(unsigned), s), "memset tickets");
  const long long threads = (long long)h->nrb * h->ng * kRowsPerBlock;
  const int block = 256;
  const unsigned grid = (unsigned)((threads + block - 1) / block);
  if (h->bits == 2)
    pack_kernel<2><<<grid, block, 0, s>>>(sign, idx, rcode, scale, offset,
                                          (uint8_t*)h->tiles, h->rows, h->ng, h->nrb, h->flag);
  else
    pack_kernel<3><<<grid, block, 0, s>>>(sign, idx, rcode, scale, offset,
                                          (uint8_t*)h->tiles, h->rows, h->ng, h->nrb, h->flag);
  SPHQ_CUDA(cudaGetLastError(), "pack kernel launch");
  int flag = 0;
  SPHQ_CUDA(cudaMemcpyAsync(&flag, h->flag, sizeof(int), cudaMemcpyDeviceToHost, s), "read flag");
  SPHQ_CUDA(cudaStreamSynchronize(s), "pack");
  if (flag)
    return set_error(SPHQ_ERR_INVALID_ARG,
                     "sphq_pack: a direction index >= K or a radius code > 15");
  h->packed = true;
  return SPHQ_OK;
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
  if (h->bits == 2)
    decode_kernel<2><<<grid, block, 0, s>>>((const uint8_t*)h->tiles, (const uint4*)h->codebook,
                                            (uint16_t*)w, h->rows, h->cols, h->ng);
  else
    decode_kernel<3><<<grid, block, 0, s>>>((const uint8_t*)h->tiles, (const uint4*)h->codebook,
                                            (uint16_t*)w, h->rows, h->cols, h->ng);
  SPHQ_CUDA(cudaGetLastError(), "decode kernel launch");
  return SPHQ_OK;
}

sphq_status sphq_gemv(sphq_handle h, const void* x, void* y, int batch, sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv: batch must be 1..8");
  if (!x || reinterpret_cast<uintptr_t>(x) % 16)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: x must be a 16-byte aligned pointer");
  if (!y || reinterpret_cast<uintptr_t>(y) % 4)
    return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv: y must be a 4-byte aligned pointer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemv: handle not packed");
  return launch_gemv(h, x, y, batch, reinterpret_cast<cudaStream_t>(stream));
}

sphq_status sphq_gemv_host(sphq_handle h, const void* x_host, void* y_host, int batch,
                           sphq_stream stream) {
  g_last_error.clear();
  if (!h) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_host: NULL handle");
  if (batch < 1 || batch > SPHQ_MAX_BATCH)
    return set_error(SPHQ_ERR_UNSUPPORTED, "sphq_gemv_host: batch must be 1..8");
  if (!x_host || !y_host) return set_error(SPHQ_ERR_INVALID_ARG, "sphq_gemv_host: NULL buffer");
  if (!h->packed) return set_error(SPHQ_ERR_NOT_PACKED, "sphq_gemv_host: handle not packed");
  cudaStream_t s = reinterpret_cast<cudaStream_t>(stream);
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
  // payload bits per 8-D vector: 8 signs + (7B-8) index bits + 4 radius bits
  const size_t vec_bits = 8 + (7 * h->bits - 8) + 4;
  const size_t payload = weights / kVec * vec_bits / 8;
  const size_t params = (size_t)h->rows * h->ng * 4;
  const size_t codebook = (size_t)h->K * 16;
  const size_t io = 2 * (size_t)batch * (h->cols + h->rows);
  return payload + params + codebook + io;
}

sphq_status sphq_destroy(sphq_handle h) {
  g_last_error.clear();
  free_handle(h);
  return SPHQ_OK;
}

}  // extern "C"
