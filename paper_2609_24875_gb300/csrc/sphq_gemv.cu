// Launch plans and launches of the fused dequantize-GEMV (the kernel itself is
// in sphq_gemv_kernel.cuh); instantiates the W2 and W3 formats.
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include <algorithm>
#include <mutex>
#include <string>

#include "sphq_gemv_kernel.cuh"

namespace sphq {
// ---------------------------------------------------------------------------
// Host side: kernel selection, launch plans, launches
// ---------------------------------------------------------------------------

static int warps_for(int fmt) {
  return fmt_small(fmt) || fmt == kFmt4D ? KernelShape<2>::kWarps : KernelShape<3>::kWarps;
}
// shared-memory codebook image: interleaved copies (128 bytes per entry) for
// the small codebooks and 4-D, the plain 128 KiB table for W3
static uint32_t cb_bytes_for(int fmt) {
  return fmt_small(fmt) || fmt == kFmt4D ? (uint32_t)(1u << fmt_dir_bits(fmt)) * 128u
                                         : KernelShape<3>::kCbBytes;
}

static int mode_for(int batch) {
  return batch == 1 ? kFactored1 : batch == 2 ? kFactored2 : batch <= kMaxBatch ? kFull : kFull16;
}

// formats with a one-CTA-per-SM build beside the two-CTA one
static bool has_solo(int fmt) { return fmt == 2; }

static const void* select_kernel(int fmt, int mode, int strip, bool solo = false) {
  if (mode == kFull16)  // one build per format (strips of two, one CTA per SM)
    return fmt == 2 ? kptr_full16<2>() : fmt == 3 ? kptr_full16<3>()
           : fmt == kFmtW3V3 ? kptr_full16<kFmtW3V3>() : split_kernel(fmt, mode);
  return fmt == 2 ? (solo ? (strip == 4 ? kptr_mode_solo<2, 4>(mode) : kptr_mode_solo<2>(mode))
                           : kptr_mode<2>(mode))
         : fmt == 3 ? (strip == 4 ? kptr_mode<3, 4>(mode) : kptr_mode<3, 2>(mode))
         : fmt == kFmtW3V3 ? (strip == 4 ? kptr_mode<kFmtW3V3, 4>(mode) : kptr_mode<kFmtW3V3, 2>(mode))
                           : split_kernel(fmt, mode);
}

// Dynamic shared memory is sized per handle, while the attribute that permits
// it belongs to the kernel function and is process-wide: raise it once to the
// device's opt-in maximum.
static sphq_status allow_max_smem(int device, int optin) {
  static std::mutex mu;
  static bool done[64] = {};
  std::lock_guard<std::mutex> lock(mu);
  if (device < 0 || device >= 64) return set_error(SPHQ_ERR_DEVICE, "device index out of range");
  if (done[device]) return SPHQ_OK;
  for (int fmt = 2; fmt <= kFmt4D; ++fmt)
    for (int mode : kModes)
      for (int strip : {2, 4})
        for (int solo = 0; solo < 2; ++solo) {
          if (strip == 4 && !fmt_has_strip4(fmt) && !(solo && has_solo(fmt))) continue;
          if (solo && !has_solo(fmt)) continue;
          const void* k = select_kernel(fmt, mode, strip, solo);
          if (!k) continue;  // no 16-row build for 4-D vectors
          cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, optin);
          if (e != cudaSuccess) return cuda_error(e, "cudaFuncSetAttribute");
        }
  done[device] = true;
  return SPHQ_OK;
}

static size_t align_up(size_t v, size_t a) { return (v + a - 1) / a * a; }

// Shared-memory layout for a given cluster size and tile count per cluster.
struct SmemLayout {
  size_t zero, x, recv, bar, total;
  uint32_t x_pitch;
};

static SmemLayout smem_layout(const sphq_handle_s* h, int mode, int warps, int csize, int tmax) {
  SmemLayout L{};
  const int nbp = mode;  // batch rows of a partial block
  const size_t blk = (size_t)kRowsPerTile * nbp * 4;
  const int ngc_max = (h->ng + csize - 1) / csize;
  const int nown_max = (tmax + csize - 1) / csize;  // tiles one CTA owns
  size_t o = cb_bytes_for(h->fmt);
  // batch 1-2: a 256 B zero block, then the activation rows.  Rows start 320 B
  // after the zero block and 64 B apart modulo 128, so within a quarter warp
  // the suppliers' 16-byte chunks and the zero readers' chunks fall in
  // different bank groups.
  L.zero = o;
  L.x = o + 320;
  L.x_pitch = (uint32_t)((size_t)ngc_max * kGroupCols * 2 + 64);
  if (!mode_full(mode)) o = L.x + (size_t)L.x_pitch * mode;
  // receive slots: one block per (owned tile, rank, warp)
  o = align_up(o, 16);
  L.recv = o;
  o += (size_t)nown_max * csize * warps * blk;
  o = align_up(o, 8);
  L.bar = o;
  o += 32;  // three mbarriers
  L.total = align_up(o, 16);
  return L;
}

// Without `pdl` the launch waits for the previous work on the stream to
// finish; the kernel's dependency wait then returns at once.
static cudaLaunchConfig_t launch_config(const GemvPlan& p, cudaStream_t s,
                                        cudaLaunchAttribute (&attr)[2], bool pdl = true) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = dim3(p.grid);
  cfg.blockDim = dim3(p.warps_per_cta * 32);
  cfg.dynamicSmemBytes = p.smem;
  cfg.stream = s;
  attr[0].id = cudaLaunchAttributeClusterDimension;
  attr[0].val.clusterDim.x = (unsigned)p.csize;
  attr[0].val.clusterDim.y = 1;
  attr[0].val.clusterDim.z = 1;
  attr[1].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[1].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = pdl ? 2 : 1;
  return cfg;
}

// Launch plan for one batch size: the cheapest shape by the cost model, or
// the cheapest at cluster size `forced` (1, 2, 4, 8) when it is nonzero.
static sphq_status make_plan(sphq_handle h, int batch, int forced, int optin, GemvPlan& out) {
  cudaError_t e;
  {
    GemvPlan best{};
    double best_cost = 0;
    // W2: the one-CTA-per-SM build with four-tile strips, kept aside and
    // compared below by the work of the busiest SM
    GemvPlan packed{};
    double packed_load = 0;
    const int warps = warps_for(h->fmt);
    // Batch 2 reads its activations through L1 (the full mode: exact w_hat,
    // no staged copy) for the 8192-entry tables and for small matrices:
    // measured against the staged factored mode, W3 3584^2 5.57 -> 5.17 us,
    // 4096^2 6.07 -> 5.75, 8192^2 16.13 -> 15.26, 512 x 3584 2.50 -> 2.37
    // (18944 x 3584 15.28 / 15.37: equal); W2 512 x 3584 2.06 -> 1.89,
    // 3584^2 4.30 -> 4.15, 4096^2 4.48 -> 4.32, while from 32768 units up the
    // staged mode stays faster (8192^2 10.61 against 11.19).  Batch 1 keeps
    // the staged mode (the full mode within -2% to +4% of it).
    const bool full2 = batch == 2 && (!fmt_small(h->fmt) && h->fmt != kFmt4D
                                          ? true
                                          : (long long)h->nrt * h->ng <= 16384);
    for (int staged = full2 ? 0 : 1; staged >= 0; --staged) {
      int mode = mode_for(batch);
      if (!staged && !mode_full(mode)) mode = kFull;
      if (staged && mode_full(mode)) continue;
      const int nsolo = mode == kFull16 ? 1 : has_solo(h->fmt) ? 2 : 1;
      for (int solo = 0; solo < nsolo; ++solo) {
        // both strip sizes: same resources
        const void* k = select_kernel(h->fmt, mode, 2, solo);
        if (!k) continue;
        for (int csize : {1, 2, 4, 8}) {
          if (csize > h->ng) break;
          if (forced && csize != forced) continue;
          // 9-16 rows: partial blocks of 16 batch rows make the reduction in a
          // cluster twice as heavy, and strips of two tiles leave one-tile
          // strips in odd tile ranges; single CTAs measured best (8192^2 W3
          // 20.7 against 23.3 us in clusters of 2, W2 3584 x 18944 16.1 against
          // 22.3) unless the row tiles cannot fill half the SMs (512 x 3584:
          // clusters of 4, 3.5 against 4.5 us)
          if (!forced && mode == kFull16 && csize > 1 && 2 * h->nrt >= std::max(h->sm_count, 1))
            continue;
          // clusters: as many as fit at once, at most one per row tile; the
          // tile range of a cluster is limited by its shared memory
          GemvPlan p;
          p.mode = mode;
          p.warps_per_cta = warps;
          p.csize = csize;
          p.grid = csize;
          p.smem = smem_layout(h, mode, warps, csize, 1).total;
          if (p.smem > (size_t)optin) continue;
          cudaLaunchAttribute attr[2];
          cudaLaunchConfig_t cfg = launch_config(p, nullptr, attr);
          int ncl = 0;
          e = cudaOccupancyMaxActiveClusters(&ncl, k, &cfg);
          if (e != cudaSuccess) {
            (void)cudaGetLastError();
            continue;
          }
          if (ncl < 1) continue;
          int nclusters = std::min(ncl, h->nrt);
          int tmax = (h->nrt + nclusters - 1) / nclusters;
          SmemLayout L = smem_layout(h, mode, warps, csize, tmax);
          // grow the cluster count (extra waves) until a cluster's tiles fit
          while (L.total > (size_t)optin && tmax > 1) {
            nclusters = std::min(h->nrt, nclusters * 2);
            tmax = (h->nrt + nclusters - 1) / nclusters;
            L = smem_layout(h, mode, warps, csize, tmax);
          }
          if (L.total > (size_t)optin) continue;
          // with the final shared-memory size the resident count may be lower
          p.smem = L.total;
          cfg = launch_config(p, nullptr, attr);
          e = cudaOccupancyMaxActiveClusters(&ncl, k, &cfg);
          if (e != cudaSuccess || ncl < 1) {
            (void)cudaGetLastError();
            continue;
          }
          const int waves = (nclusters + ncl - 1) / ncl;
          // Estimated time per launch (us), fitted (least log-regret over a grid
          // of constants) to GB300 measurements of back-to-back launches at
          // cluster sizes 1, 2 and 4 on the decoder and square shapes (W2 and
          // W3, batch 1, 2, 4 and 8): a fixed part (launch, staging, reduction)
          // plus ~0.02 us per unit of the most loaded CTA; one-tile strips do
          // not share activation loads between two units.  With the prologue
          // free of divisions and per-tile cover masks, clusters of 2 and 4 cost
          // no more than single CTAs in every mode (worst regret against the
          // best of the three sizes: 2.3% at batch 4-8, 5.9% at batch 1-2);
          // clusters of 8 leave SMs idle (only 15 fit) and are priced out unless
          // nothing else runs.  A plan that needs a second wave of clusters (its
          // shared memory did not fit at one wave) pays the fixed part again per
          // wave (measured: W3 18944 x 3584 batch 8 in two waves of clusters of
          // 4, 22.1 us against 15.6 us in one wave of single CTAs).
          const double fixed = csize == 8 ? (mode_full(mode) ? 5.8 : 5.0) : 2.0;
          const double shallow = 1.0 + 0.33 * (2 - std::min(tmax, 2));
          const double cost = fixed * waves + waves * 0.02 * tmax * ((h->ng + csize - 1) / csize) * shallow;
          // The one-CTA-per-SM build wins ties: at equal load the row tiles
          // bound the cluster count, and no second CTA would share an SM.
          const bool better = best.grid == 0 || cost < best_cost - 1e-9 ||
                              (solo && !best.solo && cost <= best_cost + 1e-9);
          const bool strip4_ok =
              mode != kFull16 && (fmt_has_strip4(h->fmt) || (solo && has_solo(h->fmt)));
          const double load = (double)tmax * ((h->ng + csize - 1) / csize) * waves;
          const bool packed_candidate = solo && has_solo(h->fmt) && mode != kFull16 && tmax >= 3 &&
                                        (packed.grid == 0 || load < packed_load);
          if (better || packed_candidate) {
            p.grid = nclusters * csize;
            p.nclusters = nclusters;
            p.tmax = tmax;
            p.cb_bytes = cb_bytes_for(h->fmt);
            p.x_pitch = L.x_pitch;
            p.off_x = (uint32_t)L.x;
            p.off_zero = (uint32_t)L.zero;
            p.off_recv = (uint32_t)L.recv;
            p.off_bar = (uint32_t)L.bar;
            // four-tile strips once a cluster holds three tiles or more (W3)
            p.strip = strip4_ok && tmax >= 3 ? 4 : 2;
            p.solo = solo != 0 || mode == kFull16;
          p.ctas_per_sm = p.solo ? 1
                          : fmt_small(h->fmt) || h->fmt == kFmt4D ? KernelShape<2>::kMinBlocks
                                                                   : KernelShape<3>::kMinBlocks;
            if (packed_candidate) {
              packed = p;
              packed_load = load;
            }
            if (better) {
              best = p;
              best_cost = cost;
            }
          }
        }
      }
      if (best.grid > 0) break;  // staged activations fit: keep that mode
    }
    // When more CTAs of the two-per-SM build are launched than there are SMs,
    // some SMs run two of them: their work is twice a CTA's.  The one-CTA
    // build with four-tile strips takes the same tiles in fewer, longer CTAs
    // (and shares each activation load among up to four units); take it when
    // its busiest SM has clearly less work and its CTAs have long rows of work
    // (32 groups or more: with fewer, the items dealt to 8 warps are too
    // coarse to gain).  Per unit its 8 warps per SM count 7% slower than 16
    // at 1-2 rows, and 7% faster at 3-8 rows, where each strip of four shares
    // one read of the activations through L1.  Measured: W2 3584 x 18944 at
    // batch 1-8 13-14% faster, W2 8192^2 at 4-8 rows 8-11% faster; 3584^2 (14
    // groups per CTA) 2% slower, hence the row condition; 18944 x 3584
    // unchanged.
    if (packed.grid > 0 && best.grid > 0 && !best.solo && !forced &&
        (h->ng + packed.csize - 1) / packed.csize >= 32) {
      const int sms = h->sm_count > 0 ? h->sm_count : 1;
      const int per_sm = std::min(best.ctas_per_sm, (best.grid + sms - 1) / sms);
      const double best_load = (double)best.tmax * ((h->ng + best.csize - 1) / best.csize) * per_sm;
      const double per_unit = packed.mode == kFull ? 0.93 : 1.07;
      if (packed_load * per_unit < 0.95 * best_load) best = packed;
    }
    if (best.grid == 0)
      return set_error(forced ? SPHQ_ERR_UNSUPPORTED : SPHQ_ERR_CUDA,
                       forced ? "no resident launch shape at this cluster size"
                              : "no resident launch shape for the gemv kernel");
    out = best;
  }
  return SPHQ_OK;
}

static sphq_status device_optin(sphq_handle h, int* optin) {
  cudaError_t e = cudaDeviceGetAttribute(optin, cudaDevAttrMaxSharedMemoryPerBlockOptin, h->device);
  if (e != cudaSuccess) return cuda_error(e, "cudaDeviceGetAttribute");
  return allow_max_smem(h->device, *optin);
}

sphq_status make_gemv_plans(sphq_handle h) {
  if (h->fmt == kFmt16D) {  // batches 9-16: launches of 8 rows and the rest
    for (int batch = 1; batch <= SPHQ_MAX_BATCH; ++batch) {
      h->plan[batch] = GemvPlan{};
      if (batch <= kMaxBatch) {
        sphq_status st = make_gemv16_plan(h, batch, 0, h->plan[batch]);
        if (st != SPHQ_OK) return st;
      }
    }
    h->ws_floats = 0;
    return SPHQ_OK;
  }
  int optin = 0;
  sphq_status st = device_optin(h, &optin);
  if (st != SPHQ_OK) return st;
  for (int batch = 1; batch <= SPHQ_MAX_BATCH; ++batch) {
    if (batch > kMaxBatch && h->fmt == kFmt4D) {
      h->plan[batch] = GemvPlan{};  // 4-D: two launches of at most 8 rows
      continue;
    }
    st = make_plan(h, batch, 0, optin, h->plan[batch]);
    if (st != SPHQ_OK) return st;
  }
  h->ws_floats = 0;
  return SPHQ_OK;
}

sphq_status set_gemv_cluster_size(sphq_handle h, int batch, int csize) {
  if (h->fmt == kFmt16D) {
    if (batch > kMaxBatch)
      return set_error(SPHQ_ERR_UNSUPPORTED,
                       "sphq_set_cluster_size: 16-D batches above 8 run as launches of 8 and the rest");
    return make_gemv16_plan(h, batch, csize, h->plan[batch]);
  }
  int optin = 0;
  sphq_status st = device_optin(h, &optin);
  if (st != SPHQ_OK) return st;
  GemvPlan p;
  st = make_plan(h, batch, csize, optin, p);
  if (st != SPHQ_OK) return st;
  h->plan[batch] = p;
  return SPHQ_OK;
}

sphq_status launch_gemv(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s) {
  if (batch > kMaxBatch && h->plan[batch].grid == 0) {
    // no 16-row build (4-D and 16-D vectors): 8 rows, then the rest
    sphq_status st = launch_gemv(h, x, y, kMaxBatch, s);
    if (st != SPHQ_OK) return st;
    return launch_gemv(h, static_cast<const uint16_t*>(x) + (size_t)kMaxBatch * h->cols,
                       static_cast<uint16_t*>(y) + (size_t)kMaxBatch * h->rows, batch - kMaxBatch,
                       s);
  }
  if (h->fmt == kFmt16D) return launch_gemv16(h, x, y, batch, s);
  const GemvPlan& p = h->plan[batch];
  GemvArgs a;
  a.units = (const uint8_t*)h->units;
  a.cbimage = (const uint8_t*)(h->cbimage ? h->cbimage : h->codebook);
  a.x = (const uint16_t*)x;
  a.y = (uint16_t*)y;
  a.flag = h->flag + 1;
  a.rows = h->rows;
  a.cols = h->cols;
  a.ng = h->ng;
  a.nrt = h->nrt;
  a.batch = batch;
  a.nclusters = p.nclusters;
  a.cb_bytes = p.cb_bytes;
  a.x_pitch = p.x_pitch;
  a.off_x = p.off_x;
  a.off_zero = p.off_zero;
  a.zeros = (const uint16_t*)h->zeros;
  a.off_recv = p.off_recv;
  a.off_bar = p.off_bar;
  int cshift = 0;
  while ((1 << cshift) < p.csize) ++cshift;
  a.cshift = cshift;
  a.tq = h->nrt / p.nclusters;
  a.tr = h->nrt % p.nclusters;
  a.gq = h->ng >> cshift;
  a.gr = h->ng & (p.csize - 1);
  for (int k = 0; k < 2; ++k) {
    const unsigned long long d = (unsigned long long)std::max(1, a.gq + k);
    a.ngc_m[k] = ((1ull << 32) + d - 1) / d;
  }
  cudaLaunchAttribute attr[2];
  cudaLaunchConfig_t cfg = launch_config(p, s, attr, h->pdl);
  void* args[] = {&a};
  cudaError_t e = cudaLaunchKernelExC(&cfg, select_kernel(h->fmt, p.mode, p.strip, p.solo), args);
  if (e != cudaSuccess) return cuda_error(e, "gemv launch");
  return SPHQ_OK;
}

// The kernel reduces on chip and needs no global scratch; the caller's
// scratch is accepted and left untouched.  A plan that asked for scratch
// (ws_floats > 0) would have to pass `ws` and `tickets` to its kernel; no
// kernel takes them, so such a plan is refused rather than launched on the
// handle's own buffer.
sphq_status launch_gemv_scratch(sphq_handle h, const void* x, void* y, int batch, cudaStream_t s,
                                float* ws, unsigned* tickets) {
  (void)ws;
  (void)tickets;
  if (h->ws_floats > 0)
    return set_error(SPHQ_ERR_UNSUPPORTED,
                     "sphq_gemv_noalloc: this launch plan reduces through scratch that the "
                     "kernel does not take from the caller");
  return launch_gemv(h, x, y, batch, s);
}

}  // namespace sphq

