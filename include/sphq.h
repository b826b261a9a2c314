/*
 * sphq.h -- C ABI of the GB300 (sm_103a) SPHQuant decode library.
 *
 * The library runs one operation: the fused dequantize-GEMV that decodes
 * spherically quantised weights and multiplies them with fp16 activations
 * during autoregressive decode (SPHQuant, §3.4 "Efficient Kernel
 * Implementation" and App. D).  Each 8-D weight vector w_i of a row is stored
 * as 8 coordinate sign bits s_i, a direction index z_i into a codebook of
 * non-negative unit vectors c_k, and a 4-bit radius code q_i; every group of
 * 16 consecutive vectors (128 scalars) along the input dimension shares an
 * fp16 scale Delta_G and offset r_min_G (§3.1, Eq. (7)).  The library
 * reconstructs (Eq. (7) then Eq. (4))
 *
 *     r_hat_i = RN16(q_i * Delta_G + r_min_G)          one fp16 fused multiply-add
 *     w_hat_i = RN16(r_hat_i * c_{z_i})  with coordinate j negated when bit j of s_i is set
 *
 * and computes y[b][r] = sum_j w_hat[r][j] * x[b][j] with fp32 accumulation,
 * rounding y to fp16 (round to nearest even).
 *
 * Supported settings (§3.1 bit budget, App. B): bits = 2 (W2: K = 64 entries,
 * 8 sign + 6 index + 4 radius bits = 2.25 bits/weight) and bits = 3
 * (W3: K = 8192 entries, 8 + 13 + 4 = 3.125 bits/weight); batch 1..16.
 *
 * Conventions
 *   - All fp16 data are IEEE binary16 bit patterns (uint16_t storage).
 *   - Row-major everywhere.  rows = d_out, cols = d_in; cols % 128 == 0.
 *   - "device pointer": memory the current CUDA device can access
 *     (cudaMalloc, managed, or mapped pinned host memory).
 *   - Every call acts on the CUDA device that was current when the handle
 *     was created; the caller keeps that device current.
 *   - Errors: every call returns a status and launches nothing on error.
 *     sphq_last_error() gives a message for the calling thread.
 *   - No call traps, asserts or spins on the device.
 */
#ifndef SPHQ_H_
#define SPHQ_H_

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

/* Host logging: with the environment variable SPHQ_LOG set (and not "0"),
 * sphq_create prints the format and the GEMV launch plans and sphq_gemm its
 * launch shape to stderr. */

/* Opaque handle to one quantised weight matrix resident in device memory. */
typedef struct sphq_handle_s* sphq_handle;

/* A cudaStream_t (the runtime's stream type is `struct CUstream_st*`).
 * NULL means the legacy default stream. */
typedef struct CUstream_st* sphq_stream;

typedef enum sphq_status {
  SPHQ_OK = 0,
  SPHQ_ERR_INVALID_ARG = 1,   /* bad size, pointer, alignment or code value */
  SPHQ_ERR_UNSUPPORTED = 2,   /* bits/K/batch outside the supported set      */
  SPHQ_ERR_NOT_PACKED = 3,    /* gemv/decode before a successful sphq_pack   */
  SPHQ_ERR_CUDA = 4,          /* a CUDA runtime call failed                  */
  SPHQ_ERR_OOM = 5,           /* device allocation failed                    */
  SPHQ_ERR_DEVICE = 6,        /* no usable sm_103 device                     */
  SPHQ_ERR_TIMEOUT = 7        /* a kernel gave up an on-chip wait (sphq_check) */
} sphq_status;

#define SPHQ_MAX_BATCH 16
#define SPHQ_GEMM_MAX_BATCH (1 << 22)
#define SPHQ_GROUP_COLS 128   /* scalars per radius group (§3.1)   */
#define SPHQ_VECTOR_DIM 8     /* 8-D vectors (§3.1)                */

/*
 * sphq_create -- describe one quantised matrix and allocate its device storage.
 *
 *   rows, cols   d_out and d_in; rows >= 1, cols >= 128, cols % 128 == 0.
 *   bits         2 (W2) or 3 (W3), the target bit-width B of §3.1.
 *   K            codebook entries; must equal 2^(7*bits - 8) (§3.1): 64 or 8192.
 *   codebook     K x 8 fp16, entry k = direction c_k (§3.1, Eq. (5)); values are
 *                used as given (the paper's entries are non-negative unit vectors).
 *   scale        rows x (cols/128) fp16, Delta_G of Eq. (7) for group G = (row, col/128).
 *   offset       rows x (cols/128) fp16, r_min_G of Eq. (7).
 *   out          receives the handle.
 *
 * codebook, scale and offset may be host or device pointers (they are read
 * with cudaMemcpyDefault); the call is synchronous and copies them, so the
 * caller may free them on return.  The handle owns all device memory it
 * allocates (packed codes and parameters, codebook images, an error word and
 * the staging buffer of sphq_gemv_host).
 * Returns SPHQ_ERR_INVALID_ARG / SPHQ_ERR_UNSUPPORTED / SPHQ_ERR_OOM /
 * SPHQ_ERR_DEVICE / SPHQ_ERR_CUDA; *out is NULL on error.
 */
sphq_status sphq_create(int rows, int cols, int bits, int K, const void* codebook,
                        const void* scale, const void* offset, sphq_handle* out);

/*
 * sphq_create_v -- sphq_create for a general bit split (§3.1, Eq. (7),
 * Tab. 4, App. B): a vector costs 8 sign bits + D = log2(K) direction-index
 * bits + V = radius_bits radius bits, i.e. (8 + D + V) / 8 bits per weight.
 *
 *   bits = 3     K = 8192 (D = 13) with radius_bits 4 (W3, 3.125 b/w; the
 *                same as sphq_create) or 3 (3.00 b/w, radius codes q < 8).
 *   bits = 2     K = 64, 128 or 256 (D = 6, 7, 8) with D + V <= 10:
 *                8/6/4 (W2, 2.25 b/w; the same as sphq_create), 8/6/3,
 *                8/6/2 (2.00 b/w), 8/7/3, 8/7/2, 8/8/2 -- the splits of the
 *                bit-allocation ablation (Tab. 4).
 *
 * codebook is K x 8 fp16.  Other combinations give SPHQ_ERR_UNSUPPORTED.  The
 * other arguments, ownership and errors are those of sphq_create; sphq_pack
 * then rejects direction indices >= K and radius codes >= 2^V.
 */
sphq_status sphq_create_v(int rows, int cols, int bits, int radius_bits, int K,
                          const void* codebook, const void* scale, const void* offset,
                          sphq_handle* out);

/*
 * sphq_create_dim -- sphq_create_v for vectors of `dim` coordinates (§3.1
 * with k = dim; the vector-dimension comparison of Tab. 7).
 *
 *   dim 8   as sphq_create_v.
 *   dim 4   bits = 2, K = 4 (3B - 4 = 2 index bits), radius_bits = 4: 4 sign
 *           bits + 2 + 4 = 10 bits per 4 weights (2.5 bits per weight);
 *           codebook K x 4 fp16; radius groups of 128 scalars (32 vectors);
 *           sphq_pack takes sign bytes with bits 0-3 (values above 15 are
 *           rejected) and rows x cols/4 codes.  sphq_gemv, sphq_gemv_host,
 *           sphq_decode, sphq_export support it; sphq_gemm and sphq_encode
 *           do not (SPHQ_ERR_UNSUPPORTED).
 *   dim 16  bits = 2, K = 16384 (15B - 16 = 14 index bits), radius_bits = 4:
 *           16 sign bits + 14 + 4 = 34 bits per 16 weights (2.125 bits per
 *           weight); codebook K x 16 fp16 (512 KiB, beyond an SM's shared
 *           memory: the GEMV gathers its entries from global memory, so it
 *           is bound by random L2 reads, ~14% of the HBM rate on GB300);
 *           radius groups of 128 scalars (8 vectors); sphq_pack takes the
 *           sign argument as rows x cols/16 uint16 (bit j = coordinate j,
 *           2-byte aligned) and rows x cols/16 codes.  sphq_gemv (batch
 *           1..16; 9..16 as launches of 8 rows and the rest),
 *           sphq_gemv_host, sphq_gemv_noalloc, sphq_decode, sphq_export /
 *           sphq_import support it; sphq_gemm and sphq_encode do not.
 */
sphq_status sphq_create_dim(int rows, int cols, int dim, int bits, int radius_bits, int K,
                            const void* codebook, const void* scale, const void* offset,
                            sphq_handle* out);

/*
 * sphq_pack -- convert canonical codes into the library's device layout
 * (the finalise-and-pack step, App. A step 10).
 *
 *   sign   rows x (cols/8) uint8, bit j set <=> coordinate j of the vector is
 *          negative (§3.1, Eq. (3)); vector t of a row covers columns 8t..8t+7
 *          (4-D handles: rows x (cols/4), columns 4t..4t+3, bits 0-3; 16-D
 *          handles: rows x (cols/16) uint16, columns 16t..16t+15).
 *   idx    rows x (cols/8) uint16, direction index z < K (Eq. (5)).
 *   rcode  rows x (cols/8) uint8, radius code q < 2^V (Eq. (7); V = 4, or
 *          the handle's radius_bits).
 *   stream stream the pack kernel runs on.
 *
 * All three are device pointers.  The call validates every code on the
 * device and synchronises `stream` before returning; out-of-range codes give
 * SPHQ_ERR_INVALID_ARG and leave the handle unpacked.  May be called again
 * to replace the codes.  Not for use inside CUDA graph capture.
 */
sphq_status sphq_pack(sphq_handle h, const uint8_t* sign, const uint16_t* idx,
                      const uint8_t* rcode, sphq_stream stream);

/*
 * sphq_encode -- quantise a weight matrix with the handle's codebook (§3.1:
 * Eq. (3) signs / radius / direction, Eq. (5) nearest codebook direction,
 * Eq. (6) radius projection, Eq. (7) per-group radius codes) and pack it.
 *
 *   w       rows x cols fp32, device pointer, 16-byte aligned.
 *   sign    rows x (cols/8) uint8 out, idx uint16 out (2-byte aligned), rcode
 *           uint8 out: the canonical codes sphq_pack takes (device pointers).
 *   scale, offset  rows x (cols/128) fp16 out (Delta16, m16), or NULL.
 *
 * Every decision is taken in IEEE single precision in a fixed order (see
 * sphq_encode.cu): the codes equal those of a single-precision CPU encoder
 * bit for bit.  The handle's group parameters are replaced by the encoder's
 * and the codes are packed (as sphq_pack), so the handle is ready for
 * sphq_gemv / sphq_gemm on return.  Synchronous; allocates a temporary
 * rows x cols/8 fp32 buffer.  Errors as sphq_pack, plus SPHQ_ERR_TIMEOUT.
 */
sphq_status sphq_encode(sphq_handle h, const float* w, uint8_t* sign, uint16_t* idx,
                        uint8_t* rcode, void* scale, void* offset, sphq_stream stream);

/*
 * Codebook construction (the quantise side, run once per layer before
 * sphq_encode; the decode GEMV never calls these).  All pointers are device
 * pointers; every call is asynchronous on `stream` and takes its temporary
 * buffers from the stream-ordered allocator (cudaMallocAsync / cudaFreeAsync).
 * Results are deterministic (fixed summation orders).
 */

/*
 * sphq_sample_directions -- radius-weighted sampling of §3.1: 8-D vector i of
 * w is drawn with probability r_i^2 / sum_j r_j^2 (r_i = ||w_i||_2), by
 * inverse transform of caller-supplied uniforms.
 *
 *   w        nvec x 8 fp32 (the weight matrix, rows x cols with cols % 8 == 0,
 *            read as consecutive 8-D vectors), 4-byte aligned.
 *   u        samples uniforms in [0, 1), float64.
 *   dirs     samples x 8 float64 out: d = |w_i| / r_i (non-negative, unit).
 *   idx      samples int32 out (the drawn vector indices), or NULL.
 *
 * r_i^2 sums the squares in coordinate order in float64; prefix sums P of
 * r^2 run block-wise; the pick for u is the first i with P_i > u * P_total
 * (vectors of zero radius are never drawn; where u * P_total rounds up to the
 * total, the last vector of nonzero radius).  SPHQ_ERR_INVALID_ARG for NULL
 * pointers or non-positive sizes; all-zero weights give NaN directions.
 */
sphq_status sphq_sample_directions(const float* w, long long nvec, const double* u, int samples,
                                   double* dirs, int* idx, sphq_stream stream);

/*
 * sphq_kmeans_step -- one iteration of the spherical k-means that initialises
 * the codebook (§3.1, App. A step 6): every sample goes to the centre of
 * largest cosine (Eq. (5); scores d . c in float64 in coordinate order, each
 * product and sum rounded once, ties to the lowest index -- found by a
 * single-precision pass over all centres and exact re-scoring of those within
 * 1e-5 of the best), then every centre becomes the normalised sum of its
 * members (an empty cluster keeps its centre).
 *
 *   dirs         samples x 8 float64 unit directions (sphq_sample_directions).
 *   centres      K x 8 float64 centres of norm at most ~1 (unit in practice).
 *   centres_out  K x 8 float64 out; may equal `centres` (in place).
 *   assign       samples int32 out (the assignment), or NULL.
 *   objective    one float64 out: the mean assigned score before the update,
 *                or NULL.
 */
sphq_status sphq_kmeans_step(const double* dirs, int samples, const double* centres, int K,
                             double* centres_out, int* assign, double* objective,
                             sphq_stream stream);

/*
 * sphq_kmeans -- `iters` steps of sphq_kmeans_step in place on `centres`
 * (K x 8 float64: the initial centres in, the final ones out; the paper runs
 * 20 iterations on 65,536 samples, §4.1).  objective_history: `iters`
 * float64 out (the objective of each step), or NULL.
 */
sphq_status sphq_kmeans(const double* dirs, int samples, double* centres, int K, int iters,
                        double* objective_history, sphq_stream stream);

/*
 * sphq_angle_codebook -- the angle-parameterised codebook of §3.3: for entry
 * k, Eq. (sph-angle-logits) theta_j = eps + (pi/2 - 2 eps) sigmoid(phi_kj),
 * j = 1..7, and Eq. (sph-angle-codebook) c_1 = cos theta_1,
 * c_i = (prod_{j<i} sin theta_j) cos theta_i (2 <= i <= 7),
 * c_8 = prod_{j<=7} sin theta_j -- non-negative and unit by construction.
 *
 *   phi           K x 7 fp32 logits.
 *   eps           in [0, pi/4).
 *   codebook_f64  K x 8 float64 out, or NULL.
 *   codebook_f16  K x 8 fp16 out (round to nearest even: the codebook
 *                 sphq_create takes), or NULL; not both NULL.
 *
 * Computed in float64 with the device's sin, cos and exp.
 */
sphq_status sphq_angle_codebook(const float* phi, int K, double eps, double* codebook_f64,
                                void* codebook_f16, sphq_stream stream);

/*
 * sphq_gemv -- y = W_hat x for a batch of activation rows (§3.4, App. D).
 *
 *   x      batch x cols fp16, device pointer, 16-byte aligned.
 *   y      batch x rows fp16, device pointer, 4-byte aligned; written in full.
 *   batch  1..SPHQ_MAX_BATCH (16).  Each decoded weight serves every row of
 *          the batch: 1 row (and 2 rows on large small-codebook matrices)
 *          with the radius factored out of the dot products, 2-8 rows
 *          otherwise as the N dimension of the tensor-core products, 9-16
 *          rows as two such halves per decoded block (8-D vectors; 4-D and
 *          16-D handles run 9-16 rows as two launches).
 *
 * Asynchronous on `stream`: no host synchronisation and no allocation, so it
 * may be captured in a CUDA graph.  One handle should not run two gemv calls
 * concurrently (different streams): they share the handle's error word, so a
 * timeout reported by one could be charged to the other; calls on one stream,
 * or on different handles, are independent.  Numerics:
 * fp32 accumulation; |y - W_hat x| <= 1e-3 * sum_j |w_hat_j||x_j| + 2^-24 per
 * output (fp16 output rounding included), where W_hat is the exact decode
 * that sphq_decode returns.
 */
sphq_status sphq_gemv(sphq_handle h, const void* x, void* y, int batch, sphq_stream stream);

/*
 * sphq_gemv_host -- the same GEMV for host-resident activations and outputs.
 *
 *   x_host  batch x cols fp16 in host memory; y_host  batch x rows fp16.
 *
 * With page-locked (pinned) host buffers that are mapped into the device
 * address space (cudaHostAlloc / cudaHostRegister with mapping, the default
 * on this platform) and aligned like sphq_gemv's (x 16 bytes, y 4 bytes), a
 * small kernel reads x once over the CPU-GPU link into a device staging
 * buffer owned by the handle and the GEMV writes y in host memory directly:
 * two launches on `stream`, no copy operations.  Otherwise it
 * enqueues a copy of x into a device staging buffer owned by the handle, the
 * GEMV, and a copy of y back to y_host; with pageable buffers the CUDA runtime
 * makes those copies synchronous.  Either way the call returns without
 * waiting for the GPU (pageable copies aside) and y_host is valid once
 * `stream` has been synchronised.  Same numerics; the staging buffer makes
 * concurrent calls on one handle invalid, as for sphq_gemv.
 */
sphq_status sphq_gemv_host(sphq_handle h, const void* x_host, void* y_host, int batch,
                           sphq_stream stream);

/*
 * sphq_gemv_noalloc -- sphq_gemv for callers that must not allocate GPU memory
 * at run time.  (This entry point has no counterpart in the paper; it is an
 * interface choice of this library.)
 *
 * Who needs it: code that may not call cudaMalloc/cudaFree (or any allocator)
 * on its serving path -- a real-time decode loop, because cudaMalloc and
 * cudaFree synchronise the device and their latency is unbounded; programs
 * that reserve all device memory up front or run under a fixed memory budget;
 * and callers that hold their own allocator's lock or run inside a region
 * where allocation is not allowed.  sphq_gemv itself does not allocate either
 * (sphq_create allocated everything the handle needs); this variant adds a
 * guarantee that holds whatever reduction the kernel's launch plan uses: any
 * split-K scratch a plan needs comes from a single fixed 4 MiB device array
 * compiled into the library, which every GPU that loads the library holds
 * until the process exits, never from memory allocated at call time.  (The
 * current GEMV reduces its partial sums on chip, in shared and distributed
 * shared memory, so its plans need no scratch and calls only validate and
 * launch.)
 *
 * Arguments, numerics and asynchrony are those of sphq_gemv.  It calls no
 * cudaMalloc, cudaFree or other allocating routine.  Limits: a launch plan
 * that reduces through the array may cover at most 16384 row tiles (rows <=
 * 262144) and need at most 4128768 bytes of partial sums; beyond that the
 * call returns SPHQ_ERR_UNSUPPORTED with a message naming the limit.  The
 * current plans reduce on chip, so every shape sphq_gemv takes is accepted.
 * The current device must be the handle's device (else SPHQ_ERR_DEVICE).
 *
 * The first call on each device looks up the array's device address (one
 * cudaGetSymbolAddress with that device current) and caches it; make that
 * first call before any stream capture.  All calls share the one array and it
 * keeps the last call's contents: a call whose plan uses the array clears the
 * counters it needs (an asynchronous memset on `stream`), and such calls that
 * overlap on the GPU -- on different streams or from different host threads --
 * race on the array and give wrong results.  Serialise them, e.g. on one
 * stream.
 */
sphq_status sphq_gemv_noalloc(sphq_handle h, const void* x, void* y, int batch,
                              sphq_stream stream);

/*
 * sphq_gemm -- Y = X W_hat^T for any batch (prefill), on the tensor cores.
 * (The paper's kernel serves decode only; this is the large-batch form of the
 * same product, §3.4 with W_hat from Eq. (7) and Eq. (4).)
 *
 *   x      batch x cols fp16, device pointer, 16-byte aligned.
 *   y      batch x rows fp16, device pointer, 2-byte aligned; written in full.
 *   batch  1..SPHQ_GEMM_MAX_BATCH; efficient from a few dozen rows up (tiles
 *          of 128 activation rows); sphq_gemv is the fast path for batch <= 16.
 *          Batches of 9..64 run as GEMV launches of 3..16 rows (full modes:
 *          exact w_hat, fp32 accumulation of exact products) when that is
 *          estimated faster than the tensor-core kernel, y is 4-byte aligned
 *          and no shape is fixed with sphq_set_gemm_shape.
 *
 * Asynchronous on `stream`, no allocation (graph-capturable).  Numerics: each
 * weight is the exact fp16 W_hat of sphq_decode, products are exact in fp32,
 * fp32 accumulation, fp16 output rounded to nearest: the same bound as
 * sphq_gemv.  Concurrency as for sphq_gemv (the handle's error word).
 */
sphq_status sphq_gemm(sphq_handle h, const void* x, void* y, int batch, sphq_stream stream);

/*
 * sphq_gemm_workspace / sphq_gemm_ws -- the same product with a caller
 * workspace, in one of two forms (§3.4 with W_hat from Eq. (7) and Eq. (4)).
 *
 * Two-pass form, for large batches of the formats whose fused kernel is bound
 * by its codebook gathers: pass 1 decodes W_hat (rows x cols fp16, exactly
 * sphq_decode's output) into the workspace; pass 2 is a dense tensor-core
 * product that loads W_hat and X tiles with TMA.  The decode then costs one
 * write and one read of 2 bytes per weight per call instead of a
 * shared-memory gather per weight and activation tile.  Products,
 * accumulation order and rounding are those of sphq_gemm: Y is equal to
 * sphq_gemm's bit for bit.
 *
 * Split-K form, for batches of 41..256 (shape automatic) when the output
 * tiles are too few to fill the GPU and each tile's columns can be shared by
 * several CTAs of at least 16 radius groups each: every CTA multiplies its
 * share, writes an fp32 partial tile into the workspace, and the tile's last
 * CTA adds the partials in share order (a fixed order: repeatable bit for
 * bit; not equal to sphq_gemm's bits, within the same tolerance).  The
 * workspace holds the partial tiles and one counter per tile, which a memset
 * clears on the stream before the launch.  sphq_get_gemm_shape reports the
 * shares (ksplit).
 *
 * sphq_gemm_workspace sets *bytes to the split-K form's size where it
 * applies, else to rows x cols x 2 when the two-pass form is estimated
 * faster than the fused kernel for this batch, else to 0.
 *
 * sphq_gemm_ws takes the arguments of sphq_gemm plus the workspace:
 *   workspace        device pointer, 16-byte aligned, owned by the caller,
 *                    overwritten; NULL runs sphq_gemm.
 *   workspace_bytes  the split-K form runs where it applies and the
 *                    workspace holds its size; otherwise the two-pass form,
 *                    which needs rows x cols x 2 bytes (SPHQ_ERR_INVALID_ARG
 *                    otherwise).
 * Asynchronous on `stream` (two launches: the decode and the product, or the
 * counter memset and the product), no allocation.  A workspace must not be
 * shared by calls that overlap on the GPU.
 */
sphq_status sphq_gemm_workspace(sphq_handle h, int batch, size_t* bytes);
sphq_status sphq_gemm_ws(sphq_handle h, const void* x, void* y, int batch, void* workspace,
                         size_t workspace_bytes, sphq_stream stream);

/*
 * sphq_gemm_info / sphq_get_gemm_shape -- the launch shape sphq_gemm uses for
 * `batch`: activation tiles of 128 rows per CTA (1 or 2), weight rows per CTA
 * (128 or 256), columns per pipeline stage (64 or 32), ring stages, output
 * tiles (grid_x weight tiles x grid_y activation tiles of act_tiles x 128
 * rows), dynamic shared memory, and split_ctas: with two activation tiles,
 * the CTAs of one activation tile that take a final partial wave of output
 * tiles (two per output tile; 0 when the wave is not split), and ksplit: the
 * CTAs that share each output tile's columns in sphq_gemm_ws's split-K form
 * (1 where that form does not apply).  (No counterpart in the paper.)
 * sphq_set_gemm_shape -- fix act_tiles (1, 2; 0 = automatic) and weight_rows
 * (128, 256; 0 = automatic) for later sphq_gemm calls on the handle; 128 rows
 * go with one activation tile only; a fixed act_tiles also keeps the final
 * wave whole.  Invalid values give SPHQ_ERR_INVALID_ARG.
 */
typedef struct sphq_gemm_info {
  int act_tiles, weight_rows, stage_cols, stages, grid_x, grid_y;
  long long smem_bytes;
  int split_ctas, ksplit;
} sphq_gemm_info;
sphq_status sphq_get_gemm_shape(sphq_handle h, int batch, sphq_gemm_info* out);
sphq_status sphq_set_gemm_shape(sphq_handle h, int act_tiles, int weight_rows);

/*
 * sphq_check -- synchronise `stream`, then read and clear the handle's device
 * error word.  Every on-chip wait in the GEMV and GEMM kernels (mbarriers of
 * the staged copies, the cluster exchange, the tensor-core pipeline) gives up
 * after about two seconds instead of hanging, sets the word and lets the
 * kernel finish; the output of such a launch is invalid.  Returns
 * SPHQ_ERR_TIMEOUT if the word was set since the last check, SPHQ_OK
 * otherwise (or SPHQ_ERR_CUDA if the stream itself reports an error).
 */
sphq_status sphq_check(sphq_handle h, sphq_stream stream);

/*
 * sphq_export / sphq_import -- the packed device image of a handle as one
 * host blob and back (checkpointing quantised weights without re-packing).
 * (No counterpart in the paper.)
 *
 *   sphq_export(h, buf, capacity, &size): *size = blob bytes; with buf NULL
 *     only the size is returned.  Otherwise writes the blob (a 48-byte header
 *     "SPHQ" / format 1 / shape / split, then codebook, group parameters and
 *     the packed units) into host memory `buf` of `capacity` bytes
 *     (SPHQ_ERR_INVALID_ARG if smaller); the handle must be packed.
 *     Synchronous.
 *   sphq_import(buf, size, &h): a new packed handle on the current device
 *     from a blob (SPHQ_ERR_INVALID_ARG for a malformed or truncated blob).
 *     Blobs are tied to this library's layout version (format 1).
 */
sphq_status sphq_export(sphq_handle h, void* buf, size_t capacity, size_t* size);
sphq_status sphq_import(const void* buf, size_t size, sphq_handle* out);

/*
 * sphq_selftest_wait_timeout -- exercises the bounded-wait path: launches on
 * `stream` a one-CTA kernel whose single on-chip wait (an mbarrier nothing
 * arrives on) can never complete.  It gives up after about two seconds like
 * every wait of the library, sets the handle's error word and exits; the
 * next sphq_check returns SPHQ_ERR_TIMEOUT and the context stays usable.
 * For tests of the failure detection.  (No counterpart in the paper.)
 */
sphq_status sphq_selftest_wait_timeout(sphq_handle h, sphq_stream stream);

/*
 * sphq_decode -- write the decoded weights W_hat (rows x cols fp16, device
 * pointer, 16-byte aligned) on `stream`.  Bit-exact with Eq. (7) + Eq. (4) as
 * stated at the top of this header.  For verification; the GEMV never
 * materialises W_hat.  Asynchronous; no allocation.
 */
sphq_status sphq_decode(sphq_handle h, void* w, sphq_stream stream);

/*
 * sphq_bytes -- algorithmic bytes one gemv of this batch moves: packed codes
 * ((8 + log2 K + V) / 8 bits per weight: 2.25 (W2), 3.125 (W3), or the split
 * chosen with sphq_create_v) +
 * group parameters (4 bytes per 128 weights)
 * + codebook (K*16 bytes, once) + activations (2*batch*cols) + outputs
 * (2*batch*rows).  Returns 0 for a NULL handle or a batch outside 1..16.
 */
size_t sphq_bytes(sphq_handle h, int batch);

/*
 * sphq_plan_info / sphq_get_plan -- the launch shape sphq_gemv uses for one
 * batch size.  (No counterpart in the paper: introspection of this library's
 * work split.)  Row tiles of 16 rows go to thread-block clusters in contiguous
 * ranges; the CTAs of a cluster split the 128-column groups and reduce their
 * partial sums through distributed shared memory.  Fills *out; returns
 * SPHQ_ERR_INVALID_ARG for a NULL handle or out, or a batch outside 1..16
 * (4-D handles have no 16-row plan: grid 0 for batches above 8).
 */
typedef struct sphq_plan_info {
  int grid;              /* CTAs launched */
  int cluster_size;      /* CTAs per thread-block cluster: 1, 2, 4 or 8 */
  int clusters;          /* clusters, each with a contiguous range of row tiles */
  int tiles_per_cluster; /* most row tiles of one cluster */
  int warps_per_cta;
  int smem_bytes;        /* dynamic shared memory per CTA */
  int staged_x;          /* 1: activations copied to shared memory (the factored mode of batch
                            1, and of batch 2 on large small-codebook matrices), 0: read via L1 */
  int ctas_per_sm;       /* CTAs per SM the kernel is built for: 2 (W2 and the small-codebook
                            splits, at most 128 registers per thread) or 1 (W3; and W2 when
                            the row tiles bound the cluster count, with the whole register
                            file) */
} sphq_plan_info;
sphq_status sphq_get_plan(sphq_handle h, int batch, sphq_plan_info* out);

/*
 * sphq_set_cluster_size -- fix the cluster size of the launch shape used for
 * one batch size (1, 2, 4 or 8), or restore the automatic choice (0).  (No
 * counterpart in the paper: a tuning and testing knob.)  The library then
 * uses the cheapest shape at that size by its cost model.  Results do not
 * change beyond fp32 summation order.  Returns SPHQ_ERR_UNSUPPORTED when the
 * matrix has fewer 128-column groups than the size or no launch at that size
 * fits the device (the previous shape stays), SPHQ_ERR_INVALID_ARG for bad
 * arguments.  Not safe while a GEMV on the handle is being enqueued from
 * another thread; kernels already enqueued keep their shape.
 */
sphq_status sphq_set_cluster_size(sphq_handle h, int batch, int cluster_size);

/*
 * sphq_set_pdl -- launch this handle's GEMVs as programmatic dependent
 * launches (enabled = 1, the default) or as plain stream-ordered launches
 * (0).  (No counterpart in the paper: a launch option.)  With it, a GEMV's
 * CTAs may start while the previous kernel on the stream is finishing and
 * load their codes and codebook before waiting for it; the activations are
 * read only after that kernel completes, so results are the same either way
 * (bit for bit).  Applies to sphq_gemv, sphq_gemv_noalloc and
 * sphq_gemv_host; launches already enqueued or captured keep their setting.
 * SPHQ_ERR_INVALID_ARG for a NULL handle or another value.
 */
sphq_status sphq_set_pdl(sphq_handle h, int enabled);

/* Release the handle and its device memory.  NULL is accepted.  The caller
 * ensures no kernel using the handle is still running. */
sphq_status sphq_destroy(sphq_handle h);

/* Message describing the last error returned on the calling thread ("" if none). */
const char* sphq_last_error(void);

/* Library ABI version (major*10000 + minor*100 + patch). */
int sphq_version(void);

#ifdef __cplusplus
}
#endif

#endif /* SPHQ_H_ */
