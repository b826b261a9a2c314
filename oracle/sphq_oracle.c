/*
 * SPHQuant CPU oracle -- TEST INFRASTRUCTURE ONLY.
 *
 * A plain, slow, obviously correct float64 implementation of what the
 * spherical dequantize-GEMV computes.  Only tests/, __graft_entry__.smoke()
 * and the cpu_baseline / reference legs of bench.py may load this library;
 * the product path (paper_2609_24875_gb300/) never does.  It shares no code,
 * header, table or helper with the CUDA path.
 *
 * What is computed (paper notation, SPHQuant §3.1 and §3.4):
 *   per 8-D vector i of row `row`, slot t (columns 8t .. 8t+7):
 *     s_i  : 8 sign bits, bit j set  <=>  coordinate j is negative
 *     z_i  : index into the positive-direction codebook C = {c_k}
 *     q_i  : V = 4 bit radius code
 *   per group G of 16 consecutive vectors (128 scalars) along the input dim:
 *     Delta_G (scale) and r_min_G (offset), both fp16
 *   Eq. (7):  r_hat_i = r_min_G + q_i * Delta_G           (one fused multiply-add)
 *   Eq. (4):  w_hat_i = r_hat_i * s_i (.) c_{z_i}
 *   y[b][row] = sum_j w_hat[row][j] * x[b][j]
 *
 * Rounding reading (the paper states "a fused multiply-add applies the group's
 * scale and offset" and fp16 "half2" arithmetic, App. D; it gives no rounding
 * rule): r_hat is the exact value q*Delta + r_min rounded ONCE to binary16
 * (an fp16 FMA); each decoded weight is the exact product r_hat * c_{z,j}
 * rounded once to binary16; a set sign bit flips the binary16 sign bit.
 * Every intermediate here is exact in float64 (q*Delta + r_min needs at most
 * 45 significant bits; a product of two binary16 values needs 22), so the
 * only roundings are the ones named above.
 *
 * binary16 rounding is written from the IEEE 754 definition: nearest
 * representable value, ties to the value with an even significand,
 * gradual underflow (subnormals), overflow to infinity at or above 65520.
 *
 * Build (done by __graft_entry__.build()):
 *   gcc -O2 -fopenmp -ffp-contract=off -shared -fPIC sphq_oracle.c -o libsphq_oracle.so -lm
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define SPHQO_VEC 8      /* vector dimension k = 8 (§3.1)                     */
#define SPHQO_GROUP 16   /* vectors per radius group: 128 scalars (§3.1, §3.4) */

/* ------------------------------------------------------------------------- */
/* threads                                                                    */
/* ------------------------------------------------------------------------- */

static int g_threads = 1;

void sphqo_set_threads(int n) {
  g_threads = n < 1 ? 1 : n;
#ifdef _OPENMP
  omp_set_num_threads(g_threads);
#endif
}

int sphqo_get_threads(void) { return g_threads; }

int sphqo_max_threads(void) {
#ifdef _OPENMP
  return omp_get_num_procs();
#else
  return 1;
#endif
}

/* ------------------------------------------------------------------------- */
/* IEEE 754 binary16                                                          */
/* ------------------------------------------------------------------------- */

/* Value of a binary16 bit pattern. */
double sphqo_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1F;
  int m = h & 0x3FF;
  double v;
  if (e == 0) {
    v = ldexp((double)m, -24);                 /* zero or subnormal: m * 2^-24 */
  } else if (e == 31) {
    v = m ? NAN : INFINITY;
  } else {
    v = ldexp((double)(1024 + m), e - 25);     /* (1 + m/1024) * 2^(e-15) */
  }
  return sign ? -v : v;
}

/* Round a real value (given exactly as a double) to binary16, nearest-even. */
uint16_t sphqo_round_half(double v) {
  uint16_t sign = signbit(v) ? 0x8000u : 0u;
  if (isnan(v)) return (uint16_t)(sign | 0x7E00u);
  double a = fabs(v);
  if (a >= 65520.0) return (uint16_t)(sign | 0x7C00u);  /* to infinity */
  if (a == 0.0) return sign;

  /* exponent of the leading bit: a in [2^e, 2^(e+1)) */
  int E;
  frexp(a, &E);          /* a = f * 2^E, f in [0.5, 1) */
  int e = E - 1;
  /* spacing of binary16 values around a */
  int qexp = (e < -14) ? -24 : e - 10;
  double n = ldexp(a, -qexp);      /* a in units of the spacing; exact */
  double fl = floor(n);
  double frac = n - fl;
  double r;
  if (frac > 0.5) {
    r = fl + 1.0;
  } else if (frac < 0.5) {
    r = fl;
  } else {
    r = (fmod(fl, 2.0) == 0.0) ? fl : fl + 1.0;  /* tie: keep the even one */
  }
  double R = ldexp(r, qexp);       /* the rounded value, exact */
  if (R >= 65536.0) return (uint16_t)(sign | 0x7C00u);
  if (R < ldexp(1.0, -14)) {
    /* subnormal (or zero): significand field = R / 2^-24 */
    return (uint16_t)(sign | (uint16_t)ldexp(R, 24));
  }
  int E2;
  double f2 = frexp(R, &E2);       /* R = f2 * 2^E2, f2 in [0.5, 1) */
  int e2 = E2 - 1;
  int mant = (int)ldexp(f2 * 2.0 - 1.0, 10);  /* (R / 2^e2 - 1) * 1024 */
  return (uint16_t)(sign | (uint16_t)((e2 + 15) << 10) | (uint16_t)mant);
}

void sphqo_round_half_array(const double* v, uint16_t* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = sphqo_round_half(v[i]);
}

void sphqo_half_to_double_array(const uint16_t* h, double* out, int64_t n) {
  for (int64_t i = 0; i < n; ++i) out[i] = sphqo_half_to_double(h[i]);
}

/* ------------------------------------------------------------------------- */
/* Eq. (7) and Eq. (4): decode                                               */
/* ------------------------------------------------------------------------- */

/* r_hat = RN16(q * Delta + r_min), Eq. (7) with one fused multiply-add. */
uint16_t sphqo_radius(int q, uint16_t scale, uint16_t offset) {
  double delta = sphqo_half_to_double(scale);
  double rmin = sphqo_half_to_double(offset);
  double exact = (double)q * delta + rmin;   /* exact in float64 */
  return sphqo_round_half(exact);
}

/* One 8-D block: w_hat_j = s_j * RN16(r_hat * c_{z,j}), Eq. (4). */
void sphqo_decode_vector(uint8_t sign, const uint16_t* c /* 8 fp16 */, uint16_t r_hat,
                         uint16_t* out /* 8 fp16 */) {
  double r = sphqo_half_to_double(r_hat);
  for (int j = 0; j < SPHQO_VEC; ++j) {
    double prod = r * sphqo_half_to_double(c[j]);    /* exact */
    uint16_t w = sphqo_round_half(prod);
    if ((sign >> j) & 1) w ^= 0x8000u;
    out[j] = w;
  }
}

/*
 * Decode a rows x cols matrix into binary16 bit patterns, row-major.
 *   codebook : K x 8 binary16
 *   scale, offset : rows x (cols/128) binary16 (Delta_G, r_min_G)
 *   sign, rcode : rows x (cols/8) bytes; idx : rows x (cols/8) u16
 * Returns 0, or -1 on a bad shape or an out-of-range code.
 */
int sphqo_decode(int rows, int cols, int K, const uint16_t* codebook,
                 const uint16_t* scale, const uint16_t* offset,
                 const uint8_t* sign, const uint16_t* idx, const uint8_t* rcode,
                 uint16_t* w_out) {
  if (rows < 0 || cols < 0 || cols % (SPHQO_VEC * SPHQO_GROUP) != 0 || K <= 0) return -1;
  const int nv = cols / SPHQO_VEC;
  const int ng = cols / (SPHQO_VEC * SPHQO_GROUP);
  int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
  for (int row = 0; row < rows; ++row) {
    for (int t = 0; t < nv; ++t) {
      int64_t v = (int64_t)row * nv + t;
      int64_t g = (int64_t)row * ng + t / SPHQO_GROUP;
      int k = idx[v];
      int q = rcode[v];
      if (k >= K || q > 15) { bad = 1; continue; }
      uint16_t r_hat = sphqo_radius(q, scale[g], offset[g]);
      sphqo_decode_vector(sign[v], codebook + (int64_t)k * SPHQO_VEC, r_hat,
                          w_out + (int64_t)row * cols + (int64_t)t * SPHQO_VEC);
    }
  }
  return bad ? -1 : 0;
}

/* ------------------------------------------------------------------------- */
/* dense matvec in float64                                                    */
/* ------------------------------------------------------------------------- */

/*
 * y[b][row] = sum_j w[row][j] * x[b][j], in float64 with every product exact.
 * absdot[b][row] = sum_j |w[row][j]| * |x[b][j]|, the scale of the tolerance.
 * w : rows x cols binary16, x : B x cols binary16, y/absdot : B x rows.
 */
int sphqo_gemv(int rows, int cols, int B, const uint16_t* w, const uint16_t* x,
               double* y, double* absdot) {
  if (rows < 0 || cols < 0 || B < 1) return -1;
  double* xd = (double*)malloc(sizeof(double) * (size_t)B * (size_t)(cols ? cols : 1));
  if (!xd) return -1;
  for (int64_t i = 0; i < (int64_t)B * cols; ++i) xd[i] = sphqo_half_to_double(x[i]);
#pragma omp parallel for schedule(static)
  for (int row = 0; row < rows; ++row) {
    for (int b = 0; b < B; ++b) {
      double acc = 0.0, aacc = 0.0;
      for (int j = 0; j < cols; ++j) {
        double wv = sphqo_half_to_double(w[(int64_t)row * cols + j]);
        double xv = xd[(int64_t)b * cols + j];
        acc += wv * xv;
        aacc += fabs(wv) * fabs(xv);
      }
      y[(int64_t)b * rows + row] = acc;
      if (absdot) absdot[(int64_t)b * rows + row] = aacc;
    }
  }
  free(xd);
  return 0;
}

/*
 * Decode + matvec row by row without materialising the matrix: the plain
 * oracle path that bench.py times as the CPU baseline.  Same arithmetic as
 * sphqo_decode followed by sphqo_gemv.
 */
int sphqo_decode_gemv(int rows, int cols, int K, int B, const uint16_t* codebook,
                      const uint16_t* scale, const uint16_t* offset,
                      const uint8_t* sign, const uint16_t* idx, const uint8_t* rcode,
                      const uint16_t* x, double* y, double* absdot) {
  if (rows < 0 || cols < 0 || cols % (SPHQO_VEC * SPHQO_GROUP) != 0 || K <= 0 || B < 1 ||
      B > 8)
    return -1;
  const int nv = cols / SPHQO_VEC;
  const int ng = cols / (SPHQO_VEC * SPHQO_GROUP);
  double* xd = (double*)malloc(sizeof(double) * (size_t)B * (size_t)(cols ? cols : 1));
  if (!xd) return -1;
  for (int64_t i = 0; i < (int64_t)B * cols; ++i) xd[i] = sphqo_half_to_double(x[i]);
  int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
  for (int row = 0; row < rows; ++row) {
    double acc[8], aacc[8];
    for (int b = 0; b < B; ++b) { acc[b] = 0.0; aacc[b] = 0.0; }
    for (int t = 0; t < nv; ++t) {
      int64_t v = (int64_t)row * nv + t;
      int64_t g = (int64_t)row * ng + t / SPHQO_GROUP;
      int k = idx[v];
      int q = rcode[v];
      if (k >= K || q > 15) { bad = 1; continue; }
      uint16_t blk[SPHQO_VEC];
      sphqo_decode_vector(sign[v], codebook + (int64_t)k * SPHQO_VEC,
                          sphqo_radius(q, scale[g], offset[g]), blk);
      for (int j = 0; j < SPHQO_VEC; ++j) {
        double wv = sphqo_half_to_double(blk[j]);
        for (int b = 0; b < B; ++b) {
          double xv = xd[(int64_t)b * cols + t * SPHQO_VEC + j];
          acc[b] += wv * xv;
          aacc[b] += fabs(wv) * fabs(xv);
        }
      }
    }
    for (int b = 0; b < B; ++b) {
      y[(int64_t)b * rows + row] = acc[b];
      if (absdot) absdot[(int64_t)b * rows + row] = aacc[b];
    }
  }
  free(xd);
  return bad ? -1 : 0;
}

/* ------------------------------------------------------------------------- */
/* The paper's W2 word format (§3.4, Fig. 3(b), App. A step 10)               */
/* ------------------------------------------------------------------------- */

/*
 * Per vector one 16-bit base word: bits [0,8) signs, [8,14) the 6-bit
 * direction index, [14,16) the two low bits of the 4-bit radius code.
 * Per group of 16 vectors one 32-bit word holding the two high radius bits
 * of each vector; vector j of the group (j = t mod 16) owns bits [2j, 2j+2).
 */
int sphqo_pack_w2_words(int rows, int cols, const uint8_t* sign, const uint16_t* idx,
                        const uint8_t* rcode, uint16_t* base, uint32_t* extra) {
  if (rows < 0 || cols % (SPHQO_VEC * SPHQO_GROUP) != 0) return -1;
  const int nv = cols / SPHQO_VEC;
  const int ng = nv / SPHQO_GROUP;
  for (int row = 0; row < rows; ++row) {
    for (int g = 0; g < ng; ++g) extra[(int64_t)row * ng + g] = 0u;
    for (int t = 0; t < nv; ++t) {
      int64_t v = (int64_t)row * nv + t;
      if (idx[v] >= 64 || rcode[v] > 15) return -1;
      base[v] = (uint16_t)(sign[v] | (idx[v] << 8) | ((rcode[v] & 3) << 14));
      extra[(int64_t)row * ng + t / SPHQO_GROUP] |=
          (uint32_t)((rcode[v] >> 2) & 3) << (2 * (t % SPHQO_GROUP));
    }
  }
  return 0;
}

int sphqo_unpack_w2_words(int rows, int cols, const uint16_t* base, const uint32_t* extra,
                          uint8_t* sign, uint16_t* idx, uint8_t* rcode) {
  if (rows < 0 || cols % (SPHQO_VEC * SPHQO_GROUP) != 0) return -1;
  const int nv = cols / SPHQO_VEC;
  const int ng = nv / SPHQO_GROUP;
  for (int row = 0; row < rows; ++row) {
    for (int t = 0; t < nv; ++t) {
      int64_t v = (int64_t)row * nv + t;
      uint32_t e = extra[(int64_t)row * ng + t / SPHQO_GROUP];
      sign[v] = (uint8_t)(base[v] & 0xFF);
      idx[v] = (uint16_t)((base[v] >> 8) & 0x3F);
      rcode[v] = (uint8_t)(((base[v] >> 14) & 3) | (((e >> (2 * (t % SPHQO_GROUP))) & 3) << 2));
    }
  }
  return 0;
}

/* ------------------------------------------------------------------------- */
/* Eqs. (3), (5), (6), (7) in IEEE binary32: the encoder                      */
/* ------------------------------------------------------------------------- */

/*
 * The encoder of §3.1 (Eq. (3) decomposition, Eq. (5) nearest direction,
 * Eq. (6) radius projection, Eq. (7) group quantisation) with every decision
 * taken in single precision, in this order (the float64 encoder in
 * oracle/__init__.py is the same algorithm in double precision):
 *   p_j = |w_j|, sign bit j = (w_j < 0)
 *   r = sqrt(fma(p_7, p_7, ... fma(p_0, p_0, 0)))     (correctly rounded sqrt)
 *   d_j = p_j / max(r, 1e-12)                          (correctly rounded division)
 *   score_k = fma(d_7, c_k7, ... fma(d_0, c_k0, 0)); z = argmax, ties -> lowest k
 *   r~ = fma(p_7, c_z7, ... fma(p_0, c_z0, 0))
 *   per group of 16 vectors: Delta = (max r~ - min r~) / (2^V - 1),
 *   Delta16 = RN16(Delta), m16 = RN16(min r~),
 *   q = 0 if Delta16 = 0, else clip(floor((r~ - m16) / Delta16 + 0.5), 0, 2^V - 1)
 * fma is the fused multiply-add (one rounding).  `codebook` is K x 8 binary16.
 */
static float sphqo_half_to_float(uint16_t h) { return (float)sphqo_half_to_double(h); }

int sphqo_encode_f32(int rows, int cols, int K, int V, const uint16_t* codebook, const float* w,
                     uint8_t* sign, uint16_t* idx, uint8_t* rcode, uint16_t* scale,
                     uint16_t* offset) {
  if (rows < 0 || cols % (SPHQO_VEC * SPHQO_GROUP) != 0 || K < 1 || V < 1 || V > 8) return -1;
  const int nv = cols / SPHQO_VEC;
  const int ng = nv / SPHQO_GROUP;
  const int qmax = (1 << V) - 1;
  float* cf = (float*)malloc(sizeof(float) * (size_t)K * SPHQO_VEC);
  if (!cf) return -2;
  for (int64_t i = 0; i < (int64_t)K * SPHQO_VEC; ++i) cf[i] = sphqo_half_to_float(codebook[i]);
#pragma omp parallel for schedule(dynamic, 4) num_threads(g_threads)
  for (int row = 0; row < rows; ++row) {
    for (int g = 0; g < ng; ++g) {
      float rt[SPHQO_GROUP];
      for (int v = 0; v < SPHQO_GROUP; ++v) {
        const int64_t t = (int64_t)row * nv + (int64_t)g * SPHQO_GROUP + v;
        const float* x = w + t * SPHQO_VEC;
        float p[SPHQO_VEC], d[SPHQO_VEC];
        uint8_t s = 0;
        float acc = 0.0f;
        for (int j = 0; j < SPHQO_VEC; ++j) {
          p[j] = fabsf(x[j]);
          if (x[j] < 0.0f) s |= (uint8_t)(1u << j);
          acc = fmaf(p[j], p[j], acc);
        }
        const float r = sqrtf(acc);
        const float den = r > 1e-12f ? r : 1e-12f;
        for (int j = 0; j < SPHQO_VEC; ++j) d[j] = p[j] / den;
        int best = 0;
        float bs = 0.0f;
        for (int k = 0; k < K; ++k) {
          float sc = 0.0f;
          for (int j = 0; j < SPHQO_VEC; ++j) sc = fmaf(d[j], cf[(int64_t)k * SPHQO_VEC + j], sc);
          if (k == 0 || sc > bs) {
            bs = sc;
            best = k;
          }
        }
        float rr = 0.0f;
        for (int j = 0; j < SPHQO_VEC; ++j) rr = fmaf(p[j], cf[(int64_t)best * SPHQO_VEC + j], rr);
        rt[v] = rr;
        sign[t] = s;
        idx[t] = (uint16_t)best;
      }
      float mn = rt[0], mx = rt[0];
      for (int v = 1; v < SPHQO_GROUP; ++v) {
        mn = fminf(mn, rt[v]);
        mx = fmaxf(mx, rt[v]);
      }
      const float delta = (mx - mn) / (float)qmax;
      const uint16_t d16 = sphqo_round_half((double)delta);
      const uint16_t m16 = sphqo_round_half((double)mn);
      const float df = sphqo_half_to_float(d16), mf = sphqo_half_to_float(m16);
      scale[(int64_t)row * ng + g] = d16;
      offset[(int64_t)row * ng + g] = m16;
      for (int v = 0; v < SPHQO_GROUP; ++v) {
        int q = 0;
        if (df != 0.0f) {
          const float u = floorf((rt[v] - mf) / df + 0.5f);
          q = u < 0.0f ? 0 : (u > (float)qmax ? qmax : (int)u);
        }
        rcode[(int64_t)row * nv + (int64_t)g * SPHQO_GROUP + v] = (uint8_t)q;
      }
    }
  }
  free(cf);
  return 0;
}

/* ------------------------------------------------------------------------- */
/* Eq. (7) and Eq. (4) for vectors of `dim` coordinates (Tab. 7)               */
/* ------------------------------------------------------------------------- */

/*
 * The decode of sphqo_decode for vectors of dim = 4, 8 or 16 coordinates (§3.1
 * with k = dim; the 4-D and 16-D configurations of Tab. 7).  Radius groups
 * span 128 scalars (128 / dim vectors) as for 8-D vectors; radius codes have V
 * bits.  sign is rows x (cols/dim) u16 (bit j = coordinate j negative),
 * idx u16, rcode u8; codebook is K x dim binary16.
 */
int sphqo_decode_dim(int rows, int cols, int dim, int K, int V, const uint16_t* codebook,
                     const uint16_t* scale, const uint16_t* offset, const uint16_t* sign,
                     const uint16_t* idx, const uint8_t* rcode, uint16_t* w_out) {
  if (rows < 0 || cols < 0 || cols % 128 != 0 || K <= 0 || V < 1 || V > 8 ||
      (dim != 4 && dim != 8 && dim != 16))
    return -1;
  const int nv = cols / dim;
  const int ng = cols / 128;
  const int per_group = 128 / dim;
  int bad = 0;
#pragma omp parallel for schedule(static) reduction(| : bad)
  for (int row = 0; row < rows; ++row) {
    for (int t = 0; t < nv; ++t) {
      const int64_t v = (int64_t)row * nv + t;
      const int64_t g = (int64_t)row * ng + t / per_group;
      const int k = idx[v];
      const int q = rcode[v];
      if (k >= K || q >= (1 << V)) {
        bad = 1;
        continue;
      }
      const double r = sphqo_half_to_double(sphqo_radius(q, scale[g], offset[g]));
      for (int j = 0; j < dim; ++j) {
        uint16_t w = sphqo_round_half(r * sphqo_half_to_double(codebook[(int64_t)k * dim + j]));
        if ((sign[v] >> j) & 1) w ^= 0x8000u;
        w_out[(int64_t)row * cols + (int64_t)t * dim + j] = w;
      }
    }
  }
  return bad ? -1 : 0;
}
