/*
 * zo_oracle.c -- plain, slow, single-threaded CPU oracle for the parameter-space
 * hot path of 1.5-SPSA ("Probe-Space Preconditioning for Fast and Stable
 * Zero-Order Training", Chaubard, Kochenderfer, Re).
 *
 * THIS IS TEST INFRASTRUCTURE. Only the test suite, __graft_entry__.smoke() and
 * the CPU-baseline leg of bench.py may load or run it. The product library
 * (paper_2609_38095_gb300) shares no code, header, table or constant with this
 * file and never loads it.
 *
 * Every routine is the definition written out in the most direct form, in the
 * order the paper states it: no blocking, no caching of random blocks, no
 * vectorisation. Floating point follows plain C semantics; build with
 * -ffp-contract=off and without -ffast-math so that every float operation is a
 * single IEEE-754 operation rounded to nearest-even.
 *
 * Parity status of each function (what pins it, see tests/test_oracle_*.py):
 *   philox4x32_10        pinned: Triton's independent Philox (CPU interpreter),
 *                        uniformity / independence statistics.
 *   probe_bit/bytes      pinned: brute force unpack rule (Appendix F layout),
 *                        statistics.
 *   dtype conversions    pinned: numpy float16 and torch bfloat16 casts, on
 *                        edge cases and (property tests) arbitrary fp32 bits;
 *                        NaN results in the one encoding read above (NaN-ness
 *                        pinned against numpy, the encoding is a reading).
 *   perturb              pinned: brute force, exact-grid restore identity,
 *                        restore drift bound, numpy fp32 addition (property).
 *   precondition         pinned: worked value of Sec. 6 (|c|=1e8, alpha=0.1),
 *                        alpha=0 / alpha=1 special cases, quadratic closed form,
 *                        invariants on arbitrary triples (property); relative
 *                        curvature: alpha=1 closed form, equal magnitudes,
 *                        scale invariance, degenerate cases.
 *   update               pinned: K=1 equals perturb, fp64 brute force sum,
 *                        update(c) then update(-c), quadratic gradient identity.
 *   update_sequential    pinned: equals K perturb passes.
 *   quadratic_loss       pinned: closed form on constant inputs, math.fsum.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>

#define ORC_F32 0
#define ORC_BF16 1
#define ORC_F16 2

#define ORC_OK 0
#define ORC_ERR_ARG (-1)
#define ORC_ERR_NONFINITE (-4)

/* ------------------------------------------------------------------------- */
/* Philox4x32-10 (Salmon, Moraes, Dror, Shaw, "Parallel Random Numbers: As   */
/* Easy as 1, 2, 3", SC'11). The paper only asks for a seed-driven packed     */
/* Rademacher generator (Sec. 4.3, "Bit-Packed perturbations"; Algorithm 1,  */
/* PackedPerturbation(s_i)); Philox is the counter-based generator chosen    */
/* here so that any element of any probe can be produced on its own.          */
/* ------------------------------------------------------------------------- */

/* Round multipliers and key increments as published for Philox4x32. */
static const uint32_t PHILOX_M0 = 0xD2511F53u;
static const uint32_t PHILOX_M1 = 0xCD9E8D57u;
static const uint32_t PHILOX_W0 = 0x9E3779B9u; /* golden ratio */
static const uint32_t PHILOX_W1 = 0xBB67AE85u; /* sqrt(3) - 1 */

/* One Philox S-box round: two 32x32->64 products, the high halves xored with
 * the other counter words and the key, the low halves passed through. */
static void philox_round(uint32_t x[4], const uint32_t k[2]) {
  uint64_t p0 = (uint64_t)PHILOX_M0 * (uint64_t)x[0];
  uint64_t p1 = (uint64_t)PHILOX_M1 * (uint64_t)x[2];
  uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
  uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
  uint32_t y0 = hi1 ^ x[1] ^ k[0];
  uint32_t y1 = lo1;
  uint32_t y2 = hi0 ^ x[3] ^ k[1];
  uint32_t y3 = lo0;
  x[0] = y0;
  x[1] = y1;
  x[2] = y2;
  x[3] = y3;
}

/* Ten rounds; the key is bumped by the Weyl increments between rounds. */
void oracle_philox4x32_10(const uint32_t ctr[4], const uint32_t key[2], uint32_t out[4]) {
  uint32_t x[4] = {ctr[0], ctr[1], ctr[2], ctr[3]};
  uint32_t k[2] = {key[0], key[1]};
  for (int r = 0; r < 10; ++r) {
    if (r > 0) {
      k[0] += PHILOX_W0;
      k[1] += PHILOX_W1;
    }
    philox_round(x, k);
  }
  out[0] = x[0];
  out[1] = x[1];
  out[2] = x[2];
  out[3] = x[3];
}

/* ------------------------------------------------------------------------- */
/* Probe definition.                                                          */
/*                                                                           */
/* z_k is Rademacher, one bit per parameter (Sec. 2 "1SPSA", Sec. 4.3        */
/* "Bit-Packed perturbations"), with the unpack rule of Appendix F: bit 1    */
/* means +1, bit 0 means -1.                                                 */
/*                                                                           */
/* Element index g is the "virtual" flattened index: tensor t starts at      */
/* S_t = sum over earlier tensors of numel rounded up to a multiple of 16.   */
/*                                                                           */
/* Packing 1 (default, one generated bit per (element, probe)): Philox block */
/* b = g / 16 with probe group q = k / 8 gives 128 bits; byte (g mod 16) of  */
/* that output (little-endian within each 32-bit word) holds the signs of    */
/* probes 8q..8q+7 of element g, probe k in bit (k mod 8).                   */
/*                                                                           */
/* Packing 8 (one generated byte per (element, probe)): Philox block         */
/* b = g / 16 with the probe id k itself in the counter; the sign of element */
/* g is bit 0 of byte (g mod 16).                                            */
/* ------------------------------------------------------------------------- */

static int g_packing = 1; /* 1 or 8, see above */

/* Select the probe packing (1 or 8); returns ORC_ERR_ARG otherwise. */
int oracle_set_packing(int bits_per_value) {
  if (bits_per_value != 1 && bits_per_value != 8) return -1;
  g_packing = bits_per_value;
  return 0;
}

int oracle_get_packing(void) { return g_packing; }

/* The 16 output bytes of Philox(counter = (b_lo, b_hi, q, 0), key = seed). */
static void philox_block_bytes(uint64_t seed, uint64_t b, uint32_t q, uint8_t bytes[16]) {
  uint32_t ctr[4] = {(uint32_t)(b & 0xFFFFFFFFu), (uint32_t)(b >> 32), q, 0u};
  uint32_t key[2] = {(uint32_t)(seed & 0xFFFFFFFFu), (uint32_t)(seed >> 32)};
  uint32_t out[4];
  oracle_philox4x32_10(ctr, key, out);
  for (int m = 0; m < 16; ++m) bytes[m] = (uint8_t)((out[m / 4] >> (8 * (m % 4))) & 0xFFu);
}

/* Probe bit of element g for probe k: 1 means z = +1, 0 means z = -1. */
int oracle_probe_bit(uint64_t seed, uint32_t k, uint64_t g) {
  uint8_t bytes[16];
  if (g_packing == 8) {
    philox_block_bytes(seed, g / 16u, k, bytes);
    return bytes[g % 16u] & 1;
  }
  philox_block_bytes(seed, g / 16u, k / 8u, bytes);
  return (bytes[g % 16u] >> (k % 8u)) & 1;
}

/* z_k[g] in {-1, +1}. */
int oracle_probe_sign(uint64_t seed, uint32_t k, uint64_t g) {
  return oracle_probe_bit(seed, k, g) ? +1 : -1;
}

/* Probe k packed one bit per element, eight elements per byte, element 8j+i
 * in bit i of byte j (the layout Appendix F unpacks). Bytes first..first+n-1. */
void oracle_probe_bytes(uint64_t seed, uint32_t k, int64_t first, int64_t n, uint8_t* out) {
  for (int64_t j = 0; j < n; ++j) {
    uint64_t byte_index = (uint64_t)(first + j);
    uint8_t v = 0;
    for (int i = 0; i < 8; ++i) {
      uint64_t g = 8u * byte_index + (uint64_t)i;
      v = (uint8_t)(v | (oracle_probe_bit(seed, k, g) << i));
    }
    out[j] = v;
  }
}

/* Unpacked probe values z_k[g] as int8 for g = first..first+n-1. */
void oracle_probe_signs(uint64_t seed, uint32_t k, int64_t first, int64_t n, int8_t* out) {
  for (int64_t j = 0; j < n; ++j) out[j] = (int8_t)oracle_probe_sign(seed, k, (uint64_t)(first + j));
}

/* Virtual start S_t of every tensor (see the probe definition above). */
void oracle_virtual_offsets(int32_t n_tensors, const int64_t* numel, int64_t* start) {
  int64_t s = 0;
  for (int32_t t = 0; t < n_tensors; ++t) {
    start[t] = s;
    s += ((numel[t] + 15) / 16) * 16;
  }
}

/* ------------------------------------------------------------------------- */
/* Storage formats. Weights are stored as fp32, bf16 or fp16 (the paper      */
/* trains bf16 weights in place, Sec. 4.3). Arithmetic is fp32 and the       */
/* result is rounded once to the storage format, to nearest, ties to even.   */
/* Written from the IEEE-754 definitions: the value is scaled by the format's */
/* quantum at its exponent, rounded to an integer with rint() (the default   */
/* rounding mode is to nearest-even), and scaled back.                       */
/* ------------------------------------------------------------------------- */

/* Round finite x to a binary format with `p` significand bits (including the
 * implicit one) and minimum normal exponent emin; returns the rounded value,
 * or +-INFINITY when the rounded magnitude exceeds `maxval`. */
static double round_to_format(double x, int p, int emin, double maxval) {
  if (x == 0.0) return x;
  double ax = fabs(x);
  int e;
  frexp(ax, &e); /* ax = f * 2^e, f in [0.5, 1): unbiased exponent is e - 1 */
  int unb = e - 1;
  if (unb < emin) unb = emin; /* subnormal range uses the quantum at emin */
  double quantum = ldexp(1.0, unb - (p - 1));
  double r = rint(ax / quantum) * quantum; /* both steps exact in double */
  if (r > maxval) r = INFINITY;
  return x < 0 ? -r : r;
}

static uint32_t f32_bits(float f) {
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

static float f32_from_bits(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return f;
}

/* NaN results. The paper says nothing about NaN weights, and IEEE 754 leaves
 * the sign and payload of an arithmetic result that is NaN to the
 * implementation. Reading taken here: a NaN result is stored as the positive
 * quiet NaN with every payload bit set, in each storage format. */
#define ORC_NAN_F32 0x7FFFFFFFu
#define ORC_NAN_16 0x7FFFu

/* Storage bits of an fp32 result (fp32 storage). */
static uint32_t f32_result_bits(float f) { return isnan(f) ? ORC_NAN_F32 : f32_bits(f); }

/* bfloat16 is the upper half of an fp32 bit pattern. */
float oracle_bf16_to_f32(uint16_t h) { return f32_from_bits((uint32_t)h << 16); }

uint16_t oracle_f32_to_bf16(float f) {
  if (isnan(f)) return (uint16_t)ORC_NAN_16;
  /* 8 significand bits, fp32's exponent range; max = (2 - 2^-7) * 2^127 */
  double r = round_to_format((double)f, 8, -126, ldexp(2.0 - ldexp(1.0, -7), 127));
  /* r is exactly representable in fp32 (or infinite), so this cast is exact */
  return (uint16_t)(f32_bits((float)r) >> 16);
}

/* binary16: 1 sign, 5 exponent (bias 15), 10 fraction bits. */
float oracle_f16_to_f32(uint16_t h) {
  int s = (h >> 15) & 1, e = (h >> 10) & 0x1F, m = h & 0x3FF;
  double v;
  if (e == 0x1F) {
    v = m ? NAN : INFINITY;
  } else if (e == 0) {
    v = ldexp((double)m, -24); /* subnormal: m * 2^-24 */
  } else {
    v = ldexp(1.0 + (double)m / 1024.0, e - 15);
  }
  return (float)(s ? -v : v);
}

uint16_t oracle_f32_to_f16(float f) {
  if (isnan(f)) return (uint16_t)ORC_NAN_16;
  uint16_t sign = (uint16_t)((f32_bits(f) >> 16) & 0x8000u);
  double r = round_to_format((double)f, 11, -14, 65504.0);
  double ar = fabs(r);
  if (isinf(r)) return (uint16_t)(sign | 0x7C00u);
  if (ar == 0.0) return sign;
  if (ar < ldexp(1.0, -14)) /* subnormal: an integer multiple of 2^-24 */
    return (uint16_t)(sign | (uint16_t)(ar / ldexp(1.0, -24)));
  int e;
  double fr = frexp(ar, &e); /* ar = fr * 2^e, fr in [0.5, 1) */
  int biased = (e - 1) + 15;
  uint16_t mant = (uint16_t)((fr * 2.0 - 1.0) * 1024.0);
  return (uint16_t)(sign | (uint16_t)(biased << 10) | mant);
}

/* Read element i of a tensor stored in `dtype` as fp32 (exact widening). */
static float load_f32(const void* base, int32_t dtype, int64_t i) {
  if (dtype == ORC_F32) return ((const float*)base)[i];
  if (dtype == ORC_BF16) return oracle_bf16_to_f32(((const uint16_t*)base)[i]);
  return oracle_f16_to_f32(((const uint16_t*)base)[i]);
}

/* Store fp32 value v into element i, rounding once to the storage format. */
static void store_f32(void* base, int32_t dtype, int64_t i, float v) {
  if (dtype == ORC_F32)
    ((uint32_t*)base)[i] = f32_result_bits(v);
  else if (dtype == ORC_BF16)
    ((uint16_t*)base)[i] = oracle_f32_to_bf16(v);
  else
    ((uint16_t*)base)[i] = oracle_f32_to_f16(v);
}

/* Round a double result straight to the storage format (one rounding). */
static void store_f64(void* base, int32_t dtype, int64_t i, double v) {
  if (dtype == ORC_F32) {
    ((uint32_t*)base)[i] = f32_result_bits((float)v);
  } else if (dtype == ORC_BF16) {
    if (isnan(v)) {
      ((uint16_t*)base)[i] = (uint16_t)ORC_NAN_16;
      return;
    }
    double r = round_to_format(v, 8, -126, ldexp(2.0 - ldexp(1.0, -7), 127));
    ((uint16_t*)base)[i] = (uint16_t)(f32_bits((float)r) >> 16);
  } else {
    if (isnan(v)) {
      ((uint16_t*)base)[i] = (uint16_t)ORC_NAN_16;
      return;
    }
    double r = round_to_format(v, 11, -14, 65504.0);
    /* r is exact in fp32, so the fp32 encoder returns its exact encoding */
    ((uint16_t*)base)[i] = oracle_f32_to_f16((float)r);
  }
}

static int valid_dtype(int32_t d) { return d == ORC_F32 || d == ORC_BF16 || d == ORC_F16; }

/* ------------------------------------------------------------------------- */
/* Fused perturb (Algorithm 1: ApplyPackedPerturbation(theta, +-eps, z_i);   */
/* Appendix F: w + alpha * sign stored back in place). For every element:   */
/* theta <- round(fp32(theta) + scale * z_k[g]).                              */
/* ------------------------------------------------------------------------- */
int oracle_perturb(int32_t n_tensors, void* const* ptrs, const int64_t* numel, const int32_t* dtype,
                   uint64_t seed, uint32_t k, float scale) {
  int64_t s = 0;
  for (int32_t t = 0; t < n_tensors; ++t) {
    if (!valid_dtype(dtype[t]) || numel[t] < 0) return ORC_ERR_ARG;
    for (int64_t i = 0; i < numel[t]; ++i) {
      uint64_t g = (uint64_t)(s + i);
      float z = (float)oracle_probe_sign(seed, k, g);
      float th = load_f32(ptrs[t], dtype[t], i);
      float r = th + scale * z;
      store_f32(ptrs[t], dtype[t], i, r);
    }
    s += ((numel[t] + 15) / 16) * 16;
  }
  return ORC_OK;
}

/* Same arithmetic on a list of sampled elements: element j has virtual index
 * g[j] and stored value theta[j] (widened to fp32); its new storage bits go to
 * out_bits[j] (fp32 bits, or the 16-bit pattern zero-extended). */
int oracle_perturb_elements(int32_t dtype, int64_t n, const uint64_t* g, const float* theta,
                            uint64_t seed, uint32_t k, float scale, uint32_t* out_bits) {
  if (!valid_dtype(dtype)) return ORC_ERR_ARG;
  for (int64_t j = 0; j < n; ++j) {
    float z = (float)oracle_probe_sign(seed, k, g[j]);
    float r = theta[j] + scale * z;
    if (dtype == ORC_F32)
      out_bits[j] = f32_result_bits(r);
    else if (dtype == ORC_BF16)
      out_bits[j] = oracle_f32_to_bf16(r);
    else
      out_bits[j] = oracle_f32_to_f16(r);
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* Probe-space preconditioner, for each probe k with (L+, L-, L0):            */
/*   curvature  c_hat = (L+ - 2 L0 + L-) / eps^2          (Sec. 4.1, Eq. 3)   */
/*   weight     w     = 1 / max(lambda_reg, |c_hat|^alpha) (Sec. 4.1, Eq. 4)  */
/*   coefficient c_k  = w * (L+ - L-) / (2 eps)   two-sided (Eq. 5, Alg. 1)   */
/*                c_k = w * (L+ - L0) / eps       one-sided variant            */
/* losses is K rows of {L+, L-, L0}. Non-finite inputs or results return      */
/* ORC_ERR_NONFINITE and leave the outputs untouched.                         */
/*                                                                           */
/* flags: ORC_PRECOND_ONE_SIDED selects the one-sided coefficient;            */
/* ORC_PRECOND_RELATIVE applies Eq. 4 to the relative curvature               */
/*   r_k = c_hat_k / m,   m = (1/K) sum_j |c_hat_j|  (j in probe order),      */
/* one reading of the per-step curvature normalisation that Sec. 6 leaves to  */
/* future work; m = 0 (every curvature zero) gives r_k = 0, a non-finite m is */
/* ORC_ERR_NONFINITE. curv_out always receives Eq. 3's c_hat.                 */
/* ------------------------------------------------------------------------- */
#define ORC_PRECOND_ONE_SIDED 1
#define ORC_PRECOND_RELATIVE 2

static double curvature(const double* l, double eps) { return (l[0] - 2.0 * l[2] + l[1]) / (eps * eps); }

static double difference(const double* l, double eps, int one_sided) {
  return one_sided ? (l[0] - l[2]) / eps : (l[0] - l[1]) / (2.0 * eps);
}

int oracle_precondition(const double* losses, int32_t K, double eps, double alpha, double lambda_reg,
                        int32_t flags, double* c, double* w_out, double* curv_out) {
  if (K < 1 || !(eps > 0.0) || !isfinite(eps) || !(alpha >= 0.0) || !(alpha <= 1.0) ||
      !(lambda_reg > 0.0) || !isfinite(lambda_reg) || (flags & ~(ORC_PRECOND_ONE_SIDED | ORC_PRECOND_RELATIVE)) != 0)
    return ORC_ERR_ARG;
  const int one_sided = (flags & ORC_PRECOND_ONE_SIDED) != 0;
  const int relative = (flags & ORC_PRECOND_RELATIVE) != 0;
  /* first pass: every loss and curvature finite, and the normaliser m */
  double m = 1.0;
  if (relative) m = 0.0;
  for (int32_t k = 0; k < K; ++k) {
    const double* l = losses + 3 * k;
    if (!isfinite(l[0]) || !isfinite(l[1]) || !isfinite(l[2])) return ORC_ERR_NONFINITE;
    double curv = curvature(l, eps);
    if (!isfinite(curv)) return ORC_ERR_NONFINITE;
    if (relative) m += fabs(curv);
  }
  if (relative) {
    m = m / (double)K;
    if (!isfinite(m)) return ORC_ERR_NONFINITE;
  }
  /* second pass: weights and coefficients, all checked before any write */
  for (int32_t k = 0; k < K; ++k) {
    double curv = curvature(losses + 3 * k, eps);
    double r = relative ? (m > 0.0 ? curv / m : 0.0) : curv;
    double w = 1.0 / fmax(lambda_reg, pow(fabs(r), alpha));
    if (!isfinite(w * difference(losses + 3 * k, eps, one_sided))) return ORC_ERR_NONFINITE;
  }
  for (int32_t k = 0; k < K; ++k) {
    double curv = curvature(losses + 3 * k, eps);
    double r = relative ? (m > 0.0 ? curv / m : 0.0) : curv;
    double w = 1.0 / fmax(lambda_reg, pow(fabs(r), alpha));
    c[k] = w * difference(losses + 3 * k, eps, one_sided);
    if (w_out) w_out[k] = w;
    if (curv_out) curv_out[k] = curv;
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* Fused K-probe update (Sec. 4.2, Eqs. 5-6: Delta theta = -eta Z W dl).     */
/* With c_k from the preconditioner and step size lr:                        */
/*   theta <- theta - (lr / K) * sum_k c_k z_k                                */
/* which at lr = eps is Algorithm 1's gamma_k = g_k w_k / (2n) applied with a */
/* minus sign. Each coefficient is first rounded to fp32,                     */
/*   a_k = fp32( (-(lr / K)) * c_k ),                                         */
/* then the sum over k = 0..K-1 of a_k z_k is formed in double (exact for the */
/* sizes used here) and added to theta with one rounding to the storage type. */
/* ------------------------------------------------------------------------- */
static int update_coefficients(const double* c, int32_t K, double lr, float* a) {
  double m = -(lr / (double)K);
  for (int32_t k = 0; k < K; ++k) a[k] = (float)(m * c[k]);
  return ORC_OK;
}

#define ORC_MAX_PROBES 4096

int oracle_update(int32_t n_tensors, void* const* ptrs, const int64_t* numel, const int32_t* dtype,
                  uint64_t seed, const double* c, int32_t K, double lr) {
  if (K < 1 || K > ORC_MAX_PROBES) return ORC_ERR_ARG;
  float a[ORC_MAX_PROBES];
  update_coefficients(c, K, lr, a);
  int64_t s = 0;
  for (int32_t t = 0; t < n_tensors; ++t) {
    if (!valid_dtype(dtype[t]) || numel[t] < 0) return ORC_ERR_ARG;
    for (int64_t i = 0; i < numel[t]; ++i) {
      uint64_t g = (uint64_t)(s + i);
      double acc = 0.0;
      for (int32_t k = 0; k < K; ++k) acc += (double)a[k] * (double)oracle_probe_sign(seed, (uint32_t)k, g);
      double th = (double)load_f32(ptrs[t], dtype[t], i);
      store_f64(ptrs[t], dtype[t], i, th + acc);
    }
    s += ((numel[t] + 15) / 16) * 16;
  }
  return ORC_OK;
}

/* Sampled elements, as oracle_perturb_elements. */
int oracle_update_elements(int32_t dtype, int64_t n, const uint64_t* g, const float* theta, uint64_t seed,
                           const double* c, int32_t K, double lr, uint32_t* out_bits) {
  if (!valid_dtype(dtype) || K < 1 || K > ORC_MAX_PROBES) return ORC_ERR_ARG;
  float a[ORC_MAX_PROBES];
  update_coefficients(c, K, lr, a);
  for (int64_t j = 0; j < n; ++j) {
    double acc = 0.0;
    for (int32_t k = 0; k < K; ++k) acc += (double)a[k] * (double)oracle_probe_sign(seed, (uint32_t)k, g[j]);
    double v = (double)theta[j] + acc;
    if (dtype == ORC_F32) {
      out_bits[j] = f32_result_bits((float)v);
    } else {
      uint16_t h;
      store_f64(&h, dtype, 0, v);
      out_bits[j] = h;
    }
  }
  return ORC_OK;
}

/* Algorithm 1's rank-0 loop: for k = 0..K-1, theta <- theta - gamma_k z_k, one
 * in-place pass per probe, each rounded to storage (the comparator for the
 * fused update). Uses the same a_k as oracle_update. */
int oracle_update_sequential(int32_t n_tensors, void* const* ptrs, const int64_t* numel, const int32_t* dtype,
                             uint64_t seed, const double* c, int32_t K, double lr) {
  if (K < 1 || K > ORC_MAX_PROBES) return ORC_ERR_ARG;
  float a[ORC_MAX_PROBES];
  update_coefficients(c, K, lr, a);
  for (int32_t k = 0; k < K; ++k) {
    int rc = oracle_perturb(n_tensors, ptrs, numel, dtype, seed, (uint32_t)k, a[k]);
    if (rc != ORC_OK) return rc;
  }
  return ORC_OK;
}

/* ------------------------------------------------------------------------- */
/* Quadratic test loss f(theta) = 1/2 sum_i a_i theta_i^2 (the ill-conditioned */
/* quadratic of the small synthetic workload; the paper's stiff paraboloid,   */
/* Sec. 5.3, is of this family). Accumulated in double, in index order.       */
/* ------------------------------------------------------------------------- */
double oracle_quadratic_loss(const float* theta, const float* a, int64_t n) {
  double s = 0.0;
  for (int64_t i = 0; i < n; ++i) {
    double th = (double)theta[i];
    s += (double)a[i] * (th * th);
  }
  return 0.5 * s;
}
