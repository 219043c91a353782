/*
 * layer_math.c -- CPU oracle of the decoder-layer math -- TEST INFRASTRUCTURE ONLY.
 *
 * Only tests/, __graft_entry__.smoke() and bench.py's CPU-baseline leg may load this
 * library. It shares no code, header, table or constant with the CUDA path.
 *
 * The paper (Trident) names the operators -- rms_norm (§2.1, §2.3, Fig. 1) and silu
 * (§4.1, §4.2) -- and runs them inside the decode loops of the LLMs it evaluates
 * (§4.1: Qwen3-8B, DeepSeek-V2-Lite), but prints no formula. The functions below are
 * the standard definitions of those layer steps, written out one element at a time:
 *
 *   RMSNorm       y = x / sqrt(mean(x^2) + eps) * gamma in fp64 (the paper's running
 *                 example operator, rms_norm, §2.3 and Fig. 1).
 *   add+RMSNorm   s = x + r (fp32 add, the kernel's precision: r_out = round(s) is a
 *                 rounding decision, so both sides take it from the same fp32 value);
 *                 ms = sum(s^2)/H in fp64; y = s / sqrt(ms + eps) * gamma in fp64.
 *   q/k RMSNorm   the same over each head's D elements, without the residual.
 *   RoPE          rotate-half: for i < D/2, a = pos * theta^(-2i/D) (fp64),
 *                 x'_i = x_i cos a - x_{i+D/2} sin a, x'_{i+D/2} = x_{i+D/2} cos a + x_i sin a.
 *   KV append     k_cache[h][pos][:] = round(rope(k)), v_cache[h][pos][:] = v (bit copy).
 *   SwiGLU        out = g / (1 + exp(-g)) * u in fp64.
 *
 * Every output is returned twice: unrounded (fp64, for tolerance checks) and rounded
 * once, round-to-nearest-even, to the activation dtype (bit patterns).
 * Activations are raw bit patterns: uint16 for bf16/fp16, uint32 for fp32.
 * Build with -ffp-contract=off so that no multiply-add is fused behind our back.
 *
 * The token (or element) loops carry an OpenMP work-sharing pragma. The default build has
 * no -fopenmp, so the pragmas are ignored and every loop runs serially in order; a second
 * build with -fopenmp (liboracle_omp.so) exists only to time the oracle on all host cores.
 * Every iteration writes its own outputs, so both builds compute the same values.
 */
#include <math.h>
#include <stdint.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

/* Threads the work-sharing loops use (1 in the default build). */
int orc_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

enum { OR_BF16 = 1, OR_FP16 = 2, OR_FP32 = 3 };

/* ------------------------------------------------------------------ widening */
static double widen_bf16(uint16_t b) {
  uint32_t u = (uint32_t)b << 16;
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

static double widen_fp16(uint16_t h) {
  int sign = (h >> 15) & 1;
  int e = (h >> 10) & 0x1f;
  int m = h & 0x3ff;
  double v;
  if (e == 0) {
    v = ldexp((double)m, -24);                 /* subnormal: m * 2^-24 */
  } else if (e == 31) {
    v = (m == 0) ? INFINITY : NAN;
  } else {
    v = ldexp((double)(m + 1024), e - 15 - 10); /* (1 + m/1024) * 2^(e-15) */
  }
  return sign ? -v : v;
}

static double widen_fp32(uint32_t u) {
  float f;
  memcpy(&f, &u, 4);
  return (double)f;
}

double orc_widen(uint32_t bits, int dtype) {
  if (dtype == OR_BF16) return widen_bf16((uint16_t)bits);
  if (dtype == OR_FP16) return widen_fp16((uint16_t)bits);
  return widen_fp32(bits);
}

/* ------------------------------------------------------------------ rounding
 * Round a double to the nearest value with `sig` significant bits whose quantum is at
 * least 2^qmin (subnormals), ties to even; overflow past `maxv` goes to infinity. */
static double round_to_format(double v, int sig, int qmin, double maxv) {
  if (isnan(v) || isinf(v) || v == 0.0) return v;
  int e;
  frexp(v, &e);                 /* v = m * 2^e, 0.5 <= |m| < 1 */
  int q = e - sig;              /* quantum exponent of a normal number in that binade */
  if (q < qmin) q = qmin;
  double scaled = ldexp(v, -q); /* exact: only the exponent changes */
  double r = nearbyint(scaled); /* current rounding mode: to nearest, ties to even */
  double out = ldexp(r, q);
  if (fabs(out) > maxv) return v > 0 ? INFINITY : -INFINITY;
  return out;
}

static uint16_t bf16_bits_of_exact(double v) {
  /* v is exactly a bf16 value (or inf/nan): its float has zero low 16 bits. */
  if (isnan(v)) return 0x7fc0;
  float f = (float)v;
  uint32_t u;
  memcpy(&u, &f, 4);
  return (uint16_t)(u >> 16);
}

static uint16_t fp16_bits_of_exact(double v) {
  uint16_t sign = signbit(v) ? 0x8000 : 0;
  double a = fabs(v);
  if (isnan(v)) return 0x7e00;
  if (isinf(a)) return sign | 0x7c00;
  if (a == 0.0) return sign;
  if (a < ldexp(1.0, -14)) return sign | (uint16_t)(a / ldexp(1.0, -24)); /* subnormal */
  int e;
  frexp(a, &e);                 /* a = m * 2^e, 2^(e-1) <= a < 2^e */
  int exp_field = (e - 1) + 15;
  double mant = a / ldexp(1.0, e - 1) * 1024.0 - 1024.0; /* 0..1023, exact */
  return sign | (uint16_t)(exp_field << 10) | (uint16_t)mant;
}

uint32_t orc_round(double v, int dtype) {
  if (dtype == OR_BF16) {
    /* bf16: 8 significant bits, min normal 2^-126 so the quantum never drops below
       2^-133, max finite (2 - 2^-7) * 2^127. */
    return bf16_bits_of_exact(round_to_format(v, 8, -133, ldexp(255.0, 120)));
  }
  if (dtype == OR_FP16) {
    /* fp16: 11 significant bits, quantum >= 2^-24, max finite 65504. */
    return fp16_bits_of_exact(round_to_format(v, 11, -24, 65504.0));
  }
  float f = (float)v; /* fp32: the C conversion rounds to nearest even */
  uint32_t u;
  memcpy(&u, &f, 4);
  return u;
}

/* Element i of a raw activation array. */
static double load_act(const void* p, int64_t i, int dtype) {
  if (dtype == OR_FP32) return widen_fp32(((const uint32_t*)p)[i]);
  return orc_widen(((const uint16_t*)p)[i], dtype);
}

static void store_act(void* p, int64_t i, int dtype, uint32_t bits) {
  if (dtype == OR_FP32) ((uint32_t*)p)[i] = bits;
  else ((uint16_t*)p)[i] = (uint16_t)bits;
}

/* ------------------------------------------------------------------ add + RMSNorm
 * x, r, y_bits, r_out_bits: contiguous [T,H]; gamma [H]; y_ref [T,H] unrounded. */
void orc_add_rmsnorm(int64_t T, int64_t H, int dtype, const void* x, const void* r,
                     const float* gamma, double eps, double* y_ref, void* y_bits,
                     void* r_out_bits) {
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    double sumsq = 0.0;
    for (int64_t j = 0; j < H; ++j) {
      float s = (float)load_act(x, t * H + j, dtype) + (float)load_act(r, t * H + j, dtype);
      store_act(r_out_bits, t * H + j, dtype, orc_round((double)s, dtype));
      sumsq += (double)s * (double)s;
    }
    double ms = sumsq / (double)H;
    double inv = 1.0 / sqrt(ms + eps);
    for (int64_t j = 0; j < H; ++j) {
      float s = (float)load_act(x, t * H + j, dtype) + (float)load_act(r, t * H + j, dtype);
      double y = (double)s * inv * (double)gamma[j];
      y_ref[t * H + j] = y;
      store_act(y_bits, t * H + j, dtype, orc_round(y, dtype));
    }
  }
}

/* ------------------------------------------------------------------ RMSNorm
 * x, y_bits: contiguous [T,H]; gamma [H]; y_ref [T,H] unrounded:
 * y = x / sqrt(mean(x^2) + eps) * gamma, in fp64. */
void orc_rmsnorm(int64_t T, int64_t H, int dtype, const void* x, const float* gamma, double eps,
                 double* y_ref, void* y_bits) {
#pragma omp parallel for schedule(static)
  for (int64_t t = 0; t < T; ++t) {
    double sumsq = 0.0;
    for (int64_t j = 0; j < H; ++j) {
      double v = load_act(x, t * H + j, dtype);
      sumsq += v * v;
    }
    double inv = 1.0 / sqrt(sumsq / (double)H + eps);
    for (int64_t j = 0; j < H; ++j) {
      double y = load_act(x, t * H + j, dtype) * inv * (double)gamma[j];
      y_ref[t * H + j] = y;
      store_act(y_bits, t * H + j, dtype, orc_round(y, dtype));
    }
  }
}

/* ------------------------------------------------------------------ head RMSNorm, RoPE */
/* x[0..n-1] <- x / sqrt(mean(x^2) + eps) * gamma, in fp64. */
void orc_rms_scale(int64_t n, double* x, const float* gamma, double eps) {
  double sumsq = 0.0;
  for (int64_t j = 0; j < n; ++j) sumsq += x[j] * x[j];
  double inv = 1.0 / sqrt(sumsq / (double)n + eps);
  for (int64_t j = 0; j < n; ++j) x[j] = x[j] * inv * (double)gamma[j];
}

/* Rotate-half RoPE of one head vector x[0..D-1] at position pos, in fp64. */
void orc_rope_apply(int64_t D, double* x, int64_t pos, double theta) {
  int64_t half = D / 2;
  for (int64_t i = 0; i < half; ++i) {
    double inv_freq = pow(theta, -2.0 * (double)i / (double)D);
    double a = (double)pos * inv_freq;
    double c = cos(a), s = sin(a);
    double lo = x[i], hi = x[i + half];
    x[i] = lo * c - hi * s;
    x[i + half] = hi * c + lo * s;
  }
}

/* RoPE on q and k plus KV-cache append, optionally after per-head RMSNorm of q and k.
 *   q      [T,Hq,D] bits, rotated in place (tokens with a bad position untouched)
 *   q_ref  [T,Hq,D] unrounded rotated q (NaN for skipped tokens)
 *   k, v   [T,Hkv,D] bits;   k_ref [T,Hkv,D] unrounded rotated k (NaN if skipped)
 *   pos    [T];  k_cache, v_cache [Hkv,S,D] bits, written only at valid positions
 * Returns 1 if some position was outside [0,S), else 0. */
int orc_rope_kv(int64_t T, int64_t Hq, int64_t Hkv, int64_t D, int64_t S, int dtype,
                double theta, int qknorm, const float* gamma_q, const float* gamma_k,
                double eps, void* q, double* q_ref, const void* k, const void* v,
                const int32_t* pos, void* k_cache, void* v_cache, double* k_ref) {
  int bad = 0;
  if (D > 1024) return -1;
  /* positions are distinct within a call, so tokens write disjoint cache rows */
#pragma omp parallel for schedule(static) reduction(| : bad)
  for (int64_t t = 0; t < T; ++t) {
    double buf[1024];
    int64_t p = pos[t];
    if (p < 0 || p >= S) {
      bad = 1;
      for (int64_t j = 0; j < Hq * D; ++j) q_ref[t * Hq * D + j] = NAN;
      for (int64_t j = 0; j < Hkv * D; ++j) k_ref[t * Hkv * D + j] = NAN;
      continue;
    }
    for (int64_t h = 0; h < Hq; ++h) {
      int64_t base = (t * Hq + h) * D;
      for (int64_t j = 0; j < D; ++j) buf[j] = load_act(q, base + j, dtype);
      if (qknorm) orc_rms_scale(D, buf, gamma_q, eps);
      orc_rope_apply(D, buf, p, theta);
      for (int64_t j = 0; j < D; ++j) {
        q_ref[base + j] = buf[j];
        store_act(q, base + j, dtype, orc_round(buf[j], dtype));
      }
    }
    for (int64_t h = 0; h < Hkv; ++h) {
      int64_t base = (t * Hkv + h) * D;
      int64_t cbase = (h * S + p) * D;
      for (int64_t j = 0; j < D; ++j) buf[j] = load_act(k, base + j, dtype);
      if (qknorm) orc_rms_scale(D, buf, gamma_k, eps);
      orc_rope_apply(D, buf, p, theta);
      for (int64_t j = 0; j < D; ++j) {
        k_ref[base + j] = buf[j];
        store_act(k_cache, cbase + j, dtype, orc_round(buf[j], dtype));
        ((uint16_t*)v_cache)[cbase + j] = ((const uint16_t*)v)[base + j];
      }
    }
  }
  return bad;
}

/* ------------------------------------------------------------------ pointwise operators
 * The FlagGems-style operators of the paper's kernel benchmark (§4.1): silu, add, neg,
 * masked_fill, over n contiguous elements; ref = unrounded result, out = its rounding.
 *   silu(x) = x / (1 + exp(-x))                     (fp64)
 *   add     = a + b, summed in fp32 (the kernels' precision: the rounding of the sum is a
 *             rounding decision, taken from the same fp32 value on both sides)
 *   neg     = -x                                    (exact)
 *   masked_fill: mask != 0 ? value : x, with value converted to fp32 and then rounded to
 *             the activation type */
void orc_silu(int64_t n, int dtype, const void* x, double* ref, void* out_bits) {
  for (int64_t i = 0; i < n; ++i) {
    double v = load_act(x, i, dtype);
    double o = v / (1.0 + exp(-v));
    ref[i] = o;
    store_act(out_bits, i, dtype, orc_round(o, dtype));
  }
}

void orc_add(int64_t n, int dtype, const void* a, const void* b, double* ref, void* out_bits) {
  for (int64_t i = 0; i < n; ++i) {
    float s = (float)load_act(a, i, dtype) + (float)load_act(b, i, dtype);
    ref[i] = (double)s;
    store_act(out_bits, i, dtype, orc_round((double)s, dtype));
  }
}

void orc_neg(int64_t n, int dtype, const void* x, double* ref, void* out_bits) {
  for (int64_t i = 0; i < n; ++i) {
    double v = -load_act(x, i, dtype);
    ref[i] = v;
    store_act(out_bits, i, dtype, orc_round(v, dtype));
  }
}

void orc_masked_fill(int64_t n, int dtype, const void* x, const uint8_t* mask, double value,
                     double* ref, void* out_bits) {
  /* the fill value is converted to fp32 first, then rounded to the activation type, as a
     framework scalar reaches a bf16/fp16 tensor */
  uint32_t vbits = orc_round((double)(float)value, dtype);
  for (int64_t i = 0; i < n; ++i) {
    if (mask[i]) {
      ref[i] = orc_widen(vbits, dtype);
      store_act(out_bits, i, dtype, vbits);
    } else {
      ref[i] = load_act(x, i, dtype);
      store_act(out_bits, i, dtype, (dtype == OR_FP32) ? ((const uint32_t*)x)[i] : ((const uint16_t*)x)[i]);
    }
  }
}

/* ------------------------------------------------------------------ SwiGLU
 * g, u, out_bits: n contiguous elements; ref: n unrounded results. */
void orc_swiglu(int64_t n, int dtype, const void* g, const void* u, double* ref,
                void* out_bits) {
#pragma omp parallel for schedule(static)
  for (int64_t i = 0; i < n; ++i) {
    double gv = load_act(g, i, dtype);
    double uv = load_act(u, i, dtype);
    double silu = gv / (1.0 + exp(-gv));
    double o = silu * uv;
    ref[i] = o;
    store_act(out_bits, i, dtype, orc_round(o, dtype));
  }
}
