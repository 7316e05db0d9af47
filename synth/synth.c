/*
 * Seeded synthetic inputs for the QTEA GEMV (ternary codes, scales, activations, salient
 * columns and the 1:4 residual). This module draws numbers and rounds them to the input
 * formats; it contains none of the GEMV's arithmetic. Both the oracle and the GPU library
 * are fed the bytes it writes.
 *
 * Generator: SplitMix64 (Steele, Lea and Flood, "Fast Splittable Pseudorandom Number
 * Generators", OOPSLA 2014) used as a counter-based generator: draw i of stream (seed, id)
 * is mix(base + (i + 1) * GAMMA) with base = mix(seed * GAMMA ^ mix(id)). Every value
 * depends only on (seed, stream, index), so the tensors are identical whatever the
 * thread count and on every host.
 *
 * Distributions: uniform doubles in [0, 1) from the top 53 bits; normals by Box-Muller
 * (cosine branch, draws 2i and 2i+1); Laplace by inverse CDF; ternary codes by
 * thresholds (t = -1 if u < p_neg, 0 if u < p_neg + p_zero, else +1); salient columns by a
 * partial Fisher-Yates shuffle then an ascending sort; 1:4 residual positions as
 * floor(4u). Reals are drawn in double and rounded to binary16 with round-to-nearest-even.
 */
#include <math.h>
#include <pthread.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#include <unistd.h>

#define GAMMA 0x9E3779B97F4A7C15ULL

static uint64_t mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

static uint64_t stream_base(uint64_t seed, uint64_t stream) { return mix64(seed * GAMMA ^ mix64(stream)); }

static uint64_t draw(uint64_t base, uint64_t i) { return mix64(base + (i + 1) * GAMMA); }

static double u01(uint64_t base, uint64_t i) { return (double)(draw(base, i) >> 11) * 0x1.0p-53; }

/* double -> IEEE binary16 bits, round to nearest, ties to even; overflow -> inf. */
uint16_t synth_f16_from_double(double v) {
  uint16_t sign = signbit(v) ? 0x8000 : 0;
  double a = fabs(v);
  if (isnan(v)) return 0x7e00;
  if (a == 0.0) return sign;
  int e;
  frexp(a, &e); /* a = f * 2^e, f in [0.5, 1) => unbiased exponent of a is e - 1 */
  int ue = e - 1;
  if (ue < -14) {
    /* subnormal range: units of 2^-24 */
    double q = nearbyint(a * 0x1.0p24); /* default rounding mode is to-nearest-even */
    if (q >= 1024.0) return sign | 0x0400; /* rounded up to the smallest normal */
    return sign | (uint16_t)q;
  }
  double q = nearbyint(ldexp(a, 10 - ue)); /* significand in [1024, 2048] */
  if (q >= 2048.0) {
    q = 1024.0;
    ue += 1;
  }
  if (ue > 15) return sign | 0x7c00;
  return sign | (uint16_t)((ue + 15) << 10) | (uint16_t)((int)q - 1024);
}

/* double -> FP8 E4M3 bits (sign, 4 exponent bits with bias 7, 3 mantissa bits; no infinity),
 * round to nearest, ties to even; magnitudes beyond the largest finite value 448 saturate. */
uint8_t synth_e4m3_from_double(double v) {
  uint8_t sign = signbit(v) ? 0x80 : 0;
  double a = fabs(v);
  if (isnan(v)) return 0x7f;
  if (a == 0.0) return sign;
  if (a >= 448.0) return sign | 0x7e;
  int e;
  frexp(a, &e);
  int ue = e - 1;
  if (ue < -6) {
    /* subnormal range: units of 2^-9 */
    double q = nearbyint(a * 0x1.0p9);
    if (q >= 8.0) return sign | 0x08; /* rounded up to the smallest normal */
    return sign | (uint8_t)q;
  }
  double q = nearbyint(ldexp(a, 3 - ue)); /* significand in [8, 16] */
  if (q >= 16.0) {
    q = 8.0;
    ue += 1;
  }
  if (ue > 8 || (ue == 8 && q > 14.0)) return sign | 0x7e; /* 448 is the largest finite value */
  return sign | (uint8_t)((ue + 7) << 3) | (uint8_t)((int)q - 8);
}

/* ------------------------------------------------------------------ threads */

typedef struct {
  int kind;
  uint64_t base;
  size_t lo, hi;
  double a, b;
  void* out;
} job_t;

enum { K_CODES = 0, K_UNIFORM = 1, K_NORMAL = 2, K_LAPLACE = 3, K_NORMAL_E4M3 = 4 };

static void run_job(job_t* j) {
  for (size_t i = j->lo; i < j->hi; ++i) {
    switch (j->kind) {
      case K_CODES: {
        double u = u01(j->base, i);
        ((int8_t*)j->out)[i] = (int8_t)(u < j->a ? -1 : (u < j->a + j->b ? 0 : 1));
        break;
      }
      case K_UNIFORM: {
        double u = u01(j->base, i);
        ((uint16_t*)j->out)[i] = synth_f16_from_double(j->a + (j->b - j->a) * u);
        break;
      }
      case K_NORMAL: {
        double u1 = 1.0 - u01(j->base, 2 * i); /* (0, 1] */
        double u2 = u01(j->base, 2 * i + 1);
        double z = sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
        ((uint16_t*)j->out)[i] = synth_f16_from_double(j->a + j->b * z);
        break;
      }
      case K_NORMAL_E4M3: {
        double u1 = 1.0 - u01(j->base, 2 * i); /* (0, 1] */
        double u2 = u01(j->base, 2 * i + 1);
        double z = sqrt(-2.0 * log(u1)) * cos(6.283185307179586 * u2);
        ((uint8_t*)j->out)[i] = synth_e4m3_from_double(j->a + j->b * z);
        break;
      }
      case K_LAPLACE: {
        double u = u01(j->base, i) - 0.5; /* [-0.5, 0.5) */
        double m = 1.0 - 2.0 * fabs(u);   /* (0, 1] */
        double z = (u < 0 ? 1.0 : -1.0) * log(m);
        ((uint16_t*)j->out)[i] = synth_f16_from_double(j->a + j->b * z);
        break;
      }
    }
  }
}

static void* thread_main(void* arg) {
  run_job((job_t*)arg);
  return NULL;
}

static void run_parallel(int kind, uint64_t base, size_t n, double a, double b, void* out) {
  long ncpu = sysconf(_SC_NPROCESSORS_ONLN);
  int nt = (int)(ncpu < 1 ? 1 : (ncpu > 32 ? 32 : ncpu));
  if (n < (size_t)1 << 20) nt = 1;
  job_t jobs[32];
  pthread_t th[32];
  size_t chunk = (n + nt - 1) / nt;
  for (int t = 0; t < nt; ++t) {
    size_t lo = (size_t)t * chunk, hi = lo + chunk < n ? lo + chunk : n;
    if (lo > n) lo = n;
    jobs[t] = (job_t){kind, base, lo, hi, a, b, out};
  }
  int started = 0;
  for (int t = 1; t < nt; ++t) {
    if (pthread_create(&th[t], NULL, thread_main, &jobs[t]) != 0) break;
    started = t;
  }
  run_job(&jobs[0]);
  for (int t = started + 1; t < nt; ++t) run_job(&jobs[t]); /* threads that failed to start */
  for (int t = 1; t <= started; ++t) pthread_join(th[t], NULL);
}

/* ------------------------------------------------------------------ exports */

void synth_codes(uint64_t seed, uint64_t stream, size_t n, double p_neg, double p_zero, int8_t* out) {
  run_parallel(K_CODES, stream_base(seed, stream), n, p_neg, p_zero, out);
}

void synth_uniform_f16(uint64_t seed, uint64_t stream, size_t n, double lo, double hi, uint16_t* out) {
  run_parallel(K_UNIFORM, stream_base(seed, stream), n, lo, hi, out);
}

void synth_normal_f16(uint64_t seed, uint64_t stream, size_t n, double mean, double std, uint16_t* out) {
  run_parallel(K_NORMAL, stream_base(seed, stream), n, mean, std, out);
}

void synth_normal_e4m3(uint64_t seed, uint64_t stream, size_t n, double mean, double std, uint8_t* out) {
  run_parallel(K_NORMAL_E4M3, stream_base(seed, stream), n, mean, std, out);
}

void synth_laplace_f16(uint64_t seed, uint64_t stream, size_t n, double loc, double scale, uint16_t* out) {
  run_parallel(K_LAPLACE, stream_base(seed, stream), n, loc, scale, out);
}

static int cmp_i32(const void* a, const void* b) {
  int32_t x = *(const int32_t*)a, y = *(const int32_t*)b;
  return (x > y) - (x < y);
}

/* s distinct columns of [0, K), ascending. Returns 0, or 1 if s > K or allocation fails. */
int synth_salient(uint64_t seed, uint64_t stream, int K, int s, int32_t* out) {
  if (s < 0 || s > K) return 1;
  int32_t* perm = (int32_t*)malloc(sizeof(int32_t) * (size_t)(K > 0 ? K : 1));
  if (!perm) return 1;
  for (int i = 0; i < K; ++i) perm[i] = i;
  uint64_t base = stream_base(seed, stream);
  for (int i = 0; i < s; ++i) {
    int j = i + (int)(u01(base, (uint64_t)i) * (double)(K - i));
    if (j >= K) j = K - 1;
    int32_t t = perm[i];
    perm[i] = perm[j];
    perm[j] = t;
  }
  memcpy(out, perm, sizeof(int32_t) * (size_t)s);
  free(perm);
  qsort(out, (size_t)s, sizeof(int32_t), cmp_i32);
  return 0;
}

/* 1:4 residual positions, idx = floor(4u) per (group q, salient column c), written in the
 * residual_idx input format: [n_groups][ceil(s/4)] bytes, entry (q, c) at bits 2*(c%4) of
 * byte c/4; unused high bits of a row's last byte are zero. */
void synth_residual_idx(uint64_t seed, uint64_t stream, int n_groups, int s, uint8_t* out) {
  int stride = (s + 3) / 4;
  uint64_t base = stream_base(seed, stream);
  memset(out, 0, (size_t)n_groups * (size_t)stride);
  for (int q = 0; q < n_groups; ++q)
    for (int c = 0; c < s; ++c) {
      int idx = (int)(u01(base, (uint64_t)q * (uint64_t)s + (uint64_t)c) * 4.0);
      if (idx > 3) idx = 3;
      out[(size_t)q * stride + c / 4] |= (uint8_t)(idx << (2 * (c % 4)));
    }
}
