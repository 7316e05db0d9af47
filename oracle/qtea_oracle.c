/*
 * QTEA oracle: plain, slow, fp64 CPU reference of the decode-time GEMV.
 *
 * TEST INFRASTRUCTURE ONLY. This library exists to check the GPU library. It is
 * loaded by the tests, by the smoke check in __graft_entry__ and by the CPU-baseline
 * leg of bench.py, and by nothing else: the GPU library never links, loads or calls
 * it, and it shares no code, header or table with the GPU library.
 *
 * Every routine is a direct transcription of a definition from the QTEA paper
 * ("Ternary LLMs with Sparse Residual Salient Weight and By-Column Optimization"):
 *
 *   Eq. 1 / Eq. 4   dequantized weight   W^[r][j] = beta[r][g] + v[j] * alpha[r][g] * T[r][j]
 *   Eq. 10          group output         y_r^(g) = alpha[r][g] * sum_{j in g} T[r][j] v[j] x[j]
 *                                                  + beta[r][g] * sum_{j in g} x[j]
 *   Eq. 11          full output          y_r = sum_g y_r^(g) + sum_{j in S} R[r][j] x[j]
 *   Sec. 3.5        residual storage     per salient column, per group of four rows:
 *                                        one value and a 2-bit position inside the group
 *   Sec. 3.5        LUT                  five ternary digits per byte (3^5 < 2^8); the table
 *                                        holds every pattern's dot product with v*x
 *   Appendix A      ASIC latency model   T_tern = ceil(K/128)(652+977+N), T_dense = K N / 26
 *
 * Storage formats the oracle reads (shared with the GPU library only as a written
 * specification, never as code):
 *   fp16 values           IEEE 754 binary16 bit patterns (uint16_t)
 *   ternary codes         int8 T[N][K], values -1, 0, +1
 *   2-bit layout          K_pad = K rounded up to a multiple of 64. Row r occupies bytes
 *                         [r*K_pad/4, (r+1)*K_pad/4). Column k sits in byte r*K_pad/4 + k/4 at
 *                         bits 2*(k%4), 2*(k%4)+1 (least significant first) as code T+1.
 *                         Columns k >= K hold code 1 (T = 0). Code 3 never occurs.
 *   base-3 layout         K_pad3 = K rounded up to a multiple of 128. Each row is K_pad3/128
 *                         groups of 26 bytes. Byte p of group h holds columns
 *                         128h + 5p + d, d = 0..4, as sum_d (T+1) * 3^d (lowest column in the
 *                         least significant digit). Byte 25 covers 3 real columns and 2 pad
 *                         digits; pad digits and columns >= K hold digit 1 (T = 0).
 *   salient_idx           int32 [s], strictly ascending, each < K
 *   salient bitmap        Sec. 3.5 stores the salient set as a bitmap over the input columns:
 *                         uint32 words [ceil(K/32)], column j at bit j % 32 of word j / 32 (least
 *                         significant bit first); bits of columns >= K are ignored on input and
 *                         zero on output
 *   residual_vals         fp16 [N/4][s]: value of group q (rows 4q..4q+3) in salient column c;
 *                         or, where the paper's storage is used (Sec. 4.1: FP8 residual), one
 *                         byte per value in the FP8 E4M3 format: sign bit 7, exponent bits 6-3
 *                         with bias 7, mantissa bits 2-0; exponent 0 is subnormal (m * 2^-9);
 *                         0x7F and 0xFF are NaN; there is no infinity
 *   residual_idx          uint8 [N/4][ceil(s/4)]: 2-bit position of that value inside its
 *                         group, entry (q, c) at bits 2*(c%4) of byte q*ceil(s/4) + c/4
 *
 * Return codes: 0 success, 1 invalid argument, 2 invalid code or index.
 */
#include <math.h>
#include <stddef.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

#define QO_OK 0
#define QO_BAD_ARG 1
#define QO_BAD_DATA 2

/* IEEE 754 binary16 -> double, exact (every binary16 value is a double). */
double qo_half_to_double(uint16_t h) {
  int sign = (h >> 15) & 1;
  int expo = (h >> 10) & 0x1f;
  int frac = h & 0x3ff;
  double mag;
  if (expo == 0) {
    mag = ldexp((double)frac, -24); /* subnormal: frac * 2^-24 */
  } else if (expo == 31) {
    mag = frac ? NAN : INFINITY;
  } else {
    mag = ldexp((double)(1024 + frac), expo - 25); /* (1 + frac/1024) * 2^(expo-15) */
  }
  return sign ? -mag : mag;
}

/* FP8 E4M3 -> double, exact (every E4M3 value is a double). */
double qo_e4m3_to_double(uint8_t b) {
  int sign = (b >> 7) & 1;
  int expo = (b >> 3) & 0xf;
  int frac = b & 7;
  double mag;
  if (expo == 0xf && frac == 7) {
    mag = NAN;
  } else if (expo == 0) {
    mag = ldexp((double)frac, -9); /* subnormal: frac/8 * 2^-6 */
  } else {
    mag = ldexp((double)(8 + frac), expo - 10); /* (1 + frac/8) * 2^(expo-7) */
  }
  return sign ? -mag : mag;
}

/* Value of residual entry (q, c): fp16 or, with fp8 set, FP8 E4M3. */
static double residual_value(const void* residual_vals, int fp8, int s, int q, int c) {
  size_t i = (size_t)q * s + c;
  return fp8 ? qo_e4m3_to_double(((const uint8_t*)residual_vals)[i])
             : qo_half_to_double(((const uint16_t*)residual_vals)[i]);
}

static int residual_stride(int s) { return (s + 3) / 4; }

static int residual_position(const uint8_t* ridx, int s, int q, int c) {
  return (ridx[(size_t)q * residual_stride(s) + c / 4] >> (2 * (c % 4))) & 3;
}

/*
 * The GEMV of Eq. 10 and Eq. 11 with Eq. 4's weights, y = x * W^T, in fp64.
 *
 *   x      fp16 [M][K]         alpha  fp16 [N][G]        beta  fp16 [N][G] or NULL (= 0)
 *   T      int8 [N][K]         v      fp16 [K]           G = ceil(K / group_size)
 *   rows   NULL for all rows, else the n_rows output rows to evaluate, in that order
 *   y      double [M][n_out]   bound  double [M][n_out] or NULL; n_out = N or n_rows
 *
 * y[m][o]     = sum_g ( alpha[o][g] sum_{j in g} T[o][j] v[j] x[m][j] + beta[o][g] sum_{j in g} x[m][j] )
 *             + sum_{c < s} [ residual position of (o/4, c) == o % 4 ] R[o/4][c] x[m][S_c]
 * bound[m][o] = sum_j | x[m][j] * W^[o][j] |, W^ the dense dequantized row including the
 *               residual entries, the scale of the comparison tolerance.
 * residual_fp8 selects FP8 E4M3 residual values (one byte each) instead of fp16.
 */
int qo_gemv_ex(int M, int N, int K, int group_size, const int8_t* T, const uint16_t* x,
               const uint16_t* alpha, const uint16_t* beta, const uint16_t* v, int s,
               const int32_t* salient_idx, const void* residual_vals, int residual_fp8,
               const uint8_t* residual_idx, const int32_t* rows, int n_rows, double* y, double* bound) {
  if (M < 0 || N < 0 || K < 0 || s < 0 || group_size <= 0) return QO_BAD_ARG;
  if (s > 0 && (N % 4 != 0 || !salient_idx || !residual_vals || !residual_idx)) return QO_BAD_ARG;
  for (int c = 0; c < s; ++c) {
    if (salient_idx[c] < 0 || salient_idx[c] >= K) return QO_BAD_DATA;
    if (c > 0 && salient_idx[c] <= salient_idx[c - 1]) return QO_BAD_DATA;
  }
  int G = (K + group_size - 1) / group_size;
  int n_out = rows ? n_rows : N;
  double* w_row = (double*)malloc(sizeof(double) * (size_t)(K > 0 ? K : 1));
  if (!w_row) return QO_BAD_ARG;
  int status = QO_OK;
  for (int i = 0; i < n_out && status == QO_OK; ++i) {
    int o = rows ? rows[i] : i;
    if (o < 0 || o >= N) { status = QO_BAD_ARG; break; }
    for (int j = 0; j < K; ++j) {
      int t = T[(size_t)o * K + j];
      if (t < -1 || t > 1) { status = QO_BAD_DATA; break; }
    }
    if (status != QO_OK) break;
    /* dense dequantized row W^[o][:] (Eq. 4 plus the residual of Eq. 11), for the bound */
    for (int j = 0; j < K; ++j) {
      int g = j / group_size;
      double a = qo_half_to_double(alpha[(size_t)o * G + g]);
      double b = beta ? qo_half_to_double(beta[(size_t)o * G + g]) : 0.0;
      w_row[j] = b + qo_half_to_double(v[j]) * a * (double)T[(size_t)o * K + j];
    }
    for (int c = 0; c < s; ++c) {
      if (residual_position(residual_idx, s, o / 4, c) == o % 4)
        w_row[salient_idx[c]] += residual_value(residual_vals, residual_fp8, s, o / 4, c);
    }
    for (int m = 0; m < M; ++m) {
      const uint16_t* xm = x + (size_t)m * K;
      double acc = 0.0;
      /* Eq. 10, group by group */
      for (int g = 0; g < G; ++g) {
        int j0 = g * group_size;
        int j1 = j0 + group_size < K ? j0 + group_size : K;
        double tvx = 0.0, sx = 0.0;
        for (int j = j0; j < j1; ++j) {
          double xj = qo_half_to_double(xm[j]);
          tvx += (double)T[(size_t)o * K + j] * qo_half_to_double(v[j]) * xj;
          sx += xj;
        }
        double a = qo_half_to_double(alpha[(size_t)o * G + g]);
        double b = beta ? qo_half_to_double(beta[(size_t)o * G + g]) : 0.0;
        acc += a * tvx + b * sx;
      }
      /* Eq. 11, the sparse residual over the salient columns */
      for (int c = 0; c < s; ++c) {
        if (residual_position(residual_idx, s, o / 4, c) == o % 4)
          acc += residual_value(residual_vals, residual_fp8, s, o / 4, c) *
                 qo_half_to_double(xm[salient_idx[c]]);
      }
      y[(size_t)m * n_out + i] = acc;
      if (bound) {
        double bsum = 0.0;
        for (int j = 0; j < K; ++j) bsum += fabs(qo_half_to_double(xm[j]) * w_row[j]);
        bound[(size_t)m * n_out + i] = bsum;
      }
    }
  }
  free(w_row);
  return status;
}

/* The same with fp16 residual values. */
int qo_gemv(int M, int N, int K, int group_size, const int8_t* T, const uint16_t* x,
            const uint16_t* alpha, const uint16_t* beta, const uint16_t* v, int s,
            const int32_t* salient_idx, const uint16_t* residual_vals, const uint8_t* residual_idx,
            const int32_t* rows, int n_rows, double* y, double* bound) {
  return qo_gemv_ex(M, N, K, group_size, T, x, alpha, beta, v, s, salient_idx, residual_vals, 0, residual_idx,
                    rows, n_rows, y, bound);
}

/* ---------------------------- packed layouts ---------------------------- */

static int round_up(int a, int b) { return (a + b - 1) / b * b; }

size_t qo_packed_bytes_2bit(int N, int K) { return (size_t)N * (size_t)round_up(K, 64) / 4; }

size_t qo_packed_bytes_base3(int N, int K) { return (size_t)N * (size_t)(round_up(K, 128) / 128) * 26; }

int qo_pack_2bit(const int8_t* T, int N, int K, uint8_t* out) {
  if (N < 0 || K < 0) return QO_BAD_ARG;
  int kp = round_up(K, 64);
  memset(out, 0, qo_packed_bytes_2bit(N, K));
  for (int r = 0; r < N; ++r) {
    for (int k = 0; k < kp; ++k) {
      int code = 1;
      if (k < K) {
        int t = T[(size_t)r * K + k];
        if (t < -1 || t > 1) return QO_BAD_DATA;
        code = t + 1;
      }
      out[(size_t)r * (kp / 4) + k / 4] |= (uint8_t)(code << (2 * (k % 4)));
    }
  }
  return QO_OK;
}

int qo_unpack_2bit(const uint8_t* packed, int N, int K, int8_t* T) {
  if (N < 0 || K < 0) return QO_BAD_ARG;
  int kp = round_up(K, 64);
  for (int r = 0; r < N; ++r) {
    for (int k = 0; k < kp; ++k) {
      int code = (packed[(size_t)r * (kp / 4) + k / 4] >> (2 * (k % 4))) & 3;
      if (code == 3) return QO_BAD_DATA;
      if (k < K) T[(size_t)r * K + k] = (int8_t)(code - 1);
      else if (code != 1) return QO_BAD_DATA;
    }
  }
  return QO_OK;
}

int qo_pack_base3(const int8_t* T, int N, int K, uint8_t* out) {
  if (N < 0 || K < 0) return QO_BAD_ARG;
  int groups = round_up(K, 128) / 128;
  for (int r = 0; r < N; ++r) {
    for (int h = 0; h < groups; ++h) {
      for (int p = 0; p < 26; ++p) {
        int value = 0, weight = 1;
        for (int d = 0; d < 5; ++d) {
          int col_in_group = 5 * p + d;
          int k = 128 * h + col_in_group;
          int digit = 1;
          if (col_in_group < 128 && k < K) {
            int t = T[(size_t)r * K + k];
            if (t < -1 || t > 1) return QO_BAD_DATA;
            digit = t + 1;
          }
          value += digit * weight;
          weight *= 3;
        }
        out[((size_t)r * groups + h) * 26 + p] = (uint8_t)value;
      }
    }
  }
  return QO_OK;
}

int qo_unpack_base3(const uint8_t* packed, int N, int K, int8_t* T) {
  if (N < 0 || K < 0) return QO_BAD_ARG;
  int groups = round_up(K, 128) / 128;
  for (int r = 0; r < N; ++r) {
    for (int h = 0; h < groups; ++h) {
      for (int p = 0; p < 26; ++p) {
        int value = packed[((size_t)r * groups + h) * 26 + p];
        if (value >= 243) return QO_BAD_DATA;
        for (int d = 0; d < 5; ++d) {
          int digit = value % 3;
          value /= 3;
          int col_in_group = 5 * p + d;
          int k = 128 * h + col_in_group;
          if (col_in_group < 128 && k < K) T[(size_t)r * K + k] = (int8_t)(digit - 1);
          else if (digit != 1) return QO_BAD_DATA;
        }
      }
    }
  }
  return QO_OK;
}

/*
 * Sec. 3.5 lookup table for one five-column pack: entry c (0 <= c < 243) is the dot
 * product of the pattern whose base-3 digits are d_0..d_4 (T = d - 1) with the scaled
 * activations xs[0..4] (xs = v * x).
 */
/* Sec. 3.5: the salient columns marked in the bitmap, ascending; returns their number (-1 for a
 * negative K) and writes the first max_s of them to out. */
int qo_salient_from_bitmap(const uint32_t* bitmap, int K, int32_t* out, int max_s) {
  if (K < 0) return -1;
  int n = 0;
  for (int j = 0; j < K; ++j) {
    if ((bitmap[j / 32] >> (j % 32)) & 1u) {
      if (n < max_s) out[n] = j;
      ++n;
    }
  }
  return n;
}

/* The bitmap of a salient index list (strictly ascending, each in [0, K)). */
int qo_salient_to_bitmap(const int32_t* idx, int s, int K, uint32_t* bitmap) {
  if (K < 0 || s < 0) return QO_BAD_ARG;
  memset(bitmap, 0, sizeof(uint32_t) * (size_t)((K + 31) / 32));
  for (int i = 0; i < s; ++i) {
    if (idx[i] < 0 || idx[i] >= K || (i > 0 && idx[i] <= idx[i - 1])) return QO_BAD_DATA;
    bitmap[idx[i] / 32] |= 1u << (idx[i] % 32);
  }
  return QO_OK;
}

void qo_lut5(const double xs[5], double lut[243]) {
  for (int c = 0; c < 243; ++c) {
    int rest = c;
    double dot = 0.0;
    for (int d = 0; d < 5; ++d) {
      dot += (double)(rest % 3 - 1) * xs[d];
      rest /= 3;
    }
    lut[c] = dot;
  }
}

/*
 * Appendix A latency model of the ternary-LUT engine and the 26-lane FP16 baseline, at
 * the stated 1 GHz clock, for y = x W with x [1, K] and W [K, N]. Results in microseconds.
 */
void qo_asic_latency_us(int K, int N, double* t_ternary_us, double* t_dense_us) {
  double groups = (double)((K + 127) / 128);
  *t_ternary_us = groups * (652.0 + 977.0 + (double)N) / 1000.0;
  *t_dense_us = (double)K * (double)N / 26.0 / 1000.0;
}
