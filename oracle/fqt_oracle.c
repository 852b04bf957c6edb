/*
 * fqt_oracle.c -- CPU oracle for the quantized backward pass of one linear
 * (or im2col-lowered conv) layer under fully quantized training (FQT), from
 * "A Statistical Framework for Low-bitwidth Training of Deep Neural Networks"
 * (Chen, Gai, Yao, Mahoney, Gonzalez, NeurIPS 2020, arXiv 2010.14298).
 *
 * TEST INFRASTRUCTURE ONLY.  This is a plain, slow, single-threaded CPU
 * restatement of the method, used to check the CUDA library.  Only the test
 * suite, the smoke check and the benchmark's CPU-baseline leg may load it.
 * It shares no code, header, table or constant generator with the CUDA
 * library, and the library never calls it.
 *
 * Build: gcc -O2 -std=c11 -ffp-contract=off -fPIC -shared (no -ffast-math):
 * every float expression below is evaluated as written, one IEEE rounding
 * per operation, without fused multiply-add.
 *
 * Readings taken where the paper leaves a detail open (each is argued in the
 * design notes of the repository):
 *  R1  Stochastic rounding SR (Sec. 3.3): the probability X - floor(X) is
 *      realised with a 16-bit uniform u from Philox4x32-10:
 *      code = (floor(v * 2^16) + u) >> 16, so P(round up) =
 *      floor(frac(v) * 2^16) / 2^16 (a downward bias below 2^-16 of a bin).
 *  R2  Uniform layout: key = (seed lo, seed hi); counter = (q lo, q hi,
 *      stream, 0) with q = i / 8 for the row-major flat index i; the 16-bit
 *      uniform is half (i mod 2) of word (i / 2) mod 4.  Stream 0 draws the
 *      Q_b2 codes, stream 1 the Q_b1 codes (App. E bifurcation).
 *  R3  The affine map and the rounding decision are FP32, as the paper's
 *      O(ND) FP32 transform (Sec. 4.1, 4.2): v = (h - z) * s for PTQ/PSQ.
 *      R = 0 (or B/R not finite) takes s = 1 and codes 0.
 *  R4  BHQ groups are contiguous blocks of `block` rows in original order;
 *      the lead row p of a block is the first row of largest infinity norm;
 *      lambda1 = R(h_p), lambda2 = 2 max_{k != p} ||h_k||_inf (Sec. 4.2),
 *      N in s1, s2 (App. D.4) is the actual block size.  lambda2 = 0 uses
 *      the limit s2 -> inf (small rows are zero), lambda1 = 0 uses
 *      lambda1 = 2 ||h_p||_inf, an all-zero block gives codes 0, scales 0.
 *  R5  BHQ zero point: the row-constant z' = min_j T_kj of the transformed
 *      block T = Q diag(s) H, so that every row maps into [0, B] (the range
 *      bound of App. D.4).  The transform is evaluated in double and rounded
 *      to FP32 before the FP32 rounding decision.
 *  R6  Stored metadata: value = inv_s * (Q_blk (code + zero)), with inv_s =
 *      1 / s and zero = s * z (PTQ/PSQ; Q_blk = I) or z' (BHQ).
 *  R7  Forward quantizers Q_f, Q_theta (Sec. 2.1, App. E): deterministic
 *      8-bit PTQ, round half to even, codes clamped to [0, B].
 *  R9  Shift quantizer (Sec. 4.3, left open by the paper): the range is
 *      per tensor and symmetric, [-M, M], so that every row shares the
 *      integer midpoint code 2^(b-1) as its zero point; a per-row zero point
 *      would add a per-row offset that shifted integer accumulators cannot
 *      absorb, and a per-tensor minimum as zero point leaves no room to
 *      shift rows that straddle 0.  Shifts are capped at 4 (the paper's
 *      [0, 4]).
 *  R8  Adaptive BHQ groups (App. D.5): as printed, the variance estimate
 *      sum_i M_i^2 / size_i with size_i = (N - G) M_i / sum M equals
 *      (sum_{i<=G} M_i)^2 / (N - G), which grows with G, so it would always
 *      pick one group.  It is the small-row-free limit of App. D.4's bound;
 *      the oracle keeps that bound's second term (see orc_bhq_grouping).
 */
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>

/* ------------------------------------------------------------------------ */
/* Philox4x32-10: J. K. Salmon, M. A. Moraes, R. O. Dror, D. E. Shaw,        */
/* "Parallel Random Numbers: As Easy as 1, 2, 3", SC'11.  Ten rounds of the  */
/* 4x32 S-box with multipliers 0xD2511F53 / 0xCD9E8D57 and the Weyl key      */
/* increments 0x9E3779B9 / 0xBB67AE85 (golden ratio, sqrt(3) - 1).           */
/* ------------------------------------------------------------------------ */
void orc_philox4x32_10(const uint32_t ctr_in[4], const uint32_t key_in[2],
                       uint32_t out[4]) {
  uint32_t x0 = ctr_in[0], x1 = ctr_in[1], x2 = ctr_in[2], x3 = ctr_in[3];
  uint32_t k0 = key_in[0], k1 = key_in[1];
  for (int round = 0; round < 10; ++round) {
    if (round > 0) {
      k0 += 0x9E3779B9u;
      k1 += 0xBB67AE85u;
    }
    uint64_t p0 = (uint64_t)0xD2511F53u * (uint64_t)x0;
    uint64_t p1 = (uint64_t)0xCD9E8D57u * (uint64_t)x2;
    uint32_t hi0 = (uint32_t)(p0 >> 32), lo0 = (uint32_t)p0;
    uint32_t hi1 = (uint32_t)(p1 >> 32), lo1 = (uint32_t)p1;
    uint32_t y0 = hi1 ^ x1 ^ k0;
    uint32_t y1 = lo1;
    uint32_t y2 = hi0 ^ x3 ^ k1;
    uint32_t y3 = lo0;
    x0 = y0; x1 = y1; x2 = y2; x3 = y3;
  }
  out[0] = x0; out[1] = x1; out[2] = x2; out[3] = x3;
}

/* 16-bit uniform for flat element index `idx` of stream `stream` (R2). */
uint32_t orc_u16(uint64_t seed, uint32_t stream, uint64_t idx) {
  uint64_t q = idx >> 3;
  uint32_t ctr[4] = {(uint32_t)q, (uint32_t)(q >> 32), stream, 0u};
  uint32_t key[2] = {(uint32_t)seed, (uint32_t)(seed >> 32)};
  uint32_t w[4];
  orc_philox4x32_10(ctr, key, w);
  uint32_t word = w[(idx >> 1) & 3u];
  return (idx & 1u) ? (word >> 16) : (word & 0xFFFFu);
}

/* Stochastic rounding SR(v) of v >= 0 onto the integers 0..B (Sec. 3.3, R1). */
uint32_t orc_sr(float v, uint32_t u16, uint32_t B) {
  float cap = (float)(B + 1u);
  if (!(v < cap)) v = cap; /* guards the fixed-point form; such v clamps to B */
  float scaled = v * 65536.0f; /* exact: power-of-two scaling */
  uint32_t fixed = (uint32_t)scaled; /* floor for v >= 0 */
  uint32_t code = (fixed + u16) >> 16;
  return code > B ? B : code;
}

/* Mean and variance of SR(v) by enumerating all 2^16 uniforms (brute force). */
void orc_sr_moments(float v, uint32_t B, double *mean, double *var) {
  double s1 = 0.0, s2 = 0.0;
  for (uint32_t u = 0; u < 65536u; ++u) {
    double c = (double)orc_sr(v, u, B);
    s1 += c;
    s2 += c * c;
  }
  double m = s1 / 65536.0;
  *mean = m;
  *var = s2 / 65536.0 - m * m;
}

/* Min and max of `count` floats; returns the number of non-finite entries. */
int64_t orc_range(const float *h, int64_t count, float *mn, float *mx) {
  float lo = INFINITY, hi = -INFINITY;
  int64_t bad = 0;
  for (int64_t i = 0; i < count; ++i) {
    float x = h[i];
    if (!isfinite(x)) { ++bad; continue; }
    if (x < lo) lo = x;
    if (x > hi) hi = x;
  }
  *mn = lo;
  *mx = hi;
  return bad;
}

/* Scale s = B / R(X) of PTQ and PSQ (Sec. 3.3, Sec. 4.1), with R3's guard. */
static float affine_scale(float mn, float mx, uint32_t B) {
  float R = mx - mn;
  if (!(R > 0.0f)) return 1.0f;
  float s = (float)B / R;
  if (!isfinite(s)) return 1.0f;
  return s;
}

/* ------------------------------------------------------------------------ */
/* Per-tensor quantizer PTQ (Sec. 3.3): z = min dH, s = B / R(dH),           */
/* Q = SR(s (dH - z)) / s + z.  Optional `vout` receives s (dH - z).         */
/* Returns the number of non-finite inputs (outputs untouched when > 0).     */
/* ------------------------------------------------------------------------ */
int64_t orc_quant_ptq(const float *h, int64_t n, int64_t c, int bits,
                      uint64_t seed, uint32_t stream, uint8_t *codes,
                      float *inv_s, float *zero, float *vout) {
  uint32_t B = (1u << bits) - 1u;
  float mn, mx;
  int64_t bad = orc_range(h, n * c, &mn, &mx);
  if (bad) return bad;
  float s = affine_scale(mn, mx, B);
  for (int64_t i = 0; i < n * c; ++i) {
    float v = (h[i] - mn) * s;
    if (vout) vout[i] = v;
    codes[i] = (uint8_t)orc_sr(v, orc_u16(seed, stream, (uint64_t)i), B);
  }
  inv_s[0] = 1.0f / s;
  zero[0] = s * mn;
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Per-sample quantizer PSQ (Sec. 4.1): S = diag(s_i), s_i = B / R(h_i),     */
/* z_i = min h_i, one affine map per row (sample).                           */
/* ------------------------------------------------------------------------ */
int64_t orc_quant_psq(const float *h, int64_t n, int64_t c, int bits,
                      uint64_t seed, uint32_t stream, uint8_t *codes,
                      float *inv_s, float *zero, float *vout) {
  uint32_t B = (1u << bits) - 1u;
  float gmn, gmx;
  int64_t bad = orc_range(h, n * c, &gmn, &gmx);
  if (bad) return bad;
  for (int64_t r = 0; r < n; ++r) {
    const float *row = h + r * c;
    float mn, mx;
    orc_range(row, c, &mn, &mx);
    float s = affine_scale(mn, mx, B);
    for (int64_t j = 0; j < c; ++j) {
      int64_t i = r * c + j;
      float v = (row[j] - mn) * s;
      if (vout) vout[i] = v;
      codes[i] = (uint8_t)orc_sr(v, orc_u16(seed, stream, (uint64_t)i), B);
    }
    inv_s[r] = 1.0f / s;
    zero[r] = s * mn;
  }
  return 0;
}

/* Householder reflection Q = I - 2 n n^T / ||n||^2 with n = 1/sqrt(N) 1 - e_p
 * (Sec. 4.2, App. D.4), written out as a dense N x N row-major matrix.
 * N = 1 has n = 0; the block is then left as is (Q = I). */
void orc_householder(int nb, int p, double *Q) {
  for (int a = 0; a < nb; ++a)
    for (int b = 0; b < nb; ++b) Q[a * nb + b] = (a == b) ? 1.0 : 0.0;
  if (nb <= 1) return;
  double *nv = (double *)malloc(sizeof(double) * (size_t)nb);
  double r = 1.0 / sqrt((double)nb), nn = 0.0;
  for (int a = 0; a < nb; ++a) {
    nv[a] = r - (a == p ? 1.0 : 0.0);
    nn += nv[a] * nv[a];
  }
  for (int a = 0; a < nb; ++a)
    for (int b = 0; b < nb; ++b) Q[a * nb + b] -= 2.0 * nv[a] * nv[b] / nn;
  free(nv);
}

/* Householder scales of App. D.4 for one group of N rows:
 *   s1 = B lambda1^{-1/3} N^{1/6} / (lambda1^{2/3} N^{-1/3} + lambda2^{2/3} N^{2/3})
 *   s2 = B lambda2^{-1/3} N^{1/6} / (same denominator).
 * lambda2 = 0 returns the limit s1 = B sqrt(N) / lambda1 and s2 = +inf.    */
void orc_bhq_scales(double lambda1, double lambda2, int nb, uint32_t B,
                    double *s1, double *s2) {
  double N = (double)nb;
  if (lambda2 <= 0.0) {
    *s1 = (double)B * sqrt(N) / lambda1;
    *s2 = INFINITY;
    return;
  }
  double c1 = cbrt(lambda1), c2 = cbrt(lambda2);
  double den = c1 * c1 * pow(N, -1.0 / 3.0) + c2 * c2 * pow(N, 2.0 / 3.0);
  *s1 = (double)B * pow(N, 1.0 / 6.0) / (c1 * den);
  *s2 = (double)B * pow(N, 1.0 / 6.0) / (c2 * den);
}

/* ------------------------------------------------------------------------ */
/* Block Householder quantizer BHQ (Sec. 4.2, App. D.4; R4, R5) for one      */
/* group of nb rows: src[k] is the row of h that becomes stored row k0 + k,  */
/* p the lead row within the group.  S = Q diag(s1, s2, ..., s2) with the    */
/* lead row carrying s1, T = S H_grp, z'_k = min_j T_kj,                     */
/* codes = SR(T - z' 1^T), drawn with the stored flat index (k0 + k) c + j.  */
/* Scratch: Q nb*nb, g and t nb*c, mnr/mxr/nrm nb entries.                   */
/* ------------------------------------------------------------------------ */
static void bhq_group(const float *h, int64_t c, const int64_t *src, int nb,
                      int p, int64_t k0, uint32_t B, uint64_t seed,
                      uint32_t stream, uint8_t *codes, float *inv_s,
                      float *zero, float *vout, double *Q, double *g, float *t,
                      float *mnr, float *mxr, float *nrm) {
  for (int k = 0; k < nb; ++k) {
    orc_range(h + src[k] * c, c, &mnr[k], &mxr[k]);
    float a = fabsf(mnr[k]), m = fabsf(mxr[k]);
    nrm[k] = a > m ? a : m; /* ||h_k||_inf */
  }
  if (!(nrm[p] > 0.0f)) { /* whole group is zero */
    for (int k = 0; k < nb; ++k) {
      for (int64_t j = 0; j < c; ++j) {
        codes[(k0 + k) * c + j] = 0;
        if (vout) vout[(k0 + k) * c + j] = 0.0f;
      }
      inv_s[k0 + k] = 0.0f;
      zero[k0 + k] = 0.0f;
    }
    return;
  }
  float lambda1 = mxr[p] - mnr[p];
  if (!(lambda1 > 0.0f)) lambda1 = 2.0f * nrm[p];
  float lambda2 = 0.0f;
  for (int k = 0; k < nb; ++k)
    if (k != p && nrm[k] > lambda2) lambda2 = nrm[k];
  lambda2 = 2.0f * lambda2;
  double s1, s2;
  orc_bhq_scales((double)lambda1, (double)lambda2, nb, B, &s1, &s2);
  float s1f = (float)s1;
  float s2f = lambda2 > 0.0f ? (float)s2 : 0.0f; /* 0 marks the s2 -> inf limit */
  /* g = diag(s) H_grp; rows other than p are zero when lambda2 = 0. */
  for (int k = 0; k < nb; ++k) {
    double sk = (k == p) ? (double)s1f : (double)s2f;
    for (int64_t j = 0; j < c; ++j)
      g[(size_t)k * c + j] = (k == p || lambda2 > 0.0f)
                                 ? sk * (double)h[src[k] * c + j]
                                 : 0.0;
  }
  orc_householder(nb, p, Q);
  for (int k = 0; k < nb; ++k) {
    for (int64_t j = 0; j < c; ++j) {
      double acc = 0.0;
      for (int m = 0; m < nb; ++m) acc += Q[k * nb + m] * g[(size_t)m * c + j];
      t[(size_t)k * c + j] = (float)acc;
    }
  }
  for (int k = 0; k < nb; ++k) {
    float zk = INFINITY;
    for (int64_t j = 0; j < c; ++j)
      if (t[(size_t)k * c + j] < zk) zk = t[(size_t)k * c + j];
    for (int64_t j = 0; j < c; ++j) {
      int64_t i = (k0 + k) * c + j;
      float v = t[(size_t)k * c + j] - zk;
      if (vout) vout[i] = v;
      codes[i] = (uint8_t)orc_sr(v, orc_u16(seed, stream, (uint64_t)i), B);
    }
    zero[k0 + k] = zk;
    if (k == p)
      inv_s[k0 + k] = 1.0f / s1f;
    else
      inv_s[k0 + k] = lambda2 > 0.0f ? 1.0f / s2f : 0.0f;
  }
}

/* BHQ with contiguous blocks of `block` rows in original order (R4): the   */
/* lead row p of a block is its first row of largest infinity norm.         */
/* `lead` receives p for every block.                                        */
int64_t orc_quant_bhq(const float *h, int64_t n, int64_t c, int bits,
                      int block, uint64_t seed, uint32_t stream,
                      uint8_t *codes, float *inv_s, float *zero, int32_t *lead,
                      float *vout) {
  uint32_t B = (1u << bits) - 1u;
  float gmn, gmx;
  int64_t bad = orc_range(h, n * c, &gmn, &gmx);
  if (bad) return bad;
  double *Q = (double *)malloc(sizeof(double) * (size_t)block * (size_t)block);
  double *g = (double *)malloc(sizeof(double) * (size_t)block * (size_t)c);
  float *t = (float *)malloc(sizeof(float) * (size_t)block * (size_t)c);
  float *mnr = (float *)malloc(sizeof(float) * (size_t)block);
  float *mxr = (float *)malloc(sizeof(float) * (size_t)block);
  float *nrm = (float *)malloc(sizeof(float) * (size_t)block);
  int64_t *src = (int64_t *)malloc(sizeof(int64_t) * (size_t)block);
  int64_t nblocks = (n + block - 1) / block;
  for (int64_t b = 0; b < nblocks; ++b) {
    int64_t r0 = b * block;
    int nb = (int)((n - r0) < block ? (n - r0) : block);
    int p = 0;
    float best = -1.0f;
    for (int k = 0; k < nb; ++k) {
      float mn, mx;
      orc_range(h + (r0 + k) * c, c, &mn, &mx);
      float a = fabsf(mn), m = fabsf(mx);
      float nk = a > m ? a : m;
      if (nk > best) { best = nk; p = k; }
      src[k] = r0 + k;
    }
    lead[b] = p;
    bhq_group(h, c, src, nb, p, r0, B, seed, stream, codes, inv_s, zero, vout,
              Q, g, t, mnr, mxr, nrm);
  }
  free(Q); free(g); free(t); free(mnr); free(mxr); free(nrm); free(src);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Adaptive BHQ grouping (App. D.5; R8).                                     */
/*  1. M_i = ||h_i||_inf; rows in descending M, ties by ascending row index. */
/*  2. For G = 1 .. n-1 the first G rows are large and the other n - G      */
/*     small; group i holds the i-th large row and size_i = (n - G) M_i /    */
/*     S_G small rows, S_G = sum of the G large M_i.  The variance of the    */
/*     grouping is estimated with App. D.4's bound per group,                */
/*       V(G) = sum_i (M_i^(2/3) size_i^(-1/3) + L^(2/3) size_i^(2/3))^3,    */
/*     L = M_(G+1), the largest small row: every group's small rows are at   */
/*     most that large.  L -> 0 leaves sum_i M_i^2 / size_i, App. D.5's own  */
/*     estimate.  A large row with M_i = 0 adds 0; S_G = 0 gives V = 0.      */
/*     G = argmin V (the smallest G on ties); n = 1 gives G = 1.             */
/*  3. Integer sizes by cumulative rounding: e_0 = 0,                        */
/*     e_i = floor((n - G) (C_i / S_G) + 1/2) with C_i the sum of the first  */
/*     i large M, e_G = n - G; group i takes e_i - e_(i-1) small rows.  The  */
/*     small rows are dealt from the smallest up: group 1 takes the          */
/*     e_1 smallest, group 2 the next e_2 - e_1, and so on.                  */
/*  4. Stored order: group after group, each lead row first, then its small  */
/*     rows in descending M.  perm[k] = row of h stored at k; gstart[i] =    */
/*     first stored row of group i (i < G), gstart[G .. n] = n; gsize[k] =   */
/*     size of the group holding stored row k.  V[G-1] = V(G) when V is     */
/*     non-NULL (n - 1 entries).  Returns the number of non-finite entries.  */
/* ------------------------------------------------------------------------ */
typedef struct {
  float m;
  int64_t i;
} orc_mrow;

static int cmp_mrow(const void *a, const void *b) {
  const orc_mrow *x = (const orc_mrow *)a, *y = (const orc_mrow *)b;
  if (x->m != y->m) return x->m > y->m ? -1 : 1;
  return x->i < y->i ? -1 : (x->i > y->i ? 1 : 0);
}

int64_t orc_bhq_grouping(const float *h, int64_t n, int64_t c, int32_t *perm,
                         int32_t *gstart, int32_t *gsize, int64_t *G_out,
                         double *V) {
  float gmn, gmx;
  int64_t bad = orc_range(h, n * c, &gmn, &gmx);
  if (bad) return bad;
  orc_mrow *r = (orc_mrow *)malloc(sizeof(orc_mrow) * (size_t)(n > 0 ? n : 1));
  for (int64_t i = 0; i < n; ++i) {
    float mn, mx;
    orc_range(h + i * c, c, &mn, &mx);
    float a = fabsf(mn), m = fabsf(mx);
    r[i].m = a > m ? a : m;
    r[i].i = i;
  }
  qsort(r, (size_t)n, sizeof(orc_mrow), cmp_mrow);
  int64_t G = 1;
  if (n >= 2) {
    double best = INFINITY;
    for (int64_t g = 1; g < n; ++g) {
      double S = 0.0;
      for (int64_t i = 0; i < g; ++i) S += (double)r[i].m;
      double v = 0.0;
      if (S > 0.0) {
        double L = (double)r[g].m, cl = cbrt(L);
        for (int64_t i = 0; i < g; ++i) {
          double Mi = (double)r[i].m;
          if (!(Mi > 0.0)) continue;
          double size = (double)(n - g) * Mi / S;
          double cm = cbrt(Mi), cs = cbrt(size);
          double term = cm * cm / cs + cl * cl * cs * cs;
          v += term * term * term;
        }
      }
      if (V) V[g - 1] = v;
      if (v < best) {
        best = v;
        G = g;
      }
    }
  }
  /* cumulative rounding of the sizes */
  int64_t *e = (int64_t *)malloc(sizeof(int64_t) * (size_t)(G + 1));
  double SG = 0.0;
  for (int64_t i = 0; i < G; ++i) SG += (double)r[i].m;
  e[0] = 0;
  double Ci = 0.0;
  for (int64_t i = 1; i <= G; ++i) {
    Ci += (double)r[i - 1].m;
    if (i == G)
      e[i] = n - G;
    else if (SG > 0.0)
      e[i] = (int64_t)floor((double)(n - G) * (Ci / SG) + 0.5);
    else
      e[i] = 0;
  }
  for (int64_t i = 0; i < G; ++i) {
    int64_t k0 = i + e[i], ns = e[i + 1] - e[i];
    gstart[i] = (int32_t)k0;
    perm[k0] = (int32_t)r[i].i;
    for (int64_t t = 0; t < ns; ++t) perm[k0 + 1 + t] = (int32_t)r[n - e[i + 1] + t].i;
    for (int64_t t = 0; t <= ns; ++t) gsize[k0 + t] = (int32_t)(ns + 1);
  }
  for (int64_t i = G; i <= n; ++i) gstart[i] = (int32_t)n;
  *G_out = G;
  free(e);
  free(r);
  return 0;
}

/* BHQ over explicit groups (App. D.5 grouping, R8): group i is stored rows */
/* gstart[i] .. gstart[i+1]-1, read from rows perm[k] of h, lead first.     */
int64_t orc_quant_bhq_groups(const float *h, int64_t n, int64_t c, int bits,
                             const int32_t *perm, const int32_t *gstart,
                             int64_t G, uint64_t seed, uint32_t stream,
                             uint8_t *codes, float *inv_s, float *zero,
                             float *vout) {
  uint32_t B = (1u << bits) - 1u;
  float gmn, gmx;
  int64_t bad = orc_range(h, n * c, &gmn, &gmx);
  if (bad) return bad;
  int64_t mx = 1;
  for (int64_t i = 0; i < G; ++i)
    if (gstart[i + 1] - gstart[i] > mx) mx = gstart[i + 1] - gstart[i];
  double *Q = (double *)malloc(sizeof(double) * (size_t)mx * (size_t)mx);
  double *g = (double *)malloc(sizeof(double) * (size_t)mx * (size_t)c);
  float *t = (float *)malloc(sizeof(float) * (size_t)mx * (size_t)c);
  float *mnr = (float *)malloc(sizeof(float) * (size_t)mx);
  float *mxr = (float *)malloc(sizeof(float) * (size_t)mx);
  float *nrm = (float *)malloc(sizeof(float) * (size_t)mx);
  int64_t *src = (int64_t *)malloc(sizeof(int64_t) * (size_t)mx);
  for (int64_t i = 0; i < G; ++i) {
    int64_t k0 = gstart[i];
    int nb = (int)(gstart[i + 1] - k0);
    for (int k = 0; k < nb; ++k) src[k] = perm[k0 + k];
    bhq_group(h, c, src, nb, 0, k0, B, seed, stream, codes, inv_s, zero, vout,
              Q, g, t, mnr, mxr, nrm);
  }
  free(Q); free(g); free(t); free(mnr); free(mxr); free(nrm); free(src);
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Per-sample power-of-two shift quantizer (Sec. 4.3; R9): one symmetric     */
/* per-tensor range [-M, M], M = max |dH|, base scale s = (2^(b-1) - 1) / M, */
/* and per row a shift sh_i, the largest integer in [0, 4] with              */
/* 2^sh_i ||h_i||_inf <= M.  Row i is quantized with s 2^sh_i around the     */
/* integer midpoint z0 = 2^(b-1): v = (s 2^sh_i) h + z0, code = SR(v), so    */
/* value = (code - z0) / (s 2^sh_i): inv_s_i = (1/s) 2^-sh_i, zero_i = -z0   */
/* (R6's encoding, per row).  M = 0 (or s not finite) takes s = 1.           */
/* `shift` receives sh_i.                                                    */
/* ------------------------------------------------------------------------ */
int64_t orc_quant_shift(const float *h, int64_t n, int64_t c, int bits,
                        uint64_t seed, uint32_t stream, uint8_t *codes,
                        float *inv_s, float *zero, int32_t *shift, float *vout) {
  uint32_t B = (1u << bits) - 1u;
  float z0 = (float)(1u << (bits - 1));
  float gmn, gmx;
  int64_t bad = orc_range(h, n * c, &gmn, &gmx);
  if (bad) return bad;
  float M = fabsf(gmn) > fabsf(gmx) ? fabsf(gmn) : fabsf(gmx);
  float s = (float)((1u << (bits - 1)) - 1u) / M;
  if (!(M > 0.0f) || !isfinite(s)) s = 1.0f;
  float inv = 1.0f / s;
  for (int64_t r = 0; r < n; ++r) {
    const float *row = h + r * c;
    float mn, mx;
    orc_range(row, c, &mn, &mx);
    float Mi = fabsf(mn) > fabsf(mx) ? fabsf(mn) : fabsf(mx);
    int sh = 0;
    while (sh < 4 && ldexpf(Mi, sh + 1) <= M) ++sh;
    float sr = ldexpf(s, sh); /* exact: a power-of-two multiple */
    for (int64_t j = 0; j < c; ++j) {
      int64_t i = r * c + j;
      float v = sr * row[j] + z0;
      if (vout) vout[i] = v;
      codes[i] = (uint8_t)orc_sr(v, orc_u16(seed, stream, (uint64_t)i), B);
    }
    inv_s[r] = ldexpf(inv, -sh);
    zero[r] = -z0;
    shift[r] = sh;
  }
  return 0;
}

/* Gradient quantizer dispatch: kind 0 = PTQ, 1 = PSQ, 2 = BHQ, 3 = the shift
 * quantizer (`lead` then receives the per-row shifts). */
int64_t orc_quantize_grad(const float *h, int64_t n, int64_t c, int kind,
                          int bits, int block, uint64_t seed, uint32_t stream,
                          uint8_t *codes, float *inv_s, float *zero,
                          int32_t *lead, float *vout) {
  if (kind == 0)
    return orc_quant_ptq(h, n, c, bits, seed, stream, codes, inv_s, zero, vout);
  if (kind == 1)
    return orc_quant_psq(h, n, c, bits, seed, stream, codes, inv_s, zero, vout);
  if (kind == 3)
    return orc_quant_shift(h, n, c, bits, seed, stream, codes, inv_s, zero, lead, vout);
  return orc_quant_bhq(h, n, c, bits, block, seed, stream, codes, inv_s, zero,
                       lead, vout);
}

/* ------------------------------------------------------------------------ */
/* Deterministic PTQ of the forward operands X~ = Q_f(X), W~ = Q_theta(W)    */
/* (Sec. 2.1, App. E; R7): v = (x - min) s, code = round-half-even(v).       */
/* ------------------------------------------------------------------------ */
int64_t orc_quant_det(const float *x, int64_t n, int64_t c, int bits,
                      uint8_t *codes, float *inv_s, float *zero) {
  uint32_t B = (1u << bits) - 1u;
  float mn, mx;
  int64_t bad = orc_range(x, n * c, &mn, &mx);
  if (bad) return bad;
  float s = affine_scale(mn, mx, B);
  for (int64_t i = 0; i < n * c; ++i) {
    float v = (x[i] - mn) * s;
    float r = nearbyintf(v); /* default rounding mode: half to even */
    if (r < 0.0f) r = 0.0f;
    if (r > (float)B) r = (float)B;
    codes[i] = (uint8_t)r;
  }
  inv_s[0] = 1.0f / s;
  zero[0] = s * mn;
  return 0;
}

/* ------------------------------------------------------------------------ */
/* Dequantization: the value a code represents (Eq. 9 with R6),              */
/*   Q(dH) = S^{-1} (codes + z' 1^T) = diag(inv_s) Q_blk (codes + z' 1^T).   */
/* kind 0 reads inv_s[0], zero[0]; kind 1 one pair per row; kind 2 one pair  */
/* per row and the block reflections built from `lead`.                      */
/* ------------------------------------------------------------------------ */
void orc_dequant_f64(const double *codes, int64_t n, int64_t c, int kind,
                     int block, const float *inv_s, const float *zero,
                     const int32_t *lead, double *out) {
  if (kind != 2) {
    for (int64_t r = 0; r < n; ++r) {
      double is = (double)inv_s[kind == 0 ? 0 : r];
      double z = (double)zero[kind == 0 ? 0 : r];
      for (int64_t j = 0; j < c; ++j)
        out[r * c + j] = is * (codes[r * c + j] + z);
    }
    return;
  }
  double *Q = (double *)malloc(sizeof(double) * (size_t)block * (size_t)block);
  int64_t nblocks = (n + block - 1) / block;
  for (int64_t b = 0; b < nblocks; ++b) {
    int64_t r0 = b * block;
    int nb = (int)((n - r0) < block ? (n - r0) : block);
    orc_householder(nb, lead[b], Q);
    for (int k = 0; k < nb; ++k) {
      double is = (double)inv_s[r0 + k];
      for (int64_t j = 0; j < c; ++j) {
        double acc = 0.0;
        for (int m = 0; m < nb; ++m)
          acc += Q[k * nb + m] *
                 (codes[(r0 + m) * c + j] + (double)zero[r0 + m]);
        out[(r0 + k) * c + j] = is * acc;
      }
    }
  }
  free(Q);
}

/* Dequantization over explicit groups (R8), rows in stored order:        */
/* out_k = inv_s_k (Q_grp (codes + z' 1^T))_k, the lead first in its group. */
void orc_dequant_groups_f64(const double *codes, int64_t n, int64_t c,
                            const int32_t *gstart, int64_t G,
                            const float *inv_s, const float *zero,
                            double *out) {
  for (int64_t i = 0; i < G; ++i) {
    int64_t r0 = gstart[i];
    int nb = (int)(gstart[i + 1] - r0);
    double *Q = (double *)malloc(sizeof(double) * (size_t)nb * (size_t)nb);
    orc_householder(nb, 0, Q);
    for (int k = 0; k < nb; ++k) {
      double is = (double)inv_s[r0 + k];
      for (int64_t j = 0; j < c; ++j) {
        double acc = 0.0;
        for (int m = 0; m < nb; ++m)
          acc += Q[k * nb + m] *
                 (codes[(r0 + m) * c + j] + (double)zero[r0 + m]);
        out[(r0 + k) * c + j] = is * acc;
      }
    }
    free(Q);
  }
  (void)n;
}

/* Same map for uint8 codes. */
void orc_dequant(const uint8_t *codes, int64_t n, int64_t c, int kind,
                 int block, const float *inv_s, const float *zero,
                 const int32_t *lead, double *out) {
  double *cd = (double *)malloc(sizeof(double) * (size_t)(n * c));
  for (int64_t i = 0; i < n * c; ++i) cd[i] = (double)codes[i];
  orc_dequant_f64(cd, n, c, kind, block, inv_s, zero, lead, out);
  free(cd);
}

/* Exact integer contraction P_ij = sum_k (A_ik - oa)(B_kj - ob) in int64.
 * A is M x K, stored row-major (a_kmajor = 1) or as its K x M transpose;
 * B is K x N, stored row-major as K x N (b_kmajor = 0) or as N x K.        */
void orc_int_gemm(const uint8_t *A, int a_kmajor, const uint8_t *Bm,
                  int b_kmajor, int64_t M, int64_t N, int64_t K, int oa, int ob,
                  int64_t *out) {
  for (int64_t i = 0; i < M; ++i)
    for (int64_t j = 0; j < N; ++j) {
      int64_t acc = 0;
      for (int64_t k = 0; k < K; ++k) {
        int64_t a = a_kmajor ? A[i * K + k] : A[k * M + i];
        int64_t b = b_kmajor ? Bm[j * K + k] : Bm[k * N + j];
        acc += (a - oa) * (b - ob);
      }
      out[i * N + j] = acc;
    }
}

/* Plain double matrix product out = op(A) Bm, op(A) = A (M x K) or A^T when
 * a_trans (A stored K x M); Bm is K x N row-major. */
void orc_matmul_f64(const double *A, int a_trans, const double *Bm, int64_t M,
                    int64_t K, int64_t N, double *out) {
  for (int64_t i = 0; i < M; ++i)
    for (int64_t j = 0; j < N; ++j) out[i * N + j] = 0.0;
  for (int64_t i = 0; i < M; ++i)
    for (int64_t k = 0; k < K; ++k) {
      double a = a_trans ? A[k * M + i] : A[i * K + k];
      for (int64_t j = 0; j < N; ++j) out[i * N + j] += a * Bm[k * N + j];
    }
}

/* ------------------------------------------------------------------------ */
/* col2im of an im2col-space gradient (the adjoint of im2col; a conv layer   */
/* as a linear layer on im2col rows, Sec. 2.1): G has one row per output     */
/* pixel (n, oy, ox) and columns (ky, kx, c); the result is NHWC,            */
/* out[n, y, x, c] = sum of G[(n, oy, ox), (ky, kx, c)] over the output      */
/* pixels and taps with y = oy stride + ky - pad, x = ox stride + kx - pad.  */
/* ------------------------------------------------------------------------ */
void orc_col2im_nhwc(const double *G, int64_t n, int64_t h, int64_t w, int64_t c, int kh,
                     int kw, int stride, int pad, double *out) {
  int64_t oh = (h + 2 * pad - kh) / stride + 1;
  int64_t ow = (w + 2 * pad - kw) / stride + 1;
  for (int64_t i = 0; i < n * h * w * c; ++i) out[i] = 0.0;
  for (int64_t b = 0; b < n; ++b)
    for (int64_t oy = 0; oy < oh; ++oy)
      for (int64_t ox = 0; ox < ow; ++ox) {
        const double *row = G + ((b * oh + oy) * ow + ox) * (int64_t)(kh * kw) * c;
        for (int ky = 0; ky < kh; ++ky)
          for (int kx = 0; kx < kw; ++kx) {
            int64_t y = oy * stride + ky - pad, x = ox * stride + kx - pad;
            if (y < 0 || y >= h || x < 0 || x >= w) continue; /* a padding entry */
            const double *g = row + (int64_t)(ky * kw + kx) * c;
            double *o = out + ((b * h + y) * w + x) * c;
            for (int64_t ch = 0; ch < c; ++ch) o[ch] += g[ch];
          }
      }
}
