/*
 * awsrc_oracle.c — plain, slow CPU oracle of AWSRC's encoder, selection and
 * decoder (Activation-Weighted Seeded Residual Coding, arXiv 2608.23144).
 *
 * TEST INFRASTRUCTURE ONLY. Nothing in the product path may call this file:
 * only tests/, __graft_entry__.smoke() and bench.py's cpu_baseline leg load it.
 * It shares no code, header, table or constant with the CUDA library; both are
 * written independently from the paper and from the numeric convention stated
 * in the public header.
 *
 * Two modes:
 *  - spec mode (float): the paper's steps in the paper's order, in binary32 with
 *    one rounding per operation. Integer decisions (seed, exponent, codes) are
 *    taken in binary32, the precision the GPU path decides them in.
 *  - definition mode (double): Eq. 3 solved by Gaussian elimination on the
 *    normal equations and Eq. 4 evaluated directly from the reconstructed tile;
 *    used to validate spec mode and to adjudicate near-ties.
 *
 * Built with -ffp-contract=off so that no multiply-add is fused unless written
 * as fmaf().
 *
 * Readings of points the paper leaves open, all stated in the library header:
 * the generator (SplitMix64, Sec. 3.1 only says encoder and decoder share one),
 * a relative ridge eps = ridge_rel * mean(d) (Sec. 3.2 gives no value), the
 * symmetric code range [-qmax, qmax], the smallest non-clipping power-of-two
 * exponent, the 40 + 8*n_mod byte header (Sec. 4 gives 904 B for 108 modules).
 *
 * Parity unpinned by the paper: the generator (orc_gen_basis). The paper
 * prints no generator values, so it is pinned only to SplitMix64's published
 * outputs, to an independent restatement of the draw schedule in the tests,
 * and to the basis structure (bijective permutation, distinct columns, exact
 * orthonormality).
 */
#include <float.h>
#include <math.h>
#include <stdint.h>
#include <stdlib.h>
#include <string.h>
#ifdef _OPENMP
#include <omp.h>
#endif

#define ORC_MAXP 8
#define ORC_GAMMA 0x9E3779B97F4A7C15ULL


/* Candidate record layout mirrors the ABI's 16-byte struct (an interface, not code). */
typedef struct {
  float gain;
  uint16_t seed;
  int16_t scale;
  int8_t code[8];
} orc_candidate;

typedef struct {
  int32_t C, P, b, S;
  int32_t b_e, e_bias;
  int32_t scale_mode, permute, variant;
  float ridge_rel;
  uint64_t gen_seed;
} orc_params;

/* ------------------------------------------------------------------------ */
/* SplitMix64 (Steele, Lea & Flood, "Fast splittable pseudorandom number     */
/* generators", OOPSLA 2014): state advances by the golden gamma and each    */
/* output is the MurmurHash3-style 64-bit finaliser of the state.           */
/* ------------------------------------------------------------------------ */
static uint64_t orc_mix64(uint64_t z) {
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ULL;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBULL;
  return z ^ (z >> 31);
}

/* Host threads the oracle's parallel loops use. */
int orc_num_threads(void) {
#ifdef _OPENMP
  return omp_get_max_threads();
#else
  return 1;
#endif
}

/* n-th output (n >= 1) of the SplitMix64 stream whose initial state is x. */
uint64_t orc_splitmix64_output(uint64_t x, uint64_t n) { return orc_mix64(x + n * ORC_GAMMA); }

/* ------------------------------------------------------------------------ */
/* GenBasis(s, C, P)  — Eq. 2 and the sentence after it (Sec. 3.1): a seed    */
/* selects a sign pattern, a coordinate permutation and P columns of the     */
/* order-C (Sylvester) Hadamard matrix; the basis is normalised.             */
/* Outputs: sign[C] in {0,1} (1 = negative), perm[C], cols[P], and           */
/* negmask[p*C + j] = 1 where entry (j, p) of B_s is negative.              */
/* ------------------------------------------------------------------------ */
static int orc_popcount(uint32_t v) {
  int n = 0;
  while (v) { n += (int)(v & 1u); v >>= 1; }
  return n;
}

void orc_gen_basis(uint64_t gen_seed, uint32_t s, int C, int P, int permute,
                   uint8_t* sign, int32_t* perm, int32_t* cols, uint8_t* negmask) {
  uint64_t key = orc_splitmix64_output(gen_seed, (uint64_t)s + 1);
  uint64_t n = 1;
  /* sign pattern: one 64-bit draw per 64 coordinates */
  for (int w = 0; w * 64 < C; ++w) {
    uint64_t word = orc_splitmix64_output(key, n++);
    for (int j = w * 64; j < C && j < w * 64 + 64; ++j) sign[j] = (uint8_t)((word >> (j - w * 64)) & 1u);
  }
  /* coordinate permutation: Fisher-Yates (Durstenfeld), index by multiply-shift */
  for (int j = 0; j < C; ++j) perm[j] = j;
  if (permute) {
    for (int i = C - 1; i >= 1; --i) {
      uint64_t x = orc_splitmix64_output(key, n++) >> 32;
      int k = (int)((x * (uint64_t)(i + 1)) >> 32);
      int32_t t = perm[i]; perm[i] = perm[k]; perm[k] = t;
    }
  }
  /* P distinct Hadamard columns: partial Fisher-Yates over 0..C-1, draw order kept */
  int32_t pool[256];
  for (int j = 0; j < C; ++j) pool[j] = j;
  for (int p = 0; p < P; ++p) {
    uint64_t x = orc_splitmix64_output(key, n++) >> 32;
    int k = p + (int)((x * (uint64_t)(C - p)) >> 32);
    int32_t t = pool[p]; pool[p] = pool[k]; pool[k] = t;
    cols[p] = pool[p];
  }
  /* B_s[j][p] = C^-1/2 * sigma_j * H[pi(j), c_p],  H[i][k] = (-1)^popcount(i & k) */
  for (int p = 0; p < P; ++p)
    for (int j = 0; j < C; ++j)
      negmask[p * C + j] = (uint8_t)((sign[j] + orc_popcount((uint32_t)(perm[j] & cols[p]))) & 1);
}

/* ------------------------------------------------------------------------ */
/* Rounding helpers (IEEE binary16 / bfloat16, round to nearest even).       */
/* ------------------------------------------------------------------------ */
static uint32_t orc_f2u(float f) { uint32_t u; memcpy(&u, &f, 4); return u; }
static float orc_u2f(uint32_t u) { float f; memcpy(&f, &u, 4); return f; }

uint16_t orc_f32_to_f16(float f) {
  uint32_t x = orc_f2u(f);
  uint16_t sign = (uint16_t)((x >> 16) & 0x8000u);
  uint32_t ax = x & 0x7fffffffu;
  if (ax > 0x7f800000u) return (uint16_t)(sign | 0x7e00u);  /* NaN */
  if (ax == 0x7f800000u) return (uint16_t)(sign | 0x7c00u); /* inf */
  float a = orc_u2f(ax);
  if (a < 6.103515625e-05f) {            /* below 2^-14: binary16 subnormal range */
    float n = rintf(a * 16777216.0f);    /* multiple of 2^-24, exact scaling then RNE */
    return (uint16_t)(sign | (uint16_t)n);  /* n == 1024 encodes 2^-14, the smallest normal */
  }
  int e = (int)(ax >> 23) - 127 + 15;
  if (e >= 31) return (uint16_t)(sign | 0x7c00u);
  uint32_t m = ax & 0x7fffffu;
  uint32_t h = ((uint32_t)e << 10) | (m >> 13);
  uint32_t rem = m & 0x1fffu;
  if (rem > 0x1000u || (rem == 0x1000u && (h & 1u))) h += 1u; /* carry may reach inf: correct */
  return (uint16_t)(sign | h);
}

float orc_f16_to_f32(uint16_t h) {
  uint32_t sign = (uint32_t)(h & 0x8000u) << 16;
  int e = (h >> 10) & 0x1f;
  uint32_t m = h & 0x3ffu;
  if (e == 0) {
    float v = ldexpf((float)m, -24);
    return sign ? -v : v;
  }
  if (e == 31) return orc_u2f(sign | 0x7f800000u | (m << 13));
  return orc_u2f(sign | ((uint32_t)(e - 15 + 127) << 23) | (m << 13));
}

uint16_t orc_f32_to_bf16(float f) {
  uint32_t x = orc_f2u(f);
  if ((x & 0x7fffffffu) > 0x7f800000u) return (uint16_t)((x >> 16) | 0x40u);
  uint32_t lsb = (x >> 16) & 1u;
  return (uint16_t)((x + 0x7fffu + lsb) >> 16);
}

/* ------------------------------------------------------------------------ */
/* Spec-mode score of one (tile, seed) candidate: Eq. 3 fit, Sec. 3.2        */
/* quantisation, Eq. 4 gain. Returns 1 if the candidate is valid.            */
/* r, d: the tile's residual and weights (C floats). negmask: GenBasis(s).   */
/* alpha_out (may be NULL): the float fit alpha*.                            */
/* ------------------------------------------------------------------------ */
static int orc_qmax(int b) { return (1 << (b - 1)) - 1; }

static void orc_exp_range(const orc_params* prm, int* lo, int* hi) {
  int half = 1 << (prm->b_e - 1);
  *lo = prm->e_bias - half;
  *hi = prm->e_bias + half - 1;
  if (*lo < -126) *lo = -126;
  if (*hi > 126) *hi = 126;
}

/* Per-tile fixed point: q = ilogb(max |x_j|) - 20 so that max |x| 2^-q lies in
 * [2^20, 2^21), and X_j = rint(x_j 2^-q) (exact scaling, one rounding), so
 * |X_j| <= 2^21. A vector whose largest magnitude is below 2^-100 is all zero
 * (q = 0). Returns q. */
int orc_fixed_point(int C, const float* x, int32_t* X) {
  float m = 0.0f;
  for (int j = 0; j < C; ++j)
    if (fabsf(x[j]) > m) m = fabsf(x[j]);
  if (!(m >= 0x1p-100f)) {
    for (int j = 0; j < C; ++j) X[j] = 0;
    return 0;
  }
  int q = ilogbf(m) - 20;
  for (int j = 0; j < C; ++j) X[j] = (int32_t)rintf(ldexpf(x[j], -q));
  return q;
}

int orc_tile_valid(int C, const float* r, const float* d) {
  for (int j = 0; j < C; ++j) {
    if (!(fabsf(r[j]) <= 65536.0f)) return 0;                  /* also rejects NaN */
    if (!(d[j] >= 0.0f && d[j] <= 4294967296.0f)) return 0;
  }
  return 1;
}

int orc_score_candidate(const orc_params* prm, const float* r, const float* d,
                        const uint8_t* negmask, float* gain_out, int16_t* scale_out,
                        int8_t* codes_out, float* alpha_out) {
  const int C = prm->C, P = prm->P;
  const int qmax = orc_qmax(prm->b);
  const float c = (float)(1.0 / sqrt((double)C));  /* RN(C^-1/2) */
  const float c2 = 1.0f / (float)C;                  /* exact: C is a power of two */
  float y[256];
  for (int j = 0; j < C; ++j) y[j] = d[j] * r[j];

  /* Correlations of Eq. 3 on a per-tile fixed-point grid: y and d become
   * integers Y = rint(y 2^-qy), D = rint(d 2^-qd) with at most 21 bits, their
   * +-1 correlations are summed exactly (integers) and rounded once. */
  int32_t Y[256], Dq[256];
  int qy = orc_fixed_point(C, y, Y);
  int qd = orc_fixed_point(C, d, Dq);

  /* right-hand side b = B_s^T D r  (Eq. 3 normal equations) */
  float bvec[ORC_MAXP];
  for (int p = 0; p < P; ++p) {
    int64_t su = 0;
    for (int j = 0; j < C; ++j) su += negmask[p * C + j] ? -(int64_t)Y[j] : (int64_t)Y[j];
    float u = ldexpf((float)su, qy);
    bvec[p] = c * u;
  }
  /* Gram G = B_s^T D B_s */
  float G[ORC_MAXP][ORC_MAXP];
  int64_t sd = 0;
  for (int j = 0; j < C; ++j) sd += Dq[j];
  float gd = c2 * ldexpf((float)sd, qd);
  for (int p = 0; p < P; ++p) {
    G[p][p] = gd;
    for (int q = p + 1; q < P; ++q) {
      int64_t sv = 0;
      for (int j = 0; j < C; ++j)
        sv += (negmask[p * C + j] ^ negmask[q * C + j]) ? -(int64_t)Dq[j] : (int64_t)Dq[j];
      G[p][q] = G[q][p] = c2 * ldexpf((float)sv, qd);
    }
  }
  /* ridge (Eq. 3): A = G + eps I */
  float eps = prm->ridge_rel * gd;
  float A[ORC_MAXP][ORC_MAXP];
  for (int p = 0; p < P; ++p)
    for (int q = 0; q < P; ++q) A[p][q] = G[p][q];
  for (int p = 0; p < P; ++p) A[p][p] = gd + eps;

  /* LDL^T factorisation */
  float L[ORC_MAXP][ORC_MAXP], E[ORC_MAXP][ORC_MAXP], invD[ORC_MAXP];
  for (int k = 0; k < P; ++k) {
    for (int j = 0; j < k; ++j) {
      float v = A[k][j];
      for (int i = 0; i < j; ++i) v = fmaf(-L[k][i], E[j][i], v);
      E[k][j] = v;
      L[k][j] = v * invD[j];
    }
    float dk = A[k][k];
    for (int i = 0; i < k; ++i) dk = fmaf(-L[k][i], E[k][i], dk);
    if (!(dk > 0.0f && dk <= FLT_MAX)) return 0;
    invD[k] = 1.0f / dk;
  }
  /* solve A alpha = b */
  float z[ORC_MAXP], alpha[ORC_MAXP];
  for (int k = 0; k < P; ++k) {
    float v = bvec[k];
    for (int i = 0; i < k; ++i) v = fmaf(-L[k][i], z[i], v);
    z[k] = v;
  }
  for (int k = P - 1; k >= 0; --k) {
    float v = z[k] * invD[k];
    for (int i = k + 1; i < P; ++i) v = fmaf(-L[i][k], alpha[i], v);
    alpha[k] = v;
  }
  if (alpha_out)
    for (int p = 0; p < P; ++p) alpha_out[p] = alpha[p];

  /* coefficient-wise RTN with one scale per tile (Sec. 3.2) */
  float amax = 0.0f;
  for (int p = 0; p < P; ++p) {
    float a = fabsf(alpha[p]);
    if (a != a || a > amax) amax = a;
    if (amax != amax) break;
  }
  if (!(amax >= 0x1p-100f && amax <= 4294967296.0f)) return 0;
  float sc;
  int16_t scale_field;
  int codes[ORC_MAXP];
  if (prm->scale_mode == 0) {
    int lo, hi;
    orc_exp_range(prm, &lo, &hi);
    int e0 = ilogbf(amax) - (prm->b - 2);   /* ilogb(qmax) = b - 2 */
    int e = e0 + (amax > ldexpf((float)qmax, e0) ? 1 : 0);
    if (e < lo) e = lo;
    if (e > hi) e = hi;
    float inv = ldexpf(1.0f, -e);
    for (int p = 0; p < P; ++p) {
      float q = rintf(alpha[p] * inv);
      if (q > (float)qmax) q = (float)qmax;
      if (q < (float)-qmax) q = (float)-qmax;
      codes[p] = (int)q;
    }
    sc = ldexpf(1.0f, e);
    scale_field = (int16_t)e;
  } else {
    uint16_t h = orc_f32_to_f16(amax / (float)qmax);
    sc = orc_f16_to_f32(h);
    if (!(sc > 0.0f && sc <= FLT_MAX)) return 0;
    for (int p = 0; p < P; ++p) {
      float q = rintf(alpha[p] / sc);
      if (q > (float)qmax) q = (float)qmax;
      if (q < (float)-qmax) q = (float)-qmax;
      codes[p] = (int)q;
    }
    scale_field = (int16_t)h;
  }
  /* Eq. 4 gain: sum_j d_j [r_j^2 - (r_j - rhat_j)^2] = 2 ahat^T b - ahat^T G ahat */
  float Aq = 0.0f;
  for (int p = 0; p < P; ++p) Aq = fmaf((float)codes[p], bvec[p], Aq);
  float Qq = 0.0f;
  for (int p = 0; p < P; ++p) {
    Qq = fmaf((float)(codes[p] * codes[p]), G[p][p], Qq);
    for (int q = p + 1; q < P; ++q) Qq = fmaf((float)(2 * codes[p] * codes[q]), G[p][q], Qq);
  }
  float t = sc * Qq;
  float g = sc * (2.0f * Aq - t);
  *gain_out = g;
  *scale_out = scale_field;
  for (int p = 0; p < ORC_MAXP; ++p) codes_out[p] = (int8_t)(p < P ? codes[p] : 0);
  return 1;
}

/* Per-tile weights and residual (Sec. 3.2): U uses the activation diagonal,
 * shared by rows; PF blends it with the row-specific Fisher diagonal. */
static void orc_tile_inputs(const orc_params* prm, int64_t cols, const float* W, const float* W0,
                            const float* act, const float* fisher, float w_act, float w_fisher,
                            int64_t row, int64_t cb, float* r, float* d) {
  const int C = prm->C;
  for (int j = 0; j < C; ++j) {
    int64_t idx = row * cols + cb * C + j;
    r[j] = W[idx] - W0[idx];
    float a = act[cb * C + j];
    if (prm->variant == 0) d[j] = a;
    else d[j] = w_act * a + w_fisher * fisher[idx];
  }
}

/* Encode tiles [tile_begin, tile_end) of one module in spec mode: every seed,
 * keep the largest gain (ties: smallest seed). out is indexed from tile_begin.
 * masks: S*P*C bytes from orc_gen_basis (negmask per seed). */
void orc_encode_tiles(const orc_params* prm, int64_t rows, int64_t cols, const float* W,
                      const float* W0, const float* act, const float* fisher, float w_act,
                      float w_fisher, const uint8_t* masks, int64_t tile_begin, int64_t tile_end,
                      orc_candidate* out) {
  const int C = prm->C, P = prm->P;
  const int64_t n_cb = cols / C;
  (void)rows;
#pragma omp parallel for schedule(dynamic, 4)
  for (int64_t t = tile_begin; t < tile_end; ++t) {
    float r[256], d[256];
    orc_tile_inputs(prm, cols, W, W0, act, fisher, w_act, w_fisher, t / n_cb, t % n_cb, r, d);
    orc_candidate best;
    memset(&best, 0, sizeof best);
    best.gain = -INFINITY;
    if (orc_tile_valid(C, r, d)) {
      for (int s = 0; s < prm->S; ++s) {
        float g; int16_t sf; int8_t codes[8];
        if (!orc_score_candidate(prm, r, d, masks + (size_t)s * P * C, &g, &sf, codes, NULL)) continue;
        if (g > best.gain) {
          best.gain = g;
          best.seed = (uint16_t)s;
          best.scale = sf;
          memcpy(best.code, codes, 8);
        }
      }
    }
    out[t - tile_begin] = best;
  }
}

/* Same, for an explicit list of tile indices (sampled parity at full size). */
void orc_encode_tile_list(const orc_params* prm, int64_t rows, int64_t cols, const float* W,
                          const float* W0, const float* act, const float* fisher, float w_act,
                          float w_fisher, const uint8_t* masks, const int64_t* tiles, int64_t n,
                          orc_candidate* out) {
  (void)rows;
#pragma omp parallel for schedule(dynamic, 1)
  for (int64_t i = 0; i < n; ++i)
    orc_encode_tiles(prm, rows, cols, W, W0, act, fisher, w_act, w_fisher, masks, tiles[i],
                     tiles[i] + 1, out + i);
}

/* ------------------------------------------------------------------------ */
/* Definition mode (double)                                                 */
/* ------------------------------------------------------------------------ */

/* Eq. 3 by Gaussian elimination with partial pivoting on (B^T D B + eps I) a = B^T D r.
 * eps = ridge_rel * mean(d). Returns 0 if the system is singular. */
int orc_def_fit(int C, int P, double ridge_rel, const double* r, const double* d,
                const uint8_t* negmask, double* alpha) {
  double Bm[256][ORC_MAXP];
  double c = 1.0 / sqrt((double)C);
  for (int j = 0; j < C; ++j)
    for (int p = 0; p < P; ++p) Bm[j][p] = negmask[p * C + j] ? -c : c;
  double mean = 0.0;
  for (int j = 0; j < C; ++j) mean += d[j];
  mean /= C;
  double M[ORC_MAXP][ORC_MAXP + 1];
  for (int p = 0; p < P; ++p) {
    for (int q = 0; q < P; ++q) {
      double s = 0.0;
      for (int j = 0; j < C; ++j) s += Bm[j][p] * d[j] * Bm[j][q];
      M[p][q] = s + (p == q ? ridge_rel * mean : 0.0);
    }
    double s = 0.0;
    for (int j = 0; j < C; ++j) s += Bm[j][p] * d[j] * r[j];
    M[p][P] = s;
  }
  for (int k = 0; k < P; ++k) {
    int piv = k;
    for (int i = k + 1; i < P; ++i)
      if (fabs(M[i][k]) > fabs(M[piv][k])) piv = i;
    if (M[piv][k] == 0.0) return 0;
    if (piv != k)
      for (int q = 0; q <= P; ++q) { double t = M[k][q]; M[k][q] = M[piv][q]; M[piv][q] = t; }
    for (int i = k + 1; i < P; ++i) {
      double f = M[i][k] / M[k][k];
      for (int q = k; q <= P; ++q) M[i][q] -= f * M[k][q];
    }
  }
  for (int k = P - 1; k >= 0; --k) {
    double s = M[k][P];
    for (int q = k + 1; q < P; ++q) s -= M[k][q] * alpha[q];
    alpha[k] = s / M[k][k];
  }
  return 1;
}

/* Eq. 4 numerator evaluated directly: sum_j d_j [r_j^2 - (r_j - rhat_j)^2],
 * rhat = B_s * (codes * scale). */
double orc_def_gain(int C, int P, const double* r, const double* d, const uint8_t* negmask,
                    const int32_t* codes, double scale) {
  double c = 1.0 / sqrt((double)C);
  double g = 0.0;
  for (int j = 0; j < C; ++j) {
    double rh = 0.0;
    for (int p = 0; p < P; ++p) rh += (negmask[p * C + j] ? -c : c) * codes[p] * scale;
    double e = r[j] - rh;
    g += d[j] * (r[j] * r[j] - e * e);
  }
  return g;
}

/* ------------------------------------------------------------------------ */
/* Serialized rate (Sec. 3.4, Eq. 5)                                        */
/* ------------------------------------------------------------------------ */
static int orc_ceil_log2(uint64_t x) {  /* bits to index 0..x-1 */
  int n = 0;
  while (n < 64 && (1ULL << n) < x) ++n;
  return n;
}

int64_t orc_header_bytes(int32_t n_mod) { return 40 + 8 * (int64_t)n_mod; }

int64_t orc_record_bytes(const orc_params* prm, int64_t T) {
  int64_t bits = orc_ceil_log2((uint64_t)T) + orc_ceil_log2((uint64_t)prm->S) + prm->b_e +
                 (int64_t)prm->P * prm->b;
  return (bits + 7) / 8;
}

int64_t orc_budget_bytes(double rate_bpw, int64_t n_scope) {
  return (int64_t)floor(rate_bpw * (double)n_scope / 8.0);
}

static void orc_put_bits(uint8_t* rec, int* pos, uint64_t value, int nbits) {
  for (int k = 0; k < nbits; ++k, ++*pos)
    if ((value >> k) & 1u) rec[*pos / 8] |= (uint8_t)(1u << (*pos % 8));
}

static uint64_t orc_get_bits(const uint8_t* rec, int* pos, int nbits) {
  uint64_t v = 0;
  for (int k = 0; k < nbits; ++k, ++*pos)
    if ((rec[*pos / 8] >> (*pos % 8)) & 1u) v |= 1ULL << k;
  return v;
}

static void orc_put_le(uint8_t* p, uint64_t v, int n) {
  for (int i = 0; i < n; ++i) p[i] = (uint8_t)(v >> (8 * i));
}

/* One record: tile, seed, scale field, P codes — LSB-first, zero padded. */
void orc_pack_record(const orc_params* prm, int64_t T, int64_t tile, const orc_candidate* cd,
                     uint8_t* rec) {
  int64_t L = orc_record_bytes(prm, T);
  memset(rec, 0, (size_t)L);
  int pos = 0;
  orc_put_bits(rec, &pos, (uint64_t)tile, orc_ceil_log2((uint64_t)T));
  orc_put_bits(rec, &pos, cd->seed, orc_ceil_log2((uint64_t)prm->S));
  uint64_t sf;
  if (prm->scale_mode == 0) sf = (uint64_t)(int64_t)(cd->scale - prm->e_bias);
  else sf = (uint16_t)cd->scale;
  orc_put_bits(rec, &pos, sf & ((prm->b_e >= 64) ? ~0ULL : ((1ULL << prm->b_e) - 1)), prm->b_e);
  for (int p = 0; p < prm->P; ++p)
    orc_put_bits(rec, &pos, (uint64_t)(int64_t)cd->code[p] & ((1ULL << prm->b) - 1), prm->b);
}

static int64_t orc_sign_extend(uint64_t v, int bits) {
  if (bits == 0) return 0;
  uint64_t m = 1ULL << (bits - 1);
  return (int64_t)((v ^ m) - m);
}

void orc_unpack_record(const orc_params* prm, int64_t T, const uint8_t* rec, int64_t* tile,
                       orc_candidate* cd) {
  int pos = 0;
  memset(cd, 0, sizeof *cd);
  *tile = (int64_t)orc_get_bits(rec, &pos, orc_ceil_log2((uint64_t)T));
  cd->seed = (uint16_t)orc_get_bits(rec, &pos, orc_ceil_log2((uint64_t)prm->S));
  uint64_t sf = orc_get_bits(rec, &pos, prm->b_e);
  if (prm->scale_mode == 0) cd->scale = (int16_t)(orc_sign_extend(sf, prm->b_e) + prm->e_bias);
  else cd->scale = (int16_t)(uint16_t)sf;
  for (int p = 0; p < prm->P; ++p) cd->code[p] = (int8_t)orc_sign_extend(orc_get_bits(rec, &pos, prm->b), prm->b);
}

typedef struct { float gain; int64_t tile; } orc_key;

static int orc_key_cmp(const void* a, const void* b) {
  const orc_key* x = (const orc_key*)a;
  const orc_key* y = (const orc_key*)b;
  if (x->gain > y->gain) return -1;   /* rho = gain / L with one L: gain descending */
  if (x->gain < y->gain) return 1;
  return (x->tile > y->tile) - (x->tile < y->tile);  /* ties: tile ascending */
}

/*
 * Byte-aware allocation (Sec. 3.3) and serialisation (Sec. 3.4).
 * mod_tiles[m]: tiles of module m (concatenated in cands); mod_weights[m] = N_m.
 * U: one rate, per-module quotas; PF: global ranking, prefixes per rate.
 * stream: capacity bytes; counts: n_mod (U) or n_rates (PF); bytes_out: n_rates.
 * Returns 0 on success, 4 if a budget is below the header, 7 if capacity is short.
 */
int orc_select_records(const orc_params* prm, int32_t n_mod, const int64_t* mod_tiles,
                       const int64_t* mod_weights, const orc_candidate* cands,
                       const double* rates, int32_t n_rates, uint8_t* stream, int64_t capacity,
                       int64_t* counts, int64_t* bytes_out) {
  int64_t T = 0, Nscope = 0;
  for (int m = 0; m < n_mod; ++m) { T += mod_tiles[m]; Nscope += mod_weights[m]; }
  const int64_t h = orc_header_bytes(n_mod), L = orc_record_bytes(prm, T);
  orc_key* keys = (orc_key*)malloc(sizeof(orc_key) * (size_t)(T > 0 ? T : 1));
  int64_t* mod_K = (int64_t*)calloc((size_t)n_mod, sizeof(int64_t));
  int64_t K_stream = 0;
  int rc = 0;
  /* eligibility: non-positive (or non-finite) records are discarded (Sec. 3.3) */
  int64_t npos = 0;
  for (int64_t t = 0; t < T; ++t)
    if (cands[t].gain > 0.0f && cands[t].gain <= FLT_MAX) { keys[npos].gain = cands[t].gain; keys[npos].tile = t; ++npos; }
  int64_t* order = (int64_t*)malloc(sizeof(int64_t) * (size_t)(T > 0 ? T : 1));
  if (prm->variant == 0) {
    /* U: within each module, the best records that fit its quota */
    int64_t B = orc_budget_bytes(rates[0], Nscope);
    if (B < h) { rc = 4; goto done; }
    int64_t off = 0, kbeg = 0;
    for (int m = 0; m < n_mod; ++m) {
      int64_t kend = kbeg;
      while (kend < npos && keys[kend].tile < off + mod_tiles[m]) ++kend;
      qsort(keys + kbeg, (size_t)(kend - kbeg), sizeof(orc_key), orc_key_cmp);
      unsigned __int128 q = (unsigned __int128)(uint64_t)(B - h) * (uint64_t)mod_weights[m];
      int64_t quota = (int64_t)(q / (uint64_t)Nscope);
      int64_t K = quota / L;
      if (K > kend - kbeg) K = kend - kbeg;
      for (int64_t k = 0; k < K; ++k) order[K_stream++] = keys[kbeg + k].tile;
      mod_K[m] = K;
      counts[m] = K;
      off += mod_tiles[m];
      kbeg = kend;
    }
    bytes_out[0] = h + K_stream * L;
  } else {
    qsort(keys, (size_t)npos, sizeof(orc_key), orc_key_cmp);
    for (int r = 0; r < n_rates; ++r) {
      int64_t B = orc_budget_bytes(rates[r], Nscope);
      if (B < h) { rc = 4; goto done; }
      int64_t K = (B - h) / L;
      if (K > npos) K = npos;
      counts[r] = K;
      bytes_out[r] = h + K * L;
      if (K > K_stream) K_stream = K;
    }
    for (int64_t k = 0; k < K_stream; ++k) {
      order[k] = keys[k].tile;
      int64_t off = 0;
      for (int m = 0; m < n_mod; ++m) {
        if (order[k] < off + mod_tiles[m]) { mod_K[m]++; break; }
        off += mod_tiles[m];
      }
    }
  }
  if (h + K_stream * L > capacity) { rc = 7; goto done; }
  /* header */
  memset(stream, 0, (size_t)h);
  orc_put_le(stream + 0, 0x52535741u, 4);
  orc_put_le(stream + 4, 1, 2);
  stream[6] = (uint8_t)prm->variant;
  stream[7] = (uint8_t)prm->scale_mode;
  orc_put_le(stream + 8, (uint64_t)prm->C, 2);
  stream[10] = (uint8_t)prm->P;
  stream[11] = (uint8_t)prm->b;
  stream[12] = (uint8_t)prm->b_e;
  stream[13] = (uint8_t)(int8_t)prm->e_bias;
  stream[14] = (uint8_t)prm->permute;
  orc_put_le(stream + 16, (uint64_t)prm->S, 4);
  orc_put_le(stream + 20, (uint64_t)n_mod, 4);
  orc_put_le(stream + 24, prm->gen_seed, 8);
  orc_put_le(stream + 32, (uint64_t)K_stream, 8);
  for (int m = 0; m < n_mod; ++m) {
    orc_put_le(stream + 40 + 8 * m, (uint64_t)mod_tiles[m], 4);
    orc_put_le(stream + 44 + 8 * m, (uint64_t)mod_K[m], 4);
  }
  for (int64_t k = 0; k < K_stream; ++k)
    orc_pack_record(prm, T, order[k], &cands[order[k]], stream + h + k * L);
done:
  free(keys);
  free(order);
  free(mod_K);
  return rc;
}

/* ------------------------------------------------------------------------ */
/* Decoder (Sec. 3.2): regenerate B_s alpha_hat for each record and add it   */
/* to W0; tiles without a record keep W0.                                    */
/* W0 and out are float arrays of each module; out must hold a copy of W0.   */
/* out_bf16 != 0: each element is then rounded to bfloat16 (stored widened). */
/* ------------------------------------------------------------------------ */
int orc_decode_apply(const orc_params* prm, int32_t n_mod, const int64_t* mod_rows,
                     const int64_t* mod_cols, const uint8_t* stream, int64_t K,
                     float* const* out, int out_bf16) {
  const int C = prm->C, P = prm->P;
  int64_t T = 0;
  for (int m = 0; m < n_mod; ++m) T += mod_rows[m] * mod_cols[m] / C;
  const int64_t h = orc_header_bytes(n_mod), L = orc_record_bytes(prm, T);
  const float c = (float)(1.0 / sqrt((double)C));
  uint8_t sign[256], neg[8 * 256];
  int32_t perm[256], cols[8];
  int bad = 0;
  for (int64_t k = 0; k < K; ++k) {
    int64_t tile;
    orc_candidate cd;
    orc_unpack_record(prm, T, stream + h + k * L, &tile, &cd);
    if (tile >= T || cd.seed >= prm->S) { bad = 1; continue; }
    int64_t m = 0, off = 0;
    while (tile >= off + mod_rows[m] * mod_cols[m] / C) { off += mod_rows[m] * mod_cols[m] / C; ++m; }
    int64_t lt = tile - off, n_cb = mod_cols[m] / C;
    int64_t base = (lt / n_cb) * mod_cols[m] + (lt % n_cb) * C;
    orc_gen_basis(prm->gen_seed, cd.seed, C, P, prm->permute, sign, perm, cols, neg);
    float sc = prm->scale_mode == 0 ? ldexpf(1.0f, cd.scale) : orc_f16_to_f32((uint16_t)cd.scale);
    for (int j = 0; j < C; ++j) {
      int kj = 0;
      for (int p = 0; p < P; ++p) kj += neg[p * C + j] ? -cd.code[p] : cd.code[p];
      float rh = ((float)kj * c) * sc;
      out[m][base + j] = out[m][base + j] + rh;
    }
  }
  if (out_bf16) {
    for (int m = 0; m < n_mod; ++m)
      for (int64_t i = 0; i < mod_rows[m] * mod_cols[m]; ++i)
        out[m][i] = orc_u2f((uint32_t)orc_f32_to_bf16(out[m][i]) << 16);
  }
  return bad;
}

/* ------------------------------------------------------------------------ */
/* RTN-INT4 backbone (Eq. 1's W0 = Q(W); Sec. 4: round to nearest, groups of */
/* `group` consecutive input coordinates of a row) and scale double          */
/* quantisation (SDQ, Sec. 3.3: the group scales are themselves quantised,   */
/* after QLoRA's double quantisation; the paper gives no format):            */
/*  first level, group g (groups are consecutive runs since cols % group ==  */
/*  0): s_g = binary16(max|w| / 7); q = clamp(rint(w / s_g), -8, 7), q = 0    */
/*  when s_g == 0;                                                            */
/*  second level (sdq != 0), per block of `block` consecutive groups:        */
/*  mu = binary32((sum of the block's s_g, exact in double) / n), d = s_g -   */
/*  mu, a = max|d|, step = a / 127, c_g = clamp(rint(d / step), -127, 127)   */
/*  (0 when step == 0), s~_g = mu + c_g * step (two roundings);              */
/*  W0 = q * s_eff in binary32, s_eff = s_g, or s~_g with SDQ.               */
/* Outputs: q (rows*cols), s16 (G), c8 and consts (mu, step per block; SDQ   */
/* only), s_eff (G), W0 (rows*cols).                                         */
/* ------------------------------------------------------------------------ */
void orc_rtn_quantize(int64_t rows, int64_t cols, int group, int sdq, int block, const float* W, int8_t* q,
                      uint16_t* s16, int8_t* c8, float* consts, float* s_eff, float* W0) {
  const int64_t G = rows * cols / group;
  for (int64_t g = 0; g < G; ++g) {
    const float* w = W + g * group;
    float amax = 0.0f;
    for (int j = 0; j < group; ++j) {
      const float a = fabsf(w[j]);
      if (a > amax) amax = a;
    }
    const uint16_t h = orc_f32_to_f16(amax / 7.0f);
    s16[g] = h;
    const float s = orc_f16_to_f32(h);
    for (int j = 0; j < group; ++j) {
      float v = 0.0f;
      if (s > 0.0f) {
        v = rintf(w[j] / s);
        if (v < -8.0f) v = -8.0f;
        if (v > 7.0f) v = 7.0f;
      }
      q[g * group + j] = (int8_t)v;
    }
    s_eff[g] = s;
  }
  if (sdq) {
    for (int64_t b0 = 0; b0 < G; b0 += block) {
      const int64_t n = G - b0 < block ? G - b0 : block;
      double sum = 0.0;
      for (int64_t g = b0; g < b0 + n; ++g) sum += (double)s_eff[g];
      const float mu = (float)(sum / (double)n);
      float a = 0.0f;
      for (int64_t g = b0; g < b0 + n; ++g) {
        const float d = fabsf(s_eff[g] - mu);
        if (d > a) a = d;
      }
      const float step = a / 127.0f;
      consts[2 * (b0 / block)] = mu;
      consts[2 * (b0 / block) + 1] = step;
      for (int64_t g = b0; g < b0 + n; ++g) {
        float cv = 0.0f;
        if (step > 0.0f) {
          cv = rintf((s_eff[g] - mu) / step);
          if (cv < -127.0f) cv = -127.0f;
          if (cv > 127.0f) cv = 127.0f;
        }
        c8[g] = (int8_t)cv;
        s_eff[g] = mu + cv * step;
      }
    }
  }
  for (int64_t i = 0; i < rows * cols; ++i) W0[i] = (float)q[i] * s_eff[i / group];
}

/* ------------------------------------------------------------------------ */
/* Definition of the packed product (the decoded weights applied to x        */
/* without forming them) for module m of a stream over n_mod modules:        */
/* y[v][i] = sum_j (W0_ij + r_ij) x[v][j] in double, W0_ij = q_ij * s_eff    */
/* (the backbone's binary32 value), r the decoder's residual (Sec. 3.2) on    */
/* the module's tiles named by the first K records, in double:                */
/* k_j * C^-1/2 * scale. yabs = sum_j (|W0_ij x[v][j]| + |r_ij x[v][j]|),    */
/* the magnitude a binary32 evaluation that sums the backbone's and the      */
/* residual's terms separately is rounded against. x: M x cols, y and yabs:  */
/* M x rows.                                                                  */
/* ------------------------------------------------------------------------ */
int orc_packed_gemv(const orc_params* prm, int32_t n_mod, const int64_t* mod_rows, const int64_t* mod_cols,
                    int32_t m, int group, const int8_t* q, const float* s_eff, const uint8_t* stream, int64_t K,
                    int M, const float* x, double* y, double* yabs) {
  const int C = prm->C, P = prm->P;
  int64_t T = 0, off = 0;
  for (int i = 0; i < n_mod; ++i) {
    if (i == m) off = T;
    T += mod_rows[i] * mod_cols[i] / C;
  }
  const int64_t rows = mod_rows[m], cols = mod_cols[m], Tm = rows * cols / C, n_cb = cols / C;
  const int64_t h = orc_header_bytes(n_mod), L = orc_record_bytes(prm, T);
  double* Wt = (double*)malloc(sizeof(double) * (size_t)(rows * cols));
  double* Rt = (double*)calloc((size_t)(rows * cols), sizeof(double));
  if (!Wt || !Rt) {
    free(Wt);
    free(Rt);
    return -1;
  }
  for (int64_t i = 0; i < rows * cols; ++i) Wt[i] = (double)((float)q[i] * s_eff[i / group]);
  const double c = 1.0 / sqrt((double)C);
  uint8_t sign[256], neg[8 * 256];
  int32_t perm[256], colsel[8];
  int bad = 0;
  for (int64_t k = 0; k < K; ++k) {
    int64_t tile;
    orc_candidate cd;
    orc_unpack_record(prm, T, stream + h + k * L, &tile, &cd);
    if (tile >= T || cd.seed >= prm->S) { bad = 1; continue; }
    if (tile < off || tile >= off + Tm) continue;  /* another module's record */
    const int64_t lt = tile - off;
    const int64_t base = (lt / n_cb) * cols + (lt % n_cb) * C;
    orc_gen_basis(prm->gen_seed, cd.seed, C, P, prm->permute, sign, perm, colsel, neg);
    const double sc = prm->scale_mode == 0 ? ldexp(1.0, cd.scale) : (double)orc_f16_to_f32((uint16_t)cd.scale);
    for (int j = 0; j < C; ++j) {
      int kj = 0;
      for (int p = 0; p < P; ++p) kj += neg[p * C + j] ? -cd.code[p] : cd.code[p];
      Rt[base + j] = (double)kj * c * sc;  /* a later record of the tile replaces it */
    }
  }
  for (int v = 0; v < M; ++v)
    for (int64_t i = 0; i < rows; ++i) {
      double acc = 0.0, aabs = 0.0;
      for (int64_t j = 0; j < cols; ++j) {
        const double xj = (double)x[(int64_t)v * cols + j];
        acc += (Wt[i * cols + j] + Rt[i * cols + j]) * xj;
        aabs += fabs(Wt[i * cols + j] * xj) + fabs(Rt[i * cols + j] * xj);
      }
      y[(int64_t)v * rows + i] = acc;
      yabs[(int64_t)v * rows + i] = aabs;
    }
  free(Wt);
  free(Rt);
  return bad;
}
