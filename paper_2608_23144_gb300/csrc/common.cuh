// common.cuh — device-side building blocks shared by the AWSRC kernels:
// the shared basis generator (Sec. 3.1, Eq. 2), the binary32 fit / quantise /
// gain epilogue (Eq. 3, Sec. 3.2, Eq. 4) and small launch descriptors.
//
// Every floating-point operation that decides an integer output is written
// with an explicit round-to-nearest intrinsic (__fmaf_rn, __fmul_rn, ...), and
// the library is compiled with --fmad=false, so the compiler cannot fuse or
// reorder them: the order is the one the public header fixes.
#pragma once

#include <cstdint>
#include <cuda_bf16.h>
#include <cuda_fp16.h>
#include <cuda_runtime.h>

#include "awsrc.h"

namespace awsrc {

constexpr int kMaxP = 8;
constexpr int kMaxC = 256;
constexpr int kMaxModsPerLaunch = 16;

// Fault bits of the device status word kept at the start of every workspace.
constexpr uint32_t kFaultRecord = 1u;     // decoder: record names a tile/seed out of range
constexpr uint32_t kFaultSelfCheck = 2u;  // encoder: the winner's recomputation disagrees with the search
constexpr uint32_t kFaultTimeout = 4u;    // a bounded wait gave up
constexpr size_t kStatusBytes = 256;

// Host-validated parameters plus derived constants, passed by value.
struct Prm {
  int C, P, b, S, b_e, e_bias, scale_mode, permute, variant;
  float ridge_rel;
  uint64_t gen_seed;
  int qmax;       // 2^(b-1) - 1
  float qmaxf;
  int e_lo, e_hi; // POW2 exponent range, within [-126, 126]
  float c;        // RN(C^-1/2)
  float c2;       // 1/C (exact)
  int W;          // 64-bit mask words per (seed, atom)
  int S_pad;      // seeds rounded up to the search chunk
  int logC;       // log2(C)
  int fast_pow2;  // POW2 scale whose exponent range can never bind for a valid candidate
  uint32_t mant_q;  // mantissa field of (float)qmax
  int prune;        // 1: the C = 64, P = 4 U search skips candidates its bound rules out
  int stall_chunk;  // test of the bounded waits: the U search's producer issues no copies from
                    // this chunk of its block's range on (-1: never)
  uint64_t wait_ns; // limit of every bounded wait inside a kernel (2 s)
};

constexpr uint64_t kWaitLimitNs = 2000000000ull;

// ---------------------------------------------------------------- generator --
// SplitMix64 (Steele, Lea & Flood 2014): n-th output of the stream at state x.
__host__ __device__ __forceinline__ uint64_t sm64_output(uint64_t x, uint64_t n) {
  uint64_t z = x + n * 0x9E3779B97F4A7C15ull;
  z = (z ^ (z >> 30)) * 0xBF58476D1CE4E5B9ull;
  z = (z ^ (z >> 27)) * 0x94D049BB133111EBull;
  return z ^ (z >> 31);
}

// --------------------------------------------------------------- numerics --
__device__ __forceinline__ float sign_f(uint64_t bit) {  // bit 1 -> -1.0f, 0 -> +1.0f
  return __int_as_float(0x3f800000u | ((uint32_t)(bit & 1u) << 31));
}

// max with NaN propagation (PTX max.NaN.f32)
__device__ __forceinline__ float fmax_nan(float a, float b) {
  float r;
  asm("max.NaN.f32 %0, %1, %2;" : "=f"(r) : "f"(a), "f"(b));
  return r;
}

__device__ __forceinline__ float load_elem(const void* p, int64_t i, int dtype) {
  if (dtype == AWSRC_DTYPE_F32) return static_cast<const float*>(p)[i];
  return __bfloat162float(static_cast<const __nv_bfloat16*>(p)[i]);
}

// Per-tile fixed point of the correlations: for m = max_j |x_j| >= 2^-100,
// q = ilogb(m) - 20, and x_j is represented by X_j = rint(x_j * 2^-q), |X_j| <= 2^21.
// Smaller (or NaN) m: the vector counts as zero (q = 0). Returns 2^-q, or 0 for a
// zero vector; *q receives q.
__device__ __forceinline__ float fixed_point_inv(float m, int* q) {
  if (!(m >= 0x1p-100f)) {
    *q = 0;
    return 0.0f;
  }
  const int e = (int)((__float_as_uint(m) >> 23) & 0xffu) - 127;  // m is normal here
  const int qq = min(e, 126) - 20;
  *q = qq;
  return __int_as_float((127 - qq) << 23);
}

__device__ __forceinline__ float pow2f(int q) { return __int_as_float((127 + q) << 23); }

// X = rint(x * inv), exact scaling then round half to even.
__device__ __forceinline__ int fixed_point_int(float x, float inv) {
  return __float2int_rn(__fmul_rn(x, inv));
}

// Tile-domain check: |r| <= 2^16 and 0 <= d <= 2^32 (NaN fails both).
__device__ __forceinline__ bool in_domain(float r, float d) {
  return (fabsf(r) <= 65536.0f) && (d >= 0.0f) && (d <= 4294967296.0f);
}

// Packed strict-lower-triangle index of (k, i), k > i.
__host__ __device__ constexpr int tri(int k, int i) { return k * (k - 1) / 2 + i; }

// Floats per (column block, seed) entry of the U Gram table:
// L (P(P-1)/2), invD (P), G off-diagonal (P(P-1)/2), gd (1), padded to 4.
__host__ __device__ constexpr int gram_stride(int P) {
  return ((P * (P - 1) + P + 1) + 3) / 4 * 4;
}

// float2 entries per (column block, seed pair) of the paired table the C = 64,
// P = 4 search streams: -L, invD rounded up after multiplying by the seed's
// pruning-bound multiplier (used only by the bound), invD, G off-diagonal
// (2*G_pq on the fast power-of-two path), gd, zero padding to an even count;
// seed 2i in component x and seed 2i+1 in y.
__host__ __device__ constexpr int pair_stride(int P) {
  return ((P * (P - 1) + 2 * P + 1) + 1) / 2 * 2;
}

// Correctly rounded binary32 reciprocal, as __frcp_rn, cheaper on the range
// the LDL^T pivots live in. For positive normal x in [2^-125, 2^125) the
// hardware approximation y (rcp.approx, within one ulp) is corrected once,
// y + y (1 - x y) with both steps fused (Markstein's final correction: P.
// Markstein, "Computation of elementary functions on the IBM RISC System/6000
// processor", IBM J. Res. Dev. 34(1), 1990): 1 - x y is exact and the fused
// update rounds the corrected value once. Every other input takes __frcp_rn.
// The fast path equals __frcp_rn on every float of its range, checked
// exhaustively on the GPU (awsrc_verify_reciprocal).
__device__ __forceinline__ float rcp_rn(float x) {
  const uint32_t b = __float_as_uint(x);
  if (b - 0x01000000u < 0x7D000000u - 0x01000000u) {
    float y;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(y) : "f"(x));
    return __fmaf_rn(y, __fmaf_rn(-x, y, 1.0f), y);
  }
  return __frcp_rn(x);
}

// LDL^T of A = G + eps I with G_pp = gd, G_pq = Goff[tri(q, p)]. Writes L and
// invD; returns false if some pivot is not in (0, FLT_MAX].
template <int P>
__device__ __forceinline__ bool ldl_factor(float gd, float eps, const float* Goff, float* L,
                                           float* invD) {
  float E[P * (P - 1) / 2 + 1];
  bool ok = true;
  const float diag = __fadd_rn(gd, eps);
#pragma unroll
  for (int k = 0; k < P; ++k) {
#pragma unroll
    for (int j = 0; j < k; ++j) {
      float v = Goff[tri(k, j)];
#pragma unroll
      for (int i = 0; i < j; ++i) v = __fmaf_rn(-L[tri(k, i)], E[tri(j, i)], v);
      E[tri(k, j)] = v;
      L[tri(k, j)] = __fmul_rn(v, invD[j]);
    }
    float dk = diag;
#pragma unroll
    for (int i = 0; i < k; ++i) dk = __fmaf_rn(-L[tri(k, i)], E[tri(k, i)], dk);
    ok = ok && (dk > 0.0f) && (dk <= 3.402823466e38f);
    invD[k] = rcp_rn(dk);
  }
  return ok;
}

// Solve (L D L^T) alpha = b.
template <int P>
__device__ __forceinline__ void ldl_solve(const float* L, const float* invD, const float* bv,
                                          float* alpha) {
  float z[P];
#pragma unroll
  for (int k = 0; k < P; ++k) {
    float v = bv[k];
#pragma unroll
    for (int i = 0; i < k; ++i) v = __fmaf_rn(-L[tri(k, i)], z[i], v);
    z[k] = v;
  }
#pragma unroll
  for (int k = P - 1; k >= 0; --k) {
    float v = __fmul_rn(z[k], invD[k]);
#pragma unroll
    for (int i = k + 1; i < P; ++i) v = __fmaf_rn(-L[tri(i, k)], alpha[i], v);
    alpha[k] = v;
  }
}

// Quantise alpha (Sec. 3.2) and return the Eq. 4 gain with the unregularised
// Gram; -inf when the candidate is invalid. q receives the codes as floats and
// *sf the scale field (exponent or binary16 bits).
template <int P>
__device__ __forceinline__ float quant_gain(const Prm& pr, const float* alpha, const float* bv,
                                            float gd, const float* Goff, float* q, int* sf) {
  float amax = fabsf(alpha[0]);
#pragma unroll
  for (int p = 1; p < P; ++p) amax = fmax_nan(amax, fabsf(alpha[p]));
  bool ok = (amax >= 0x1p-100f) && (amax <= 4294967296.0f);
  float sc;
  if (pr.scale_mode == AWSRC_SCALE_POW2) {
    const int E = (int)((__float_as_uint(amax) >> 23) & 0xffu) - 127;
    const int e0 = E - (pr.b - 2);  // ilogb(qmax) = b - 2
    const int e0c = min(max(e0, -126), 126);
    const float thr = __fmul_rn(pr.qmaxf, __int_as_float((e0c + 127) << 23));
    int e = e0 + (amax > thr ? 1 : 0);
    e = min(max(e, pr.e_lo), pr.e_hi);
    sc = __int_as_float((e + 127) << 23);
    const float inv = __int_as_float((127 - e) << 23);
#pragma unroll
    for (int p = 0; p < P; ++p) {
      float x = __fmul_rn(alpha[p], inv);
      x = fminf(fmaxf(x, -pr.qmaxf), pr.qmaxf);
      q[p] = __fsub_rn(__fadd_rn(x, 12582912.0f), 12582912.0f);  // RNE to integer
    }
    *sf = e;
  } else {
    const __half h = __float2half_rn(__fdiv_rn(amax, pr.qmaxf));
    sc = __half2float(h);
    ok = ok && (sc > 0.0f) && (sc <= 3.402823466e38f);
#pragma unroll
    for (int p = 0; p < P; ++p) {
      float x = __fdiv_rn(alpha[p], sc);
      x = fminf(fmaxf(x, -pr.qmaxf), pr.qmaxf);
      q[p] = __fsub_rn(__fadd_rn(x, 12582912.0f), 12582912.0f);
    }
    *sf = (int)(int16_t)__half_as_ushort(h);
  }
  float Aq = 0.0f;
#pragma unroll
  for (int p = 0; p < P; ++p) Aq = __fmaf_rn(q[p], bv[p], Aq);
  float Qq = 0.0f;
#pragma unroll
  for (int p = 0; p < P; ++p) {
    Qq = __fmaf_rn(__fmul_rn(q[p], q[p]), gd, Qq);
#pragma unroll
    for (int r = p + 1; r < P; ++r)
      Qq = __fmaf_rn(__fmul_rn(__fmul_rn(2.0f, q[p]), q[r]), Goff[tri(r, p)], Qq);
  }
  const float t = __fmul_rn(sc, Qq);
  const float g = __fmul_rn(sc, __fsub_rn(__fmul_rn(2.0f, Aq), t));
  return ok ? g : -__int_as_float(0x7f800000);
}

// The POW2 branch of quant_gain when the exponent range never binds (fast_pow2):
// the same results with integer work on the bit pattern of amax. For a valid
// candidate amax = f_a*2^E is normal and the smallest e with amax <= qmax*2^e is
// E - ilogb(qmax) + [f_a > f_qmax] (compare mantissa fields); |alpha_p|*2^-e then
// never exceeds qmax, so the code clamps are no-ops and are left out. Goff2
// holds 2*G_pq (exact), which gives the same fma as (2*code_p*code_q)*G_pq
// because the fused product is exact.
template <int P>
__device__ __forceinline__ float quant_gain_fast(const Prm& pr, const float* alpha, const float* bv,
                                                 float gd, const float* Goff2, float* q, int* e_out) {
  float amax = fabsf(alpha[0]);
#pragma unroll
  for (int p = 1; p < P; ++p) amax = fmax_nan(amax, fabsf(alpha[p]));
  const uint32_t ab = __float_as_uint(amax);
  // 2^-100 <= amax <= 2^32 (NaN and inf fail: their bit patterns lie above)
  const bool ok = (ab - 0x0D800000u) <= (0x4F800000u - 0x0D800000u);
  const uint32_t sc_bits = (ab & 0x7F800000u) - ((uint32_t)(pr.b - 2) << 23) +
                           (((ab & 0x007FFFFFu) > pr.mant_q) ? 0x00800000u : 0u);
  const float sc = __uint_as_float(sc_bits);
  const float inv = __uint_as_float(0x7F000000u - sc_bits);
#pragma unroll
  for (int p = 0; p < P; ++p)
    q[p] = __fsub_rn(__fadd_rn(__fmul_rn(alpha[p], inv), 12582912.0f), 12582912.0f);
  *e_out = (int)(sc_bits >> 23) - 127;
  float Aq = 0.0f;
#pragma unroll
  for (int p = 0; p < P; ++p) Aq = __fmaf_rn(q[p], bv[p], Aq);
  float Qq = 0.0f;
#pragma unroll
  for (int p = 0; p < P; ++p) {
    Qq = __fmaf_rn(__fmul_rn(q[p], q[p]), gd, Qq);
#pragma unroll
    for (int r = p + 1; r < P; ++r) Qq = __fmaf_rn(__fmul_rn(q[p], q[r]), Goff2[tri(r, p)], Qq);
  }
  const float t = __fmul_rn(sc, Qq);
  const float g = __fmul_rn(sc, __fmaf_rn(2.0f, Aq, -t));
  return ok ? g : -__int_as_float(0x7f800000);
}

// ------------------------------------------------------- paired epilogue --
// The same solve and power-of-two quantiser for two candidates at once, one per
// component of a float2, on the packed binary32 instructions of sm_100-class
// GPUs (__ffma2_rn, __fmul2_rn, __fadd2_rn round each component exactly like
// their scalar forms). nL holds -L (exact), so every step is one packed fma.
template <int P>
__device__ __forceinline__ void ldl_solve2(const float2* nL, const float2* invD, const float2* bv,
                                           float2* alpha) {
  float2 z[P];
#pragma unroll
  for (int k = 0; k < P; ++k) {
    float2 v = bv[k];
#pragma unroll
    for (int i = 0; i < k; ++i) v = __ffma2_rn(nL[tri(k, i)], z[i], v);
    z[k] = v;
  }
#pragma unroll
  for (int k = P - 1; k >= 0; --k) {
    float2 v = __fmul2_rn(z[k], invD[k]);
#pragma unroll
    for (int i = k + 1; i < P; ++i) v = __ffma2_rn(nL[tri(i, k)], alpha[i], v);
    alpha[k] = v;
  }
}

// Scale bits 2^e of a candidate for quant_gain_fast2 from amax's bits ab,
// valid when ab is in range (amax in [2^-100, 2^32]; inf and NaN patterns are
// not): adding 0x7FFFFF - mant_q carries into the exponent field exactly when
// the mantissa field of amax exceeds that of qmax, which is the
// [f_a > f_qmax] step of quant_gain_fast.
__device__ __forceinline__ bool fast_scale_in_range(uint32_t ab) {
  return (ab - 0x0D800000u) <= (0x4F800000u - 0x0D800000u);
}
__device__ __forceinline__ uint32_t fast_scale_bits(const Prm& pr, uint32_t ab) {
  return ((ab + (0x007FFFFFu - pr.mant_q)) & 0x7F800000u) - ((uint32_t)(pr.b - 2) << 23);
}

// quant_gain_fast on two candidates. Each code is RN(alpha*2^-e + 1.5*2^23) -
// 1.5*2^23 with the product fused: alpha*2^-e is exact whenever it can reach
// a rounding boundary, so this is the code of the scalar form. -t is formed as
// (-sc)*Qq, the exact negation of sc*Qq. amax ignores NaN: a candidate with a
// NaN coefficient but a valid amax gets a NaN gain (its code and Aq are NaN),
// which no comparison of the seed argmax accepts, just as it accepts no -inf.
template <int P>
__device__ __forceinline__ float2 quant_gain_fast2(const Prm& pr, const float2* alpha, const float2* bv,
                                                   float2 gd, const float2* Goff2) {
  float m0 = fabsf(alpha[0].x), m1 = fabsf(alpha[0].y);
#pragma unroll
  for (int p = 1; p < P; ++p) {
    m0 = fmaxf(m0, fabsf(alpha[p].x));
    m1 = fmaxf(m1, fabsf(alpha[p].y));
  }
  // an amax out of range gets a gain of -inf below, whatever its bits give
  const uint32_t ab0 = __float_as_uint(m0), ab1 = __float_as_uint(m1);
  const bool in0 = fast_scale_in_range(ab0), in1 = fast_scale_in_range(ab1);
  const uint32_t s0 = fast_scale_bits(pr, ab0), s1 = fast_scale_bits(pr, ab1);
  const float2 sc = make_float2(__uint_as_float(s0), __uint_as_float(s1));
  const float2 nsc = make_float2(__uint_as_float(s0 | 0x80000000u), __uint_as_float(s1 | 0x80000000u));
  const float2 inv = make_float2(__uint_as_float(0x7F000000u - s0), __uint_as_float(0x7F000000u - s1));
  const float2 magic = make_float2(12582912.0f, 12582912.0f);
  const float2 nmagic = make_float2(-12582912.0f, -12582912.0f);
  float2 q[P];
#pragma unroll
  for (int p = 0; p < P; ++p) q[p] = __fadd2_rn(__ffma2_rn(alpha[p], inv, magic), nmagic);
  float2 Aq = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int p = 0; p < P; ++p) Aq = __ffma2_rn(q[p], bv[p], Aq);
  float2 Qq = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int p = 0; p < P; ++p) {
    Qq = __ffma2_rn(__fmul2_rn(q[p], q[p]), gd, Qq);
#pragma unroll
    for (int r = p + 1; r < P; ++r) Qq = __ffma2_rn(__fmul2_rn(q[p], q[r]), Goff2[tri(r, p)], Qq);
  }
  const float2 tn = __fmul2_rn(nsc, Qq);
  float2 g = __fmul2_rn(sc, __ffma2_rn(make_float2(2.0f, 2.0f), Aq, tn));
  if (!in0) g.x = -__int_as_float(0x7f800000);
  if (!in1) g.y = -__int_as_float(0x7f800000);
  return g;
}

// Candidate comparison of the seed argmax: larger gain wins, equal gains keep
// the smaller selector.
__device__ __forceinline__ bool better(float g, uint32_t s, float bg, uint32_t bs) {
  return g > bg || (g == bg && s < bs);
}

// ------------------------------------------------------------- descriptors --
struct ModDesc {
  const void* W;
  const void* W0;
  const float* act;
  const float* fisher;
  int64_t rows, cols, n_cb, n_rb;
  int64_t tile_off;   // first global tile of the module
  int64_t gram_off;   // U: first Gram-table entry of the module ([cb][S_pad])
  int64_t block_off;  // first block of the module in the launch
  int32_t w_dtype, w0_dtype, nsplit, pad_;
  float w_act, w_fisher;
};

struct LaunchDesc {
  int n;
  int64_t T;          // tiles in the whole call (partials stride)
  ModDesc m[kMaxModsPerLaunch];
};

__device__ __forceinline__ int find_mod(const LaunchDesc& ld, int64_t block) {
  int mi = 0;
  for (int i = 1; i < ld.n; ++i)
    if (block >= ld.m[i].block_off) mi = i;
  return mi;
}

}  // namespace awsrc
