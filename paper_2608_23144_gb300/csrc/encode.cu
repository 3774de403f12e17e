// encode.cu — the seed search of Sec. 3.2 for any supported (C, P) and both
// variants, plus the two kernels around every search:
//
//  gram_u      U only. The activation diagonal is shared by all rows of a module
//              (Sec. 3.2), so the Gram matrix B_s^T D B_s of Eq. 3 and its LDL^T
//              depend on (column block, seed) only. They are computed once per
//              (cb, s) and reused by every row.
//  search      per (tile, seed): correlation b = B_s^T D r, solve, quantise,
//              gain; running argmax over the seeds of one split.
//  finalize    per tile: argmax over splits, then recomputation of the winning
//              seed's codes and scale with the same operations; the recomputed
//              gain must equal the searched one bit for bit (self-check bit).
#include <cfloat>

#include "internal.h"

namespace awsrc {

namespace {

constexpr int kGenRows = 32;      // rows per block of the generic search
constexpr int kGenLanes = 8;      // seed lanes per row
constexpr int kGenThreads = kGenRows * kGenLanes;

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

// ------------------------------------------------------------- seed bound --
// Multiplier m of the search's pruning bound for one (column block, seed).
//
// For any coefficients x, the Eq. 4 gain 2x^T b - x^T G x is at most
// U_G = b^T G^-1 b (its maximum over x), so the quantised gain of a candidate
// can never exceed U_G. The search computes U = b^T alpha with alpha from the
// ridge solve, i.e. U_eps = b^T (G + eps I)^-1 b up to rounding, and
// U_G <= (1 + eps/lambda_min) U_eps <= (1 + eps tr(G^-1)) U_eps. With
// kappa = tr(G) tr(G^-1) >= cond(G + eps I), the binary32 errors of the
// solve, of b^T alpha and of the gain itself are each below a small multiple
// of kappa*2^-24 relative to U (plus a few ulps), far inside the factor
// 1 + 2^-10 + 2^-14 kappa. So a candidate with U * m < g_best cannot score
// above g_best. m is +inf (no pruning) when G is not positive definite in
// double precision or kappa > 2^16. Computed in double and rounded up.
template <int P>
__device__ float bound_multiplier(float gd, const float* Goff, float eps) {
  // LDL^T of G in double; tr(G^-1) = sum_k |row k of L^-1|^2 / D_k
  double L[P][P], d[P], inv_d[P];
#pragma unroll
  for (int k = 0; k < P; ++k) {
    double dk = gd;
#pragma unroll
    for (int i = 0; i < k; ++i) dk -= L[k][i] * L[k][i] * d[i];
    if (!(dk > 0.0)) return __int_as_float(0x7f800000);
    d[k] = dk;
    inv_d[k] = 1.0 / dk;
#pragma unroll
    for (int j = k + 1; j < P; ++j) {
      double v = Goff[tri(j, k)];
#pragma unroll
      for (int i = 0; i < k; ++i) v -= L[j][i] * L[k][i] * d[i];
      L[j][k] = v * inv_d[k];
    }
  }
  double tr_inv = 0.0;
#pragma unroll
  for (int i = 0; i < P; ++i) {  // column i of X = L^-1, rows k >= i
    double x[P];
    x[i] = 1.0;
    tr_inv += inv_d[i];
#pragma unroll
    for (int k = i + 1; k < P; ++k) {
      double v = 0.0;
#pragma unroll
      for (int j = i; j < k; ++j) v -= L[k][j] * x[j];
      x[k] = v;
      tr_inv += v * v * inv_d[k];
    }
  }
  const double kappa = (double)P * gd * tr_inv;
  if (!(kappa <= 65536.0)) return __int_as_float(0x7f800000);
  const double m = (1.0 + (double)eps * tr_inv) * (1.0 + 0x1p-10 + 0x1p-14 * kappa);
  return __double2float_ru(m);
}

// ----------------------------------------------------------------- gram_u --
template <int P>
__global__ void __launch_bounds__(128) gram_u_kernel(Prm pr, LaunchDesc ld,
                                                     const uint64_t* __restrict__ masks,
                                                     float* __restrict__ gram,
                                                     float2* __restrict__ pairs) {
  // blockIdx.y enumerates the column blocks of all modules of the launch
  int mi = 0;
  int64_t cb = blockIdx.y;
  while (mi < ld.n - 1 && cb >= ld.m[mi].n_cb) { cb -= ld.m[mi].n_cb; ++mi; }
  const ModDesc& md = ld.m[mi];
  const int C = pr.C;
  __shared__ float d[kMaxC];
  __shared__ int Dq[kMaxC];
  __shared__ int dok;
  __shared__ float dmax;
  __shared__ float two_qd;
  if (threadIdx.x == 0) dok = 1;
  __syncthreads();
  for (int j = threadIdx.x; j < C; j += blockDim.x) {
    const float v = md.act[cb * C + j];
    d[j] = v;
    if (!(v >= 0.0f && v <= 4294967296.0f)) dok = 0;
  }
  __syncthreads();
  if (threadIdx.x == 0) {
    float m = 0.0f;
    for (int j = 0; j < C; ++j) m = fmaxf(m, fabsf(d[j]));
    dmax = m;
  }
  __syncthreads();
  int qd;
  const float inv = fixed_point_inv(dmax, &qd);
  for (int j = threadIdx.x; j < C; j += blockDim.x) Dq[j] = inv == 0.0f ? 0 : fixed_point_int(d[j], inv);
  if (threadIdx.x == 0) two_qd = pow2f(qd);
  __syncthreads();
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= pr.S_pad) return;
  constexpr int NL = P * (P - 1) / 2 > 0 ? P * (P - 1) / 2 : 1;
  int sd = 0;
  for (int j = 0; j < C; ++j) sd += Dq[j];
  const float gd = __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(sd), two_qd));
  float Goff[NL], L[NL], invD[P];
  const uint64_t* mk = masks + (size_t)s * P * pr.W;
#pragma unroll
  for (int q = 1; q < P; ++q) {
#pragma unroll
    for (int p = 0; p < q; ++p) {
      int v = 0;
      for (int wd = 0; wd < pr.W; ++wd) {
        const uint64_t x = mk[p * pr.W + wd] ^ mk[q * pr.W + wd];
        const int jn = min(64, C - 64 * wd);
        for (int jj = 0; jj < jn; ++jj) {
          const int dj = Dq[64 * wd + jj];
          v += ((x >> jj) & 1ull) ? -dj : dj;
        }
      }
      Goff[tri(q, p)] = __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(v), two_qd));
    }
  }
  const float eps = __fmul_rn(pr.ridge_rel, gd);
  bool ok = ldl_factor<P>(gd, eps, Goff, L, invD);
  ok = ok && dok && (s < pr.S);
  const float qnan = __int_as_float(0x7fc00000);
  if (gram) {
    float* out = gram + (size_t)(md.gram_off + cb * pr.S_pad + s) * gram_stride(P);
#pragma unroll
    for (int i = 0; i < P * (P - 1) / 2; ++i) out[i] = L[i];
#pragma unroll
    for (int k = 0; k < P; ++k) out[P * (P - 1) / 2 + k] = ok ? invD[k] : qnan;
#pragma unroll
    for (int i = 0; i < P * (P - 1) / 2; ++i) out[P * (P - 1) / 2 + P + i] = Goff[i];
    out[P * (P - 1) + P] = gd;
  }
  if (pairs) {
    // seed s is component s & 1 of seed pair s >> 1 (entries start on even seeds)
    float* po = reinterpret_cast<float*>(pairs) +
                (size_t)((md.gram_off + cb * pr.S_pad + s) >> 1) * pair_stride(P) * 2 + (s & 1);
    constexpr int nl = P * (P - 1) / 2;
#pragma unroll
    for (int i = 0; i < nl; ++i) po[2 * i] = -L[i];
#pragma unroll
    for (int k = 0; k < P; ++k) po[2 * (nl + k)] = ok ? invD[k] : qnan;
#pragma unroll
    for (int i = 0; i < nl; ++i) po[2 * (nl + P + i)] = pr.fast_pow2 ? __fmul_rn(2.0f, Goff[i]) : Goff[i];
    po[2 * (2 * nl + P)] = gd;
    for (int i = 2 * nl + P + 1; i < pair_stride(P) - 1; ++i) po[2 * i] = 0.0f;
    po[2 * (pair_stride(P) - 1)] = ok ? bound_multiplier<P>(gd, Goff, eps) : __int_as_float(0x7f800000);
  }
}

// Tile staging shared by search and finalisation: r = W - W0, d, y = d*r.
__device__ __forceinline__ void tile_elem(const Prm& pr, const ModDesc& md, int64_t row,
                                          int64_t cb, int j, float* y, float* d, bool* ok) {
  const int64_t idx = row * md.cols + cb * pr.C + j;
  const float r = __fsub_rn(load_elem(md.W, idx, md.w_dtype), load_elem(md.W0, idx, md.w0_dtype));
  const float a = md.act[cb * pr.C + j];
  float dv;
  if (pr.variant == AWSRC_VARIANT_U) dv = a;
  else dv = __fadd_rn(__fmul_rn(md.w_act, a), __fmul_rn(md.w_fisher, md.fisher[idx]));
  *ok = in_domain(r, dv);
  *d = dv;
  *y = __fmul_rn(dv, r);
}

// Score of seed s for one tile from its fixed-point Y (and D for PF): the +-1
// correlations are exact integer sums, rounded once and scaled by 2^q.
template <int P, int VAR, bool ALLOW_FAST = true>
__device__ __forceinline__ float score_seed(const Prm& pr, const int* Yi, const int* Di, float two_qy,
                                            float two_qd, float gd_row, const uint64_t* __restrict__ masks,
                                            const float* __restrict__ gram_cb, uint32_t s, float* q,
                                            int* sf) {
  constexpr int NL = P * (P - 1) / 2 > 0 ? P * (P - 1) / 2 : 1;
  const uint64_t* mk = masks + (size_t)s * P * pr.W;
  int u[P];
#pragma unroll
  for (int p = 0; p < P; ++p) u[p] = 0;
  int v[NL];
#pragma unroll
  for (int i = 0; i < NL; ++i) v[i] = 0;
  for (int wd = 0; wd < pr.W; ++wd) {
    uint64_t m[P];
#pragma unroll
    for (int p = 0; p < P; ++p) m[p] = mk[p * pr.W + wd];
    const int jn = min(64, pr.C - 64 * wd);
    for (int jj = 0; jj < jn; ++jj) {
      const int yj = Yi[64 * wd + jj];
#pragma unroll
      for (int p = 0; p < P; ++p) u[p] += ((m[p] >> jj) & 1ull) ? -yj : yj;
      if (VAR == AWSRC_VARIANT_PF) {
        const int dj = Di[64 * wd + jj];
#pragma unroll
        for (int qq = 1; qq < P; ++qq)
#pragma unroll
          for (int p = 0; p < qq; ++p) v[tri(qq, p)] += (((m[p] ^ m[qq]) >> jj) & 1ull) ? -dj : dj;
      }
    }
  }
  float bv[P], alpha[P];
#pragma unroll
  for (int p = 0; p < P; ++p) bv[p] = __fmul_rn(pr.c, __fmul_rn(__int2float_rn(u[p]), two_qy));
  if (VAR == AWSRC_VARIANT_U) {
    const float* gt = gram_cb + (size_t)s * gram_stride(P);
    float L[NL], invD[P], Goff[NL];
#pragma unroll
    for (int i = 0; i < P * (P - 1) / 2; ++i) L[i] = gt[i];
#pragma unroll
    for (int k = 0; k < P; ++k) invD[k] = gt[P * (P - 1) / 2 + k];
#pragma unroll
    for (int i = 0; i < P * (P - 1) / 2; ++i) Goff[i] = gt[P * (P - 1) / 2 + P + i];
    const float gd = gt[P * (P - 1) + P];
    ldl_solve<P>(L, invD, bv, alpha);
    if (ALLOW_FAST && pr.fast_pow2) {
#pragma unroll
      for (int i = 0; i < P * (P - 1) / 2; ++i) Goff[i] = __fmul_rn(2.0f, Goff[i]);
      return quant_gain_fast<P>(pr, alpha, bv, gd, Goff, q, sf);
    }
    return quant_gain<P>(pr, alpha, bv, gd, Goff, q, sf);
  } else {
    float Goff[NL], L[NL], invD[P];
#pragma unroll
    for (int i = 0; i < P * (P - 1) / 2; ++i) Goff[i] = __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(v[i]), two_qd));
    const float eps = __fmul_rn(pr.ridge_rel, gd_row);
    const bool ok = ldl_factor<P>(gd_row, eps, Goff, L, invD);
    ldl_solve<P>(L, invD, bv, alpha);
    float g;
    if (ALLOW_FAST && pr.fast_pow2) {
#pragma unroll
      for (int i = 0; i < P * (P - 1) / 2; ++i) Goff[i] = __fmul_rn(2.0f, Goff[i]);
      g = quant_gain_fast<P>(pr, alpha, bv, gd_row, Goff, q, sf);
    } else {
      g = quant_gain<P>(pr, alpha, bv, gd_row, Goff, q, sf);
    }
    return ok ? g : neg_inf();
  }
}

// Turn a staged row of C floats (y or d) into its fixed-point integers in place
// (one thread per row); returns 2^q. The integer array aliases the floats.
__device__ __forceinline__ float row_to_fixed(float* x, int C) {
  float m = 0.0f;
  for (int j = 0; j < C; ++j) m = fmaxf(m, fabsf(x[j]));
  int q;
  const float inv = fixed_point_inv(m, &q);
  int* X = reinterpret_cast<int*>(x);
  for (int j = 0; j < C; ++j) X[j] = inv == 0.0f ? 0 : fixed_point_int(x[j], inv);
  return pow2f(q);
}

// gd = c2 * 2^qd * RN(sum_j D_j) for a row of fixed-point D.
__device__ __forceinline__ float row_gd(const Prm& pr, const int* D, float two_qd) {
  int sd = 0;
  for (int j = 0; j < pr.C; ++j) sd += D[j];
  return __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(sd), two_qd));
}

// Seed range of split z in units of `chunk` seeds.
__device__ __forceinline__ void split_range(int S, int chunk, int nsplit, int z, int* s0, int* s1) {
  const int nck = (S + chunk - 1) / chunk;
  const int per = (nck + nsplit - 1) / nsplit;
  *s0 = min(S, z * per * chunk);
  *s1 = min(S, (z + 1) * per * chunk);
}

// ---------------------------------------------------------- generic search --
template <int P, int VAR>
__global__ void __launch_bounds__(kGenThreads) search_generic_kernel(
    Prm pr, LaunchDesc ld, const uint64_t* __restrict__ masks, const float* __restrict__ gram,
    float2* __restrict__ partials) {
  extern __shared__ float smem[];
  const int mi = find_mod(ld, blockIdx.x);
  const ModDesc& md = ld.m[mi];
  const int64_t b = blockIdx.x - md.block_off;
  const int z = (int)(b % md.nsplit);
  const int64_t rest = b / md.nsplit;
  const int64_t rb = rest % md.n_rb;
  const int64_t cb = rest / md.n_rb;
  const int C = pr.C, ldc = C + 1;
  float* ys = smem;
  float* ds = smem + kGenRows * ldc;
  __shared__ int rowok[kGenRows];
  __shared__ float gds[kGenRows];
  const int tid = threadIdx.x;
  if (tid < kGenRows) rowok[tid] = 1;
  __syncthreads();
  for (int e = tid; e < kGenRows * C; e += kGenThreads) {
    const int r = e / C, j = e % C;
    const int64_t row = rb * kGenRows + r;
    float y = 0.0f, d = 0.0f;
    if (row < md.rows) {
      bool ok;
      tile_elem(pr, md, row, cb, j, &y, &d, &ok);
      if (!ok) rowok[r] = 0;
    }
    ys[r * ldc + j] = y;
    if (VAR == AWSRC_VARIANT_PF) ds[r * ldc + j] = d;
  }
  __syncthreads();
  __shared__ float tqy[kGenRows], tqd[kGenRows];
  if (tid < kGenRows) {
    tqy[tid] = row_to_fixed(ys + tid * ldc, C);
    if (VAR == AWSRC_VARIANT_PF) {
      tqd[tid] = row_to_fixed(ds + tid * ldc, C);
      gds[tid] = row_gd(pr, reinterpret_cast<const int*>(ds + tid * ldc), tqd[tid]);
    }
  }
  __syncthreads();
  const int r = tid / kGenLanes, sl = tid % kGenLanes;
  const int64_t row = rb * kGenRows + r;
  int s0, s1;
  split_range(pr.S, kGenLanes, md.nsplit, z, &s0, &s1);
  float bg = neg_inf();
  uint32_t bs = 0xffffffffu;
  const float* gram_cb = (VAR == AWSRC_VARIANT_U)
                             ? gram + (size_t)(md.gram_off + cb * pr.S_pad) * gram_stride(P)
                             : nullptr;
  if (row < md.rows && rowok[r]) {
    for (int s = s0 + sl; s < s1; s += kGenLanes) {
      float q[P];
      int sf;
      const float g = score_seed<P, VAR>(pr, reinterpret_cast<const int*>(ys + r * ldc),
                                         reinterpret_cast<const int*>(ds + r * ldc), tqy[r],
                                         VAR == AWSRC_VARIANT_PF ? tqd[r] : 0.0f,
                                         VAR == AWSRC_VARIANT_PF ? gds[r] : 0.0f, masks, gram_cb,
                                         (uint32_t)s, q, &sf);
      if (better(g, (uint32_t)s, bg, bs)) { bg = g; bs = (uint32_t)s; }
    }
  }
#pragma unroll
  for (int off = 1; off < kGenLanes; off <<= 1) {
    const float og = __shfl_xor_sync(0xffffffffu, bg, off);
    const uint32_t os = __shfl_xor_sync(0xffffffffu, bs, off);
    if (better(og, os, bg, bs)) { bg = og; bs = os; }
  }
  if (sl == 0 && row < md.rows) {
    const int64_t t = md.tile_off + row * md.n_cb + cb;
    partials[(size_t)z * ld.T + t] = make_float2(rowok[r] ? bg : neg_inf(), __uint_as_float(bs));
  }
}

// V consecutive elements (V = 4 or 8) of a weight array as floats; idx is a
// multiple of V. Vector loads when the array is 16-byte aligned.
template <int V>
__device__ __forceinline__ void load_run(const void* p, int64_t idx, int dtype, bool aligned, float* out) {
  if (aligned && dtype == AWSRC_DTYPE_F32) {
#pragma unroll
    for (int i = 0; i < V; i += 4) {
      const float4 f = *reinterpret_cast<const float4*>(static_cast<const float*>(p) + idx + i);
      out[i] = f.x; out[i + 1] = f.y; out[i + 2] = f.z; out[i + 3] = f.w;
    }
  } else if (aligned && V == 8) {
    const uint4 u = *reinterpret_cast<const uint4*>(static_cast<const __nv_bfloat16*>(p) + idx);
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      out[2 * i] = __uint_as_float(w[i] << 16);
      out[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  } else {
#pragma unroll
    for (int i = 0; i < V; ++i) out[i] = load_elem(p, idx + i, dtype);
  }
}

// --------------------------------------------------------------- finalize --
// One thread per tile; a block stages its tiles' y (and d) in shared memory with
// coalesced loads: tiles are numbered row-major, so consecutive tiles of a
// module are consecutive C-element runs of its weight arrays.
__host__ __device__ inline int fin_tiles(int C) { return C <= 64 ? 128 : 16384 / C; }

// Stage y = d*(W - W0) (and d) of tiles [t0, t0 + TB) in shared memory, V
// elements per load, loads of four runs issued before any is used.
template <int V, int VAR>
__device__ __forceinline__ void stage_tiles(const Prm& pr, const LaunchDesc& ld, int64_t t0, int64_t last,
                                            int TB, const int* tmod, int* tok, float* ys, float* ds) {
  const int C = pr.C, ldc = C + 1;
  const int nrun = TB * C / V;
#pragma unroll 4
  for (int g = threadIdx.x; g < nrun; g += blockDim.x) {
    const int lt = (g * V) >> pr.logC, j0 = (g * V) & (C - 1);
    const int64_t t = t0 + lt;
    float y[V], d[V];
    if (t < last) {
      const ModDesc& md = ld.m[tmod[lt]];
      const int64_t ltm = t - md.tile_off;
      const int64_t idx = ltm * C + j0;  // a module's tiles are consecutive runs of C elements
      const int64_t cb = ltm % md.n_cb;
      const bool alW = ((reinterpret_cast<uintptr_t>(md.W) | reinterpret_cast<uintptr_t>(md.W0)) & 15) == 0;
      float w[V], w0[V], a[V];
      load_run<V>(md.W, idx, md.w_dtype, alW, w);
      load_run<V>(md.W0, idx, md.w0_dtype, alW, w0);
      load_run<V>(md.act, cb * C + j0, AWSRC_DTYPE_F32, (reinterpret_cast<uintptr_t>(md.act) & 15) == 0, a);
      float f[V];
      if (VAR == AWSRC_VARIANT_PF)
        load_run<V>(md.fisher, idx, AWSRC_DTYPE_F32, (reinterpret_cast<uintptr_t>(md.fisher) & 15) == 0, f);
      bool ok = true;
#pragma unroll
      for (int i = 0; i < V; ++i) {
        const float r = __fsub_rn(w[i], w0[i]);
        const float dv = VAR == AWSRC_VARIANT_U
                             ? a[i]
                             : __fadd_rn(__fmul_rn(md.w_act, a[i]), __fmul_rn(md.w_fisher, f[i]));
        ok = ok && in_domain(r, dv);
        d[i] = dv;
        y[i] = __fmul_rn(dv, r);
      }
      if (!ok) tok[lt] = 0;
    } else {
#pragma unroll
      for (int i = 0; i < V; ++i) { y[i] = 0.0f; d[i] = 0.0f; }
    }
#pragma unroll
    for (int i = 0; i < V; ++i) {
      ys[lt * ldc + j0 + i] = y[i];
      if (VAR == AWSRC_VARIANT_PF) ds[lt * ldc + j0 + i] = d[i];
    }
  }
}

template <int P, int VAR>
__global__ void __launch_bounds__(128) finalize_kernel(Prm pr, LaunchDesc ld,
                                                       const uint64_t* __restrict__ masks,
                                                       const float* __restrict__ gram,
                                                       const float2* __restrict__ partials,
                                                       awsrc_candidate* __restrict__ out,
                                                       uint32_t* __restrict__ status) {
  extern __shared__ float fsm[];
  const int C = pr.C, ldc = C + 1, TB = fin_tiles(C);
  float* ys = fsm;
  float* ds = fsm + TB * ldc;
  __shared__ int tmod[128];
  __shared__ int tok[128];
  const int64_t first = ld.m[0].tile_off;
  const int64_t last = ld.m[ld.n - 1].tile_off + ld.m[ld.n - 1].rows * ld.m[ld.n - 1].n_cb;
  const int64_t t0 = first + (int64_t)blockIdx.x * TB;
  const int tid = threadIdx.x;
  if (tid < TB) {
    const int64_t t = t0 + tid;
    int mi = 0;
    for (int i = 1; i < ld.n; ++i)
      if (t >= ld.m[i].tile_off) mi = i;
    tmod[tid] = mi;
    tok[tid] = 1;
  }
  __syncthreads();
  if (C >= 8) stage_tiles<8, VAR>(pr, ld, t0, last, TB, tmod, tok, ys, ds);
  else stage_tiles<4, VAR>(pr, ld, t0, last, TB, tmod, tok, ys, ds);
  __syncthreads();
  if (tid >= TB) return;
  const int64_t t = t0 + tid;
  if (t >= last) return;
  const ModDesc& md = ld.m[tmod[tid]];
  const int64_t cb = (t - md.tile_off) % md.n_cb;
  float bg = neg_inf();
  uint32_t bs = 0xffffffffu;
  for (int z = 0; z < md.nsplit; ++z) {
    const float2 pz = partials[(size_t)z * ld.T + t];
    const float g = pz.x;
    const uint32_t s = __float_as_uint(pz.y);
    if (better(g, s, bg, bs)) { bg = g; bs = s; }
  }
  awsrc_candidate cd;
  cd.gain = neg_inf();
  cd.seed = 0;
  cd.scale = 0;
#pragma unroll
  for (int p = 0; p < 8; ++p) cd.code[p] = 0;
  if (bg > neg_inf() && bs < (uint32_t)pr.S) {
    const bool ok = tok[tid] != 0;
    const float two_qy = row_to_fixed(ys + tid * ldc, C);
    float two_qd = 0.0f, gd_row = 0.0f;
    if (VAR == AWSRC_VARIANT_PF) {
      two_qd = row_to_fixed(ds + tid * ldc, C);
      gd_row = row_gd(pr, reinterpret_cast<const int*>(ds + tid * ldc), two_qd);
    }
    const float* gram_cb = (VAR == AWSRC_VARIANT_U)
                               ? gram + (size_t)(md.gram_off + cb * pr.S_pad) * gram_stride(P)
                               : nullptr;
    float q[P];
    int sf = 0;
    // the general quantiser here, so the self-check also compares it with the
    // fast path the search used
    const float g = score_seed<P, VAR, false>(pr, reinterpret_cast<const int*>(ys + tid * ldc),
                                              reinterpret_cast<const int*>(ds + tid * ldc), two_qy, two_qd,
                                              gd_row, masks, gram_cb, bs, q, &sf);
    if (!ok || __float_as_uint(g) != __float_as_uint(bg)) atomicOr(status, kFaultSelfCheck);
    if (ok && g > neg_inf()) {
      cd.gain = g;
      cd.seed = (uint16_t)bs;
      cd.scale = (int16_t)sf;
#pragma unroll
      for (int p = 0; p < P; ++p) cd.code[p] = (int8_t)(int)q[p];
    }
  }
  out[t] = cd;
}

template <int P>
cudaError_t launch_gram_p(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks, float* gram,
                          float2* pairs, cudaStream_t st) {
  int64_t ncb = 0;
  for (int i = 0; i < ld.n; ++i) ncb += ld.m[i].n_cb;
  dim3 grid((pr.S_pad + 127) / 128, (unsigned)ncb);
  gram_u_kernel<P><<<grid, 128, 0, st>>>(pr, ld, masks, gram, pairs);
  note_launches(1);
  return cudaGetLastError();
}

template <int P, int VAR>
cudaError_t launch_search_pv(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                             const float* gram, int64_t n_blocks, float2* partials,
                             cudaStream_t st) {
  const size_t smem = (size_t)kGenRows * (pr.C + 1) * sizeof(float) * (VAR == AWSRC_VARIANT_PF ? 2 : 1);
  auto k = search_generic_kernel<P, VAR>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<(unsigned)n_blocks, kGenThreads, smem, st>>>(pr, ld, masks, gram, partials);
  note_launches(1);
  return cudaGetLastError();
}

template <int P, int VAR>
cudaError_t launch_finalize_pv(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                               const float* gram, const float2* partials, awsrc_candidate* out,
                               uint32_t* status, cudaStream_t st) {
  const int64_t first = ld.m[0].tile_off;
  const int64_t last = ld.m[ld.n - 1].tile_off + ld.m[ld.n - 1].rows * ld.m[ld.n - 1].n_cb;
  const int TB = fin_tiles(pr.C);
  const size_t smem = (size_t)TB * (pr.C + 1) * sizeof(float) * (VAR == AWSRC_VARIANT_PF ? 2 : 1);
  auto k = finalize_kernel<P, VAR>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<(unsigned)((last - first + TB - 1) / TB), 128, smem, st>>>(pr, ld, masks, gram, partials, out, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

#define AWSRC_DISPATCH_P(P_, EXPR) \
  switch (P_) {                    \
    case 1: { constexpr int PP = 1; return EXPR; } \
    case 2: { constexpr int PP = 2; return EXPR; } \
    case 3: { constexpr int PP = 3; return EXPR; } \
    case 4: { constexpr int PP = 4; return EXPR; } \
    case 5: { constexpr int PP = 5; return EXPR; } \
    case 6: { constexpr int PP = 6; return EXPR; } \
    case 7: { constexpr int PP = 7; return EXPR; } \
    case 8: { constexpr int PP = 8; return EXPR; } \
    default: return cudaErrorInvalidValue;          \
  }

cudaError_t launch_gram_u(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks, float* gram,
                          float2* pairs, cudaStream_t st) {
  AWSRC_DISPATCH_P(pr.P, (launch_gram_p<PP>(pr, ld, masks, gram, pairs, st)));
}

cudaError_t launch_search_generic(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                                  const float* gram, int64_t n_blocks, float2* partials,
                                  cudaStream_t st) {
  if (pr.variant == AWSRC_VARIANT_U) {
    AWSRC_DISPATCH_P(pr.P, (launch_search_pv<PP, AWSRC_VARIANT_U>(pr, ld, masks, gram, n_blocks, partials, st)));
  }
  AWSRC_DISPATCH_P(pr.P, (launch_search_pv<PP, AWSRC_VARIANT_PF>(pr, ld, masks, gram, n_blocks, partials, st)));
}

cudaError_t launch_finalize(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                            const float* gram, const float2* partials, int nsplit_max,
                            awsrc_candidate* out, uint32_t* status, cudaStream_t st) {
  (void)nsplit_max;
  if (pr.variant == AWSRC_VARIANT_U) {
    AWSRC_DISPATCH_P(pr.P, (launch_finalize_pv<PP, AWSRC_VARIANT_U>(pr, ld, masks, gram, partials, out, status, st)));
  }
  AWSRC_DISPATCH_P(pr.P, (launch_finalize_pv<PP, AWSRC_VARIANT_PF>(pr, ld, masks, gram, partials, out, status, st)));
}

int generic_rows() { return kGenRows; }
int generic_chunk() { return kGenLanes; }

}  // namespace awsrc
