// encode.cu — the seed search of Sec. 3.2 for any supported (C, P) and both
// variants, and the U Gram tables every U search reads:
//
//  gram_u      U only. The activation diagonal is shared by all rows of a module
//              (Sec. 3.2), so the Gram matrix B_s^T D B_s of Eq. 3 and its LDL^T
//              depend on (column block, seed) only. They are computed once per
//              (cb, s) and reused by every row.
//  search      per (tile, seed): correlation b = B_s^T D r, solve, quantise,
//              gain; the best seed of each tile (over one seed split) is
//              written as a whole candidate.
#include <cfloat>

#include "internal.h"

namespace awsrc {

namespace {


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
// above g_best. m is +inf (no pruning) when G is not positive definite or
// kappa > 2^16.
//
// Evaluated in binary32 (the GPU's double rate is low): the LDL^T of G and
// tr(G^-1) = sum_k |row k of L^-1|^2 / D_k. For kappa <= 2^16 the computed
// factors are those of G + dG with |dG| <= ~5 P 2^-24 kappa |G| (<= ~8% in
// eigenvalue terms), and the inverse trace from them is within ~10% of the
// exact one; it enters m inflated by 1.5, with every operation of m rounded
// up, so m is at least the value the exact trace gives.
template <int P>
__device__ float bound_multiplier(float gd, const float* Goff, float eps) {
  float L[P][P], d[P], inv_d[P];
#pragma unroll
  for (int k = 0; k < P; ++k) {
    float dk = gd;
#pragma unroll
    for (int i = 0; i < k; ++i) dk = __fmaf_rn(-L[k][i] * L[k][i], d[i], dk);
    if (!(dk > 0.0f)) return __int_as_float(0x7f800000);
    d[k] = dk;
    inv_d[k] = __frcp_rn(dk);
#pragma unroll
    for (int j = k + 1; j < P; ++j) {
      float v = Goff[tri(j, k)];
#pragma unroll
      for (int i = 0; i < k; ++i) v = __fmaf_rn(-L[j][i] * L[k][i], d[i], v);
      L[j][k] = __fmul_rn(v, inv_d[k]);
    }
  }
  float tr_inv = 0.0f;
#pragma unroll
  for (int i = 0; i < P; ++i) {  // column i of X = L^-1, rows k >= i
    float x[P];
    x[i] = 1.0f;
    tr_inv = __fadd_rn(tr_inv, inv_d[i]);
#pragma unroll
    for (int k = i + 1; k < P; ++k) {
      float v = 0.0f;
#pragma unroll
      for (int j = i; j < k; ++j) v = __fmaf_rn(-L[k][j], x[j], v);
      x[k] = v;
      tr_inv = __fmaf_rn(__fmul_rn(v, v), inv_d[k], tr_inv);
    }
  }
  if (!(tr_inv > 0.0f && tr_inv < 3.0e38f)) return __int_as_float(0x7f800000);
  const float kappa = __fmul_rn(__fmul_rn((float)P, gd), tr_inv);
  if (!(kappa <= 65536.0f)) return __int_as_float(0x7f800000);
  const float ts = __fmul_ru(1.5f, tr_inv), ks = __fmul_ru(1.5f, __fmul_ru(__fmul_ru((float)P, gd), tr_inv));
  const float f1 = __fmaf_ru(eps, ts, 1.0f);
  const float f2 = __fmaf_ru(0x1p-14f, ks, 1.0f + 0x1p-10f);
  return __fmul_ru(f1, f2);
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
  __shared__ int Dt[kMaxC / 4][16];  // subset sums of each 4-input group of Dq
  __shared__ int dok;
  __shared__ float dmax;
  __shared__ float two_qd;
  __shared__ int sdq;  // sum of the fixed-point weights (exact)
  if (threadIdx.x == 0) dok = 1;
  __syncthreads();
  for (int j = threadIdx.x; j < C; j += blockDim.x) {
    const float v = md.act[cb * C + j];
    d[j] = v;
    if (!(v >= 0.0f && v <= 4294967296.0f)) dok = 0;
  }
  __syncthreads();
  if (threadIdx.x < 32) {  // the column block's largest |d|, one warp
    float m = 0.0f;
    for (int j = threadIdx.x; j < C; j += 32) m = fmaxf(m, fabsf(d[j]));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    if (threadIdx.x == 0) dmax = m;
  }
  __syncthreads();
  int qd;
  const float inv = fixed_point_inv(dmax, &qd);
  for (int j = threadIdx.x; j < C; j += blockDim.x) Dq[j] = inv == 0.0f ? 0 : fixed_point_int(d[j], inv);
  if (threadIdx.x == 0) two_qd = pow2f(qd);
  __syncthreads();
  if (threadIdx.x < 32) {  // integer sum, so the order does not matter
    int t = 0;
    for (int j = threadIdx.x; j < C; j += 32) t += Dq[j];
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) t += __shfl_xor_sync(0xffffffffu, t, off);
    if (threadIdx.x == 0) sdq = t;
  }
  for (int i = threadIdx.x; i < (C / 4) * 16; i += blockDim.x) {
    const int g = i >> 4, nb = i & 15;
    int v = 0;
#pragma unroll
    for (int bb = 0; bb < 4; ++bb)
      if ((nb >> bb) & 1) v += Dq[4 * g + bb];
    Dt[g][nb] = v;
  }
  __syncthreads();
  // threads past S_pad (the last block of a small S_pad) score a dummy seed
  // whose entries are never written; every thread reaches the barrier below
  const int s_raw = blockIdx.x * blockDim.x + threadIdx.x;
  if (s_raw >= pr.S_pad && !pairs) return;
  const int s = min(s_raw, pr.S_pad - 1);
  constexpr int NL = P * (P - 1) / 2 > 0 ? P * (P - 1) / 2 : 1;
  const int sd = sdq;
  const float gd = __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(sd), two_qd));
  float Goff[NL], L[NL], invD[P];
  const uint64_t* mk = masks + (size_t)s * P * pr.W;
#pragma unroll
  for (int q = 1; q < P; ++q) {
#pragma unroll
    for (int p = 0; p < q; ++p) {
      // sum_j (+-1) Dq_j with the sign of atom product p*q: the total minus
      // twice the inputs where the two masks differ, by nibble-table reads
      int v = sd, neg = 0;
      for (int wd = 0; wd < pr.W; ++wd) {
        const uint64_t x = mk[p * pr.W + wd] ^ mk[q * pr.W + wd];
        const int gn = min(16, (C - 64 * wd) >> 2);
        for (int g = 0; g < gn; ++g) neg += Dt[16 * wd + g][(int)((x >> (4 * g)) & 15ull)];
      }
      v -= 2 * neg;
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
    // seed s is component s & 1 of seed pair s >> 1 (entries start on even
    // seeds); the block's 64 pairs are one contiguous run of the table, built
    // in shared memory and written out in 16-byte stores
    constexpr int ps = pair_stride(P);
    __shared__ __align__(16) float stage[128 / 2 * ps * 2];
    float* po = stage + (threadIdx.x >> 1) * ps * 2 + (threadIdx.x & 1);
    constexpr int nl = P * (P - 1) / 2;
    // pr.prune == 0 scores every candidate (the same results, for tests of the bound)
    const float m = ok && pr.prune ? bound_multiplier<P>(gd, Goff, eps) : __int_as_float(0x7f800000);
#pragma unroll
    for (int i = 0; i < nl; ++i) po[2 * i] = -L[i];
    // invD * m rounded up: the bound's terms z_k (z_k invD_k m) are then never
    // below the exact z_k^2 invD_k m (m = +inf disables pruning)
#pragma unroll
    for (int k = 0; k < P; ++k) po[2 * (nl + k)] = ok ? __fmul_ru(invD[k], m) : qnan;
#pragma unroll
    for (int k = 0; k < P; ++k) po[2 * (nl + P + k)] = ok ? invD[k] : qnan;
#pragma unroll
    for (int i = 0; i < nl; ++i) po[2 * (nl + 2 * P + i)] = pr.fast_pow2 ? __fmul_rn(2.0f, Goff[i]) : Goff[i];
    po[2 * (2 * nl + 2 * P)] = gd;
    for (int i = 2 * nl + 2 * P + 1; i < ps; ++i) po[2 * i] = 0.0f;
    __syncthreads();
    // seeds s0 .. s0 + 127 of this column block (s0 even, S_pad a multiple of 32)
    const int s0 = blockIdx.x * blockDim.x;
    const int npairs = min((int)blockDim.x, pr.S_pad - s0) / 2;
    float4* dst = reinterpret_cast<float4*>(reinterpret_cast<float*>(pairs) +
                                            (size_t)((md.gram_off + cb * pr.S_pad + s0) >> 1) * ps * 2);
    const float4* src = reinterpret_cast<const float4*>(stage);
    for (int i = threadIdx.x; i < npairs * ps / 2; i += blockDim.x) dst[i] = src[i];
  }
}

// The score of seed s for one tile works on its fixed-point Y (and D for PF):
// the +-1 correlations are exact integer sums, rounded once and scaled by 2^q.
template <int P>
__host__ __device__ constexpr int n_off() { return P * (P - 1) / 2 > 0 ? P * (P - 1) / 2 : 1; }

// The +-1 correlations of seed s with the tile's fixed-point Y (u) and, for
// PF, of the pairwise atom products with D (v), element by element.
template <int P, int VAR>
__device__ __forceinline__ void seed_sums(const Prm& pr, const int* Yi, const int* Di,
                                          const uint64_t* __restrict__ masks, uint32_t s, int* u, int* v) {
  constexpr int NL = n_off<P>();
  const uint64_t* mk = masks + (size_t)s * P * pr.W;
#pragma unroll
  for (int p = 0; p < P; ++p) u[p] = 0;
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
}

// The same sums from per-tile nibble tables (C <= 64, one mask word):
// Ty[16 g + m] = sum_{i<4} (bit i of m ? -Y : Y)[4 g + i], likewise Td for D,
// so each correlation is C/4 table reads. Integer sums: exact in any order.
template <int P, int VAR>
__device__ __forceinline__ void seed_sums_tab(const Prm& pr, const int* Ty, const int* Td,
                                              const uint64_t* __restrict__ masks, uint32_t s, int* u, int* v) {
  const uint64_t* mk = masks + (size_t)s * P;
  uint64_t m[P];
#pragma unroll
  for (int p = 0; p < P; ++p) {
    m[p] = mk[p];
    u[p] = 0;
  }
  if (VAR == AWSRC_VARIANT_PF) {
#pragma unroll
    for (int i = 0; i < n_off<P>(); ++i) v[i] = 0;
  }
  const int ng = pr.C >> 2;
  for (int g = 0; g < ng; ++g) {
    const int* ty = Ty + 16 * g;
#pragma unroll
    for (int p = 0; p < P; ++p) u[p] += ty[(uint32_t)(m[p] >> (4 * g)) & 15u];
    if (VAR == AWSRC_VARIANT_PF) {
      const int* td = Td + 16 * g;
#pragma unroll
      for (int qq = 1; qq < P; ++qq)
#pragma unroll
        for (int p = 0; p < qq; ++p) v[tri(qq, p)] += td[(uint32_t)((m[p] ^ m[qq]) >> (4 * g)) & 15u];
    }
  }
}

// Score of a seed from its correlation sums: b and (PF) the Gram off-diagonals
// rounded once and scaled, the ridge solve, quantiser and gain.
template <int P, int VAR>
__device__ __forceinline__ float score_sums(const Prm& pr, const int* u, const int* v, float two_qy,
                                            float two_qd, float gd_row, const float* __restrict__ gram_cb,
                                            uint32_t s, float* q, int* sf) {
  constexpr int NL = n_off<P>();
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
    if (pr.fast_pow2) {
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
    if (pr.fast_pow2) {
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

// ---------------------------------------------------------- generic search --
// Nibble tables pay off when a tile is one mask word (C <= 64) and each table
// serves several seeds.
__host__ __device__ inline bool gen_tables(const Prm& pr) { return pr.C <= 64 && pr.S >= 4; }

// Shared memory per tile: staged y (and d), plus the nibble tables.
__host__ __device__ inline size_t gen_tile_smem(const Prm& pr) {
  const size_t nb = pr.variant == AWSRC_VARIANT_PF ? 2 : 1;
  return (nb * (size_t)(pr.C + 1) + (gen_tables(pr) ? nb * 4 * (size_t)pr.C + 1 : 0)) * sizeof(float);
}

// Any (C, P, variant): a block takes TB consecutive tiles of the launch (a
// module's tiles are consecutive C-element runs of its weight arrays, so the
// staging loads are coalesced vectors), converts each tile to its fixed-point
// grid, and `lanes` threads per tile score interleaved seeds with score_seed;
// the best seed of each tile (larger gain, then smaller seed) is merged across
// lanes with its codes and scale field and written as a whole candidate (seed
// split z of it when the seeds are split over blocks).
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
__global__ void __launch_bounds__(256) search_tiles_kernel(Prm pr, LaunchDesc ld, const uint64_t* __restrict__ masks,
                                                           const float* __restrict__ gram,
                                                           awsrc_candidate* __restrict__ cands, int lanes, int TB) {
  extern __shared__ float fsm[];
  const int C = pr.C, ldc = C + 1;
  const int nb = VAR == AWSRC_VARIANT_PF ? 2 : 1;
  float* ys = fsm;
  float* ds = fsm + TB * ldc;
  const bool tab = gen_tables(pr);
  // nibble tables when tab: per tile [Y, D][C/4 groups][16], tiles one word
  // apart beyond their size so that tiles read from different banks
  const int tstride = nb * 4 * C + 1;
  int* tabs = reinterpret_cast<int*>(fsm + (size_t)nb * TB * ldc);
  __shared__ int tmod[256];
  __shared__ int tok[256];
  __shared__ float tqy[256], tqd[256], gds[256];
  const int nsplit = ld.m[0].nsplit;
  const int z = (int)(blockIdx.x % nsplit);
  const int64_t first = ld.m[0].tile_off;
  const int64_t last = ld.m[ld.n - 1].tile_off + ld.m[ld.n - 1].rows * ld.m[ld.n - 1].n_cb;
  const int64_t t0 = first + (int64_t)(blockIdx.x / nsplit) * TB;
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
  if (tid < TB) {
    tqy[tid] = row_to_fixed(ys + tid * ldc, C);
    if (VAR == AWSRC_VARIANT_PF) {
      tqd[tid] = row_to_fixed(ds + tid * ldc, C);
      gds[tid] = row_gd(pr, reinterpret_cast<const int*>(ds + tid * ldc), tqd[tid]);
    }
  }
  __syncthreads();
  const int lt = tid / lanes, sl = tid % lanes;
  if (tab) {  // the tile's lanes build its nibble tables
    const int per = 4 * C;  // C/4 groups x 16 patterns
    int* T = tabs + lt * tstride;
    for (int k = sl; k < nb * per; k += lanes) {
      const int which = k >= per ? 1 : 0, kk = k - which * per;
      const int g = kk >> 4, m = kk & 15;
      const int* X = reinterpret_cast<const int*>((which ? ds : ys) + lt * ldc) + 4 * g;
      int acc = 0;
#pragma unroll
      for (int i = 0; i < 4; ++i) acc += ((m >> i) & 1) ? -X[i] : X[i];
      T[k] = acc;
    }
    __syncthreads();
  }
  const int64_t t = t0 + lt;
  float bg = neg_inf();
  uint32_t bs = 0xffffffffu;
  float bq[P];
#pragma unroll
  for (int p = 0; p < P; ++p) bq[p] = 0.0f;
  int bsf = 0;
  const bool live = t < last && tok[lt] != 0;
  if (live) {
    const ModDesc& md = ld.m[tmod[lt]];
    const int64_t cb = (t - md.tile_off) % md.n_cb;
    const float* gram_cb = (VAR == AWSRC_VARIANT_U)
                               ? gram + (size_t)(md.gram_off + cb * pr.S_pad) * gram_stride(P)
                               : nullptr;
    int s0, s1;
    split_range(pr.S, lanes, nsplit, z, &s0, &s1);
    const int* Ty = tabs + (size_t)lt * tstride;
    for (int s = s0 + sl; s < s1; s += lanes) {
      float q[P];
      int sf;
      int u[P], v[n_off<P>()];
      if (tab) seed_sums_tab<P, VAR>(pr, Ty, Ty + 4 * C, masks, (uint32_t)s, u, v);
      else
        seed_sums<P, VAR>(pr, reinterpret_cast<const int*>(ys + lt * ldc),
                          reinterpret_cast<const int*>(ds + lt * ldc), masks, (uint32_t)s, u, v);
      const float g = score_sums<P, VAR>(pr, u, v, tqy[lt], VAR == AWSRC_VARIANT_PF ? tqd[lt] : 0.0f,
                                         VAR == AWSRC_VARIANT_PF ? gds[lt] : 0.0f, gram_cb, (uint32_t)s, q, &sf);
      if (better(g, (uint32_t)s, bg, bs)) {
        bg = g;
        bs = (uint32_t)s;
        bsf = sf;
#pragma unroll
        for (int p = 0; p < P; ++p) bq[p] = q[p];
      }
    }
  }
  // lanes of a tile are consecutive threads of one warp (lanes <= 8, blockDim a multiple of 32)
  for (int off = 1; off < lanes; off <<= 1) {
    const float og = __shfl_xor_sync(0xffffffffu, bg, off);
    const uint32_t os = __shfl_xor_sync(0xffffffffu, bs, off);
    const int osf = __shfl_xor_sync(0xffffffffu, bsf, off);
    float oq[P];
#pragma unroll
    for (int p = 0; p < P; ++p) oq[p] = __shfl_xor_sync(0xffffffffu, bq[p], off);
    if (better(og, os, bg, bs)) {
      bg = og;
      bs = os;
      bsf = osf;
#pragma unroll
      for (int p = 0; p < P; ++p) bq[p] = oq[p];
    }
  }
  if (sl == 0 && t < last) {
    awsrc_candidate cd;
    const bool valid = live && bg > neg_inf() && bs < (uint32_t)pr.S;
    cd.gain = valid ? bg : neg_inf();
    cd.seed = valid ? (uint16_t)bs : (uint16_t)0;
    cd.scale = valid ? (int16_t)bsf : (int16_t)0;
#pragma unroll
    for (int p = 0; p < 8; ++p) cd.code[p] = (p < P && valid) ? (int8_t)(int)bq[p < P ? p : 0] : (int8_t)0;
    cands[(size_t)z * ld.T + t] = cd;
  }
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
cudaError_t launch_search_pv(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks, const float* gram,
                             int64_t n_blocks, awsrc_candidate* cands, cudaStream_t st) {
  const GenShape gs = gen_shape(pr);
  const size_t smem = (size_t)gs.tiles * gen_tile_smem(pr);
  auto k = search_tiles_kernel<P, VAR>;
  cudaError_t e = cudaFuncSetAttribute(k, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  k<<<(unsigned)n_blocks, gs.tiles * gs.lanes, smem, st>>>(pr, ld, masks, gram, cands, gs.lanes, gs.tiles);
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
                                  const float* gram, int64_t n_blocks, awsrc_candidate* cands,
                                  cudaStream_t st) {
  if (pr.variant == AWSRC_VARIANT_U) {
    AWSRC_DISPATCH_P(pr.P, (launch_search_pv<PP, AWSRC_VARIANT_U>(pr, ld, masks, gram, n_blocks, cands, st)));
  }
  AWSRC_DISPATCH_P(pr.P, (launch_search_pv<PP, AWSRC_VARIANT_PF>(pr, ld, masks, gram, n_blocks, cands, st)));
}

GenShape gen_shape(const Prm& pr) {
  // one lane per four seeds (at most 8), 256 threads, shared memory for the
  // staged tiles (and nibble tables) at most 96 KB (but at least 32 threads)
  int lanes = 1;
  while (lanes < 8 && lanes * 4 < pr.S) lanes <<= 1;
  int tiles = 256 / lanes;
  while (tiles * lanes > 32 && tiles * gen_tile_smem(pr) > 96 * 1024) tiles >>= 1;
  return {lanes, tiles};
}

}  // namespace awsrc
