// search_pf_c64p4.cu — seed search (Sec. 3.2) for AWSRC-P_F with C = 64, P = 4
// on the tcgen05 tensor cores.
//
// P_F weights every element (d_ij = w_act a_j + w_fisher F_ij), so the Gram
// matrix G = B_s^T D B_s / C differs per (tile, seed): its off-diagonal entries
// are the +-1 correlations of the tile's D with the pairwise products
// m_p * m_q of the seed's atoms, and its diagonal is the tile's gd. Both the
// correlations b_p (with y = d r) and the six off-diagonals are exact integer
// sums on the tile's fixed-point grids (|Y|, |D| <= 2^21, FP16 halves
// hi = X >> 11, lo = X & 2047), computed by tcgen05.mma and rounded once in the
// epilogue, which then factors G + eps I (LDL^T), solves, quantises and scores
// every candidate exactly as the binary32 recipe does.
//
// Block: 128 tiles of one column block (row m = TMEM lane m), 13 warps. The
// producer warp streams 12-seed chunks (FP16 atoms 6 KB, a slice of the U
// search's atom table, and FP16 atom products 10 KB) through a 4-stage
// bulk-copy ring and issues per chunk 16 MMAs into one of two TMEM
// accumulators: Y_hi, Y_lo x atoms (N = 48) and D_hi, D_lo x products (N = 80,
// the last 8 columns zero). The search is bound by this MMA chain, so a chunk
// is as many seeds as two accumulators of 256 columns hold. Epilogue warp w
// takes TMEM lanes 32(w%4).. and seed pairs 2(w/4), 2(w/4) + 1 of each chunk,
// each as a float2 stream over the pair's two seeds, the two pairs factored
// side by side so that their dependency chains interleave. Every mbarrier
// wait is bounded.
#include "internal.h"
#include "tc05.cuh"

namespace awsrc {

namespace {

using namespace tc05;

constexpr int BM = 128;             // rows (tiles) per block = TMEM lanes
constexpr int CH = 12;              // seeds per chunk
constexpr int NA = 4 * CH;          // atom columns per chunk (MMA N = 48)
constexpr int NQ = 6 * CH;          // product columns per chunk
constexpr int NQP = 80;             // product columns padded to a multiple of 16 (MMA N)
constexpr int EW = 12;              // epilogue warps: 4 lane quarters x 3 groups of 2 seed pairs
constexpr int PPW = CH / 2 / (EW / 4);  // seed pairs per epilogue warp and chunk
constexpr int NT = 32 * (EW + 1);
constexpr int STAGES = 4;
constexpr uint32_t kABytes = NA * 64 * 2;      // 6 KB
constexpr uint32_t kQBytes = NQP * 64 * 2;     // 10 KB (the last 8 columns zero)
constexpr uint32_t kStageBytes = kABytes + kQBytes;
constexpr uint32_t kTmemCols = 512;            // 2 accumulators of 256 columns
constexpr int kYH = 0, kYL = NA, kDH = 2 * NA, kDL = 2 * NA + NQP;  // columns within an accumulator
static_assert(kDL + NQP <= 256, "accumulator of 256 columns");
constexpr uint32_t kIdA = idesc_f16(BM, NA);
constexpr uint32_t kIdQ = idesc_f16(BM, NQP);
static_assert(PPW == 2 && (EW / 4) * PPW * 2 == CH, "two seed pairs per epilogue warp and chunk");
static_assert(kStageBytes % 1024 == 0 && kABytes % 1024 == 0, "stage layout");

struct Smem {
  __half A[4][BM * 64];  // Y_hi, Y_lo, D_hi, D_lo: canonical K-major, no swizzle
  unsigned char stage[STAGES][kStageBytes];
  float Yst[BM][65];
  float Dst[BM][65];
  float tqc[BM];      // 2^qy * c
  float tqdc[BM];     // 2^qd * c2
  float gd[BM];       // G_pp
  float diag[BM];     // fl(gd + eps)
  float invd0[BM];    // 1 / D_0 = 1 / diag
  float inv_qy[BM], inv_qd[BM];
  int rowok[BM];
  float red_g[EW / 4][BM];
  uint32_t red_s[EW / 4][BM];
  unsigned long long full[STAGES], afull[2], tempty[2];
  uint32_t tmem_base;
};

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

__device__ __forceinline__ int a_offset(int m, int k) {
  return (((m >> 3) * 8 + (k >> 3)) << 7) + ((m & 7) << 4) + ((k & 7) << 1);
}

// Exact sums RN(2048*hi + lo) of two seeds, scaled by a power of two.
__device__ __forceinline__ float2 pair_sum(const float* hi, const float* lo, int i, float2 scale) {
  const float2 u = __ffma2_rn(make_float2(2048.0f, 2048.0f), make_float2(hi[i], hi[i + 1]),
                              make_float2(lo[i], lo[i + 1]));
  return __fmul2_rn(u, scale);
}

__device__ __forceinline__ float2 neg2(float2 v) { return make_float2(-v.x, -v.y); }

__device__ __forceinline__ bool pivot_ok(float d) { return d > 0.0f && d <= 3.402823466e38f; }

// Pivots k of NP pairs: the validity of each (pivot_ok) and rcp_rn of each
// component. When every component of the warp's pairs is in [2^-125, 2^125)
// (positive, normal, finite: hence valid), the hardware approximation and
// Markstein's fused correction y + y (1 - x y) as two packed fmas (each
// component rounds as the scalar form does); otherwise, in a branch the lanes
// take together, the exact checks and __frcp_rn for the components outside.
template <int NP>
__device__ __forceinline__ void pivots_rcp(const float2* x, float2* r, bool* okx, bool* oky) {
  bool fx[NP], fy[NP], in = true;
#pragma unroll
  for (int j = 0; j < NP; ++j) {
    float yx, yy;
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(yx) : "f"(x[j].x));
    asm("rcp.approx.ftz.f32 %0, %1;" : "=f"(yy) : "f"(x[j].y));
    const float2 y = make_float2(yx, yy);
    const float2 e = __ffma2_rn(make_float2(-x[j].x, -x[j].y), y, make_float2(1.0f, 1.0f));
    r[j] = __ffma2_rn(y, e, y);
    fx[j] = __float_as_uint(x[j].x) - 0x01000000u < 0x7D000000u - 0x01000000u;
    fy[j] = __float_as_uint(x[j].y) - 0x01000000u < 0x7D000000u - 0x01000000u;
    in = in && fx[j] && fy[j];
  }
  if (__any_sync(__activemask(), !in)) {
#pragma unroll
    for (int j = 0; j < NP; ++j) {
      okx[j] = okx[j] && pivot_ok(x[j].x);
      oky[j] = oky[j] && pivot_ok(x[j].y);
      if (!fx[j]) r[j].x = __frcp_rn(x[j].x);
      if (!fy[j]) r[j].y = __frcp_rn(x[j].y);
    }
  }
}

// quant_gain_fast2 with the off-diagonal G as it is rather than doubled: each
// off-diagonal term takes q_p * (2 q_r), the exact double of q_p q_r (codes
// are small integers), so that fma(q_p (2 q_r), G, Qq) rounds the same exact
// value as fma(q_p q_r, 2 G, Qq) (|G| <= 2^38 on the tile domain: 2 G is exact).
template <int P>
__device__ __forceinline__ float2 quant_gain_fast2_g(const Prm& pr, const float2* alpha, const float2* bv,
                                                     float2 gd, const float2* Goff) {
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
  float2 q[P], q2[P];
#pragma unroll
  for (int p = 0; p < P; ++p) {
    q[p] = __fadd2_rn(__ffma2_rn(alpha[p], inv, magic), nmagic);
    q2[p] = __fadd2_rn(q[p], q[p]);
  }
  float2 Aq = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int p = 0; p < P; ++p) Aq = __ffma2_rn(q[p], bv[p], Aq);
  float2 Qq = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int p = 0; p < P; ++p) {
    Qq = __ffma2_rn(__fmul2_rn(q[p], q[p]), gd, Qq);
#pragma unroll
    for (int r = p + 1; r < P; ++r) Qq = __ffma2_rn(__fmul2_rn(q[p], q2[r]), Goff[tri(r, p)], Qq);
  }
  const float2 tn = __fmul2_rn(nsc, Qq);
  float2 g = __fmul2_rn(sc, __ffma2_rn(make_float2(2.0f, 2.0f), Aq, tn));
  if (!in0) g.x = -__int_as_float(0x7f800000);
  if (!in1) g.y = -__int_as_float(0x7f800000);
  return g;
}

// Fits of NP seed pairs of this thread's row, factored side by side so that
// their chains interleave; ah/al[j]: atom p of pair j's two seeds at [2p],
// [2p+1]; qh/ql[j]: product q (tri order) at [2q], [2q+1]. Gives b, the
// off-diagonal G, alpha and whether each candidate's pivots are valid.
template <int NP>
__device__ __forceinline__ void pf_fit(const float (*ah)[8], const float (*al)[8], const float (*qh)[12],
                                       const float (*ql)[12], float tqc, float tqdc, float diag, float invd0,
                                       float2 (*bv)[4], float2 (*G)[6], float2 (*alpha)[4], bool* okx, bool* oky) {
  const float2 tq2 = make_float2(tqc, tqc), td2 = make_float2(tqdc, tqdc);
  const float2 dg = make_float2(diag, diag);
  float2 nL[NP][6], E[NP][6], invD[NP][4];
#pragma unroll
  for (int j = 0; j < NP; ++j) {
#pragma unroll
    for (int p = 0; p < 4; ++p) bv[j][p] = pair_sum(ah[j], al[j], 2 * p, tq2);
#pragma unroll
    for (int q = 0; q < 6; ++q) G[j][q] = pair_sum(qh[j], ql[j], 2 * q, td2);
    invD[j][0] = make_float2(invd0, invd0);  // D_0 = diag for every seed
    okx[j] = true;
    oky[j] = true;
  }
  // LDL^T of G + eps I in the recipe's order
#pragma unroll
  for (int k = 1; k < 4; ++k) {
    float2 dk[NP], rk[NP];
#pragma unroll
    for (int jp = 0; jp < NP; ++jp) {
#pragma unroll
      for (int j = 0; j < k; ++j) {
        float2 v = G[jp][tri(k, j)];
#pragma unroll
        for (int i = 0; i < j; ++i) v = __ffma2_rn(nL[jp][tri(k, i)], E[jp][tri(j, i)], v);
        E[jp][tri(k, j)] = v;
        nL[jp][tri(k, j)] = __fmul2_rn(v, neg2(invD[jp][j]));  // -(v * invD_j), exact negation
      }
      dk[jp] = dg;
#pragma unroll
      for (int i = 0; i < k; ++i) dk[jp] = __ffma2_rn(nL[jp][tri(k, i)], E[jp][tri(k, i)], dk[jp]);
    }
    pivots_rcp<NP>(dk, rk, okx, oky);
#pragma unroll
    for (int jp = 0; jp < NP; ++jp) invD[jp][k] = rk[jp];
  }
#pragma unroll
  for (int j = 0; j < NP; ++j) ldl_solve2<4>(nL[j], invD[j], bv[j], alpha[j]);
}

// Gains of NP seed pairs (operands as for pf_fit).
template <bool FAST, int NP>
__device__ __forceinline__ void pf_gain(const Prm& pr, const float (*ah)[8], const float (*al)[8],
                                        const float (*qh)[12], const float (*ql)[12], float tqc, float tqdc,
                                        float gd, float diag, float invd0, float2* g,
                                        float2 (*alpha_out)[4] = nullptr) {
  float2 bv[NP][4], G[NP][6], alpha[NP][4];
  bool okx[NP], oky[NP];
  pf_fit<NP>(ah, al, qh, ql, tqc, tqdc, diag, invd0, bv, G, alpha, okx, oky);
#pragma unroll
  for (int j = 0; j < NP; ++j) {
    if (alpha_out) {
#pragma unroll
      for (int p = 0; p < 4; ++p) alpha_out[j][p] = alpha[j][p];
    }
    if constexpr (FAST) {
      g[j] = quant_gain_fast2_g<4>(pr, alpha[j], bv[j], make_float2(gd, gd), G[j]);
    } else {
      float q4[4];
      int sf;
      float Gx[6], a[4], b[4];
#pragma unroll
      for (int i = 0; i < 6; ++i) Gx[i] = G[j][i].x;
#pragma unroll
      for (int p = 0; p < 4; ++p) { a[p] = alpha[j][p].x; b[p] = bv[j][p].x; }
      g[j].x = quant_gain<4>(pr, a, b, gd, Gx, q4, &sf);
#pragma unroll
      for (int i = 0; i < 6; ++i) Gx[i] = G[j][i].y;
#pragma unroll
      for (int p = 0; p < 4; ++p) { a[p] = alpha[j][p].y; b[p] = bv[j][p].y; }
      g[j].y = quant_gain<4>(pr, a, b, gd, Gx, q4, &sf);
    }
    if (!okx[j]) g[j].x = neg_inf();
    if (!oky[j]) g[j].y = neg_inf();
  }
}

// Codes and scale field of the winning seed of row m. The search keeps only
// (gain, seed), so the seed's correlations with Y (atoms) and D (atom
// products) are formed again as the exact integer sums the tensor cores
// accumulate, split into hi/lo so that 2048*hi + lo is the sum and the fma of
// pair_sum rounds it once, and go through the same fit and quantiser. Both
// halves of the pair get the winner's sums; one is read. Returns the gain
// once more, which must equal the one the search found.
template <bool FAST>
__device__ __forceinline__ float pf_winner(const Prm& pr, const Smem& sm, int m, const uint64_t* mk, bool odd,
                                           uint32_t* cw, int* sf) {
  const float iy = sm.inv_qy[m], idd = sm.inv_qd[m];
  uint64_t w[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) w[p] = mk[p];
  uint64_t wq[6];
#pragma unroll
  for (int a = 1, q = 0; a < 4; ++a)
#pragma unroll
    for (int c = 0; c < a; ++c, ++q) wq[q] = w[a] ^ w[c];  // products in tri order
  int ty = 0, td = 0, ny[4] = {0, 0, 0, 0}, nd[6] = {0, 0, 0, 0, 0, 0};
  for (int j = 0; j < 64; ++j) {
    const int y = iy == 0.0f ? 0 : fixed_point_int(sm.Yst[m][j], iy);
    const int d = idd == 0.0f ? 0 : fixed_point_int(sm.Dst[m][j], idd);
    ty += y;
    td += d;
#pragma unroll
    for (int p = 0; p < 4; ++p) ny[p] += ((w[p] >> j) & 1ull) ? y : 0;
#pragma unroll
    for (int q = 0; q < 6; ++q) nd[q] += ((wq[q] >> j) & 1ull) ? d : 0;
  }
  float ah[1][8], al[1][8], qh[1][12], ql[1][12];
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const int u = ty - 2 * ny[p];  // |u| <= 64 * 2^21
    ah[0][2 * p] = ah[0][2 * p + 1] = (float)(u >> 11);
    al[0][2 * p] = al[0][2 * p + 1] = (float)(u & 2047);
  }
#pragma unroll
  for (int q = 0; q < 6; ++q) {
    const int u = td - 2 * nd[q];
    qh[0][2 * q] = qh[0][2 * q + 1] = (float)(u >> 11);
    ql[0][2 * q] = ql[0][2 * q + 1] = (float)(u & 2047);
  }
  float2 alpha[1][4], g;
  pf_gain<FAST, 1>(pr, ah, al, qh, ql, sm.tqc[m], sm.tqdc[m], sm.gd[m], sm.diag[m], sm.invd0[m], &g, alpha);
  float a[4], q4[4], zero[6] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int p = 0; p < 4; ++p) a[p] = odd ? alpha[0][p].y : alpha[0][p].x;
  if constexpr (FAST) (void)quant_gain_fast<4>(pr, a, zero, 0.0f, zero, q4, sf);
  else (void)quant_gain<4>(pr, a, zero, 0.0f, zero, q4, sf);
  uint32_t c = 0u;
#pragma unroll
  for (int p = 0; p < 4; ++p) c |= ((uint32_t)(int)q4[p] & 0xFFu) << (8 * p);
  *cw = c;
  return odd ? g.y : g.x;
}

template <bool FAST>
__global__ void __launch_bounds__(NT, 1)
    search_pf_kernel(Prm pr, LaunchDesc ld, const unsigned char* __restrict__ atoms,
                     const unsigned char* __restrict__ prods, const uint64_t* __restrict__ masks,
                     awsrc_candidate* __restrict__ cands, uint32_t* __restrict__ status) {
  extern __shared__ unsigned char smem_raw[];
  // 1 KB aligned through an integer cast, which leaves the accesses generic:
  // measured faster here than the shared-space form the U search uses
  Smem& sm = *reinterpret_cast<Smem*>((reinterpret_cast<uintptr_t>(smem_raw) + 1023) & ~uintptr_t(1023));
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int mi = find_mod(ld, blockIdx.x);
  const ModDesc& md = ld.m[mi];
  const int64_t b = blockIdx.x - md.block_off;
  const int z = (int)(b % md.nsplit);
  const int64_t rest = b / md.nsplit;
  const int64_t rb = rest % md.n_rb;
  const int64_t cb = rest / md.n_rb;

  const int nchunks = pr.S_pad / CH;
  const int per = (nchunks + md.nsplit - 1) / md.nsplit;
  const int c0 = min(nchunks, z * per);
  const int c1 = min(nchunks, c0 + per);
  const int nck = c1 - c0;
  const unsigned char* a_src = atoms + (size_t)c0 * kABytes;
  const unsigned char* q_src = prods + (size_t)c0 * kQBytes;

  if (warp == EW) {
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(&sm.tmem_base)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
    if (lane == 0) {
      for (int i = 0; i < STAGES; ++i) mbar_init(&sm.full[i], 1);
      for (int i = 0; i < 2; ++i) {
        mbar_init(&sm.afull[i], 1);
        mbar_init(&sm.tempty[i], EW);
      }
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    tc_fence_before();
  }
  if (tid < BM) sm.rowok[tid] = 1;
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  int issued = 0;
  if (warp == EW && lane == 0) {
    for (; issued < STAGES && issued < nck; ++issued) {
      mbar_expect_tx(&sm.full[issued], kStageBytes);
      bulk_g2s(&sm.stage[issued][0], a_src + (size_t)issued * kABytes, kABytes, &sm.full[issued]);
      bulk_g2s(&sm.stage[issued][kABytes], q_src + (size_t)issued * kQBytes, kQBytes, &sm.full[issued]);
    }
  }
  // stage y = d * r and d, d = w_act * a + w_fisher * F (per element)
  for (int e = tid; e < BM * 64; e += NT) {
    const int r = e >> 6, j = e & 63;
    const int64_t row = rb * BM + r;
    float y = 0.0f, d = 0.0f;
    if (row < md.rows) {
      const int64_t idx = row * md.cols + cb * 64 + j;
      const float rr = __fsub_rn(load_elem(md.W, idx, md.w_dtype), load_elem(md.W0, idx, md.w0_dtype));
      d = __fadd_rn(__fmul_rn(md.w_act, md.act[cb * 64 + j]), __fmul_rn(md.w_fisher, md.fisher[idx]));
      if (!in_domain(rr, d)) sm.rowok[r] = 0;
      y = __fmul_rn(d, rr);
    }
    sm.Yst[r][j] = y;
    sm.Dst[r][j] = d;
  }
  __syncthreads();
  if (tid < BM) {  // per row: fixed-point exponents, gd, eps and the first pivot
    float my = 0.0f, mdd = 0.0f;
    for (int j = 0; j < 64; ++j) {
      my = fmaxf(my, fabsf(sm.Yst[tid][j]));
      mdd = fmaxf(mdd, fabsf(sm.Dst[tid][j]));
    }
    int qy, qd;
    const float iy = fixed_point_inv(my, &qy);
    const float idd = fixed_point_inv(mdd, &qd);
    const float two_qd = pow2f(qd);
    int sd = 0;
    for (int j = 0; j < 64; ++j) sd += idd == 0.0f ? 0 : fixed_point_int(sm.Dst[tid][j], idd);
    const float gd = __fmul_rn(pr.c2, __fmul_rn(__int2float_rn(sd), two_qd));
    const float eps = __fmul_rn(pr.ridge_rel, gd);
    const float diag = __fadd_rn(gd, eps);
    const bool ok = sm.rowok[tid] && pivot_ok(diag);
    sm.rowok[tid] = ok ? 1 : 0;
    sm.inv_qy[tid] = ok ? iy : 0.0f;
    sm.inv_qd[tid] = ok ? idd : 0.0f;
    sm.tqc[tid] = __fmul_rn(pow2f(qy), pr.c);
    sm.tqdc[tid] = __fmul_rn(two_qd, pr.c2);
    sm.gd[tid] = gd;
    sm.diag[tid] = diag;
    sm.invd0[tid] = __frcp_rn(diag);
  }
  __syncthreads();
  // A operands: one thread writes one 16-byte core-matrix row of both halves
  for (int e = tid; e < 2 * BM * 8; e += NT) {
    const int which = e >= BM * 8;  // 0: Y, 1: D
    const int ee = e - which * BM * 8;
    const int m = ee >> 3, k0 = (ee & 7) * 8;
    const float inv = which ? sm.inv_qd[m] : sm.inv_qy[m];
    const float* src = which ? &sm.Dst[m][k0] : &sm.Yst[m][k0];
    uint32_t wh[4], wl[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int x0 = inv == 0.0f ? 0 : fixed_point_int(src[2 * i], inv);
      const int x1 = inv == 0.0f ? 0 : fixed_point_int(src[2 * i + 1], inv);
      wh[i] = (uint32_t)__half_as_ushort(__int2half_rn(x0 >> 11)) |
              ((uint32_t)__half_as_ushort(__int2half_rn(x1 >> 11)) << 16);
      wl[i] = (uint32_t)__half_as_ushort(__int2half_rn(x0 & 2047)) |
              ((uint32_t)__half_as_ushort(__int2half_rn(x1 & 2047)) << 16);
    }
    const int off = a_offset(m, k0);
    *reinterpret_cast<uint4*>(reinterpret_cast<unsigned char*>(sm.A[2 * which]) + off) =
        make_uint4(wh[0], wh[1], wh[2], wh[3]);
    *reinterpret_cast<uint4*>(reinterpret_cast<unsigned char*>(sm.A[2 * which + 1]) + off) =
        make_uint4(wl[0], wl[1], wl[2], wl[3]);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
  __syncthreads();

  bool timed_out = false;
  if (warp == EW) {
    // ------------------------------------------------------------ producer --
    if (lane == 0) {
      uint32_t ab[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) ab[i] = smem_addr(sm.A[i]);
      int k = 0;
      for (; k < nck; ++k) {
        const int st = k % STAGES, tb = k & 1;
        if (!mbar_wait(&sm.full[st], (uint32_t)((k / STAGES) & 1), pr.wait_ns)) { timed_out = true; break; }
        if (k >= 2 && !mbar_wait(&sm.tempty[tb], (uint32_t)(((k - 2) >> 1) & 1), pr.wait_ns)) { timed_out = true; break; }
        tc_fence_after();
        const uint32_t sa = smem_addr(&sm.stage[st][0]), sq = sa + kABytes;
        const uint32_t acc = tmem + (uint32_t)(tb * 256);
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          const uint32_t kb = (uint32_t)ks * 256u, en = ks > 0 ? 1u : 0u;
          umma_f16(acc + kYH, smem_desc(ab[0] + kb), smem_desc(sa + kb), kIdA, en);
          umma_f16(acc + kYL, smem_desc(ab[1] + kb), smem_desc(sa + kb), kIdA, en);
          umma_f16(acc + kDH, smem_desc(ab[2] + kb), smem_desc(sq + kb), kIdQ, en);
          umma_f16(acc + kDL, smem_desc(ab[3] + kb), smem_desc(sq + kb), kIdQ, en);
        }
        umma_commit(&sm.afull[tb]);
        if (k >= 2 && issued < nck) {
          // chunk k+2 takes the stage of chunk k-2, whose MMAs completed before
          // its accumulator was loaded (tempty above)
          const int ps = (k - 2) % STAGES;
          mbar_expect_tx(&sm.full[ps], kStageBytes);
          bulk_g2s(&sm.stage[ps][0], a_src + (size_t)issued * kABytes, kABytes, &sm.full[ps]);
          bulk_g2s(&sm.stage[ps][kABytes], q_src + (size_t)issued * kQBytes, kQBytes, &sm.full[ps]);
          ++issued;
        }
      }
      if (timed_out) {
        for (int j = max(0, issued - STAGES); j < issued; ++j)
          (void)mbar_wait(&sm.full[j % STAGES], (uint32_t)((j / STAGES) & 1), pr.wait_ns);
        if (k > 0) (void)mbar_wait(&sm.afull[(k - 1) & 1], (uint32_t)(((k - 1) >> 1) & 1), pr.wait_ns);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue --
    const int m = 32 * (warp & 3) + lane;
    const int grp = warp >> 2;  // seed pairs 2 grp and 2 grp + 1 of each chunk
    const uint32_t lane_base = (uint32_t)(32 * (warp & 3)) << 16;
    const float tqc = sm.tqc[m], tqdc = sm.tqdc[m], gd = sm.gd[m], diag = sm.diag[m], invd0 = sm.invd0[m];
    float bg = neg_inf();
    uint32_t bsd = 0xffffffffu;
    for (int k = 0; k < nck; ++k) {
      const int tb = k & 1;
      if (!mbar_wait(&sm.afull[tb], (uint32_t)((k >> 1) & 1), pr.wait_ns)) { timed_out = true; break; }
      tc_fence_after();
      const uint32_t base = tmem + lane_base + (uint32_t)(tb * 256);
      // both pairs' columns are loaded before the accumulator is released, so
      // the next MMAs into it wait for no scoring; a pair's 12 product columns
      // start at 12 pi, 8-aligned for the even pair, 4 past for the odd one
      float ah[2][8], al[2][8], qh[2][12], ql[2][12];
      const int p0 = 2 * grp, p1 = p0 + 1;
      tmem_ld8(base + kYH + 8 * p0, ah[0]);
      tmem_ld8(base + kYL + 8 * p0, al[0]);
      tmem_ld8(base + kDH + 12 * p0, qh[0]);
      tmem_ld4(base + kDH + 12 * p0 + 8, qh[0] + 8);
      tmem_ld8(base + kDL + 12 * p0, ql[0]);
      tmem_ld4(base + kDL + 12 * p0 + 8, ql[0] + 8);
      tmem_ld8(base + kYH + 8 * p1, ah[1]);
      tmem_ld8(base + kYL + 8 * p1, al[1]);
      tmem_ld4(base + kDH + 12 * p1, qh[1]);
      tmem_ld8(base + kDH + 12 * p1 + 4, qh[1] + 4);
      tmem_ld4(base + kDL + 12 * p1, ql[1]);
      tmem_ld8(base + kDL + 12 * p1 + 4, ql[1] + 4);
      asm volatile("tcgen05.wait::ld.sync.aligned;" ::: "memory");
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        tmem_tie8(ah[j]);
        tmem_tie8(al[j]);
#pragma unroll
        for (int i = 0; i < 3; ++i) { tmem_tie4(qh[j] + 4 * i); tmem_tie4(ql[j] + 4 * i); }
      }
      tc_fence_before();
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.tempty[tb]);
      float2 g2[2];
      pf_gain<FAST, 2>(pr, ah, al, qh, ql, tqc, tqdc, gd, diag, invd0, g2);
#pragma unroll
      for (int j = 0; j < 2; ++j) {
        float2 g = g2[j];
        const int sx = (c0 + k) * CH + 2 * (p0 + j);
        if (sx + 1 >= pr.S) {  // padding selectors (all-zero masks) are not candidates
          if (sx >= pr.S) g.x = neg_inf();
          g.y = neg_inf();
        }
        // seeds reach a thread in increasing order: a strictly greater gain wins
        const float cm = fmaxf(g.x, g.y);
        if (cm > bg) {
          bg = cm;
          bsd = (uint32_t)(sx + (g.x == cm ? 0 : 1));
        }
      }
    }
    sm.red_g[grp][m] = bg;
    sm.red_s[grp][m] = bsd;
  }
  tc_fence_before();
  if (__syncthreads_or(timed_out)) {
    if (tid == 0) atomicOr(status, kFaultTimeout);
  } else if (tid < BM) {
    float g = sm.red_g[0][tid];
    uint32_t s = sm.red_s[0][tid];
#pragma unroll
    for (int i = 1; i < EW / 4; ++i) {
      if (better(sm.red_g[i][tid], sm.red_s[i][tid], g, s)) { g = sm.red_g[i][tid]; s = sm.red_s[i][tid]; }
    }
    const int64_t row = rb * BM + tid;
    if (row < md.rows) {
      const int64_t tt = md.tile_off + row * md.n_cb + cb;
      const bool valid = sm.rowok[tid] && g > neg_inf();
      uint32_t cw = 0u;
      int sf = 0;
      if (valid) {
        const float gw = pf_winner<FAST>(pr, sm, tid, masks + (size_t)s * 4, (s & 1u) != 0u, &cw, &sf);
        if (__float_as_uint(gw) != __float_as_uint(g)) atomicOr(status, kFaultSelfCheck);
      }
      awsrc_candidate cd;
      cd.gain = valid ? g : neg_inf();
      cd.seed = valid ? (uint16_t)s : (uint16_t)0;
      cd.scale = (int16_t)sf;
#pragma unroll
      for (int p = 0; p < 4; ++p) cd.code[p] = (int8_t)(cw >> (8 * p));
#pragma unroll
      for (int p = 4; p < 8; ++p) cd.code[p] = 0;
      cands[(size_t)z * ld.T + tt] = cd;
    }
  }
  if (warp == EW) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(tmem), "r"(kTmemCols)
                 : "memory");
  }
}

// FP16 products of atom pairs in the order the MMAs read them: chunk c
// (12 seeds) is an 80 x 64 K-major operand in 10 KB; item i (16 bytes, one
// core-matrix row) is chunk i / 640, column group n8 = (i >> 6) % 10, k group
// (i >> 3) & 7, row i & 7; column n = 8*n8 + r < 72 carries product q =
// (n % 12) / 2 (pairs (1,0), (2,0), (2,1), (3,0), (3,1), (3,2)) of seed
// 12c + 2*(n / 12) + n % 2, and columns 72 .. 79 are zero.
constexpr int kQItems = NQP * 8;  // 16-byte items per chunk

__global__ void products_kernel(const uint64_t* __restrict__ masks, uint4* __restrict__ out, int S_pad) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t n_items = (int64_t)(S_pad / CH) * kQItems;
  if (i >= n_items) return;
  const int64_t chunk = i / kQItems;
  const int w = (int)(i % kQItems);
  const int r = w & 7, kg = (w >> 3) & 7, n8 = w >> 6;
  const int n = 8 * n8 + r;
  if (n >= NQ) {
    out[i] = make_uint4(0u, 0u, 0u, 0u);
    return;
  }
  const int q = (n % 12) >> 1;
  const int64_t seed = chunk * CH + 2 * (n / 12) + (n & 1);
  const int pa = q < 1 ? 1 : (q < 3 ? 2 : 3);
  const int pb = q - (pa * (pa - 1)) / 2;
  const uint64_t m = masks[(size_t)seed * 4 + pa] ^ masks[(size_t)seed * 4 + pb];
  uint32_t wv[4];
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    const int k = 8 * kg + 2 * h;
    const uint32_t lo = ((m >> k) & 1ull) ? 0xBC00u : 0x3C00u;  // -1 : +1 in FP16
    const uint32_t hi = ((m >> (k + 1)) & 1ull) ? 0xBC00u : 0x3C00u;
    wv[h] = lo | (hi << 16);
  }
  out[i] = make_uint4(wv[0], wv[1], wv[2], wv[3]);
}

}  // namespace

int search_pf_c64p4_chunk() { return CH; }
size_t search_pf_c64p4_table_bytes(int S_pad) { return (size_t)(S_pad / CH) * kQBytes; }

cudaError_t launch_products_pf_c64p4(const Prm& pr, const uint64_t* masks, void* out, cudaStream_t st) {
  const int64_t n = (int64_t)(pr.S_pad / CH) * kQItems;
  products_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(masks, static_cast<uint4*>(out), pr.S_pad);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_search_pf_c64p4(const Prm& pr, const LaunchDesc& ld, const void* atoms, const void* prods,
                                   const uint64_t* masks, int64_t n_blocks, awsrc_candidate* cands,
                                   uint32_t* status, cudaStream_t st) {
  const size_t smem = sizeof(Smem) + 1024;
  auto kern = pr.fast_pow2 ? search_pf_kernel<true> : search_pf_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<(unsigned)n_blocks, NT, smem, st>>>(pr, ld, static_cast<const unsigned char*>(atoms),
                                             static_cast<const unsigned char*>(prods), masks, cands, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
