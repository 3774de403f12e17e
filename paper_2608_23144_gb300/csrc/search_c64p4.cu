// search_c64p4.cu — seed search (Sec. 3.2) specialised for C = 64, P = 4, AWSRC-U,
// with the correlation on the fifth-generation tensor cores (tcgen05, TMEM).
//
// The correlation u = B_s^T (D r) of Eq. 3 is an exact integer sum on the
// tile's fixed-point grid: Y_j = rint(y_j 2^-q) with |Y_j| <= 2^21, split as
// Y = 2048*Y_hi + Y_lo with Y_hi in [-1024, 1024] and Y_lo in [0, 2047]. Both
// halves and the +-1 atoms are exact in FP16, every product is exact, and every
// partial sum of 64 terms is an integer below 2^17, so FP32 accumulation on the
// tensor cores is exact in any order. The epilogue forms
// b = RN(2048*S_hi + S_lo) * (2^q c) — the correctly rounded exact sum, one
// rounding, scaled exactly (c = 1/8 and 2^q >= 2^-120 keep the product normal).
//
// Block: 128 rows (tiles of one column block; row m = TMEM lane m) and 17 warps.
//  * Warp 16 (producer): one thread streams each chunk of 32 seeds — FP16 atoms
//    in the canonical K-major layout (16 KB) and the chunk's paired Gram factors
//    (2.8 KB) — by bulk copies into a 4-stage shared-memory ring, and issues the
//    chunk's 8 MMAs (M = 128, N = 128, K = 16; halves hi and lo, 4 k-steps) into
//    one of two 256-column TMEM accumulators, committed to an mbarrier. Chunk
//    k's MMAs wait only until every epilogue warp has loaded chunk k-2 from
//    that accumulator; chunk k-2's stage is refilled once every warp has also
//    finished reading its factors (two release barriers).
//  * Warps 0..15 (epilogue): warp w reads TMEM lanes 32(w%4).. (its threads'
//    rows) and the columns of seeds 8(w/4)..8(w/4)+7 of each chunk, and runs the
//    fit / quantise / score epilogue on seed pairs as float2 streams, keeping a
//    running (gain, seed) argmax per row. The four warps of a row publish
//    their running best gains in shared memory and prune against the largest;
//    they merge at the end, form the winner's codes again and write the
//    tile's candidate.
// Columns of a chunk are seed-pair major: column 8i + 2p + e holds atom p of
// seed 2i + e, so one 32x32b.x8 TMEM load gives a thread one seed pair with
// each atom's two seeds in adjacent registers; the next pair's loads (and
// bound factors) are in flight while a pair is scored.
// One CTA per SM takes tile blocks blockIdx.x, blockIdx.x + gridDim.x, ...:
// it holds its TMEM allocation across them, initialises its barriers again
// for each, and prefetches the next tile block's W and W0 rows into L2 while
// one is searched.
// Every mbarrier wait is bounded in time; on expiry the CTA records a timeout
// fault, waits (bounded) for its own copies and MMAs in flight, takes no
// further tile block, frees its TMEM and returns. A test of that path
// (Prm::stall_chunk >= 0) makes the producer issue no copies from that chunk
// of its range on, with a short limit, so that the producer's wait for the
// chunk's copies and the epilogue's wait for its MMAs both run out.
#include "internal.h"
#include "tc05.cuh"

namespace awsrc {

namespace {

using namespace tc05;

constexpr int BM = 128;             // rows (tiles) per block = TMEM lanes
constexpr int CH = 32;              // seeds per chunk
constexpr int NCOL = 4 * CH;        // MMA N: 128 columns per half
constexpr int EW = 16;              // epilogue warps
constexpr int NT = 32 * (EW + 1);   // + the producer warp
constexpr int SUBS = EW / 4;        // epilogue warps per TMEM lane quarter
constexpr int SUB_PAIRS = CH / 2 / SUBS;  // seed pairs of a chunk per epilogue warp
static_assert(EW % 4 == 0 && SUB_PAIRS >= 1, "epilogue mapping");
constexpr int STAGES = 4;
constexpr int PS = pair_stride(4);  // 22 float2 per seed pair
constexpr uint32_t kBBytes = NCOL * 64 * 2;        // 16 KB of FP16 atoms per chunk
constexpr uint32_t kPBytes = (CH / 2) * PS * 8u;   // 2816 B of paired factors per chunk
constexpr uint32_t kStageBytes = 19456;            // B at 0, factors at kBBytes (1 KB multiple)
constexpr uint32_t kTmemCols = 512;                // 2 accumulators x (hi, lo) x 128 columns
static_assert(kBBytes + kPBytes <= kStageBytes, "stage layout");

constexpr uint32_t kIdesc = idesc_f16(BM, NCOL);

struct Smem {
  __half A[2][BM * 64];                   // Y_hi, Y_lo: canonical K-major, no swizzle
  unsigned char stage[STAGES][kStageBytes];
  float Yst[BM][65];
  float two_q[BM];
  float inv_q[BM];
  int rowok[BM];
  float red_g[SUBS][BM];
  uint32_t red_s[SUBS][BM];
  float cur_g[SUBS][BM];                  // running best gain of each (sub, row) in u units, for pruning
  unsigned long long full[STAGES];        // bulk copies of a chunk landed
  unsigned long long afull[2];            // MMAs of a chunk completed (tcgen05.commit)
  unsigned long long aempty[2];           // epilogue warps done loading an accumulator
  unsigned long long sempty[STAGES];      // epilogue warps done with a stage's factors
  uint32_t tmem_base;
};

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

// Byte offset of element (m, k) of a 128x64 FP16 operand in the canonical
// K-major no-swizzle layout: core matrix (m/8, k/8) at ((m/8)*8 + k/8)*128.
__device__ __forceinline__ int a_offset(int m, int k) {
  return (((m >> 3) * 8 + (k >> 3)) << 7) + ((m & 7) << 4) + ((k & 7) << 1);
}

// Pruning bound of one seed pair for this thread's row, in the units of the
// unscaled correlations u = b / (2^q c) (c 2^q is a power of two for C = 64,
// so the comparison against a threshold scaled by (2^q c)^-2 is exact). hi/lo
// hold atom p of the two seeds at [2p], [2p+1]; u = RN(2048 hi + lo) is the
// exact integer correlation rounded once. pe points at the pair's factors
// (-L, then invD m rounded up). Returns U = u^T (G + eps I)^-1 u times the
// seed's bound multiplier, as z^T (z * invD m) with z = L^-1 u: a sum of
// non-negative terms.
__device__ __forceinline__ float2 pair_bound(const float* hi, const float* lo, const float4* pf, float2* u) {
  float2 pv[10];
#pragma unroll
  for (int i = 0; i < 5; ++i) {
    const float4 v = pf[i];
    pv[2 * i] = make_float2(v.x, v.y);
    pv[2 * i + 1] = make_float2(v.z, v.w);
  }
  const float2* nL = pv;
  const float2* invDm = pv + 6;
#pragma unroll
  for (int p = 0; p < 4; ++p)
    u[p] = __ffma2_rn(make_float2(2048.0f, 2048.0f), make_float2(hi[2 * p], hi[2 * p + 1]),
                      make_float2(lo[2 * p], lo[2 * p + 1]));
  float2 z[4];
  float2 U = make_float2(0.0f, 0.0f);
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    float2 v = u[k];
#pragma unroll
    for (int i = 0; i < k; ++i) v = __ffma2_rn(nL[tri(k, i)], z[i], v);
    z[k] = v;
    const float2 wm = __fmul2_rn(v, invDm[k]);
    U = k == 0 ? __fmul2_rn(v, wm) : __ffma2_rn(v, wm, U);
  }
  return U;
}

// Forward half of the ridge solve in the recipe's units: b = u (2^q c),
// z = L^-1 b and w = D^-1 z, so that alpha = L^-T w.
__device__ __forceinline__ void pair_forward(const float2* u, float2 tqc, const float4* pl, const float4* pe,
                                             float2* bv, float2* w) {
  float2 nL[6], invD[4];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const float4 v = pl[i];
    nL[2 * i] = make_float2(v.x, v.y);
    nL[2 * i + 1] = make_float2(v.z, v.w);
  }
#pragma unroll
  for (int i = 0; i < 2; ++i) {
    const float4 v = pe[5 + i];
    invD[2 * i] = make_float2(v.x, v.y);
    invD[2 * i + 1] = make_float2(v.z, v.w);
  }
#pragma unroll
  for (int p = 0; p < 4; ++p) bv[p] = __fmul2_rn(u[p], tqc);
  float2 z[4];
#pragma unroll
  for (int k = 0; k < 4; ++k) {
    float2 v = bv[k];
#pragma unroll
    for (int i = 0; i < k; ++i) v = __ffma2_rn(nL[tri(k, i)], z[i], v);
    z[k] = v;
    w[k] = __fmul2_rn(v, invD[k]);
  }
}

// Back half of the solve: alpha = L^-T w, in the order of ldl_solve2.
__device__ __forceinline__ void pair_back(const float4* pl, const float2* w, float2* alpha) {
  float2 nL[6];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const float4 v = pl[i];
    nL[2 * i] = make_float2(v.x, v.y);
    nL[2 * i + 1] = make_float2(v.z, v.w);
  }
#pragma unroll
  for (int k = 3; k >= 0; --k) {
    float2 v = w[k];
#pragma unroll
    for (int i = k + 1; i < 4; ++i) v = __ffma2_rn(nL[tri(i, k)], alpha[i], v);
    alpha[k] = v;
  }
}

template <bool FAST>
__device__ __forceinline__ float2 pair_gain(const Prm& pr, const float2* bv, const float2* alpha,
                                            const float4* pe) {
  float2 Go[6];
#pragma unroll
  for (int i = 0; i < 3; ++i) {
    const float4 v = pe[7 + i];
    Go[2 * i] = make_float2(v.x, v.y);
    Go[2 * i + 1] = make_float2(v.z, v.w);
  }
  const float4 v10 = pe[10];
  const float2 gd = make_float2(v10.x, v10.y);
  if constexpr (FAST) {
    return quant_gain_fast2<4>(pr, alpha, bv, gd, Go);  // G off-diagonal doubled
  } else {
    float2 g;
    float q[4];
    int sf;
    float G[6], a[4], bb[4];
#pragma unroll
    for (int i = 0; i < 6; ++i) G[i] = Go[i].x;
#pragma unroll
    for (int p = 0; p < 4; ++p) { a[p] = alpha[p].x; bb[p] = bv[p].x; }
    g.x = quant_gain<4>(pr, a, bb, gd.x, G, q, &sf);
#pragma unroll
    for (int i = 0; i < 6; ++i) G[i] = Go[i].y;
#pragma unroll
    for (int p = 0; p < 4; ++p) { a[p] = alpha[p].y; bb[p] = bv[p].y; }
    g.y = quant_gain<4>(pr, a, bb, gd.y, G, q, &sf);
    return g;
  }
}

// Codes and scale field of the winning seed of row m. The search keeps only
// (gain, seed), so the seed's correlations are formed again here as the exact
// integer sums sum_j +-Y_j that the tensor cores accumulate (hi/lo split so
// that 2048*hi + lo is that sum and the fma of pair_forward rounds it once),
// then go through the same solve and quantiser instructions as in the search.
// The pair's other half gets the same correlations and is ignored. Returns the
// gain once more, which must equal the one the search found.
template <bool FAST>
__device__ __forceinline__ float winner_codes(const Prm& pr, const Smem& sm, int m, const uint64_t* mk,
                                              const float4* pe, bool odd, uint32_t* cw, int* sf) {
  const float inv = sm.inv_q[m];
  uint64_t w[4];
#pragma unroll
  for (int p = 0; p < 4; ++p) w[p] = mk[p];
  int tot = 0, neg[4] = {0, 0, 0, 0};
  for (int j = 0; j < 64; ++j) {
    const int y = inv == 0.0f ? 0 : fixed_point_int(sm.Yst[m][j], inv);
    tot += y;
#pragma unroll
    for (int p = 0; p < 4; ++p) neg[p] += ((w[p] >> j) & 1ull) ? y : 0;
  }
  float hi[8], lo[8];
#pragma unroll
  for (int p = 0; p < 4; ++p) {
    const int u = tot - 2 * neg[p];  // |u| <= 64 * 2^21
    hi[2 * p] = hi[2 * p + 1] = (float)(u >> 11);
    lo[2 * p] = lo[2 * p + 1] = (float)(u & 2047);
  }
  const float tq = __fmul_rn(sm.two_q[m], pr.c);
  float2 u[4], bv[4], wv[4], al[4];
#pragma unroll
  for (int p = 0; p < 4; ++p)
    u[p] = __ffma2_rn(make_float2(2048.0f, 2048.0f), make_float2(hi[2 * p], hi[2 * p + 1]),
                      make_float2(lo[2 * p], lo[2 * p + 1]));
  pair_forward(u, make_float2(tq, tq), pe, pe, bv, wv);
  pair_back(pe, wv, al);
  float a[4], q[4], zero[6] = {0.0f, 0.0f, 0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
  for (int p = 0; p < 4; ++p) a[p] = odd ? al[p].y : al[p].x;
  if constexpr (FAST) (void)quant_gain_fast<4>(pr, a, zero, 0.0f, zero, q, sf);
  else (void)quant_gain<4>(pr, a, zero, 0.0f, zero, q, sf);
  uint32_t c = 0u;
#pragma unroll
  for (int p = 0; p < 4; ++p) c |= ((uint32_t)(int)q[p] & 0xFFu) << (8 * p);
  *cw = c;
  const float2 g = pair_gain<FAST>(pr, bv, al, pe);
  return odd ? g.y : g.x;
}

// Tile block blk of the launch: rows 128 rb .. of column block cb of its
// module, split z of the seeds.
struct BlockPos {
  int mi, z;
  int64_t rb, cb;
};

__device__ __forceinline__ BlockPos block_pos(const LaunchDesc& ld, int64_t blk) {
  BlockPos p;
  p.mi = find_mod(ld, blk);
  const ModDesc& md = ld.m[p.mi];
  const int64_t b = blk - md.block_off;
  p.z = (int)(b % md.nsplit);
  const int64_t rest = b / md.nsplit;
  p.rb = rest % md.n_rb;
  p.cb = rest / md.n_rb;
  return p;
}

// Starts the L2 fills of tile block blk's W and W0 rows (one 128-byte row
// segment per thread and matrix), so that its staging finds them on chip.
__device__ __forceinline__ void prefetch_block(const LaunchDesc& ld, int64_t blk, int tid) {
  if (tid >= BM) return;
  const BlockPos p = block_pos(ld, blk);
  const ModDesc& md = ld.m[p.mi];
  const int64_t row = p.rb * BM + tid;
  if (row >= md.rows) return;
  const int64_t idx = row * md.cols + p.cb * 64;
  const char* w = static_cast<const char*>(md.W) + idx * (md.w_dtype == AWSRC_DTYPE_F32 ? 4 : 2);
  const char* w0 = static_cast<const char*>(md.W0) + idx * (md.w0_dtype == AWSRC_DTYPE_F32 ? 4 : 2);
  asm volatile("prefetch.global.L2 [%0];" ::"l"(w));
  asm volatile("prefetch.global.L2 [%0];" ::"l"(w0));
  if (md.w_dtype == AWSRC_DTYPE_F32) asm volatile("prefetch.global.L2 [%0];" ::"l"(w + 128));
  if (md.w0_dtype == AWSRC_DTYPE_F32) asm volatile("prefetch.global.L2 [%0];" ::"l"(w0 + 128));
}

template <bool FAST>
__device__ __forceinline__ bool search_block(const Prm& pr, const LaunchDesc& ld, int64_t blk, Smem& sm,
                                             const uint4* __restrict__ atoms, const float2* __restrict__ pairs,
                                             const uint64_t* __restrict__ masks, awsrc_candidate* __restrict__ cands,
                                             uint32_t* __restrict__ status) {
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int mi = find_mod(ld, blk);
  const ModDesc& md = ld.m[mi];
  const int64_t b = blk - md.block_off;
  const int z = (int)(b % md.nsplit);
  const int64_t rest = b / md.nsplit;
  const int64_t rb = rest % md.n_rb;
  const int64_t cb = rest / md.n_rb;

  // chunk range of this split
  const int nchunks = pr.S_pad / CH;
  const int per = (nchunks + md.nsplit - 1) / md.nsplit;
  const int c0 = min(nchunks, z * per);
  const int c1 = min(nchunks, c0 + per);
  const int nck = c1 - c0;
  const unsigned char* at_src = reinterpret_cast<const unsigned char*>(atoms) + (size_t)c0 * kBBytes;
  const unsigned char* pf_src =
      reinterpret_cast<const unsigned char*>(pairs) +
      (size_t)((md.gram_off + cb * pr.S_pad + (int64_t)c0 * CH) / 2) * PS * 8;

  if (warp == EW) {
    if (lane == 0) {
      for (int i = 0; i < STAGES; ++i) mbar_init(&sm.full[i], 1);
      for (int i = 0; i < 2; ++i) {
        mbar_init(&sm.afull[i], 1);
        mbar_init(&sm.aempty[i], EW);
      }
      for (int i = 0; i < STAGES; ++i) mbar_init(&sm.sempty[i], EW);
      asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
    }
    tc_fence_before();
  }
  if (tid < BM) {
    sm.rowok[tid] = 1;
#pragma unroll
    for (int i = 0; i < SUBS; ++i) sm.cur_g[i][tid] = neg_inf();
  }
  __syncthreads();
  tc_fence_after();
  const uint32_t tmem = sm.tmem_base;

  int issued = 0;  // chunks whose copies the producer issued
  if (warp == EW && lane == 0) {
    for (; issued < STAGES && issued < nck && issued != pr.stall_chunk; ++issued) {
      mbar_expect_tx(&sm.full[issued], kBBytes + kPBytes);
      bulk_g2s(&sm.stage[issued][0], at_src + (size_t)issued * kBBytes, kBBytes, &sm.full[issued]);
      bulk_g2s(&sm.stage[issued][kBBytes], pf_src + (size_t)issued * kPBytes, kPBytes, &sm.full[issued]);
    }
  }
  // stage y = d * (W - W0): consecutive threads take consecutive columns of a row
  for (int e = tid; e < BM * 64; e += NT) {
    const int r = e >> 6, j = e & 63;
    const int64_t row = rb * BM + r;
    float y = 0.0f;
    if (row < md.rows) {
      const int64_t idx = row * md.cols + cb * 64 + j;
      const float rr = __fsub_rn(load_elem(md.W, idx, md.w_dtype), load_elem(md.W0, idx, md.w0_dtype));
      const float d = md.act[cb * 64 + j];
      if (!in_domain(rr, d)) sm.rowok[r] = 0;
      y = __fmul_rn(d, rr);
    }
    sm.Yst[r][j] = y;
  }
  __syncthreads();
  if (tid < BM) {  // the row's fixed-point exponent
    float m = 0.0f;
    for (int j = 0; j < 64; ++j) m = fmaxf(m, fabsf(sm.Yst[tid][j]));
    int q;
    const float inv = fixed_point_inv(m, &q);
    sm.inv_q[tid] = sm.rowok[tid] ? inv : 0.0f;
    sm.two_q[tid] = pow2f(q);
  }
  __syncthreads();
  // A operands: one thread writes one 16-byte core-matrix row (8 values of k)
  // of both halves
  for (int e = tid; e < BM * 8; e += NT) {
    const int m = e >> 3, k0 = (e & 7) * 8;
    const float inv = sm.inv_q[m];
    uint32_t wh[4], wl[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const int y0 = inv == 0.0f ? 0 : fixed_point_int(sm.Yst[m][k0 + 2 * i], inv);
      const int y1 = inv == 0.0f ? 0 : fixed_point_int(sm.Yst[m][k0 + 2 * i + 1], inv);
      wh[i] = (uint32_t)__half_as_ushort(__int2half_rn(y0 >> 11)) |
              ((uint32_t)__half_as_ushort(__int2half_rn(y1 >> 11)) << 16);
      wl[i] = (uint32_t)__half_as_ushort(__int2half_rn(y0 & 2047)) |
              ((uint32_t)__half_as_ushort(__int2half_rn(y1 & 2047)) << 16);
    }
    const int off = a_offset(m, k0);
    *reinterpret_cast<uint4*>(reinterpret_cast<unsigned char*>(sm.A[0]) + off) =
        make_uint4(wh[0], wh[1], wh[2], wh[3]);
    *reinterpret_cast<uint4*>(reinterpret_cast<unsigned char*>(sm.A[1]) + off) =
        make_uint4(wl[0], wl[1], wl[2], wl[3]);
  }
  asm volatile("fence.proxy.async.shared::cta;" ::: "memory");  // A is read by the tensor cores
  __syncthreads();

  bool timed_out = false;
  if (warp == EW) {
    // ------------------------------------------------------------ producer --
    if (lane == 0) {
      const uint32_t a0 = smem_addr(sm.A[0]), a1 = smem_addr(sm.A[1]);
      int k = 0;
      for (; k < nck; ++k) {
        const int st = k % STAGES, tb = k & 1;
        if (!mbar_wait(&sm.full[st], (uint32_t)((k / STAGES) & 1), pr.wait_ns)) { timed_out = true; break; }
        // every epilogue warp has loaded chunk k-2 from its accumulator
        if (k >= 2 && !mbar_wait(&sm.aempty[tb], (uint32_t)(((k - 2) >> 1) & 1), pr.wait_ns)) { timed_out = true; break; }
        tc_fence_after();
        const uint32_t bsm = smem_addr(&sm.stage[st][0]);
#pragma unroll
        for (int h = 0; h < 2; ++h) {
#pragma unroll
          for (int ks = 0; ks < 4; ++ks) {
            umma_f16(tmem + (uint32_t)(tb * 256 + h * 128), smem_desc((h ? a1 : a0) + ks * 256),
                     smem_desc(bsm + ks * 256), kIdesc, ks > 0 ? 1u : 0u);
          }
        }
        umma_commit(&sm.afull[tb]);
        if (k >= 2 && issued < nck && issued != pr.stall_chunk) {
          // chunk k-2's factors are no longer read: its stage takes chunk k+2
          const int ps = (k - 2) % STAGES;
          if (!mbar_wait(&sm.sempty[ps], (uint32_t)(((k - 2) / STAGES) & 1), pr.wait_ns)) { timed_out = true; ++k; break; }
          const int ns = issued % STAGES;
          mbar_expect_tx(&sm.full[ns], kBBytes + kPBytes);
          bulk_g2s(&sm.stage[ns][0], at_src + (size_t)issued * kBBytes, kBBytes, &sm.full[ns]);
          bulk_g2s(&sm.stage[ns][kBBytes], pf_src + (size_t)issued * kPBytes, kPBytes, &sm.full[ns]);
          ++issued;
        }
      }
      if (timed_out) {
        // wait (bounded) for this block's copies and MMAs still in flight
        for (int j = max(0, issued - STAGES); j < issued; ++j)
          (void)mbar_wait(&sm.full[j % STAGES], (uint32_t)((j / STAGES) & 1), pr.wait_ns);
        if (k > 0) (void)mbar_wait(&sm.afull[(k - 1) & 1], (uint32_t)(((k - 1) >> 1) & 1), pr.wait_ns);
      }
    }
  } else {
    // ------------------------------------------------------------ epilogue --
    const int m = 32 * (warp & 3) + lane;  // this thread's row = TMEM lane
    const int sub = warp >> 2;             // seed pairs SUB_PAIRS*sub .. of each chunk
    const float tq = __fmul_rn(sm.two_q[m], pr.c);
    const float2 tqc = make_float2(tq, tq);
    // A gain g in the units of the bound: g (2^q c)^-2 = g 2^(6 - 2q), formed
    // by two power-of-two factors (each a normal float), so exactly unless it
    // overflows (to +inf: every finite bound is then below the scaled gain,
    // as it is below the unscaled one) or falls far below every non-zero
    // bound (which is at least ~2^-36: u is integral, D_k <= 2^33).
    const int qrow = (int)((__float_as_uint(sm.two_q[m]) >> 23) & 0xffu) - 127;
    const int eu = min(250, max(-250, 6 - 2 * qrow)), eu1 = eu / 2, eu2 = eu - eu1;
    const float fu1 = __uint_as_float((uint32_t)(eu1 + 127) << 23);
    const float fu2 = __uint_as_float((uint32_t)(eu2 + 127) << 23);
    const uint32_t lane_base = (uint32_t)(32 * (warp & 3)) << 16;
    float bg = neg_inf();
    uint32_t bsd = 0xffffffffu;
    volatile float* cur_g = &sm.cur_g[0][m];  // written by the row's other warps
    // Seeds reach a thread in increasing order, so a strictly greater gain is
    // the whole tie rule within a thread.
    for (int k = 0; k < nck; ++k) {
      const int st = k % STAGES, tb = k & 1;
      if (!mbar_wait(&sm.afull[tb], (uint32_t)((k >> 1) & 1), pr.wait_ns)) { timed_out = true; break; }
      // the stage's factors landed before the chunk's MMAs were issued; this
      // wait (already complete) makes the copy visible to this warp's reads
      if (!mbar_wait(&sm.full[st], (uint32_t)((k / STAGES) & 1), pr.wait_ns)) { timed_out = true; break; }
      tc_fence_after();
      // Pruning threshold: the best gain any of the row's SUBS warps has found
      // so far. Each of them is a gain some candidate of this row reaches, so
      // a candidate whose bound is strictly below it cannot win. The entries
      // of the other warps may be stale, which only weakens the threshold.
      float thr = neg_inf();
      if constexpr (FAST) {
#pragma unroll
        for (int i = 0; i < SUBS; ++i) thr = fmaxf(thr, cur_g[i * BM]);
      }
      const float4* pbase = reinterpret_cast<const float4*>(&sm.stage[st][kBBytes]);
      // The warp's SUB_PAIRS seed pairs, one at a time, with the next pair's
      // TMEM loads in flight while a pair is scored: wait (only pair i's
      // loads are outstanding), issue pair i + 1's, then score pair i.
      const uint32_t cbase = tmem + lane_base + (uint32_t)(tb * 256 + 8 * SUB_PAIRS * sub);
      float hb[2][8], lb[2][8];
      float4 fb[2][5];  // the bound's factors (-L, invD m) of the pair and of the next one
      tmem_ld8(cbase, hb[0]);
      tmem_ld8(cbase + 128, lb[0]);
#pragma unroll
      for (int j = 0; j < 5; ++j) fb[0][j] = pbase[SUB_PAIRS * sub * (PS / 2) + j];
#pragma unroll
      for (int i = 0; i < SUB_PAIRS; ++i) {
        float* hi = hb[i & 1];
        float* lo = lb[i & 1];
        tmem_wait_ld8(hi);
        tmem_tie8(lo);
        if (i + 1 < SUB_PAIRS) {
          tmem_ld8(cbase + 8 * (i + 1), hb[(i + 1) & 1]);
          tmem_ld8(cbase + 128 + 8 * (i + 1), lb[(i + 1) & 1]);
#pragma unroll
          for (int j = 0; j < 5; ++j) fb[(i + 1) & 1][j] = pbase[(SUB_PAIRS * sub + i + 1) * (PS / 2) + j];
        } else {
          // the warp's last loads of this accumulator are complete: release it
          // now, so that chunk k+2's MMAs need not wait for the last scores
          tc_fence_before();
          __syncwarp();
          if (lane == 0) mbar_arrive(&sm.aempty[tb]);
        }
        const int pj = SUB_PAIRS * sub + i;  // seed pair within the chunk
        {
          const float4* pe = pbase + pj * (PS / 2);
          float2 u[4];
          const float2 ub = pair_bound(hi, lo, fb[i & 1], u);
          // prune: a candidate whose gain bound is below the running best
          // cannot win (NaN bounds stay live)
          const bool lx = !FAST || !(ub.x < thr), ly = !FAST || !(ub.y < thr);
          if (__any_sync(0xffffffffu, lx || ly)) {
            float2 bv[4], wv[4], al[4];
            // -L from the bound's registers, the rest from the stage
            pair_forward(u, tqc, fb[i & 1], pe, bv, wv);
            pair_back(fb[i & 1], wv, al);
            const float2 gp = pair_gain<FAST>(pr, bv, al, pe);
            // running argmax in seed order: a strictly greater gain wins
            const uint32_t s = (uint32_t)((c0 + k) * CH + 2 * pj);
            if (lx && gp.x > bg) { bg = gp.x; bsd = s; }
            if (ly && gp.y > bg) { bg = gp.y; bsd = s + 1; }
            if constexpr (FAST) {
              const float bgu = __fmul_rn(__fmul_rn(bg, fu1), fu2);
              cur_g[sub * BM] = bgu;
              thr = fmaxf(thr, bgu);
            }
          }
        }
      }
      __syncwarp();
      if (lane == 0) mbar_arrive(&sm.sempty[st]);  // done with the stage's factors
    }
    sm.red_g[sub][m] = bg;
    sm.red_s[sub][m] = bsd;
  }
  tc_fence_before();
  const bool any_timeout = __syncthreads_or(timed_out);
  if (any_timeout) {
    if (tid == 0) atomicOr(status, kFaultTimeout);
  } else if (tid < BM) {
    // merge the SUBS warps of each row (smaller seed on equal gains) and write
    // the row's candidate (split z of it when the seeds are split over blocks)
    int best = 0;
#pragma unroll
    for (int i = 1; i < SUBS; ++i)
      if (better(sm.red_g[i][tid], sm.red_s[i][tid], sm.red_g[best][tid], sm.red_s[best][tid])) best = i;
    const int64_t row = rb * BM + tid;
    if (row < md.rows) {
      const int64_t tt = md.tile_off + row * md.n_cb + cb;
      const float g = sm.red_g[best][tid];
      const uint32_t s = sm.red_s[best][tid];
      awsrc_candidate cd;
      const bool valid = sm.rowok[tid] && g > neg_inf();
      uint32_t cw = 0u;
      int sf = 0;
      if (valid) {
        const float4* pe = reinterpret_cast<const float4*>(
            pairs + (size_t)((md.gram_off + cb * pr.S_pad + s) / 2) * PS);
        const float gw = winner_codes<FAST>(pr, sm, tid, masks + (size_t)s * 4, pe, (s & 1u) != 0u, &cw, &sf);
        if (__float_as_uint(gw) != __float_as_uint(g)) atomicOr(status, kFaultSelfCheck);
      }
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
  return any_timeout;
}

// One block per SM, taking tile blocks blockIdx.x, blockIdx.x + gridDim.x, ...;
// the next tile block's W and W0 are prefetched into L2 while one is searched.
template <bool FAST>
__global__ void __launch_bounds__(NT, 1)
    search_c64p4_kernel(Prm pr, const __grid_constant__ LaunchDesc ld, int64_t n_blocks,
                        const uint4* __restrict__ atoms, const float2* __restrict__ pairs,
                        const uint64_t* __restrict__ masks, awsrc_candidate* __restrict__ cands,
                        uint32_t* __restrict__ status) {
  extern __shared__ unsigned char smem_raw[];
  // 1 KB aligned by pointer arithmetic on the shared array, so that the
  // compiler keeps the shared address space (LDS/STS, not generic accesses)
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw + ((1024u - (smem_addr(smem_raw) & 1023u)) & 1023u));
  const int warp = threadIdx.x >> 5;
  if (warp == EW) {  // the producer warp owns the TMEM allocation, held for all tile blocks
    asm volatile("tcgen05.alloc.cta_group::1.sync.aligned.shared::cta.b32 [%0], %1;" ::"r"(
                     smem_addr(&sm.tmem_base)),
                 "r"(kTmemCols)
                 : "memory");
    asm volatile("tcgen05.relinquish_alloc_permit.cta_group::1.sync.aligned;" ::: "memory");
  }
  for (int64_t blk = blockIdx.x; blk < n_blocks; blk += gridDim.x) {
    if (blk + gridDim.x < n_blocks) prefetch_block(ld, blk + gridDim.x, threadIdx.x);
    // a tile block whose waits ran out ends the CTA's work: its copies or MMAs
    // may still be in flight into this shared memory
    if (search_block<FAST>(pr, ld, blk, sm, atoms, pairs, masks, cands, status)) break;
    __syncthreads();  // the block's shared memory is reused by the next tile block
  }
  tc_fence_before();
  __syncthreads();
  if (warp == EW) {
    tc_fence_after();
    asm volatile("tcgen05.dealloc.cta_group::1.sync.aligned.b32 %0, %1;" ::"r"(sm.tmem_base), "r"(kTmemCols)
                 : "memory");
  }
}

// FP16 atoms in the order the MMAs read them: chunk c (32 seeds) is a 128x64
// K-major operand in 16 KB; item i (16 bytes = one core-matrix row) is chunk
// i >> 10, column group n8 = (i >> 6) & 15, k group (i >> 3) & 7, row i & 7,
// and column 8*n8 + r carries atom r >> 1 of seed 32c + 2*n8 + (r & 1).
__global__ void atoms_kernel(const uint64_t* __restrict__ masks, uint4* __restrict__ out, int S_pad) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t n = (int64_t)S_pad * 32;
  if (i >= n) return;
  const int r = (int)(i & 7), kg = (int)((i >> 3) & 7), n8 = (int)((i >> 6) & 15);
  const int64_t chunk = i >> 10;
  const int64_t seed = chunk * CH + 2 * n8 + (r & 1);
  const uint64_t m = masks[(size_t)seed * 4 + (r >> 1)];
  uint32_t w[4];
#pragma unroll
  for (int h = 0; h < 4; ++h) {
    const int k = 8 * kg + 2 * h;
    const uint32_t lo = ((m >> k) & 1ull) ? 0xBC00u : 0x3C00u;  // -1 : +1 in FP16
    const uint32_t hi = ((m >> (k + 1)) & 1ull) ? 0xBC00u : 0x3C00u;
    w[h] = lo | (hi << 16);
  }
  out[i] = make_uint4(w[0], w[1], w[2], w[3]);
}

// Best of the per-split candidates of tiles [t0, t1): larger gain, then the
// smaller seed (an invalid tile's candidates are all zero with gain -inf).
__global__ void merge_kernel(const awsrc_candidate* __restrict__ pc, int nsplit, int64_t T, int64_t t0,
                             int64_t t1, awsrc_candidate* __restrict__ out) {
  const int64_t t = t0 + (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= t1) return;
  awsrc_candidate b = pc[t];
  for (int z = 1; z < nsplit; ++z) {
    const awsrc_candidate c = pc[(size_t)z * T + t];
    if (better(c.gain, c.seed, b.gain, b.seed)) b = c;
  }
  out[t] = b;
}

}  // namespace

int search_c64p4_rows() { return BM; }
int search_c64p4_chunk() { return CH; }
size_t search_c64p4_table_bytes(int S_pad) { return (size_t)S_pad * 32 * 16; }

cudaError_t launch_bfrag_c64p4(const Prm& pr, const uint64_t* masks, void* out, cudaStream_t st) {
  const int64_t n = (int64_t)pr.S_pad * 32;
  atoms_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(masks, static_cast<uint4*>(out), pr.S_pad);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_merge_candidates(const awsrc_candidate* pc, int nsplit, int64_t T, int64_t t0, int64_t t1,
                                   awsrc_candidate* out, cudaStream_t st) {
  if (t1 <= t0) return cudaSuccess;
  merge_kernel<<<(unsigned)((t1 - t0 + 255) / 256), 256, 0, st>>>(pc, nsplit, T, t0, t1, out);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_search_c64p4(const Prm& pr, const LaunchDesc& ld, const void* table,
                                const float2* pairs, const uint64_t* masks, int64_t n_blocks,
                                awsrc_candidate* cands,
                                uint32_t* status, cudaStream_t st) {
  const size_t smem = sizeof(Smem) + 1024;  // + alignment of the operand tiles
  auto kern = pr.fast_pow2 ? search_c64p4_kernel<true> : search_c64p4_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  int dev = 0, nsm = 0;
  if ((e = cudaGetDevice(&dev)) != cudaSuccess) return e;
  if ((e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev)) != cudaSuccess) return e;
  const int64_t grid = std::max<int64_t>(1, std::min<int64_t>(n_blocks, nsm));
  kern<<<(unsigned)grid, NT, smem, st>>>(pr, ld, n_blocks, static_cast<const uint4*>(table), pairs, masks, cands,
                                         status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
