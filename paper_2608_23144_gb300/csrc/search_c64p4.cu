// search_c64p4.cu — seed search (Sec. 3.2) specialised for C = 64, P = 4, AWSRC-U,
// with the correlation on the tensor cores.
//
// The correlation u = B_s^T (D r) of Eq. 3 is an exact integer sum on the
// tile's fixed-point grid: Y_j = rint(y_j 2^-q) with |Y_j| <= 2^21, split as
// Y = 2048*Y_hi + Y_lo with Y_hi in [-1024, 1024] and Y_lo in [0, 2047]. Both
// halves and the +-1 atoms are exact in FP16, every product is exact, and every
// partial sum of 64 terms is an integer below 2^17, so FP32 accumulation on the
// tensor cores (mma.sync m16n8k16) is exact in any order. The epilogue forms
// u = 2^q * RN(2048*S_hi + S_lo) — the correctly rounded exact sum, one rounding.
//
// Block: 128 rows (tiles of one column block) x 32 seeds per chunk, 8 warps;
// warp w owns rows 16w..16w+15 and keeps their A fragments (both halves, K = 64)
// in registers for the whole seed loop. Per group of 4 seeds the warp issues 16
// MMAs (2 halves x 4 k-steps x 2 column tiles); the column order puts atoms
// p0,p1 of seed t in tile 0 and p2,p3 in tile 1, so lane (g, t) holds all four
// correlations of candidates (row g, seed t) and (row g+8, seed t) and runs the
// fused epilogue (solve with the (cb, s) LDL^T, quantise, score, running argmax)
// on them directly. B fragments (16 KB per chunk, pre-arranged in fragment order)
// and the chunk's Gram entries (2.5 KB) are streamed by bulk TMA copies into two
// shared-memory buffers completed by mbarrier transaction counts. Every mbarrier
// wait is bounded in time; on expiry the block records a timeout fault, drains its
// own copies (again bounded) and returns.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int BM = 128;   // rows (tiles) per block
constexpr int CH = 32;    // seeds per chunk
constexpr int NT = 256;   // threads
constexpr int PS = pair_stride(4);  // 18 float2 per (cb, s) entry of the paired table
constexpr uint32_t kBBytes = (CH / 4) * 4 * 32 * 16;  // 16 KB of B fragments per chunk
constexpr uint32_t kGsBytes = CH * PS * 8u;            // 4608 B
constexpr uint64_t kWaitNs = 2000000000ull;            // 2 s per wait

struct Smem {
  float Yst[BM][65];
  float two_q[BM];
  float inv_q[BM];
  int rowok[BM];
  uint4 Bf[2][CH / 4][4][32];
  float2 Gp[2][CH * PS];
  unsigned long long mbar[2];
};

__device__ __forceinline__ uint32_t smem_addr(const void* p) {
  return (uint32_t)__cvta_generic_to_shared(p);
}

__device__ __forceinline__ uint64_t globaltimer() {
  uint64_t t;
  asm volatile("mov.u64 %0, %%globaltimer;" : "=l"(t));
  return t;
}

__device__ __forceinline__ void mbar_init(unsigned long long* mb, uint32_t count) {
  asm volatile("mbarrier.init.shared::cta.b64 [%0], %1;" ::"r"(smem_addr(mb)), "r"(count) : "memory");
}

__device__ __forceinline__ void mbar_expect_tx(unsigned long long* mb, uint32_t bytes) {
  asm volatile("mbarrier.arrive.expect_tx.shared::cta.b64 _, [%0], %1;" ::"r"(smem_addr(mb)),
               "r"(bytes)
               : "memory");
}

__device__ __forceinline__ bool mbar_try_wait(unsigned long long* mb, uint32_t parity) {
  uint32_t ok;
  asm volatile(
      "{\n\t.reg .pred p;\n\t"
      "mbarrier.try_wait.parity.shared::cta.b64 p, [%1], %2;\n\t"
      "selp.u32 %0, 1, 0, p;\n\t}"
      : "=r"(ok)
      : "r"(smem_addr(mb)), "r"(parity)
      : "memory");
  return ok != 0;
}

// Bounded wait: true when the phase with `parity` completed within kWaitNs.
__device__ __forceinline__ bool mbar_wait(unsigned long long* mb, uint32_t parity) {
  if (mbar_try_wait(mb, parity)) return true;
  const uint64_t t0 = globaltimer();
  while (!mbar_try_wait(mb, parity)) {
    if (globaltimer() - t0 > kWaitNs) return false;
  }
  return true;
}

__device__ __forceinline__ void bulk_g2s(void* dst, const void* src, uint32_t bytes,
                                         unsigned long long* mb) {
  asm volatile(
      "cp.async.bulk.shared::cluster.global.mbarrier::complete_tx::bytes [%0], [%1], %2, [%3];" ::"r"(
          smem_addr(dst)),
      "l"(src), "r"(bytes), "r"(smem_addr(mb))
      : "memory");
}

__device__ __forceinline__ void mma16816(float* d, const uint32_t* a, uint32_t b0, uint32_t b1) {
  asm(
      "mma.sync.aligned.m16n8k16.row.col.f32.f16.f16.f32 {%0,%1,%2,%3}, {%4,%5,%6,%7}, {%8,%9}, "
      "{%0,%1,%2,%3};"
      : "+f"(d[0]), "+f"(d[1]), "+f"(d[2]), "+f"(d[3])
      : "r"(a[0]), "r"(a[1]), "r"(a[2]), "r"(a[3]), "r"(b0), "r"(b1));
}

// Two FP16 halves (exact small integers) packed low-first.
__device__ __forceinline__ uint32_t pack_h2(int lo, int hi) {
  return (uint32_t)__half_as_ushort(__int2half_rn(lo)) | ((uint32_t)__half_as_ushort(__int2half_rn(hi)) << 16);
}

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

template <bool FAST>
__global__ void __launch_bounds__(NT, 2)
    search_c64p4_kernel(Prm pr, LaunchDesc ld, const uint4* __restrict__ bfrag,
                        const float2* __restrict__ pairs, float2* __restrict__ partials,
                        uint32_t* __restrict__ status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int tid = threadIdx.x, lane = tid & 31, warp = tid >> 5;
  const int mi = find_mod(ld, blockIdx.x);
  const ModDesc& md = ld.m[mi];
  const int64_t b = blockIdx.x - md.block_off;
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
  const uint4* bf_src = bfrag + (size_t)c0 * (kBBytes / 16);
  const float2* gs_src = pairs + (size_t)(md.gram_off + cb * pr.S_pad + (int64_t)c0 * CH) * PS;

  if (tid == 0) {
    mbar_init(&sm.mbar[0], 1);
    mbar_init(&sm.mbar[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid < BM) sm.rowok[tid] = 1;
  __syncthreads();
  if (tid == 0) {
    for (int k = 0; k < 2 && k < nck; ++k) {
      mbar_expect_tx(&sm.mbar[k], kBBytes + kGsBytes);
      bulk_g2s(&sm.Bf[k][0][0][0], bf_src + (size_t)k * (kBBytes / 16), kBBytes, &sm.mbar[k]);
      bulk_g2s(&sm.Gp[k][0], gs_src + (size_t)k * CH * PS, kGsBytes, &sm.mbar[k]);
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

  // A fragments of the warp's 16 rows: Y split into hi (a_h) and lo (a_l) halves
  const int g = lane >> 2, t = lane & 3;
  const int R0 = warp * 16 + g, R1 = R0 + 8;
  uint32_t a_h[4][4], a_l[4][4];
  {
    const float i0 = sm.inv_q[R0], i1 = sm.inv_q[R1];
#pragma unroll
    for (int ks = 0; ks < 4; ++ks) {
#pragma unroll
      for (int reg = 0; reg < 4; ++reg) {
        const int row = (reg & 1) ? R1 : R0;
        const float inv = (reg & 1) ? i1 : i0;
        const int k = 16 * ks + 2 * t + ((reg & 2) ? 8 : 0);
        const int y0 = inv == 0.0f ? 0 : fixed_point_int(sm.Yst[row][k], inv);
        const int y1 = inv == 0.0f ? 0 : fixed_point_int(sm.Yst[row][k + 1], inv);
        a_h[ks][reg] = pack_h2(y0 >> 11, y1 >> 11);
        a_l[ks][reg] = pack_h2(y0 & 2047, y1 & 2047);
      }
    }
  }
  // b = c * 2^q * RN(S) = RN(S) * (2^q c): c = 1/8 and 2^q >= 2^-120 keep every
  // product exact (normal range), so one multiply per atom gives b.
  const float2 tqc = make_float2(__fmul_rn(sm.two_q[R0], pr.c), __fmul_rn(sm.two_q[R1], pr.c));
  float bg[2] = {neg_inf(), neg_inf()};
  uint32_t bs[2] = {0xffffffffu, 0xffffffffu};

  // Seeds reach a lane in increasing order (chunk by chunk, group by group), so
  // within a lane a strictly greater gain is the whole tie rule.
  bool timed_out = false;
  for (int k = 0; k < nck; ++k) {
    const int buf = k & 1;
    const bool ok = mbar_wait(&sm.mbar[buf], (uint32_t)((k >> 1) & 1));
    if (!ok) timed_out = true;
    if (!timed_out) {
      // 16 MMAs of one group of 4 seeds into acc[half][column tile][fragment]
      auto mma_group = [&](int grp, float (&acc)[2][2][4]) {
        uint32_t bb[4][4];
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          const uint4 v = sm.Bf[buf][grp][ks][lane];
          bb[ks][0] = v.x; bb[ks][1] = v.y; bb[ks][2] = v.z; bb[ks][3] = v.w;
        }
#pragma unroll
        for (int h = 0; h < 2; ++h)
#pragma unroll
          for (int n = 0; n < 2; ++n)
#pragma unroll
            for (int i = 0; i < 4; ++i) acc[h][n][i] = 0.0f;
#pragma unroll
        for (int ks = 0; ks < 4; ++ks) {
          mma16816(acc[0][0], a_h[ks], bb[ks][0], bb[ks][1]);
          mma16816(acc[0][1], a_h[ks], bb[ks][2], bb[ks][3]);
          mma16816(acc[1][0], a_l[ks], bb[ks][0], bb[ks][1]);
          mma16816(acc[1][1], a_l[ks], bb[ks][2], bb[ks][3]);
        }
      };
      auto epilogue = [&](int grp, const float (&acc)[2][2][4]) {
        // epilogue: candidates (R0, seed t) and (R1, seed t) of this group, one
        // per float2 component
        const int sl = 4 * grp + t;
        const uint32_t s = (uint32_t)((c0 + k) * CH + sl);
        const float4* pe = reinterpret_cast<const float4*>(&sm.Gp[buf][sl * PS]);
        float2 pv[PS];
#pragma unroll
        for (int i = 0; i < PS / 2; ++i) {
          const float4 v = pe[i];
          pv[2 * i] = make_float2(v.x, v.y);
          pv[2 * i + 1] = make_float2(v.z, v.w);
        }
        const float2* nL = pv;          // -L
        const float2* invD = pv + 6;
        const float2* Go = pv + 10;     // G off-diagonal (doubled on the fast path)
        const float2 gd = pv[16];
        float2 bv[4], alpha[4];
#pragma unroll
        for (int p = 0; p < 4; ++p) {
          // atoms p0, p1 sit in column tile 0, p2, p3 in tile 1; fragment
          // elements 0,1 are row R0 and 2,3 row R1
          const int n = p >> 1, e = p & 1;
          const float2 u = make_float2(__fmaf_rn(2048.0f, acc[0][n][e], acc[1][n][e]),
                                       __fmaf_rn(2048.0f, acc[0][n][2 + e], acc[1][n][2 + e]));
          bv[p] = __fmul2_rn(u, tqc);
        }
        ldl_solve2<4>(nL, invD, bv, alpha);
        float2 gn;
        if (FAST) {
          gn = quant_gain_fast2<4>(pr, alpha, bv, gd, Go);
        } else {
          float Gx[6], q[4];
#pragma unroll
          for (int i = 0; i < 6; ++i) Gx[i] = Go[i].x;
          int sf;
          float a0[4] = {alpha[0].x, alpha[1].x, alpha[2].x, alpha[3].x};
          float b0[4] = {bv[0].x, bv[1].x, bv[2].x, bv[3].x};
          float a1[4] = {alpha[0].y, alpha[1].y, alpha[2].y, alpha[3].y};
          float b1[4] = {bv[0].y, bv[1].y, bv[2].y, bv[3].y};
          gn.x = quant_gain<4>(pr, a0, b0, gd.x, Gx, q, &sf);
          gn.y = quant_gain<4>(pr, a1, b1, gd.x, Gx, q, &sf);
        }
        if (gn.x > bg[0]) { bg[0] = gn.x; bs[0] = s; }
        if (gn.y > bg[1]) { bg[1] = gn.y; bs[1] = s; }
      };
      // the MMAs of the next group are issued before the epilogue of the current
      // one, so the tensor pipe and the FP32 pipe overlap within each warp
      float accA[2][2][4], accB[2][2][4];
      mma_group(0, accA);
#pragma unroll 1
      for (int grp = 0; grp < CH / 4; grp += 2) {
        mma_group(grp + 1, accB);
        epilogue(grp, accA);
        if (grp + 2 < CH / 4) mma_group(grp + 2, accA);
        epilogue(grp + 1, accB);
      }
    }
    // every thread is done with buffer `buf`; a timeout anywhere ends the block
    if (__syncthreads_or(timed_out)) { timed_out = true; break; }
    if (tid == 0 && k + 2 < nck) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_expect_tx(&sm.mbar[buf], kBBytes + kGsBytes);
      bulk_g2s(&sm.Bf[buf][0][0][0], bf_src + (size_t)(k + 2) * (kBBytes / 16), kBBytes, &sm.mbar[buf]);
      bulk_g2s(&sm.Gp[buf][0], gs_src + (size_t)(k + 2) * CH * PS, kGsBytes, &sm.mbar[buf]);
    }
  }
  if (timed_out) {
    // drain copies this block issued (bounded), record the fault and leave
    if (tid == 0) {
      atomicOr(status, kFaultTimeout);
      for (int bb = 0; bb < 2; ++bb) (void)mbar_wait(&sm.mbar[bb], 0), (void)mbar_wait(&sm.mbar[bb], 1);
    }
    __syncthreads();
    return;
  }
  // reduce the running argmax over the 4 lanes (t) that share rows R0, R1
#pragma unroll
  for (int rr = 0; rr < 2; ++rr) {
#pragma unroll
    for (int off = 1; off < 4; off <<= 1) {
      const float og = __shfl_xor_sync(0xffffffffu, bg[rr], off);
      const uint32_t os = __shfl_xor_sync(0xffffffffu, bs[rr], off);
      if (better(og, os, bg[rr], bs[rr])) { bg[rr] = og; bs[rr] = os; }
    }
  }
  if (t == 0) {
#pragma unroll
    for (int rr = 0; rr < 2; ++rr) {
      const int r = rr ? R1 : R0;
      const int64_t row = rb * BM + r;
      if (row < md.rows) {
        const int64_t tt = md.tile_off + row * md.n_cb + cb;
        partials[(size_t)z * ld.T + tt] = make_float2(sm.rowok[r] ? bg[rr] : neg_inf(), __uint_as_float(bs[rr]));
      }
    }
  }
}

// B fragments of the +-1 atoms in the order the kernel reads them:
// out[((chunk*8 + grp)*4 + ks)*32 + lane] = {b0, b1 of column tile 0, b0, b1 of
// tile 1} for k-step ks, where lane = 4g + t holds column g (seed 4*grp + g/2,
// atom 2*tile + g%2) at rows k = 16ks + 2t (+1) and 16ks + 2t + 8 (+9).
__global__ void bfrag_kernel(const uint64_t* __restrict__ masks, uint4* __restrict__ out, int S_pad) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  const int64_t n = (int64_t)S_pad / 4 * 4 * 32;
  if (i >= n) return;
  const int ln = (int)(i & 31), ks = (int)((i >> 5) & 3);
  const int64_t grp = i >> 7;  // global group of 4 seeds
  const int g = ln >> 2, t = ln & 3;
  const int64_t seed = grp * 4 + (g >> 1);
  uint32_t w[4];
#pragma unroll
  for (int tile = 0; tile < 2; ++tile) {
    const uint64_t m = masks[(size_t)seed * 4 + 2 * tile + (g & 1)];
#pragma unroll
    for (int half = 0; half < 2; ++half) {
      const int k = 16 * ks + 2 * t + 8 * half;
      const uint32_t lo = ((m >> k) & 1ull) ? 0xBC00u : 0x3C00u;       // -1 : +1 in FP16
      const uint32_t hi = ((m >> (k + 1)) & 1ull) ? 0xBC00u : 0x3C00u;
      w[2 * tile + half] = lo | (hi << 16);
    }
  }
  out[i] = make_uint4(w[0], w[1], w[2], w[3]);
}

}  // namespace

int search_c64p4_rows() { return BM; }
int search_c64p4_chunk() { return CH; }
size_t search_c64p4_table_bytes(int S_pad) { return (size_t)S_pad * 4 * 32 * 16 / 4; }

cudaError_t launch_bfrag_c64p4(const Prm& pr, const uint64_t* masks, void* out, cudaStream_t st) {
  const int64_t n = (int64_t)pr.S_pad / 4 * 4 * 32;
  bfrag_kernel<<<(unsigned)((n + 255) / 256), 256, 0, st>>>(masks, static_cast<uint4*>(out), pr.S_pad);
  note_launches(1);
  return cudaGetLastError();
}

cudaError_t launch_search_c64p4(const Prm& pr, const LaunchDesc& ld, const void* table,
                                const float2* pairs, int64_t n_blocks, float2* partials,
                                uint32_t* status, cudaStream_t st) {
  const size_t smem = sizeof(Smem);
  auto kern = pr.fast_pow2 ? search_c64p4_kernel<true> : search_c64p4_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<(unsigned)n_blocks, NT, smem, st>>>(pr, ld, static_cast<const uint4*>(table), pairs, partials, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
