// search_c64p4.cu — seed search (Sec. 3.2) specialised for C = 64, P = 4, AWSRC-U.
//
// The correlation b = B_s^T D r of Eq. 3 for a block of 128 rows (tiles of one
// column block) and a chunk of 32 seeds is a 128 x 64 by 64 x 128 product whose
// right operand is +-1. It runs on the FP32 pipe: each thread owns an 8-row x
// 2-seed x 4-atom register tile and accumulates over j = 0..63 in ascending
// order with one FFMA per term (m*y is exact, so FFMA rounds like the canonical
// sum). The fused epilogue solves with the precomputed LDL^T of the (cb, s)
// Gram matrix, quantises and scores every candidate in registers and keeps a
// running argmax per row; a 16-lane shuffle reduction finishes the seeds.
//
// Data movement: the residual tile block is staged once per block (plain loads,
// y = d*r written j-major to shared memory). The +-1.0f atoms (32 KB per chunk)
// and the chunk's 32 Gram entries (2.5 KB) are streamed by bulk TMA copies
// (cp.async.bulk) into two shared-memory buffers completed by mbarrier
// transaction counts, so the next chunk lands while the current one computes.
// Every mbarrier wait is bounded in time; on expiry the block records a
// timeout fault, drains its own copies (again bounded) and returns.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int BM = 128;   // rows (tiles) per block
constexpr int CH = 32;    // seeds per chunk
constexpr int NT = 256;   // threads
constexpr int GS = gram_stride(4);  // 20 floats per (cb, s) entry
constexpr uint32_t kMsBytes = 64u * CH * 4u * 4u;  // 32 KB
constexpr uint32_t kGsBytes = CH * GS * 4u;        // 2560 B
constexpr uint64_t kWaitNs = 2000000000ull;        // 2 s per wait

struct Smem {
  float Ys[64][BM];
  float Ms[2][64][CH * 4];
  float Gs[2][CH * GS];
  unsigned long long mbar[2];
  int rowok[BM];
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

__device__ __forceinline__ float neg_inf() { return -__int_as_float(0x7f800000); }

template <bool FAST>
__global__ void __launch_bounds__(NT, 2)
    search_c64p4_kernel(Prm pr, LaunchDesc ld, const float* __restrict__ mexp,
                        const float* __restrict__ gram, float2* __restrict__ partials,
                        uint32_t* __restrict__ status) {
  extern __shared__ __align__(128) unsigned char smem_raw[];
  Smem& sm = *reinterpret_cast<Smem*>(smem_raw);
  const int tid = threadIdx.x;
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
  const float* ms_src = mexp + (size_t)c0 * (64 * CH * 4);
  const float* gs_src = gram + (size_t)(md.gram_off + cb * pr.S_pad + (int64_t)c0 * CH) * GS;

  if (tid == 0) {
    mbar_init(&sm.mbar[0], 1);
    mbar_init(&sm.mbar[1], 1);
    asm volatile("fence.mbarrier_init.release.cluster;" ::: "memory");
  }
  if (tid < BM) sm.rowok[tid] = 1;
  __syncthreads();
  if (tid == 0) {
    for (int k = 0; k < 2 && k < nck; ++k) {
      mbar_expect_tx(&sm.mbar[k], kMsBytes + kGsBytes);
      bulk_g2s(&sm.Ms[k][0][0], ms_src + (size_t)k * (64 * CH * 4), kMsBytes, &sm.mbar[k]);
      bulk_g2s(&sm.Gs[k][0], gs_src + (size_t)k * CH * GS, kGsBytes, &sm.mbar[k]);
    }
  }
  // stage y = d * (W - W0), j-major; consecutive threads take consecutive rows
  for (int e = tid; e < BM * 64; e += NT) {
    const int r = e % BM, j = e / BM;
    const int64_t row = rb * BM + r;
    float y = 0.0f;
    if (row < md.rows) {
      const int64_t idx = row * md.cols + cb * 64 + j;
      const float rr = __fsub_rn(load_elem(md.W, idx, md.w_dtype), load_elem(md.W0, idx, md.w0_dtype));
      const float d = md.act[cb * 64 + j];
      if (!in_domain(rr, d)) sm.rowok[r] = 0;
      y = __fmul_rn(d, rr);
    }
    sm.Ys[j][r] = y;
  }
  __syncthreads();

  const int ty = tid >> 4;  // rows ty*8 .. ty*8+7
  const int tx = tid & 15;  // seeds tx and tx+16 of the chunk
  const float c = pr.c;
  float bg[8];
  uint32_t bs[8];
#pragma unroll
  for (int i = 0; i < 8; ++i) { bg[i] = neg_inf(); bs[i] = 0xffffffffu; }

  // Seeds reach a thread in increasing order (chunk by chunk, tx before tx+16),
  // so within a thread a strictly greater gain is the whole tie rule.
  bool timed_out = false;
  for (int k = 0; k < nck; ++k) {
    const int buf = k & 1;
    const bool ok = mbar_wait(&sm.mbar[buf], (uint32_t)((k >> 1) & 1));
    if (!ok) timed_out = true;

    if (!timed_out) {
      float acc[8][8];
#pragma unroll
      for (int i = 0; i < 8; ++i)
#pragma unroll
        for (int q = 0; q < 8; ++q) acc[i][q] = 0.0f;
      const float* ysb = &sm.Ys[0][ty * 8];
      const float* msb = &sm.Ms[buf][0][0];
#pragma unroll 4
      for (int j = 0; j < 64; ++j) {
        const float4 ya = *reinterpret_cast<const float4*>(ysb + j * BM);
        const float4 yb = *reinterpret_cast<const float4*>(ysb + j * BM + 4);
        const float4 ma = *reinterpret_cast<const float4*>(msb + j * (CH * 4) + tx * 4);
        const float4 mb = *reinterpret_cast<const float4*>(msb + j * (CH * 4) + (tx + 16) * 4);
        const float yv[8] = {ya.x, ya.y, ya.z, ya.w, yb.x, yb.y, yb.z, yb.w};
        const float mv[8] = {ma.x, ma.y, ma.z, ma.w, mb.x, mb.y, mb.z, mb.w};
#pragma unroll
        for (int i = 0; i < 8; ++i)
#pragma unroll
          for (int q = 0; q < 8; ++q) acc[i][q] = __fmaf_rn(mv[q], yv[i], acc[i][q]);
      }
      // fused epilogue: solve, quantise, score, running argmax
#pragma unroll
      for (int h = 0; h < 2; ++h) {
        const int sl = tx + 16 * h;
        const uint32_t s = (uint32_t)((c0 + k) * CH + sl);
        const float* gt = &sm.Gs[buf][sl * GS];
        const float4 g0 = *reinterpret_cast<const float4*>(gt);
        const float4 g1 = *reinterpret_cast<const float4*>(gt + 4);
        const float4 g2 = *reinterpret_cast<const float4*>(gt + 8);
        const float4 g3 = *reinterpret_cast<const float4*>(gt + 12);
        const float gd = gt[16];
        const float L[6] = {g0.x, g0.y, g0.z, g0.w, g1.x, g1.y};
        const float invD[4] = {g1.z, g1.w, g2.x, g2.y};
        float Gq[6] = {g2.z, g2.w, g3.x, g3.y, g3.z, g3.w};
        if (FAST) {
#pragma unroll
          for (int i = 0; i < 6; ++i) Gq[i] = __fmul_rn(2.0f, Gq[i]);  // exact
        }
#pragma unroll
        for (int i = 0; i < 8; ++i) {
          float bv[4], alpha[4], q[4];
#pragma unroll
          for (int p = 0; p < 4; ++p) bv[p] = __fmul_rn(c, acc[i][h * 4 + p]);
          ldl_solve<4>(L, invD, bv, alpha);
          int sf;
          const float g = FAST ? quant_gain_fast<4>(pr, alpha, bv, gd, Gq, q, &sf)
                               : quant_gain<4>(pr, alpha, bv, gd, Gq, q, &sf);
          if (g > bg[i]) { bg[i] = g; bs[i] = s; }
        }
      }
    }
    // every thread is done with buffer `buf`; a timeout anywhere ends the block
    if (__syncthreads_or(timed_out)) { timed_out = true; break; }
    if (tid == 0 && k + 2 < nck) {
      asm volatile("fence.proxy.async.shared::cta;" ::: "memory");
      mbar_expect_tx(&sm.mbar[buf], kMsBytes + kGsBytes);
      bulk_g2s(&sm.Ms[buf][0][0], ms_src + (size_t)(k + 2) * (64 * CH * 4), kMsBytes, &sm.mbar[buf]);
      bulk_g2s(&sm.Gs[buf][0], gs_src + (size_t)(k + 2) * CH * GS, kGsBytes, &sm.mbar[buf]);
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
  // reduce the running argmax over the 16 threads (tx) that share rows
#pragma unroll
  for (int i = 0; i < 8; ++i) {
#pragma unroll
    for (int off = 1; off < 16; off <<= 1) {
      const float og = __shfl_xor_sync(0xffffffffu, bg[i], off);
      const uint32_t os = __shfl_xor_sync(0xffffffffu, bs[i], off);
      if (better(og, os, bg[i], bs[i])) { bg[i] = og; bs[i] = os; }
    }
  }
  if (tx == 0) {
#pragma unroll
    for (int i = 0; i < 8; ++i) {
      const int r = ty * 8 + i;
      const int64_t row = rb * BM + r;
      if (row < md.rows) {
        const int64_t t = md.tile_off + row * md.n_cb + cb;
        partials[(size_t)z * ld.T + t] =
            make_float2(sm.rowok[r] ? bg[i] : neg_inf(), __uint_as_float(bs[i]));
      }
    }
  }
}

}  // namespace

int search_c64p4_rows() { return BM; }
int search_c64p4_chunk() { return CH; }

cudaError_t launch_search_c64p4(const Prm& pr, const LaunchDesc& ld, const float* mexp,
                                const float* gram, int64_t n_blocks, float2* partials,
                                uint32_t* status, cudaStream_t st) {
  const size_t smem = sizeof(Smem);
  auto kern = pr.fast_pow2 ? search_c64p4_kernel<true> : search_c64p4_kernel<false>;
  cudaError_t e = cudaFuncSetAttribute(kern, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)smem);
  if (e != cudaSuccess) return e;
  kern<<<(unsigned)n_blocks, NT, smem, st>>>(pr, ld, mexp, gram, partials, status);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
