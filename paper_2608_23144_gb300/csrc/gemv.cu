// gemv.cu — the decoded weights of one module applied to M vectors without
// forming them: y[m] = (W0 + r_hat) x[m], with W0 = q * s_eff read from the
// packed RTN-INT4 backbone (binary16 or SDQ scales, Sec. 3.3) and r_hat the
// decoder's residual (Sec. 3.2) on the tiles a prepared sidecar names. This is
// the packed-inference use the paper leaves to future work (Sec. 5).
//
// When x fits in shared memory: gemv_warp_kernel below. Otherwise one block per
// output row, 8 warps taking interleaved runs of 4 groups of 128 inputs (lane
// l: elements 4l .. 4l + 3 of each group; its 4 codes are 16 bits).
// For each run a warp issues all independent loads first (codes, scales, tile
// map entries, x), then the dependent ones of recorded tiles (record codes and
// mask words). Per element, w = fl(q * s_eff) as in W0 and r = fl(fl(k * C^-1/2)
// * scale) as in the decoder; both are accumulated into binary32 sums with
// fma, reduced over lanes and warps.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int kGemvWarps = 8;
constexpr size_t kGemvSmemMax = 96 * 1024;  // x staged in shared memory up to this size
constexpr int kRun = 4;  // groups per warp iteration

__device__ __forceinline__ int code4(uint32_t packed, int i) {  // 4-bit two's complement
  return (int)((int32_t)(packed << (28 - 4 * i)) >> 28);
}

__device__ __forceinline__ float sidecar_scale(const Prm& pr, int16_t s) {
  if (pr.scale_mode == AWSRC_SCALE_POW2) return __int_as_float((s + 127) << 23);
  return __half2float(__ushort_as_half((unsigned short)s));
}

template <int M>
__global__ void __launch_bounds__(32 * kGemvWarps) gemv_kernel(Prm pr, GemvArgs a) {
  __shared__ float part[kGemvWarps][M];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t i = blockIdx.x;  // output row
  const int64_t gpr = a.cols >> 7;
  float acc[M];
#pragma unroll
  for (int m = 0; m < M; ++m) acc[m] = 0.0f;
  for (int64_t gb = (int64_t)warp * kRun; gb < gpr; gb += (int64_t)kGemvWarps * kRun) {
    uint32_t pk[kRun];
    float s[kRun];
    unsigned long long ent[kRun];
    float4 xv[kRun][M];
#pragma unroll
    for (int u = 0; u < kRun; ++u) {
      const int64_t g = gb + u;
      pk[u] = 0u;
      s[u] = 0.0f;
      ent[u] = 0ull;
#pragma unroll
      for (int m = 0; m < M; ++m) xv[u][m] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);  // runs past the row end
      if (g < gpr) {
        const int64_t gid = i * gpr + g;
        pk[u] = __ldg(a.codes + gid * 32 + lane);
        if (a.sdq) {
          const float2 ms = __ldg(reinterpret_cast<const float2*>(a.sdq_consts) + (gid >> 8));
          s[u] = __fadd_rn(ms.x, __fmul_rn((float)__ldg(a.sdq_codes + gid), ms.y));
        } else {
          s[u] = __half2float(__ushort_as_half(__ldg(a.scales + gid)));
        }
        const int64_t j0 = g * 128 + 4 * lane;
        if (a.map) ent[u] = __ldg(a.map + a.tile_off + (i * a.cols + j0) / pr.C);
#pragma unroll
        for (int m = 0; m < M; ++m) xv[u][m] = __ldg(reinterpret_cast<const float4*>(a.x + m * a.cols + j0));
      }
    }
#pragma unroll
    for (int u = 0; u < kRun; ++u) {
      float w[4], r[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int e = 0; e < 4; ++e) w[e] = __fmul_rn((float)code4(pk[u], e), s[u]);
      if (ent[u] != 0ull) {  // a recorded tile: its residual on these 4 elements
        const unsigned long long en = ent[u];
        const int64_t k = (int64_t)(en >> 32) - 1;
        const uint32_t seed = (uint32_t)(en >> 16) & 0xFFFFu;
        const float sc = sidecar_scale(pr, (int16_t)(uint16_t)(en & 0xFFFFull));
        const uint2 cw = __ldg(reinterpret_cast<const uint2*>(a.rcodes + k));  // the slot's codes
        const int jt = (int)(((gb + u) * 128 + 4 * lane) & (pr.C - 1));  // position in the tile
        const uint64_t* mk = a.masks + (size_t)seed * pr.P * pr.W + (jt >> 6);
        int kj[4] = {0, 0, 0, 0};
        for (int p = 0; p < pr.P; ++p) {
          const uint32_t bits = (uint32_t)(__ldg(mk + (size_t)p * pr.W) >> (jt & 63));
          const int cp = (int)(int8_t)((p < 4 ? cw.x : cw.y) >> (8 * (p & 3)));
#pragma unroll
          for (int e = 0; e < 4; ++e) kj[e] += ((bits >> e) & 1u) ? -cp : cp;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) r[e] = __fmul_rn(__fmul_rn((float)kj[e], pr.c), sc);
      }
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float xe[4] = {xv[u][m].x, xv[u][m].y, xv[u][m].z, xv[u][m].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          acc[m] = __fmaf_rn(w[e], xe[e], acc[m]);
          acc[m] = __fmaf_rn(r[e], xe[e], acc[m]);
        }
      }
    }
  }
#pragma unroll
  for (int m = 0; m < M; ++m) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc[m] = __fadd_rn(acc[m], __shfl_xor_sync(0xffffffffu, acc[m], off));
    if (lane == 0) part[warp][m] = acc[m];
  }
  __syncthreads();
  if (threadIdx.x < M) {
    float t = 0.0f;
#pragma unroll
    for (int w = 0; w < kGemvWarps; ++w) t = __fadd_rn(t, part[w][threadIdx.x]);
    a.y[(int64_t)threadIdx.x * a.rows + i] = t;
  }
}

// One warp per output row (8 rows per block). The block first stages x in
// shared memory, lane-major per 1024-column chunk: element 1024c + 32l + 4q + e
// at float index 4((8c + q) 32 + l) + e, so that lane l's 16-byte reads of its
// 32 consecutive inputs of chunk c are conflict-free. Lane l then streams
// 16-byte code words (32 weights of one group) chunk by chunk, kUnroll chunks
// in flight: nibble pairs become floats through a byte permute into 2^23 + u
// (u the offset-binary code) and one packed subtraction, and are accumulated
// with packed FMAs; each chunk's sum is scaled by its group's s. The row's
// recorded tiles follow, 32 tiles at a time: one map entry per lane, the
// recorded lanes fetch their record codes and mask words, and the warp walks
// the tiles together (elements lane + 32e, x from the staged copy).
constexpr int kUnroll = 2;
constexpr float kNibbleBias = 8388616.0f;  // 2^23 + 8
constexpr int kPrefetchWords = 4;          // mask words (P * W) a recorded lane prefetches

__device__ __forceinline__ int xs_index(int64_t j) {  // permuted position of input j
  return (int)((((j >> 10) * 8 + ((j >> 2) & 7)) * 32 + ((j >> 5) & 31)) * 4 + (j & 3));
}

// The two codes of byte b of `lo` (even elements) and `hi` (odd elements), both
// offset binary, as floats.
__device__ __forceinline__ float2 nibble_pair(uint32_t lo, uint32_t hi, int b) {
  const float2 v = make_float2(__uint_as_float(__byte_perm(lo, 0x4B000000u, 0x7540u + b)),
                               __uint_as_float(__byte_perm(hi, 0x4B000000u, 0x7540u + b)));
  return __fadd2_rn(v, make_float2(-kNibbleBias, -kNibbleBias));
}

// Loads of one row that do not depend on anything else: the first kUnroll
// chunks' code words and scales, and the first 32 tile-map entries.
struct RowHead {
  uint4 pk[kUnroll];
  float s[kUnroll];
  unsigned long long ent;
};

__device__ __forceinline__ float group_scale(const GemvArgs& a, int64_t gid) {
  if (a.sdq) {
    const float2 ms = __ldg(reinterpret_cast<const float2*>(a.sdq_consts) + (gid >> 8));
    return __fadd_rn(ms.x, __fmul_rn((float)__ldg(a.sdq_codes + gid), ms.y));
  }
  return __half2float(__ushort_as_half(__ldg(a.scales + gid)));
}

__device__ __forceinline__ void load_chunks(const GemvArgs& a, int64_t row, int c0, int nch, int lane,
                                            uint4* pk, float* s) {
  const int64_t rowe = row * a.cols;
  const uint4* cp = reinterpret_cast<const uint4*>(a.codes) + (rowe >> 5) + lane;
  const int lim = (int)a.cols - 32 * lane;  // chunk c is active for this lane when 1024c < lim
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const int c = c0 + u;
    pk[u] = make_uint4(0u, 0u, 0u, 0u);
    s[u] = 0.0f;
    if (c < nch && 1024 * c < lim) {
      pk[u] = __ldg(cp + 32 * c);
      s[u] = group_scale(a, (rowe >> 7) + 8 * c + (lane >> 2));
    }
  }
}

__device__ __forceinline__ void load_head(const GemvArgs& a, const Prm& pr, int64_t row, int nch, int n_cb,
                                          int lane, RowHead& h) {
  load_chunks(a, row, 0, nch, lane, h.pk, h.s);
  h.ent = 0ull;
  if (a.map && lane < n_cb) h.ent = __ldg(a.map + a.tile_off + row * n_cb + lane);
}

template <int M>
__device__ __forceinline__ void dense_chunks(const float* xb, int xs_stride, int c0, const uint4* pk,
                                             const float* s, float* acc) {
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    if (s[u] == 0.0f) continue;  // beyond the row, or an all-zero group (all codes 0)
    const float* xc = xb + 1024 * (c0 + u);
    const uint32_t wd[4] = {pk[u].x, pk[u].y, pk[u].z, pk[u].w};
    float2 part[M];
#pragma unroll
    for (int m = 0; m < M; ++m) part[m] = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int k = 0; k < 4; ++k) {  // word k: inputs 8k .. 8k + 7 of the lane's 32
      const uint32_t lo = (wd[k] & 0x0F0F0F0Fu) ^ 0x08080808u;
      const uint32_t hi = ((wd[k] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float4 x0 = *reinterpret_cast<const float4*>(xc + m * xs_stride + 256 * k);
        const float4 x1 = *reinterpret_cast<const float4*>(xc + m * xs_stride + 256 * k + 128);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 0), make_float2(x0.x, x0.y), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 1), make_float2(x0.z, x0.w), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 2), make_float2(x1.x, x1.y), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 3), make_float2(x1.z, x1.w), part[m]);
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] = __fmaf_rn(__fadd_rn(part[m].x, part[m].y), s[u], acc[m]);
  }
}

template <int M>
__global__ void __launch_bounds__(32 * kGemvWarps) gemv_warp_kernel(Prm pr, GemvArgs a, int xs_stride) {
  extern __shared__ float4 xs4[];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  {
    float* xw = reinterpret_cast<float*>(xs4);
    const int n4 = (int)(a.cols >> 2), tot = M * n4;
    for (int base = 0; base < tot; base += 4 * blockDim.x) {
      float4 v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int idx = base + threadIdx.x + i * blockDim.x;
        if (idx < tot) v[i] = __ldg(reinterpret_cast<const float4*>(a.x) + idx);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int idx = base + threadIdx.x + i * blockDim.x;
        if (idx < tot) {
          const int m = idx / n4, r = idx - m * n4;
          *reinterpret_cast<float4*>(xw + m * xs_stride + xs_index(4 * (int64_t)r)) = v[i];
        }
      }
    }
  }
  __syncthreads();
  const int n_cb = (int)(a.cols / pr.C);
  const int nch = (int)((a.cols + 1023) >> 10);
  const float* xsm = reinterpret_cast<const float*>(xs4);  // x in shared memory (permuted)
  const float* xb = xsm + 4 * lane;
  const int64_t stride = (int64_t)gridDim.x * kGemvWarps;
  const bool pre = a.map && pr.P * pr.W <= kPrefetchWords;  // recorded lanes prefetch their mask words
  int64_t row = (int64_t)blockIdx.x * kGemvWarps + warp;
  RowHead cur;
  if (row < a.rows) load_head(a, pr, row, nch, n_cb, lane, cur);
  for (; row < a.rows; row += stride) {
    // the next row's head is in flight while this row is computed
    RowHead nxt;
    if (row + stride < a.rows) load_head(a, pr, row + stride, nch, n_cb, lane, nxt);
    float acc[M];
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] = 0.0f;
    dense_chunks<M>(xb, xs_stride, 0, cur.pk, cur.s, acc);
    for (int c0 = kUnroll; c0 < nch; c0 += kUnroll) {
      uint4 pk[kUnroll];
      float s[kUnroll];
      load_chunks(a, row, c0, nch, lane, pk, s);
      dense_chunks<M>(xb, xs_stride, c0, pk, s, acc);
    }
    if (a.map) {
      const unsigned long long* mrow = a.map + a.tile_off + row * n_cb;
      for (int tb = 0; tb < n_cb; tb += 32) {
        const unsigned long long ent =
            tb == 0 ? cur.ent : ((tb + lane < n_cb) ? __ldg(mrow + tb + lane) : 0ull);
        unsigned rec = __ballot_sync(0xffffffffu, ent != 0ull);
        if (!rec) continue;
        // every recorded lane fetches its tile's record codes (and mask words)
        uint2 cw = make_uint2(0u, 0u);
        unsigned long long mw[kPrefetchWords];
#pragma unroll
        for (int i = 0; i < kPrefetchWords; ++i) mw[i] = 0ull;
        if (ent != 0ull) {
          cw = __ldg(reinterpret_cast<const uint2*>(a.rcodes + ((int64_t)(ent >> 32) - 1)));
          if (pre) {
            const uint64_t* mk = a.masks + (size_t)((uint32_t)(ent >> 16) & 0xFFFFu) * pr.P * pr.W;
#pragma unroll
            for (int i = 0; i < kPrefetchWords; ++i)
              if (i < pr.P * pr.W) mw[i] = __ldg(mk + i);
          }
        }
        while (rec) {
          const int src = __ffs(rec) - 1;
          rec &= rec - 1;
          const unsigned long long en = __shfl_sync(0xffffffffu, ent, src);
          const uint32_t cx = __shfl_sync(0xffffffffu, cw.x, src), cy = __shfl_sync(0xffffffffu, cw.y, src);
          unsigned long long wv[kPrefetchWords];
#pragma unroll
          for (int i = 0; i < kPrefetchWords; ++i) wv[i] = pre ? __shfl_sync(0xffffffffu, mw[i], src) : 0ull;
          const uint32_t seed = (uint32_t)(en >> 16) & 0xFFFFu;
          const float sc = sidecar_scale(pr, (int16_t)(uint16_t)(en & 0xFFFFull));
          const uint64_t* mk = a.masks + (size_t)seed * pr.P * pr.W;
          const int64_t col0 = (int64_t)(tb + src) * pr.C;
          for (int j = lane; j < pr.C; j += 32) {
            const int wj = j >> 6, sh = j & 63;
            int kj = 0;
#pragma unroll
            for (int p = 0; p < kMaxP; ++p) {
              if (p < pr.P) {
                // prefetched words are indexed statically (one word per atom when C <= 64)
                const unsigned long long word = (pre && pr.W == 1) ? wv[p] : __ldg(mk + p * pr.W + wj);
                const int cpv = (int)(int8_t)((p < 4 ? cx : cy) >> (8 * (p & 3)));
                kj += ((word >> sh) & 1ull) ? -cpv : cpv;
              }
            }
            const float r = __fmul_rn(__fmul_rn((float)kj, pr.c), sc);
#pragma unroll
            for (int m = 0; m < M; ++m) acc[m] = __fmaf_rn(r, xsm[m * xs_stride + xs_index(col0 + j)], acc[m]);
          }
        }
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) {
      float v = acc[m];
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, off));
      if (lane == 0) a.y[(int64_t)m * a.rows + row] = v;
    }
    cur = nxt;
  }
}

unsigned persistent_grid(int64_t rows, int nsm, int per_sm) {
  const int64_t need = (rows + kGemvWarps - 1) / kGemvWarps;
  const int64_t cap = (int64_t)nsm * (per_sm > 0 ? per_sm : 1);
  return (unsigned)(need < cap ? need : cap);
}

}  // namespace

cudaError_t launch_gemv(const Prm& pr, const GemvArgs& a, int M, cudaStream_t st) {
  const dim3 block(32 * kGemvWarps);
  // x staged in shared memory (whole 1024-column chunks per vector) when it fits
  const int64_t xs_stride = (a.cols + 1023) / 1024 * 1024;
  const size_t smem = (size_t)M * xs_stride * 4;
  if (smem <= kGemvSmemMax) {
    // persistent blocks: as many as fit on the device, each staging x once
    int dev = 0, nsm = 0, per_sm = 0;
    cudaError_t e = cudaGetDevice(&dev);
    if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
    if (e != cudaSuccess) return e;
#define AWSRC_GEMV_CASE(MM)                                                                              \
  case MM:                                                                                             \
    e = cudaFuncSetAttribute(gemv_warp_kernel<MM>, cudaFuncAttributeMaxDynamicSharedMemorySize,        \
                             (int)kGemvSmemMax);                                                       \
    if (e != cudaSuccess) return e;                                                                    \
    e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemv_warp_kernel<MM>, 32 * kGemvWarps, smem); \
    if (e != cudaSuccess) return e;                                                                    \
    gemv_warp_kernel<MM><<<persistent_grid(a.rows, nsm, per_sm), block, smem, st>>>(pr, a, (int)xs_stride); \
    break;
    switch (M) {
      AWSRC_GEMV_CASE(1) AWSRC_GEMV_CASE(2) AWSRC_GEMV_CASE(3) AWSRC_GEMV_CASE(4)
      AWSRC_GEMV_CASE(5) AWSRC_GEMV_CASE(6) AWSRC_GEMV_CASE(7) AWSRC_GEMV_CASE(8)
      default: return cudaErrorInvalidValue;
    }
#undef AWSRC_GEMV_CASE
    note_launches(1);
    return cudaGetLastError();
  }
  const dim3 grid((unsigned)a.rows);
  switch (M) {
    case 1: gemv_kernel<1><<<grid, block, 0, st>>>(pr, a); break;
    case 2: gemv_kernel<2><<<grid, block, 0, st>>>(pr, a); break;
    case 3: gemv_kernel<3><<<grid, block, 0, st>>>(pr, a); break;
    case 4: gemv_kernel<4><<<grid, block, 0, st>>>(pr, a); break;
    case 5: gemv_kernel<5><<<grid, block, 0, st>>>(pr, a); break;
    case 6: gemv_kernel<6><<<grid, block, 0, st>>>(pr, a); break;
    case 7: gemv_kernel<7><<<grid, block, 0, st>>>(pr, a); break;
    case 8: gemv_kernel<8><<<grid, block, 0, st>>>(pr, a); break;
    default: return cudaErrorInvalidValue;
  }
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
