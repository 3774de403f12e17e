// gemv.cu — the decoded weights of one module applied to M vectors without
// forming them: y[m] = (W0 + r_hat) x[m], with W0 = q * s_eff read from the
// packed RTN-INT4 backbone (binary16 or SDQ scales, Sec. 3.3) and r_hat the
// decoder's residual (Sec. 3.2) on the tiles a prepared sidecar names. This is
// the packed-inference use the paper leaves to future work (Sec. 5).
//
// One block per output row, 8 warps taking interleaved runs of 4 groups of 128
// inputs (lane l: elements 4l .. 4l + 3 of each group; its 4 codes are 16 bits).
// For each run a warp issues all independent loads first (codes, scales, tile
// map entries, x), then the dependent ones of recorded tiles (record codes and
// mask words). Per element, w = fl(q * s_eff) as in W0 and r = fl(fl(k * C^-1/2)
// * scale) as in the decoder; both are accumulated into binary32 sums with
// fma, reduced over lanes and warps.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int kGemvWarps = 8;
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
        const uint2 cw = __ldg(a.rcodes + k);
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

}  // namespace

cudaError_t launch_gemv(const Prm& pr, const GemvArgs& a, int M, cudaStream_t st) {
  const dim3 grid((unsigned)a.rows), block(32 * kGemvWarps);
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
