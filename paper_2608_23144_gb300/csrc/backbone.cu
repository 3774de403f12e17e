// backbone.cu — the RTN-INT4 backbone W0 = Q(W) of Eq. 1 (round to nearest,
// symmetric, groups of 128 consecutive input coordinates of a row, Sec. 4)
// with optional scale double quantisation (SDQ, Sec. 3.3).
//
// One block per SDQ block of 256 groups (32768 weights); warp w takes groups
// w, w + 8, ... of it, lane l elements 4l .. 4l + 3 of each (coalesced 8- or
// 16-byte loads, 2 bytes of packed codes per lane). The group's largest |w|
// is a warp reduction; s = binary16(max / 7) and q = clamp(rint(w / s), -8, 7)
// as binary32 operations. With SDQ the block then forms the mean of its scales
// (their sum is exact in double), the largest deviation, the step and the
// 8-bit codes, and writes W0 = q * s~ from the codes it kept in registers.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int kRtnGroup = 128;
constexpr int kSdqBlock = 256;  // groups per second-level block = groups per CUDA block
constexpr int kRtnWarps = 8;
constexpr int kGroupsPerWarp = kSdqBlock / kRtnWarps;

template <typename T> struct Elt;
template <> struct Elt<float> {
  static __device__ __forceinline__ void ld4(const float* p, float* v) {
    const float4 f = *reinterpret_cast<const float4*>(p);
    v[0] = f.x; v[1] = f.y; v[2] = f.z; v[3] = f.w;
  }
  static __device__ __forceinline__ void st4(float* p, const float* v) {
    *reinterpret_cast<float4*>(p) = make_float4(v[0], v[1], v[2], v[3]);
  }
};
template <> struct Elt<__nv_bfloat16> {
  static __device__ __forceinline__ void ld4(const __nv_bfloat16* p, float* v) {
    const uint2 u = *reinterpret_cast<const uint2*>(p);
    v[0] = __uint_as_float(u.x << 16); v[1] = __uint_as_float(u.x & 0xffff0000u);
    v[2] = __uint_as_float(u.y << 16); v[3] = __uint_as_float(u.y & 0xffff0000u);
  }
  static __device__ __forceinline__ void st4(__nv_bfloat16* p, const float* v) {
    const __nv_bfloat162 a = __floats2bfloat162_rn(v[0], v[1]), b = __floats2bfloat162_rn(v[2], v[3]);
    uint2 u;
    memcpy(&u.x, &a, 4);
    memcpy(&u.y, &b, 4);
    *reinterpret_cast<uint2*>(p) = u;
  }
};

__device__ __forceinline__ int code_at(uint32_t packed, int i) {  // 4-bit two's complement
  return (int)((int32_t)(packed << (28 - 4 * i)) >> 28);
}

template <typename TI, typename TO>
__global__ void __launch_bounds__(32 * kRtnWarps) rtn_kernel(const TI* __restrict__ W, int64_t G, int sdq,
                                                             uint16_t* __restrict__ codes,
                                                             uint16_t* __restrict__ scales,
                                                             int8_t* __restrict__ sdq_codes,
                                                             float* __restrict__ sdq_consts, TO* __restrict__ W0) {
  __shared__ float sv[kSdqBlock];
  __shared__ double red_d[kRtnWarps];
  __shared__ float red_f[kRtnWarps];
  __shared__ float mu_step[2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t g0 = (int64_t)blockIdx.x * kSdqBlock;
  const int n = G - g0 < kSdqBlock ? (int)(G - g0) : kSdqBlock;
  uint32_t qs[kGroupsPerWarp / 2];  // this lane's 4 codes of each of the warp's groups, 16 bits each
#pragma unroll
  for (int k = 0; k < kGroupsPerWarp / 2; ++k) qs[k] = 0u;
#pragma unroll
  for (int k = 0; k < kGroupsPerWarp; ++k) {
    const int lg = warp + kRtnWarps * k;
    if (lg >= n) break;
    const int64_t g = g0 + lg;
    float w[4];
    Elt<TI>::ld4(W + g * kRtnGroup + 4 * lane, w);
    float m = fmaxf(fmaxf(fabsf(w[0]), fabsf(w[1])), fmaxf(fabsf(w[2]), fabsf(w[3])));
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
    const __half h = __float2half_rn(__fdiv_rn(m, 7.0f));
    const float s = __half2float(h);
    uint32_t pk = 0u;
    float q[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      q[i] = s > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(w[i], s)), -8.0f), 7.0f) : 0.0f;
      pk |= ((uint32_t)(int)q[i] & 15u) << (4 * i);
    }
    codes[g * (kRtnGroup / 4) + lane] = (uint16_t)pk;
    qs[k >> 1] |= pk << (16 * (k & 1));
    if (lane == 0) {
      sv[lg] = s;
      if (scales) scales[g] = __half_as_ushort(h);
    }
    if (!sdq && W0) {
      float o[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) o[i] = __fmul_rn((float)(int)q[i], s);  // the integer code: no -0
      Elt<TO>::st4(W0 + g * kRtnGroup + 4 * lane, o);
    }
  }
  if (!sdq) return;
  __syncthreads();
  // second level: mean (exact sum in double), largest deviation, step, codes
  const int t = threadIdx.x;
  double sum = t < n ? (double)sv[t] : 0.0;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  if (lane == 0) red_d[warp] = sum;
  __syncthreads();
  if (t == 0) {
    double tot = 0.0;
    for (int i = 0; i < kRtnWarps; ++i) tot += red_d[i];
    mu_step[0] = __double2float_rn(__ddiv_rn(tot, (double)n));
  }
  __syncthreads();
  const float mu = mu_step[0];
  float dev = t < n ? fabsf(__fsub_rn(sv[t], mu)) : 0.0f;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) dev = fmaxf(dev, __shfl_xor_sync(0xffffffffu, dev, off));
  if (lane == 0) red_f[warp] = dev;
  __syncthreads();
  if (t == 0) {
    float a = 0.0f;
    for (int i = 0; i < kRtnWarps; ++i) a = fmaxf(a, red_f[i]);
    mu_step[1] = __fdiv_rn(a, 127.0f);
    if (sdq_consts) {
      sdq_consts[2 * blockIdx.x] = mu;
      sdq_consts[2 * blockIdx.x + 1] = mu_step[1];
    }
  }
  __syncthreads();
  const float step = mu_step[1];
  if (t < n) {
    const float c = step > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(__fsub_rn(sv[t], mu), step)), -127.0f), 127.0f)
                                : 0.0f;
    if (sdq_codes) sdq_codes[g0 + t] = (int8_t)(int)c;
    sv[t] = __fadd_rn(mu, __fmul_rn(c, step));  // s~ replaces s (each thread its own entry)
  }
  __syncthreads();
  if (!W0) return;
#pragma unroll
  for (int k = 0; k < kGroupsPerWarp; ++k) {
    const int lg = warp + kRtnWarps * k;
    if (lg >= n) break;
    const float st = sv[lg];
    const uint32_t pk = qs[k >> 1] >> (16 * (k & 1));
    float o[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) o[i] = __fmul_rn((float)code_at(pk, i), st);
    Elt<TO>::st4(W0 + (g0 + lg) * kRtnGroup + 4 * lane, o);
  }
}

template <typename TI>
cudaError_t launch_rtn_ti(const void* W, int64_t G, int sdq, uint16_t* codes, uint16_t* scales, int8_t* sc8,
                          float* consts, void* W0, int w0_dtype, cudaStream_t st) {
  const unsigned nb = (unsigned)((G + kSdqBlock - 1) / kSdqBlock);
  const TI* w = static_cast<const TI*>(W);
  if (w0_dtype == AWSRC_DTYPE_F32)
    rtn_kernel<TI, float><<<nb, 32 * kRtnWarps, 0, st>>>(w, G, sdq, codes, scales, sc8, consts,
                                                          static_cast<float*>(W0));
  else
    rtn_kernel<TI, __nv_bfloat16><<<nb, 32 * kRtnWarps, 0, st>>>(w, G, sdq, codes, scales, sc8, consts,
                                                                  static_cast<__nv_bfloat16*>(W0));
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

int rtn_group() { return kRtnGroup; }
int sdq_block() { return kSdqBlock; }

cudaError_t launch_rtn(const void* W, int w_dtype, int64_t rows, int64_t cols, int sdq, uint8_t* codes,
                       uint16_t* scales, int8_t* sdq_codes, float* sdq_consts, void* W0, int w0_dtype,
                       cudaStream_t st) {
  const int64_t G = rows * cols / kRtnGroup;
  uint16_t* c16 = reinterpret_cast<uint16_t*>(codes);
  return w_dtype == AWSRC_DTYPE_F32
             ? launch_rtn_ti<float>(W, G, sdq, c16, scales, sdq_codes, sdq_consts, W0, w0_dtype, st)
             : launch_rtn_ti<__nv_bfloat16>(W, G, sdq, c16, scales, sdq_codes, sdq_consts, W0, w0_dtype, st);
}

}  // namespace awsrc
