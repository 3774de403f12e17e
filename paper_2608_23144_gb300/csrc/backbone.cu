// backbone.cu — the RTN-INT4 backbone W0 = Q(W) of Eq. 1 (round to nearest,
// symmetric, groups of 128 consecutive input coordinates of a row, Sec. 4)
// with optional scale double quantisation (SDQ, Sec. 3.3).
//
// One block of 16 warps per SDQ block of 256 groups (32768 weights). A
// half-warp takes one group of 128 inputs, lane l its 8 consecutive inputs
// 8(l mod 16) .. + 7 (one 16- or 32-byte load, 4 bytes of packed codes); warp
// w takes groups 2w + h + 32k (h its half, k = 0..7), loads of 4 iterations in
// flight. The group's largest |w| is a half-warp reduction, s =
// binary16(max / 7). The code q = clamp(rint(w / s), -8, 7) comes from
// t = w RN(1/s), rounded to an integer by adding 1.5 * 2^23: it equals the
// code of the correctly rounded quotient unless t lies near a half-integer
// (rtn_fast), and needs no clamp when s is a normal binary16 (|w / s| <= 7.004);
// a warp iteration with any such element takes the division for all of its
// elements. With SDQ the block then forms the mean of its scales (their sum
// is exact in double), the largest deviation, the step and the 8-bit codes,
// and writes W0 = q * s~ from the codes it kept in registers.
#include "internal.h"

namespace awsrc {

namespace {

constexpr int kRtnGroup = 128;
constexpr int kSdqBlock = 256;  // groups per second-level block = groups per CUDA block
constexpr int kRtnWarps = 16;
constexpr int kIters = kSdqBlock / (2 * kRtnWarps);  // 8 group pairs per warp
constexpr int kInFlight = 4;                         // iterations whose loads are issued together

template <typename T> struct Elt;
template <> struct Elt<float> {
  struct Raw { float4 a, b; };
  static __device__ __forceinline__ Raw ld(const float* p) {
    return {__ldg(reinterpret_cast<const float4*>(p)), __ldg(reinterpret_cast<const float4*>(p) + 1)};
  }
  static __device__ __forceinline__ void cvt8(const Raw& r, float* v) {
    v[0] = r.a.x; v[1] = r.a.y; v[2] = r.a.z; v[3] = r.a.w;
    v[4] = r.b.x; v[5] = r.b.y; v[6] = r.b.z; v[7] = r.b.w;
  }
  static __device__ __forceinline__ void st8(float* p, const float* v) {
    reinterpret_cast<float4*>(p)[0] = make_float4(v[0], v[1], v[2], v[3]);
    reinterpret_cast<float4*>(p)[1] = make_float4(v[4], v[5], v[6], v[7]);
  }
};
template <> struct Elt<__nv_bfloat16> {
  using Raw = uint4;
  static __device__ __forceinline__ Raw ld(const __nv_bfloat16* p) { return __ldg(reinterpret_cast<const uint4*>(p)); }
  static __device__ __forceinline__ void cvt8(const Raw& u, float* v) {
    const uint32_t w[4] = {u.x, u.y, u.z, u.w};
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      v[2 * i] = __uint_as_float(w[i] << 16);
      v[2 * i + 1] = __uint_as_float(w[i] & 0xffff0000u);
    }
  }
  static __device__ __forceinline__ void st8(__nv_bfloat16* p, const float* v) {
    uint32_t w[4];
#pragma unroll
    for (int i = 0; i < 4; ++i) {
      const __nv_bfloat162 h = __floats2bfloat162_rn(v[2 * i], v[2 * i + 1]);
      memcpy(&w[i], &h, 4);
    }
    *reinterpret_cast<uint4*>(p) = make_uint4(w[0], w[1], w[2], w[3]);
  }
};

constexpr float kMagic = 12582912.0f;  // 1.5 * 2^23: x + kMagic rounds x to an integer (ties to even)

// Codes of two inputs for a normal binary16 s, rs = RN(1/s). t = RN(w rs) =
// (w / s)(1 + d) with |d| < 2^-23 + 2^-48 and |w / s| <= 7.004, so
// |t - RN(w / s)| < 2^-20 and rint(t) = rint(RN(w / s)) unless t is within
// 2^-20 of a half-integer; `tie` is set when |t - rint(t)| > 1/2 - 2^-16 (the
// caller then divides). |t| < 7.5 needs no clamp. The integer sits in the low
// mantissa bits of t + kMagic (two's complement, so its low nibble is the code).
__device__ __forceinline__ uint32_t rtn_fast2(float2 w, float rs, bool& tie) {
  const float2 t = __fmul2_rn(w, make_float2(rs, rs));
  const float2 u = __fadd2_rn(t, make_float2(kMagic, kMagic));
  const float2 q = __fadd2_rn(u, make_float2(-kMagic, -kMagic));
  const float2 d = __fadd2_rn(t, make_float2(-q.x, -q.y));
  tie |= fabsf(d.x) > 0.5f - 0x1p-16f || fabsf(d.y) > 0.5f - 0x1p-16f;
  return (__float_as_uint(u.x) & 15u) | ((__float_as_uint(u.y) & 15u) << 4);
}

// Exact code of one input: clamp(rint(RN(w / s)), -8, 7), 0 when s == 0.
__device__ __forceinline__ uint32_t rtn_exact(float w, float s) {
  if (!(s > 0.0f)) return 0u;
  const float q = fminf(fmaxf(rintf(__fdiv_rn(w, s)), -8.0f), 7.0f);
  return (uint32_t)(int)q & 15u;
}

__device__ __forceinline__ int code_at(uint32_t packed, int i) {  // 4-bit two's complement
  return (int)((int32_t)(packed << (28 - 4 * i)) >> 28);
}

template <typename TI, typename TO>
__global__ void __launch_bounds__(32 * kRtnWarps) rtn_kernel(const TI* __restrict__ W, int64_t G, int sdq,
                                                             uint32_t* __restrict__ codes,
                                                             uint16_t* __restrict__ scales,
                                                             int8_t* __restrict__ sdq_codes,
                                                             float* __restrict__ sdq_consts, TO* __restrict__ W0) {
  __shared__ float sv[kSdqBlock];
  __shared__ double red_d[kRtnWarps];
  __shared__ float red_f[kRtnWarps];
  __shared__ float mu_step[2];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, h = lane >> 4, hl = lane & 15;
  const int64_t g0 = (int64_t)blockIdx.x * kSdqBlock;
  const int n = G - g0 < kSdqBlock ? (int)(G - g0) : kSdqBlock;
  uint32_t qs[kIters];  // this lane's 8 codes of each iteration
#pragma unroll
  for (int k0 = 0; k0 < kIters; k0 += kInFlight) {
    typename Elt<TI>::Raw raw[kInFlight];
#pragma unroll
    for (int k = k0; k < k0 + kInFlight; ++k) {
      const int lg = 2 * warp + h + 2 * kRtnWarps * k;
      if (lg < n) raw[k - k0] = Elt<TI>::ld(W + (g0 + lg) * kRtnGroup + 8 * hl);
    }
#pragma unroll
    for (int k = k0; k < k0 + kInFlight; ++k) {
      const int lg = 2 * warp + h + 2 * kRtnWarps * k;
      const bool act = lg < n;
      float w[8];
      if (act) Elt<TI>::cvt8(raw[k - k0], w);
      else
#pragma unroll
        for (int i = 0; i < 8; ++i) w[i] = 0.0f;
      float m = fabsf(w[0]);
#pragma unroll
      for (int i = 1; i < 8; ++i) m = fmaxf(m, fabsf(w[i]));
#pragma unroll
      for (int off = 8; off > 0; off >>= 1) m = fmaxf(m, __shfl_xor_sync(0xffffffffu, m, off));
      const __half hs = __float2half_rn(__fdiv_rn(m, 7.0f));
      const float s = __half2float(hs);
      bool slow = !(s >= 0x1p-14f);  // zero or subnormal binary16 scale
      uint32_t pk = 0u;
      if (!slow) {
        const float rs = __frcp_rn(s);
#pragma unroll
        for (int i = 0; i < 4; ++i) pk |= rtn_fast2(make_float2(w[2 * i], w[2 * i + 1]), rs, slow) << (8 * i);
      }
      if (__any_sync(0xffffffffu, slow)) {
        pk = 0u;
#pragma unroll
        for (int i = 0; i < 8; ++i) pk |= rtn_exact(w[i], s) << (4 * i);
      }
      qs[k] = pk;
      if (act) {
        const int64_t g = g0 + lg;
        codes[g * (kRtnGroup / 8) + hl] = pk;
        if (hl == 0) {
          sv[lg] = s;
          if (scales) scales[g] = __half_as_ushort(hs);
        }
        if (!sdq && W0) {
          float o[8];
#pragma unroll
          for (int i = 0; i < 8; ++i) o[i] = __fmul_rn((float)code_at(pk, i), s);  // the integer code: no -0
          Elt<TO>::st8(W0 + g * kRtnGroup + 8 * hl, o);
        }
      }
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
  for (int k = 0; k < kIters; ++k) {
    const int lg = 2 * warp + h + 2 * kRtnWarps * k;
    if (lg >= n) continue;
    const float st = sv[lg];
    float o[8];
#pragma unroll
    for (int i = 0; i < 8; ++i) o[i] = __fmul_rn((float)code_at(qs[k], i), st);
    Elt<TO>::st8(W0 + (g0 + lg) * kRtnGroup + 8 * hl, o);
  }
}

template <typename TI>
cudaError_t launch_rtn_ti(const void* W, int64_t G, int sdq, uint32_t* codes, uint16_t* scales, int8_t* sc8,
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
  uint32_t* c16 = reinterpret_cast<uint32_t*>(codes);
  return w_dtype == AWSRC_DTYPE_F32
             ? launch_rtn_ti<float>(W, G, sdq, c16, scales, sdq_codes, sdq_consts, W0, w0_dtype, st)
             : launch_rtn_ti<__nv_bfloat16>(W, G, sdq, c16, scales, sdq_codes, sdq_consts, W0, w0_dtype, st);
}

}  // namespace awsrc
