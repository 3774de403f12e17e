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
// is exact as an integer count of 2^-24), the largest deviation, the step and
// the 8-bit codes,
// and writes W0 = q * s~ from the codes it kept in registers (nibbles turned
// into floats by a byte permute into 2^23 + (q + 8) and one subtraction).
// One launch serves a batch of modules: block b takes SDQ block b - block0 of
// the module whose block range holds b.
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
// The pair's codes as floats go to q; the returned word holds t + kMagic of
// each (its low byte carries the code's nibble).
__device__ __forceinline__ float2 rtn_fast2(float2 w, float rs, bool& tie, float2& q) {
  const float2 t = __fmul2_rn(w, make_float2(rs, rs));
  const float2 u = __fadd2_rn(t, make_float2(kMagic, kMagic));
  q = __fadd2_rn(u, make_float2(-kMagic, -kMagic));
  const float2 d = __fadd2_rn(t, make_float2(-q.x, -q.y));
  tie |= fmaxf(fabsf(d.x), fabsf(d.y)) > 0.5f - 0x1p-16f;
  return u;
}

// The 8 codes (element 2i in the low nibble of byte i) from the low bytes of
// t + kMagic of elements 0 .. 7.
__device__ __forceinline__ uint32_t pack_codes(const float2* u) {
  const uint32_t e01 = __byte_perm(__float_as_uint(u[0].x), __float_as_uint(u[1].x), 0x0040u);  // 0, 2
  const uint32_t e23 = __byte_perm(__float_as_uint(u[2].x), __float_as_uint(u[3].x), 0x0040u);  // 4, 6
  const uint32_t o01 = __byte_perm(__float_as_uint(u[0].y), __float_as_uint(u[1].y), 0x0040u);  // 1, 3
  const uint32_t o23 = __byte_perm(__float_as_uint(u[2].y), __float_as_uint(u[3].y), 0x0040u);  // 5, 7
  const uint32_t ev = __byte_perm(e01, e23, 0x5410u), od = __byte_perm(o01, o23, 0x5410u);
  return (ev & 0x0F0F0F0Fu) | ((od << 4) & 0xF0F0F0F0u);
}

// Codes i of a packed word as floats (two's complement nibbles): q + 8 is put
// in the low byte of 2^23 and 2^23 + 8 subtracted, exactly.
__device__ __forceinline__ void unpack_codes(uint32_t pk, float* q) {
  const uint32_t lo = (pk & 0x0F0F0F0Fu) ^ 0x08080808u, hi = ((pk >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
#pragma unroll
  for (int b = 0; b < 4; ++b) {
    const float2 v = __fadd2_rn(make_float2(__uint_as_float(__byte_perm(lo, 0x4B000000u, 0x7540u + b)),
                                            __uint_as_float(__byte_perm(hi, 0x4B000000u, 0x7540u + b))),
                                make_float2(-8388616.0f, -8388616.0f));
    q[2 * b] = v.x;
    q[2 * b + 1] = v.y;
  }
}

// Exact code of one input: clamp(rint(RN(w / s)), -8, 7), 0 when s == 0.
__device__ __forceinline__ uint32_t rtn_exact(float w, float s) {
  if (!(s > 0.0f)) return 0u;
  const float q = fminf(fmaxf(rintf(__fdiv_rn(w, s)), -8.0f), 7.0f);
  return (uint32_t)(int)q & 15u;
}

template <typename TI, typename TO>
__global__ void __launch_bounds__(32 * kRtnWarps) rtn_kernel(const __grid_constant__ RtnArgs a) {
  __shared__ float sv[kSdqBlock];
  __shared__ long long red_i[kRtnWarps];
  __shared__ float red_f[kRtnWarps];
  __shared__ float mu_step[2];
  int ti = 0;
  for (int i = 1; i < a.n; ++i)
    if ((int)blockIdx.x >= a.t[i].block0) ti = i;
  const RtnTask& tk = a.t[ti];
  const TI* __restrict__ W = static_cast<const TI*>(tk.W);
  TO* __restrict__ W0 = static_cast<TO*>(tk.W0);
  uint32_t* __restrict__ codes = tk.codes;
  uint16_t* __restrict__ scales = tk.scales;
  const int64_t G = tk.G;
  const int sdq = tk.sdq;
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5, h = lane >> 4, hl = lane & 15;
  const int64_t blk = (int64_t)blockIdx.x - tk.block0;
  const int64_t g0 = blk * kSdqBlock;
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
      float2 qf[4];
      if (!slow) {
        const float rs = rcp_rn(s);
        float2 u[4];
#pragma unroll
        for (int i = 0; i < 4; ++i) u[i] = rtn_fast2(make_float2(w[2 * i], w[2 * i + 1]), rs, slow, qf[i]);
        pk = pack_codes(u);
      }
      const bool exact = __any_sync(0xffffffffu, slow);
      if (exact) {
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
        if (!sdq && W0) {  // the integer codes (no -0) times s
          float q[8];
          if (exact) {
            unpack_codes(pk, q);
          } else {
#pragma unroll
            for (int i = 0; i < 4; ++i) {
              q[2 * i] = qf[i].x;
              q[2 * i + 1] = qf[i].y;
            }
          }
          float o[8];
#pragma unroll
          for (int i = 0; i < 8; i += 2) {
            const float2 v = __fmul2_rn(make_float2(q[i], q[i + 1]), make_float2(s, s));
            o[i] = v.x;
            o[i + 1] = v.y;
          }
          Elt<TO>::st8(W0 + g * kRtnGroup + 8 * hl, o);
        }
      }
    }
  }
  if (!sdq) return;
  __syncthreads();
  // second level: mean, largest deviation, step, codes. Every s_g is a
  // binary16 value, an integer multiple of 2^-24 below 2^16, so the block's sum
  // is exact as an integer count of 2^-24 (below 2^48, exact in double too);
  // for a whole block (n = 256) the mean is RN(sum * 2^-32), one rounding.
  const int t = threadIdx.x;
  long long sum = t < n ? __float2ll_rn(__fmul_rn(sv[t], 0x1p24f)) : 0ll;
#pragma unroll
  for (int off = 16; off > 0; off >>= 1) sum += __shfl_xor_sync(0xffffffffu, sum, off);
  if (lane == 0) red_i[warp] = sum;
  __syncthreads();
  if (t == 0) {
    long long tot = 0;
    for (int i = 0; i < kRtnWarps; ++i) tot += red_i[i];
    mu_step[0] = n == kSdqBlock ? __fmul_rn(__ll2float_rn(tot), 0x1p-32f)
                                : __double2float_rn(__ddiv_rn(__dmul_rn((double)tot, 0x1p-24), (double)n));
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
    if (tk.sdq_consts) {
      tk.sdq_consts[2 * blk] = mu;
      tk.sdq_consts[2 * blk + 1] = mu_step[1];
    }
  }
  __syncthreads();
  const float step = mu_step[1];
  if (t < n) {
    const float c = step > 0.0f ? fminf(fmaxf(rintf(__fdiv_rn(__fsub_rn(sv[t], mu), step)), -127.0f), 127.0f)
                                : 0.0f;
    if (tk.sdq_codes) tk.sdq_codes[g0 + t] = (int8_t)(int)c;
    sv[t] = __fadd_rn(mu, __fmul_rn(c, step));  // s~ replaces s (each thread its own entry)
  }
  __syncthreads();
  if (!W0) return;
#pragma unroll
  for (int k = 0; k < kIters; ++k) {
    const int lg = 2 * warp + h + 2 * kRtnWarps * k;
    if (lg >= n) continue;
    const float st = sv[lg];
    float q[8], o[8];
    unpack_codes(qs[k], q);
#pragma unroll
    for (int i = 0; i < 8; i += 2) {
      const float2 v = __fmul2_rn(make_float2(q[i], q[i + 1]), make_float2(st, st));
      o[i] = v.x;
      o[i + 1] = v.y;
    }
    Elt<TO>::st8(W0 + (g0 + lg) * kRtnGroup + 8 * hl, o);
  }
}

template <typename TI, typename TO>
cudaError_t launch_rtn_t(RtnArgs a, cudaStream_t st) {
  int blocks = 0;
  for (int i = 0; i < a.n; ++i) {
    a.t[i].block0 = blocks;
    blocks += (int)((a.t[i].G + kSdqBlock - 1) / kSdqBlock);
  }
  rtn_kernel<TI, TO><<<(unsigned)blocks, 32 * kRtnWarps, 0, st>>>(a);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

int rtn_group() { return kRtnGroup; }
int sdq_block() { return kSdqBlock; }

int64_t rtn_max_blocks() { return 1ll << 30; }

cudaError_t launch_rtn(const RtnArgs& a, int w_dtype, int w0_dtype, cudaStream_t st) {
  const bool f32in = w_dtype == AWSRC_DTYPE_F32, f32out = w0_dtype == AWSRC_DTYPE_F32;
  if (f32in && f32out) return launch_rtn_t<float, float>(a, st);
  if (f32in) return launch_rtn_t<float, __nv_bfloat16>(a, st);
  if (f32out) return launch_rtn_t<__nv_bfloat16, float>(a, st);
  return launch_rtn_t<__nv_bfloat16, __nv_bfloat16>(a, st);
}

}  // namespace awsrc
