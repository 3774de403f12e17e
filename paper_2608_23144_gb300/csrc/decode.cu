// decode.cu — the decoder of Sec. 3.2: W_hat = W0 + B_s alpha_hat on tiles
// named by records, W0 elsewhere (Eq. 1); any prefix of a progressive stream
// decodes the same way (Sec. 3.3).
//
//  scatter   one thread per record: unpack tile, seed, scale, codes; bounds-
//            check tile < T and seed < S (a bad record is skipped and flagged);
//            map[tile] = k and a 16-byte decoded record dec[k].
//  dense     streams every element of W0 to W_hat with 16-byte vector loads and
//            stores (two groups in flight per thread); a group whose tile has a
//            record adds r_hat_j = fl(fl(k_j * C^-1/2) * scale), k_j = sum_p
//            sign * code_p computed exactly in integers.
//  inplace   one warp per record touches only that tile of W_hat.
#include <algorithm>

#include "internal.h"

namespace awsrc {

namespace {

struct DecRec {   // 16 bytes
  uint16_t seed;
  int16_t scale;
  int32_t pad;
  int8_t code[8];
};

struct DecArgs {
  int n_mod;
  int64_t T, L, h, K;  // K < 0: read from the header
  int64_t kmax;        // records that fit in the stream buffer (<= T)
  DecodeMod m[kMaxModsPerLaunch];
};

__device__ __forceinline__ int ceil_log2_dev(uint64_t x) {
  return x <= 1 ? 0 : 64 - __clzll((long long)(x - 1));
}

__device__ __forceinline__ uint64_t get_bits(const uint8_t* rec, int* pos, int nbits) {
  uint64_t v = 0;
  for (int k = 0; k < nbits; ++k, ++*pos)
    if ((rec[*pos >> 3] >> (*pos & 7)) & 1u) v |= 1ull << k;
  return v;
}

__device__ __forceinline__ int64_t sign_extend(uint64_t v, int bits) {
  if (bits == 0) return 0;
  const uint64_t m = 1ull << (bits - 1);
  return (int64_t)((v ^ m) - m);
}

// Records to apply: K itself, or the header's count when K < 0; never more than
// kmax, the records that fit in the caller's stream buffer.
__device__ __forceinline__ int64_t stream_K(const uint8_t* stream, int64_t K, int64_t kmax) {
  if (K >= 0) return min(K, kmax);
  uint64_t v = 0;
  for (int i = 0; i < 8; ++i) v |= (uint64_t)stream[32 + i] << (8 * i);
  return v > (uint64_t)kmax ? kmax : (int64_t)v;
}

// Unpack record k; returns the tile or -1 when it names a tile/seed out of range.
__device__ __forceinline__ int64_t unpack(const Prm& pr, const uint8_t* stream, int64_t T, int64_t L,
                                          int64_t h, int64_t k, DecRec* d) {
  const uint8_t* rec = stream + h + k * L;
  int pos = 0;
  const int64_t tile = (int64_t)get_bits(rec, &pos, ceil_log2_dev((uint64_t)T));
  const uint32_t seed = (uint32_t)get_bits(rec, &pos, ceil_log2_dev((uint64_t)pr.S));
  const uint64_t sf = get_bits(rec, &pos, pr.b_e);
  d->seed = (uint16_t)seed;
  d->scale = pr.scale_mode == AWSRC_SCALE_POW2 ? (int16_t)(sign_extend(sf, pr.b_e) + pr.e_bias)
                                               : (int16_t)(uint16_t)sf;
  d->pad = 0;
  for (int p = 0; p < 8; ++p)
    d->code[p] = p < pr.P ? (int8_t)sign_extend(get_bits(rec, &pos, pr.b), pr.b) : (int8_t)0;
  if (tile >= T || seed >= (uint32_t)pr.S) return -1;
  return tile;
}

__global__ void scatter_kernel(Prm pr, const uint8_t* __restrict__ stream, int64_t T, int64_t L,
                               int64_t h, int64_t K, int64_t kmax, int32_t* __restrict__ map,
                               DecRec* __restrict__ dec, uint32_t* __restrict__ status) {
  const int64_t Kd = stream_K(stream, K, kmax);
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < Kd;
       k += (int64_t)gridDim.x * blockDim.x) {
    DecRec d;
    const int64_t tile = unpack(pr, stream, T, L, h, k, &d);
    if (tile < 0) { atomicOr(status, kFaultRecord); continue; }
    dec[k] = d;
    if (map) map[tile] = (int32_t)k;
  }
}

__device__ __forceinline__ float scale_of(const Prm& pr, int16_t s) {
  if (pr.scale_mode == AWSRC_SCALE_POW2) return __int_as_float((s + 127) << 23);
  return __half2float(__ushort_as_half((unsigned short)s));
}

template <typename T> struct Io;
template <> struct Io<float> {
  static __device__ __forceinline__ float ld(const float* p, int i) { return p[i]; }
  static __device__ __forceinline__ float cvt(float v) { return v; }
};
template <> struct Io<__nv_bfloat16> {
  static __device__ __forceinline__ float ld(const __nv_bfloat16* p, int i) { return __bfloat162float(p[i]); }
  static __device__ __forceinline__ __nv_bfloat16 cvt(float v) { return __float2bfloat16_rn(v); }
};

// G consecutive elements (one vector) starting at element e of a module.
template <typename TI, int G>
struct alignas(sizeof(TI) * G) Vec { TI v[G]; };

template <typename TI, typename TO, int G>
__device__ __forceinline__ void apply_group(const Prm& pr, const Vec<TI, G>& in, int j0,
                                            const DecRec* dr, const uint64_t* __restrict__ masks,
                                            Vec<TO, G>* out) {
  float w[G];
#pragma unroll
  for (int g = 0; g < G; ++g) w[g] = Io<TI>::ld(in.v, g);
  if (dr) {
    const uint64_t* mk = masks + (size_t)dr->seed * pr.P * pr.W + (j0 >> 6);
    int kj[G];
#pragma unroll
    for (int g = 0; g < G; ++g) kj[g] = 0;
    for (int p = 0; p < pr.P; ++p) {
      const uint64_t bits = mk[(size_t)p * pr.W] >> (j0 & 63);
      const int cp = dr->code[p];
#pragma unroll
      for (int g = 0; g < G; ++g) kj[g] += ((bits >> g) & 1ull) ? -cp : cp;
    }
    const float sc = scale_of(pr, dr->scale);
#pragma unroll
    for (int g = 0; g < G; ++g)
      w[g] = __fadd_rn(w[g], __fmul_rn(__fmul_rn((float)kj[g], pr.c), sc));
  }
#pragma unroll
  for (int g = 0; g < G; ++g) out->v[g] = Io<TO>::cvt(w[g]);
}

template <typename TI, typename TO, int G>
__global__ void __launch_bounds__(256) dense_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                    const int32_t* __restrict__ map,
                                                    const DecRec* __restrict__ dec,
                                                    const uint64_t* __restrict__ masks) {
  const DecodeMod& md = a.m[blockIdx.y];
  const int64_t ngroups = md.rows * md.cols / G;
  const TI* __restrict__ src = static_cast<const TI*>(md.W0);
  TO* __restrict__ dst = static_cast<TO*>(md.out);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  int64_t gi = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  for (; gi + stride < ngroups; gi += 2 * stride) {
    const int64_t g1 = gi + stride;
    const Vec<TI, G> v0 = *reinterpret_cast<const Vec<TI, G>*>(src + gi * G);
    const Vec<TI, G> v1 = *reinterpret_cast<const Vec<TI, G>*>(src + g1 * G);
    const int32_t r0 = __ldg(map + md.tile_off + ((gi * G) >> pr.logC));
    const int32_t r1 = __ldg(map + md.tile_off + ((g1 * G) >> pr.logC));
    DecRec d0, d1;
    if (r0 >= 0) d0 = dec[r0];
    if (r1 >= 0) d1 = dec[r1];
    Vec<TO, G> o0, o1;
    apply_group<TI, TO, G>(pr, v0, (int)((gi * G) & (pr.C - 1)), r0 >= 0 ? &d0 : nullptr, masks, &o0);
    apply_group<TI, TO, G>(pr, v1, (int)((g1 * G) & (pr.C - 1)), r1 >= 0 ? &d1 : nullptr, masks, &o1);
    *reinterpret_cast<Vec<TO, G>*>(dst + gi * G) = o0;
    *reinterpret_cast<Vec<TO, G>*>(dst + g1 * G) = o1;
  }
  if (gi < ngroups) {
    const Vec<TI, G> v0 = *reinterpret_cast<const Vec<TI, G>*>(src + gi * G);
    const int32_t r0 = map[md.tile_off + ((gi * G) >> pr.logC)];
    DecRec d0;
    if (r0 >= 0) d0 = dec[r0];
    Vec<TO, G> o0;
    apply_group<TI, TO, G>(pr, v0, (int)((gi * G) & (pr.C - 1)), r0 >= 0 ? &d0 : nullptr, masks, &o0);
    *reinterpret_cast<Vec<TO, G>*>(dst + gi * G) = o0;
  }
}

// One warp per record; W_hat already holds W0 (same dtype).
template <typename TO>
__global__ void inplace_kernel(Prm pr, const __grid_constant__ DecArgs a,
                               const uint8_t* __restrict__ stream, const uint64_t* __restrict__ masks,
                               uint32_t* __restrict__ status) {
  const int64_t Kd = stream_K(stream, a.K, a.kmax);
  const int lane = threadIdx.x & 31;
  const int64_t warps = (int64_t)gridDim.x * (blockDim.x >> 5);
  for (int64_t k = ((int64_t)blockIdx.x * blockDim.x + threadIdx.x) >> 5; k < Kd; k += warps) {
    DecRec d;
    const int64_t tile = unpack(pr, stream, a.T, a.L, a.h, k, &d);
    if (tile < 0) {
      if (lane == 0) atomicOr(status, kFaultRecord);
      continue;
    }
    const DecodeMod& mlast = a.m[a.n_mod - 1];
    if (tile < a.m[0].tile_off || tile >= mlast.tile_off + mlast.rows * mlast.cols / pr.C) continue;
    int mi = 0;
    for (int i = 1; i < a.n_mod; ++i)
      if (tile >= a.m[i].tile_off) mi = i;
    const DecodeMod& md = a.m[mi];
    TO* dst = static_cast<TO*>(md.out) + (tile - md.tile_off) * pr.C;
    const float sc = scale_of(pr, d.scale);
    const uint64_t* mk = masks + (size_t)d.seed * pr.P * pr.W;
    for (int j = lane; j < pr.C; j += 32) {
      int kj = 0;
      for (int p = 0; p < pr.P; ++p) {
        const uint64_t bit = (mk[(size_t)p * pr.W + (j >> 6)] >> (j & 63)) & 1ull;
        kj += bit ? -d.code[p] : d.code[p];
      }
      const float w = Io<TO>::ld(dst, j);
      dst[j] = Io<TO>::cvt(__fadd_rn(w, __fmul_rn(__fmul_rn((float)kj, pr.c), sc)));
    }
  }
}

template <typename TI, typename TO, int G>
cudaError_t launch_dense_t(const Prm& pr, const DecArgs& a, const int32_t* map, const DecRec* dec,
                           const uint64_t* masks, cudaStream_t st) {
  int64_t maxg = 0;
  for (int i = 0; i < a.n_mod; ++i) maxg = std::max<int64_t>(maxg, a.m[i].rows * a.m[i].cols / G);
  int dev = 0, nsm = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (maxg + 2 * 256 - 1) / (2 * 256);
  const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)nsm * 8));
  dense_kernel<TI, TO, G><<<dim3(gx, a.n_mod), 256, 0, st>>>(pr, a, map, dec, masks);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_dense_group(const Prm& pr, const DecArgs& a, int w0_dtype, int out_dtype,
                               const int32_t* map, const DecRec* dec, const uint64_t* masks,
                               cudaStream_t st) {
  const bool f32in = (w0_dtype == AWSRC_DTYPE_F32), f32out = (out_dtype == AWSRC_DTYPE_F32);
  if (f32in && f32out) return launch_dense_t<float, float, 4>(pr, a, map, dec, masks, st);
  if (f32in) return launch_dense_t<float, __nv_bfloat16, 4>(pr, a, map, dec, masks, st);
  if (pr.C >= 8) {
    if (f32out) return launch_dense_t<__nv_bfloat16, float, 8>(pr, a, map, dec, masks, st);
    return launch_dense_t<__nv_bfloat16, __nv_bfloat16, 8>(pr, a, map, dec, masks, st);
  }
  if (f32out) return launch_dense_t<__nv_bfloat16, float, 4>(pr, a, map, dec, masks, st);
  return launch_dense_t<__nv_bfloat16, __nv_bfloat16, 4>(pr, a, map, dec, masks, st);
}

cudaError_t launch_decode(const Prm& pr, int n_mod, const DecodeMod* mods, int64_t T, int64_t L,
                          int64_t h, const uint8_t* stream, int64_t K, int64_t kmax, int out_dtype, int mode,
                          const uint64_t* masks, int32_t* map, uint32_t* status, cudaStream_t st) {
  cudaError_t e;
  if (mode == AWSRC_DECODE_DENSE) {
    // map[T] then decoded records dec[T]
    DecRec* dec = reinterpret_cast<DecRec*>(map + align_up((size_t)T, 64));
    e = cudaMemsetAsync(map, 0xff, (size_t)T * sizeof(int32_t), st);
    if (e != cudaSuccess) return e;
    const int64_t work = (K >= 0 ? std::min(K, kmax) : kmax);
    if (work > 0) {
      const unsigned gx = (unsigned)std::min<int64_t>((work + 255) / 256, 65535);
      scatter_kernel<<<gx, 256, 0, st>>>(pr, stream, T, L, h, K, kmax, map, dec, status);
      note_launches(1);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
    // launches over runs of at most 16 modules sharing the input dtype
    int i0 = 0;
    while (i0 < n_mod) {
      int i1 = i0 + 1;
      while (i1 < n_mod && i1 - i0 < kMaxModsPerLaunch && mods[i1].w0_dtype == mods[i0].w0_dtype) ++i1;
      DecArgs a;
      a.n_mod = i1 - i0;
      a.T = T; a.L = L; a.h = h; a.K = K; a.kmax = kmax;
      for (int i = 0; i < a.n_mod; ++i) a.m[i] = mods[i0 + i];
      if ((e = launch_dense_group(pr, a, mods[i0].w0_dtype, out_dtype, map, dec, masks, st)) != cudaSuccess)
        return e;
      i0 = i1;
    }
    return cudaSuccess;
  }
  // in place: every launch walks the record list and applies the records that
  // fall in its group of modules
  for (int i0 = 0; i0 < n_mod; i0 += kMaxModsPerLaunch) {
    DecArgs a;
    a.n_mod = std::min(kMaxModsPerLaunch, n_mod - i0);
    a.T = T; a.L = L; a.h = h; a.K = K; a.kmax = kmax;
    for (int i = 0; i < a.n_mod; ++i) a.m[i] = mods[i0 + i];
    const int64_t work = K >= 0 ? std::min(K, kmax) : kmax;
    if (work == 0) continue;
    const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>((work + 7) / 8, 65535));
    if (out_dtype == AWSRC_DTYPE_F32) inplace_kernel<float><<<gx, 256, 0, st>>>(pr, a, stream, masks, status);
    else inplace_kernel<__nv_bfloat16><<<gx, 256, 0, st>>>(pr, a, stream, masks, status);
    note_launches(1);
    if ((e = cudaGetLastError()) != cudaSuccess) return e;
  }
  return cudaSuccess;
}

size_t decode_scratch_bytes(int64_t T, int mode) {
  if (mode != AWSRC_DECODE_DENSE) return 0;
  return align_up((size_t)T, 64) * sizeof(int32_t) + (size_t)T * sizeof(DecRec);
}

}  // namespace awsrc
