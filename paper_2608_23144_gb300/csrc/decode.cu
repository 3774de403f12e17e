// decode.cu — the decoder of Sec. 3.2: W_hat = W0 + B_s alpha_hat on tiles
// named by records, W0 elsewhere (Eq. 1); any prefix of a progressive stream
// decodes the same way (Sec. 3.3).
//
//  dense mode (C >= one vector):
//   prep     one block range generates the basis masks (basis_warp),
//            the other unpacks every record once: its codes go to a per-record
//            array and the tile's map entry (k + 1, seed, scale field) is
//            raised to it with atomicMax, so a tile named twice is flagged and
//            takes its later record.
//   fused    one streaming pass: 16-byte vectors, four in flight per thread
//            with their tiles' map entries; vectors of unrecorded tiles are
//            converted and stored at once, those of recorded tiles are queued
//            in shared memory and patched densely by the whole block:
//            W_hat_j = fl(W0_j + fl(fl(k_j * C^-1/2) * scale)) with
//            k_j = sum_p sign * code_p exact in integers.
//  in-place mode, and dense mode with tiles shorter than one vector (after a
//  plain copy of W0):
//   claim    one thread per record raises its tile's claim word to k + 1
//            (atomicMax), so a tile named twice is flagged and only its later
//            record is applied;
//   patch    one thread per vector of a recorded tile: unpack tile, seed, scale,
//            codes; bounds-check tile < T and seed < S (a bad record is skipped
//            and flagged); skip a record whose tile a later record claims;
//            rewrite the tile from W0, which may be W_hat itself.
#include <algorithm>
#include <utility>

#include "basis.cuh"
#include "codetab.cuh"
#include "internal.h"

namespace awsrc {

namespace {

// Programmatic dependent launch: a kernel launched with
// cudaLaunchAttributeProgrammaticStreamSerialization may start while the
// previous kernel of the stream runs; it must call pdl_wait() before touching
// anything that kernel writes. pdl_trigger() lets the next kernel launch early.
__device__ __forceinline__ void pdl_wait() { asm volatile("griddepcontrol.wait;" ::: "memory"); }
__device__ __forceinline__ void pdl_trigger() { asm volatile("griddepcontrol.launch_dependents;" ::: "memory"); }

struct DecRec {   // an unpacked record; codes packed as signed bytes, code p in byte p
  uint16_t seed;
  int16_t scale;
  uint32_t cw[2];
};

__device__ __forceinline__ int code_of(const DecRec& d, int p) {
  return (int)(int8_t)((p < 4 ? d.cw[0] : d.cw[1]) >> (8 * (p & 3)));
}

struct DecArgs {
  int n_mod;
  int64_t T, L, h, K;  // K < 0: read from the header
  int64_t kmax;        // records that fit in the stream buffer (<= T)
  const uint32_t* claim;  // record-by-record patch: per tile, 1 + the last record naming it (or null)
  DecodeMod m[kMaxModsPerLaunch];
};

__device__ __forceinline__ int ceil_log2_dev(uint64_t x) {
  return x <= 1 ? 0 : 64 - __clzll((long long)(x - 1));
}

// A record is at most 128 bits (tile < 2^32, seed < 2^16, scale <= 16 bits,
// codes <= 64 bits): read its L bytes little-endian into two words.
__device__ __forceinline__ void load_record(const uint8_t* rec, int L, uint64_t* w0, uint64_t* w1) {
  uint64_t a = 0, b = 0;
  for (int i = 0; i < L; ++i) {
    const uint64_t v = rec[i];
    if (i < 8) a |= v << (8 * i);
    else b |= v << (8 * (i - 8));
  }
  *w0 = a;
  *w1 = b;
}

// Bits [pos, pos + n) of the 128-bit value (w1:w0), n <= 64.
__device__ __forceinline__ uint64_t field(uint64_t w0, uint64_t w1, int pos, int n) {
  uint64_t v;
  if (pos >= 64) v = w1 >> (pos - 64);
  else if (pos == 0) v = w0;
  else v = (w0 >> pos) | (w1 << (64 - pos));
  return n >= 64 ? v : (v & ((1ull << n) - 1ull));
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
// `end` bounds the bytes that may be read (h + kmax*L); when the three 8-byte
// words around the record lie inside it and the stream is 8-byte aligned, the
// record is read with word loads and a funnel shift, else byte by byte.
__device__ __forceinline__ int64_t unpack(const Prm& pr, const uint8_t* stream, int64_t T, int64_t L,
                                          int64_t h, int64_t k, DecRec* d, int64_t end = -1) {
  uint64_t w0, w1;
  const int64_t off = h + k * L;
  const int64_t a0 = off & ~7ll;
  if (end >= 0 && a0 + 24 <= end && (reinterpret_cast<uintptr_t>(stream) & 7) == 0) {
    const uint64_t* q = reinterpret_cast<const uint64_t*>(stream + a0);
    const uint64_t x0 = __ldg(q), x1 = __ldg(q + 1), x2 = __ldg(q + 2);
    const int sh = (int)(off - a0) * 8;
    w0 = sh ? (x0 >> sh) | (x1 << (64 - sh)) : x0;
    w1 = sh ? (x1 >> sh) | (x2 << (64 - sh)) : x1;
  } else {
    load_record(stream + off, (int)L, &w0, &w1);
  }
  const int tb = ceil_log2_dev((uint64_t)T), sb = ceil_log2_dev((uint64_t)pr.S);
  int pos = 0;
  const int64_t tile = (int64_t)field(w0, w1, pos, tb);
  pos += tb;
  const uint32_t seed = (uint32_t)field(w0, w1, pos, sb);
  pos += sb;
  const uint64_t sf = field(w0, w1, pos, pr.b_e);
  pos += pr.b_e;
  d->seed = (uint16_t)seed;
  d->scale = pr.scale_mode == AWSRC_SCALE_POW2 ? (int16_t)(sign_extend(sf, pr.b_e) + pr.e_bias)
                                               : (int16_t)(uint16_t)sf;
  uint32_t c0 = 0u, c1 = 0u;
#pragma unroll
  for (int p = 0; p < 8; ++p) {
    if (p < pr.P) {
      const uint32_t c = (uint32_t)(uint8_t)(int8_t)sign_extend(field(w0, w1, pos, pr.b), pr.b);
      if (p < 4) c0 |= c << (8 * p);
      else c1 |= c << (8 * (p - 4));
      pos += pr.b;
    }
  }
  d->cw[0] = c0;
  d->cw[1] = c1;
  if (tile >= T || seed >= (uint32_t)pr.S) return -1;
  return tile;
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

// Raw vector type of the same width, for the streaming load/store intrinsics.
template <int BYTES> struct RawVec;
template <> struct RawVec<16> { using T = uint4; };
template <> struct RawVec<8> { using T = uint2; };

template <typename V>
__device__ __forceinline__ V ld_stream(const V* p) {
  constexpr int B = sizeof(V) >= 16 ? 16 : (int)sizeof(V);
  using R = typename RawVec<B>::T;
  V v;
#pragma unroll
  for (int i = 0; i < (int)sizeof(V) / B; ++i) {
    const R r = __ldcs(reinterpret_cast<const R*>(p) + i);
    memcpy(reinterpret_cast<char*>(&v) + i * B, &r, B);
  }
  return v;
}

template <typename V>
__device__ __forceinline__ void st_stream(V* p, const V& v) {
  constexpr int B = sizeof(V) >= 16 ? 16 : (int)sizeof(V);
  using R = typename RawVec<B>::T;
#pragma unroll
  for (int i = 0; i < (int)sizeof(V) / B; ++i) {
    R r;
    memcpy(&r, reinterpret_cast<const char*>(&v) + i * B, B);
    __stcs(reinterpret_cast<R*>(p) + i, r);
  }
}

// Pairs of converted elements: packed f32x2 arithmetic (each component
// rounded like the scalar form) and paired BF16 rounding.
template <typename T> struct Io2;
template <> struct Io2<float> {
  static __device__ __forceinline__ float2 ld(const float* p) { return make_float2(p[0], p[1]); }
  static __device__ __forceinline__ void st(float* p, float2 v) { p[0] = v.x; p[1] = v.y; }
};
template <> struct Io2<__nv_bfloat16> {
  static __device__ __forceinline__ float2 ld(const __nv_bfloat16* p) {
    return __bfloat1622float2(*reinterpret_cast<const __nv_bfloat162*>(p));
  }
  static __device__ __forceinline__ void st(__nv_bfloat16* p, float2 v) {
    *reinterpret_cast<__nv_bfloat162*>(p) = __float22bfloat162_rn(v);
  }
};

// One G-element vector of a recorded tile: o_j = fl(w_j + fl(fl(k_j * c) * sc))
// with k_j = sum_p sign_{j,p} * code_p = tot - 2 * sum_p bit_{j,p} * code_p
// (exact integers); mk points at atom 0's mask word of the vector, j0 its first
// element. PT = P when the atom count is fixed at compile time, else 0.
template <typename TI, typename TO, int G, int PT>
__device__ __forceinline__ void patch_vec(const Prm& pr, const Vec<TI, G>& w, uint2 cw,
                                          const uint64_t* __restrict__ mk, int j0, float sc, Vec<TO, G>& o) {
  const int P = PT ? PT : pr.P;
  int tot = 0, acc[G];
#pragma unroll
  for (int e = 0; e < G; ++e) acc[e] = 0;
#pragma unroll
  for (int p = 0; p < (PT ? PT : kMaxP); ++p) {
    if (p < P) {
      const uint32_t bits = (uint32_t)(__ldg(mk + (size_t)p * pr.W) >> (j0 & 63));
      const int cp = (int)(int8_t)((p < 4 ? cw.x : cw.y) >> (8 * (p & 3)));
      tot += cp;
#pragma unroll
      for (int e = 0; e < G; ++e) acc[e] += (int)((bits >> e) & 1u) * cp;
    }
  }
  const float2 c2 = make_float2(pr.c, pr.c), s2 = make_float2(sc, sc);
#pragma unroll
  for (int e = 0; e < G; e += 2) {
    const float2 k = make_float2((float)(tot - 2 * acc[e]), (float)(tot - 2 * acc[e + 1]));
    const float2 r = __fmul2_rn(__fmul2_rn(k, c2), s2);
    Io2<TO>::st(o.v + e, __fadd2_rn(Io2<TI>::ld(w.v + e), r));
  }
}

// The record slot of the dense decoder: the codes (x, y; code p in byte p)
// and, in table mode, T[0..7] (z, w).
__device__ __forceinline__ uint4 record_slot(const Prm& pr, const DecRec& d) {
  uint32_t t0 = 0u, t1 = 0u;
  if (code_tables(pr)) {
    const int c0 = code_of(d, 0), c1 = code_of(d, 1), c2 = code_of(d, 2), c3 = code_of(d, 3);
#pragma unroll
    for (int m = 0; m < 8; ++m) {
      const int v = c3 + ((m & 1) ? -c0 : c0) + ((m & 2) ? -c1 : c1) + ((m & 4) ? -c2 : c2);
      const uint32_t b = (uint32_t)(v & 0xFF) << (8 * (m & 3));
      if (m < 4) t0 |= b;
      else t1 |= b;
    }
  }
  return make_uint4(d.cw[0], d.cw[1], t0, t1);
}

// patch_vec in table mode: the same k_j, hence the same results bit for bit.
template <typename TI, typename TO, int G>
__device__ __forceinline__ void patch_vec_tab(const Prm& pr, const Vec<TI, G>& w, const uint4& slot, uint4 nb,
                                              int j0, float sc, Vec<TO, G>& o) {
  const KTab kt = k_tables(slot);
  const KMagic km = k_magic(pr);
  float k[G];  // k_j c when c is a power of two, else k_j
  if constexpr (G == 8) {
    table_k4(kt, nb.x, nb.y, km, k);
    table_k4(kt, nb.x >> 16, nb.z, km, k + 4);
  } else {
    const bool hi = (j0 & 4) != 0;
    table_k4(kt, hi ? nb.x >> 16 : nb.x, hi ? nb.z : nb.y, km, k);
  }
  if (!km.folded) {
#pragma unroll
    for (int e = 0; e < G; ++e) k[e] = __fmul_rn(k[e], pr.c);
  }
  const float2 s2 = make_float2(sc, sc);
#pragma unroll
  for (int e = 0; e < G; e += 2) {
    const float2 r = __fmul2_rn(make_float2(k[e], k[e + 1]), s2);
    Io2<TO>::st(o.v + e, __fadd2_rn(Io2<TI>::ld(w.v + e), r));
  }
}

// Dense-mode record pass: record k's slot (record_slot) goes to codes[k] and
// map[tile] is raised to (k + 1) << 32 | seed << 16 | scale field (map cleared to 0
// beforehand). Records naming a tile or seed out of range, and tiles named
// twice, raise kFaultRecord. Threads [i0, i0 + n) of a grid-stride range.
__device__ __forceinline__ void map_records(const Prm& pr, const DecArgs& a, const uint8_t* __restrict__ stream,
                                            unsigned long long* __restrict__ map, uint4* __restrict__ codes,
                                            uint32_t* __restrict__ status, int64_t i0, int64_t n) {
  const int64_t Kd = stream_K(stream, a.K, a.kmax);
  const int64_t end = a.h + a.kmax * a.L;
  for (int64_t k = i0; k < Kd; k += n) {
    DecRec d;
    const int64_t tile = unpack(pr, stream, a.T, a.L, a.h, k, &d, end);
    pdl_wait();  // the map is cleared by the previous kernel
    if (tile < 0) {
      atomicOr(status, kFaultRecord);
      continue;
    }
    codes[k] = record_slot(pr, d);
    const unsigned long long e = ((unsigned long long)(k + 1) << 32) | ((unsigned long long)d.seed << 16) |
                                 (unsigned long long)(uint16_t)d.scale;
    if (atomicMax(map + tile, e) != 0ull) atomicOr(status, kFaultRecord);
  }
}

// Dense pass: W_hat = convert(W0) for every element, a pure stream with U
// independent 16-byte vectors in flight per thread and no dependent loads.
// With `basis`, the blocks of grid slice y = 0 (dispatched first) generate the
// basis masks (8 warps per block, basis_warp), overlapping GenBasis with the
// memory-bound stream of the other slices.
template <typename TI, typename TO, int G>
__global__ void __launch_bounds__(256) copy_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                   uint64_t* __restrict__ masks, int basis) {
  constexpr int U = 4;
  int y = blockIdx.y;
  if (basis) {
    if (y == 0) {
      __shared__ __align__(16) uint8_t bsm[8][kBasisSmem];
      const int warp = threadIdx.x >> 5;
      basis_warp(pr, masks, (int64_t)blockIdx.x * 8 + warp, pr.S, bsm[warp]);
      return;
    }
    --y;
  }
  const DecodeMod& md = a.m[y];
  const int64_t ngroups = md.rows * md.cols / G;
  const Vec<TI, G>* __restrict__ src = static_cast<const Vec<TI, G>*>(md.W0);
  Vec<TO, G>* __restrict__ dst = static_cast<Vec<TO, G>*>(md.out);
  const int64_t stride = (int64_t)gridDim.x * blockDim.x;
  for (int64_t g0 = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; g0 < ngroups; g0 += U * stride) {
    Vec<TI, G> v[U];
#pragma unroll
    for (int u = 0; u < U; ++u)
      if (g0 + u * stride < ngroups) v[u] = ld_stream(src + g0 + u * stride);
#pragma unroll
    for (int u = 0; u < U; ++u) {
      if (g0 + u * stride >= ngroups) break;
      Vec<TO, G> o;
#pragma unroll
      for (int g = 0; g < G; ++g) o.v[g] = Io<TO>::cvt(Io<TI>::ld(v[u].v, g));
      st_stream(dst + g0 + u * stride, o);
    }
  }
}

// Patch pass: G-element groups of the recorded tiles, one thread per group
// (C/G threads per record, adjacent threads on the same record), so each
// record's tile moves as whole 16-byte vectors and many records are in flight.
// W_hat = fl(W0 + r_hat) is computed from W0, which may be W_hat itself.
// One thread per G-element group of a recorded tile (C/G adjacent threads per
// record), so each record's tile moves as coalesced 16-byte vectors.
template <typename TI, typename TO, int G>
__global__ void __launch_bounds__(256) patch_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                    const uint8_t* __restrict__ stream,
                                                    const uint64_t* __restrict__ masks,
                                                    uint32_t* __restrict__ status) {
  const int64_t Kd = stream_K(stream, a.K, a.kmax);
  const int gshift = pr.logC - (G == 8 ? 3 : 2);  // log2 of the groups per tile
  const int64_t total = Kd << gshift;
  const int64_t end = a.h + a.kmax * a.L;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total;
       x += (int64_t)gridDim.x * blockDim.x) {
    const int64_t k = x >> gshift;
    const int gj = (int)(x & ((1 << gshift) - 1));
    DecRec d;
    const int64_t tile = unpack(pr, stream, a.T, a.L, a.h, k, &d, end);
    if (tile < 0) {
      if (gj == 0) atomicOr(status, kFaultRecord);
      continue;
    }
    const DecodeMod& mlast = a.m[a.n_mod - 1];
    if (tile < a.m[0].tile_off || tile >= mlast.tile_off + mlast.rows * mlast.cols / pr.C) continue;
    int mi = 0;
    for (int i = 1; i < a.n_mod; ++i)
      if (tile >= a.m[i].tile_off) mi = i;
    if (a.claim && a.claim[tile] != (uint32_t)(k + 1)) continue;  // a later record names this tile
    const DecodeMod& md = a.m[mi];
    const int j0 = gj * G;
    const int64_t e0 = (tile - md.tile_off) * pr.C + j0;
    const Vec<TI, G> v = *reinterpret_cast<const Vec<TI, G>*>(static_cast<const TI*>(md.W0) + e0);
    Vec<TO, G> o;
    patch_vec<TI, TO, G, 0>(pr, v, make_uint2(d.cw[0], d.cw[1]),
                            masks + (size_t)d.seed * pr.P * pr.W + (j0 >> 6), j0, scale_of(pr, d.scale), o);
    *reinterpret_cast<Vec<TO, G>*>(static_cast<TO*>(md.out) + e0) = o;
  }
}

// Tiles smaller than one vector take one thread per element.
template <typename TI, typename TO>
__global__ void __launch_bounds__(256) patch_small_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                          const uint8_t* __restrict__ stream,
                                                          const uint64_t* __restrict__ masks,
                                                          uint32_t* __restrict__ status) {
  const int64_t Kd = stream_K(stream, a.K, a.kmax);
  const int64_t total = Kd * pr.C;
  for (int64_t x = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; x < total;
       x += (int64_t)gridDim.x * blockDim.x) {
    const int64_t k = x >> pr.logC;
    const int j = (int)(x & (pr.C - 1));
    DecRec d;
    const int64_t tile = unpack(pr, stream, a.T, a.L, a.h, k, &d);
    if (tile < 0) {
      if (j == 0) atomicOr(status, kFaultRecord);
      continue;
    }
    const DecodeMod& mlast = a.m[a.n_mod - 1];
    if (tile < a.m[0].tile_off || tile >= mlast.tile_off + mlast.rows * mlast.cols / pr.C) continue;
    int mi = 0;
    for (int i = 1; i < a.n_mod; ++i)
      if (tile >= a.m[i].tile_off) mi = i;
    if (a.claim && a.claim[tile] != (uint32_t)(k + 1)) continue;  // a later record names this tile
    const DecodeMod& md = a.m[mi];
    const int64_t e = (tile - md.tile_off) * pr.C + j;
    const uint64_t* mk = masks + (size_t)d.seed * pr.P * pr.W;
    int kj = 0;
    for (int p = 0; p < pr.P; ++p) kj += ((mk[(size_t)p * pr.W + (j >> 6)] >> (j & 63)) & 1ull) ? -code_of(d, p) : code_of(d, p);
    const float w = Io<TI>::ld(static_cast<const TI*>(md.W0) + e, 0);
    static_cast<TO*>(md.out)[e] = Io<TO>::cvt(__fadd_rn(w, __fmul_rn(__fmul_rn((float)kj, pr.c), scale_of(pr, d.scale))));
  }
}

// Claims for the record-by-record patch: claim[tile] = 1 + the largest record
// index naming the tile, so that exactly one record (the later one) rewrites
// a tile named twice, whatever the order the patch threads run in; the second
// naming is reported. One thread per record; claim holds T zeroed words.
__global__ void __launch_bounds__(256) claim_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                    const uint8_t* __restrict__ stream,
                                                    uint32_t* __restrict__ claim, uint32_t* __restrict__ status) {
  const int64_t Kd = stream_K(stream, a.K, a.kmax);
  const int64_t end = a.h + a.kmax * a.L;
  for (int64_t k = (int64_t)blockIdx.x * blockDim.x + threadIdx.x; k < Kd; k += (int64_t)gridDim.x * blockDim.x) {
    DecRec d;
    const int64_t tile = unpack(pr, stream, a.T, a.L, a.h, k, &d, end);
    if (tile < 0) continue;  // flagged by the patch pass
    if (atomicMax(claim + tile, (uint32_t)(k + 1)) != 0u) atomicOr(status, kFaultRecord);
  }
}

// Dense pass with the patches fused in. A block walks chunks of 1024 vectors (16 bytes each,
// four per thread, coalesced): vectors of tiles without a record are converted
// and stored at once; those of recorded tiles (about 16% at 0.162 bits/weight)
// go, with their W0 data and map entry, to a queue in shared memory that all
// threads then patch densely. C >= G.
constexpr int kFusedThreads = 256;
constexpr int kFusedU = 4;
constexpr int kFusedChunk = kFusedThreads * kFusedU;

struct FusedQ {
  uint4 w0;                 // the vector's W0 bits
  unsigned long long e;     // map entry
  long long g;              // vector index within the module
};

template <typename TI, typename TO, int G, int PT>
__global__ void __launch_bounds__(kFusedThreads, 4) fused_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                                 const unsigned long long* __restrict__ map,
                                                                 const uint4* __restrict__ codes,
                                                                 const uint64_t* __restrict__ masks,
                                                                 const uint4* __restrict__ nib) {
  static_assert(sizeof(Vec<TI, G>) == 16, "16-byte vectors");
  __shared__ FusedQ q[kFusedChunk];
  __shared__ int qn;
  const DecodeMod& md = a.m[blockIdx.y];
  const int64_t ngroups = md.rows * md.cols / G;
  const int vshift = pr.logC - (G == 8 ? 3 : 2);  // log2 of the vectors per tile
  const Vec<TI, G>* __restrict__ src = static_cast<const Vec<TI, G>*>(md.W0);
  Vec<TO, G>* __restrict__ dst = static_cast<Vec<TO, G>*>(md.out);
  const unsigned long long* __restrict__ mmap = map + md.tile_off;
  const int lane = threadIdx.x & 31;
  pdl_wait();  // masks, map and codes come from the preparation kernel
  for (int64_t c0 = (int64_t)blockIdx.x * kFusedChunk; c0 < ngroups; c0 += (int64_t)gridDim.x * kFusedChunk) {
    if (threadIdx.x == 0) qn = 0;
    __syncthreads();
    Vec<TI, G> v[kFusedU];
    unsigned long long r[kFusedU];
#pragma unroll
    for (int u = 0; u < kFusedU; ++u) {
      const int64_t g = c0 + u * kFusedThreads + threadIdx.x;
      r[u] = 0ull;
      if (g < ngroups) {
        v[u] = ld_stream(src + g);
        r[u] = __ldg(mmap + (g >> vshift));
      }
    }
#pragma unroll
    for (int u = 0; u < kFusedU; ++u) {
      const int64_t g = c0 + u * kFusedThreads + threadIdx.x;
      const bool in = g < ngroups;
      const bool patch = in && r[u] != 0ull;
      if (in && !patch) {
        Vec<TO, G> o;
#pragma unroll
        for (int e = 0; e < G; e += 2) Io2<TO>::st(o.v + e, Io2<TI>::ld(v[u].v + e));
        st_stream(dst + g, o);
      }
      const unsigned m = __ballot_sync(0xffffffffu, patch);  // warp-aggregated append
      if (m) {
        int base = 0;
        if (lane == 0) base = atomicAdd(&qn, __popc(m));
        base = __shfl_sync(0xffffffffu, base, 0);
        if (patch) {
          FusedQ& x = q[base + __popc(m & ((1u << lane) - 1u))];
          memcpy(&x.w0, &v[u], 16);
          x.e = r[u];
          x.g = g;
        }
      }
    }
    __syncthreads();
    const int n = qn;
    for (int i = threadIdx.x; i < n; i += kFusedThreads) {
      const FusedQ x = q[i];
      Vec<TI, G> w;
      memcpy(&w, &x.w0, 16);
      const int64_t k = (int64_t)(x.e >> 32) - 1;
      const uint32_t seed = (uint32_t)(x.e >> 16) & 0xFFFFu;
      const int j0 = (int)(x.g & ((1 << vshift) - 1)) * G;
      Vec<TO, G> o;
      const uint4 slot = __ldg(codes + k);
      const float sc = scale_of(pr, (int16_t)(uint16_t)(x.e & 0xFFFFull));
      if (PT == 4 && nib) {
        patch_vec_tab<TI, TO, G>(pr, w, slot, __ldg(nib + (size_t)seed * (pr.C >> 3) + (j0 >> 3)), j0, sc, o);
      } else {
        patch_vec<TI, TO, G, PT>(pr, w, make_uint2(slot.x, slot.y), masks + (size_t)seed * pr.P * pr.W + (j0 >> 6),
                                 j0, sc, o);
      }
      st_stream(dst + x.g, o);
    }
    __syncthreads();
  }
}

// Clears the dense tile map (16-byte stores) and lets the preparation kernel
// launch at once: its mask generation and record unpacking overlap this pass.
__global__ void __launch_bounds__(256) zero_map_kernel(uint4* __restrict__ p, int64_t n16,
                                                       uint32_t* __restrict__ status) {
  pdl_trigger();
  if (blockIdx.x == 0 && threadIdx.x == 0) *status = 0u;  // the call's fault word
  for (int64_t i = (int64_t)blockIdx.x * 256 + threadIdx.x; i < n16; i += (int64_t)gridDim.x * 256)
    p[i] = make_uint4(0u, 0u, 0u, 0u);
}

// Launch with programmatic serialisation after the previous kernel of `st`.
template <typename... KArgs, typename... Args>
cudaError_t launch_pdl(void (*kern)(KArgs...), dim3 grid, dim3 block, cudaStream_t st, Args&&... args) {
  cudaLaunchConfig_t cfg = {};
  cfg.gridDim = grid;
  cfg.blockDim = block;
  cfg.dynamicSmemBytes = 0;
  cfg.stream = st;
  cudaLaunchAttribute attr[1];
  attr[0].id = cudaLaunchAttributeProgrammaticStreamSerialization;
  attr[0].val.programmaticStreamSerializationAllowed = 1;
  cfg.attrs = attr;
  cfg.numAttrs = 1;
  return cudaLaunchKernelEx(&cfg, kern, std::forward<Args>(args)...);
}

// Dense-mode preparation for the fused pass: blocks [0, nb) generate the masks
// (8 warps per block, basis_warp), the remaining blocks fill the tile map
// (map_records).
__global__ void __launch_bounds__(256) prep_kernel(Prm pr, const __grid_constant__ DecArgs a,
                                                   const uint8_t* __restrict__ stream,
                                                   uint64_t* __restrict__ masks,
                                                   unsigned long long* __restrict__ map,
                                                   uint4* __restrict__ codes, uint32_t* __restrict__ status,
                                                   uint4* __restrict__ nib, int nb) {
  pdl_trigger();  // the fused pass may launch now; it waits for this grid
  if ((int)blockIdx.x < nb) {
    __shared__ __align__(16) uint8_t bsm[8][kBasisSmem];
    const int warp = threadIdx.x >> 5;
    const int64_t w = (int64_t)blockIdx.x * 8 + warp;
    basis_warp(pr, masks, w, pr.S, bsm[warp]);
    if (nib && w < pr.S) {  // table mode: one selector per warp (C <= 64), one mask word per atom
      __syncwarp();  // the masks this warp just wrote
      const int lane = threadIdx.x & 31;
      if (lane < (pr.C >> 3))
        nib_window(masks + (size_t)w * 4, lane, nib + (size_t)w * (pr.C >> 3) + lane);
    }
    return;
  }
  map_records(pr, a, stream, map, codes, status, (int64_t)(blockIdx.x - nb) * blockDim.x + threadIdx.x,
              (int64_t)(gridDim.x - nb) * blockDim.x);
}

template <typename TI, typename TO, int G>
cudaError_t launch_fused_t(const Prm& pr, const DecArgs& a, const unsigned long long* map,
                           const uint4* codes, const uint64_t* masks, const uint4* nib, cudaStream_t st) {
  int64_t maxg = 0;
  for (int i = 0; i < a.n_mod; ++i) maxg = std::max<int64_t>(maxg, a.m[i].rows * a.m[i].cols / G);
  int dev = 0, nsm = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (maxg + kFusedChunk - 1) / kFusedChunk;
  const int64_t gx = std::max<int64_t>(1, std::min<int64_t>(want, (int64_t)nsm * 8));
  const dim3 grid((unsigned)gx, (unsigned)a.n_mod);
  cudaError_t e = pr.P == 4 ? launch_pdl(fused_kernel<TI, TO, G, 4>, grid, dim3(kFusedThreads), st, pr, a, map,
                                         codes, masks, nib)
                            : launch_pdl(fused_kernel<TI, TO, G, 0>, grid, dim3(kFusedThreads), st, pr, a, map,
                                         codes, masks, nib);
  note_launches(1);
  return e != cudaSuccess ? e : cudaGetLastError();
}

cudaError_t launch_fused(const Prm& pr, const DecArgs& a, int w0_dtype, int out_dtype,
                         const unsigned long long* map, const uint4* codes, const uint64_t* masks,
                         const uint4* nib, cudaStream_t st) {
  const bool f32in = (w0_dtype == AWSRC_DTYPE_F32), f32out = (out_dtype == AWSRC_DTYPE_F32);
  if (f32in && f32out) return launch_fused_t<float, float, 4>(pr, a, map, codes, masks, nib, st);
  if (f32in) return launch_fused_t<float, __nv_bfloat16, 4>(pr, a, map, codes, masks, nib, st);
  if (f32out) return launch_fused_t<__nv_bfloat16, float, 8>(pr, a, map, codes, masks, nib, st);
  return launch_fused_t<__nv_bfloat16, __nv_bfloat16, 8>(pr, a, map, codes, masks, nib, st);
}

// copy: stream the modules of `a`; basis: also generate the masks (an extra
// grid slice). With copy false only the basis slice runs.
template <typename TI, typename TO, int G>
cudaError_t launch_copy_t(const Prm& pr, DecArgs a, bool copy, bool basis, uint64_t* masks,
                          cudaStream_t st) {
  int64_t maxg = 0;
  if (!copy) a.n_mod = 0;
  for (int i = 0; i < a.n_mod; ++i) maxg = std::max<int64_t>(maxg, a.m[i].rows * a.m[i].cols / G);
  int dev = 0, nsm = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int64_t want = (maxg + 4 * 256 - 1) / (4 * 256);
  int64_t gx = std::min<int64_t>(want, (int64_t)nsm * 8);
  if (basis) {
    const int per = 8 * basis_warp_seeds(pr.C);
    gx = std::max<int64_t>(gx, (pr.S + per - 1) / per);
  }
  gx = std::max<int64_t>(gx, 1);
  copy_kernel<TI, TO, G><<<dim3((unsigned)gx, a.n_mod + (basis ? 1 : 0)), 256, 0, st>>>(pr, a, masks,
                                                                                      basis ? 1 : 0);
  note_launches(1);
  return cudaGetLastError();
}

template <typename TI, typename TO>
cudaError_t launch_patch_t(const Prm& pr, const DecArgs& a, const uint8_t* stream, const uint64_t* masks,
                           uint32_t* status, cudaStream_t st) {
  const int64_t work = a.K >= 0 ? std::min(a.K, a.kmax) : a.kmax;
  if (work <= 0) return cudaSuccess;
  constexpr int G = 16 / sizeof(TI) < 16 / sizeof(TO) ? 16 / sizeof(TI) : 16 / sizeof(TO);
  if (pr.C >= G) {
    const int64_t threads = work * (pr.C / G);
    const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>((threads + 255) / 256, 1 << 20));
    patch_kernel<TI, TO, G><<<gx, 256, 0, st>>>(pr, a, stream, masks, status);
  } else {
    const int64_t threads = work * pr.C;
    const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>((threads + 255) / 256, 1 << 20));
    patch_small_kernel<TI, TO><<<gx, 256, 0, st>>>(pr, a, stream, masks, status);
  }
  note_launches(1);
  return cudaGetLastError();
}

// copy (dense) and/or the mask slice (basis), then the record-by-record patch.
cudaError_t launch_group(const Prm& pr, const DecArgs& a, int w0_dtype, int out_dtype, bool copy,
                         bool basis, const uint8_t* stream, uint64_t* masks, uint32_t* status,
                         cudaStream_t st) {
  const bool f32in = (w0_dtype == AWSRC_DTYPE_F32), f32out = (out_dtype == AWSRC_DTYPE_F32);
  cudaError_t e = cudaSuccess;
  if (copy || basis) {
    if (f32in && f32out) e = launch_copy_t<float, float, 4>(pr, a, copy, basis, masks, st);
    else if (f32in) e = launch_copy_t<float, __nv_bfloat16, 4>(pr, a, copy, basis, masks, st);
    else if (f32out) e = launch_copy_t<__nv_bfloat16, float, 8>(pr, a, copy, basis, masks, st);
    else e = launch_copy_t<__nv_bfloat16, __nv_bfloat16, 8>(pr, a, copy, basis, masks, st);
    if (e != cudaSuccess) return e;
  }
  if (f32in && f32out) return launch_patch_t<float, float>(pr, a, stream, masks, status, st);
  if (f32in) return launch_patch_t<float, __nv_bfloat16>(pr, a, stream, masks, status, st);
  if (f32out) return launch_patch_t<__nv_bfloat16, float>(pr, a, stream, masks, status, st);
  return launch_patch_t<__nv_bfloat16, __nv_bfloat16>(pr, a, stream, masks, status, st);
}

}  // namespace

DenseScratch dense_scratch(const Prm& pr, int64_t T) {
  DenseScratch d;
  d.slots_off = align_up((size_t)T * 8, 256);
  d.nib_off = d.slots_off + align_up((size_t)T * 16, 256);
  d.bytes = d.nib_off + (code_tables(pr) ? align_up((size_t)pr.S * (pr.C / 8) * 16, 256) : 0);
  return d;
}

// Dense preparation: clear the tile map (and the fault word), then generate
// the masks (and, in table mode, the nibble tables) and unpack the records
// into the map and the record slots of `scratch` (layout: dense_scratch()).
cudaError_t launch_dense_prep(const Prm& pr, int64_t T, int64_t L, int64_t h, const uint8_t* stream, int64_t K,
                              int64_t kmax, uint64_t* masks, void* scratch, uint32_t* status, cudaStream_t st) {
  const DenseScratch ds = dense_scratch(pr, T);
  unsigned long long* map = static_cast<unsigned long long*>(scratch);
  uint4* codes = reinterpret_cast<uint4*>(static_cast<uint8_t*>(scratch) + ds.slots_off);
  uint4* nib = code_tables(pr) ? reinterpret_cast<uint4*>(static_cast<uint8_t*>(scratch) + ds.nib_off) : nullptr;
  DecArgs a;
  a.n_mod = 0;
  a.T = T; a.L = L; a.h = h; a.K = K; a.kmax = kmax;
  a.claim = nullptr;
  const int64_t work = K >= 0 ? std::min(K, kmax) : kmax;
  int dev = 0, nsm = 148;
  cudaGetDevice(&dev);
  cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  const int per = 8 * basis_warp_seeds(pr.C);
  const int nb = (pr.S + per - 1) / per;  // mask blocks, then record blocks (one record per thread)
  const int64_t nr = std::max<int64_t>(1, std::min<int64_t>((work + 255) / 256, (int64_t)nsm * 64));
  // the map region is align_up(T * 8, 256) bytes, so whole 16-byte words stay inside it
  const int64_t n16 = (T * 8 + 15) / 16;
  const unsigned gz = (unsigned)std::max<int64_t>(1, std::min<int64_t>((n16 + 255) / 256, (int64_t)nsm * 8));
  zero_map_kernel<<<gz, 256, 0, st>>>(reinterpret_cast<uint4*>(map), n16, status);
  note_launches(1);
  cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return e;
  e = launch_pdl(prep_kernel, dim3((unsigned)(nb + nr)), dim3(256), st, pr, a, stream, masks, map, codes, status,
                 nib, nb);
  note_launches(1);
  if (e == cudaSuccess) e = cudaGetLastError();
  return e;
}

// Launches over runs of at most 16 modules sharing the input dtype. DENSE with
// C >= G: the first run's copy also generates the masks and fills the tile map,
// then each run is patched in tile order; otherwise (INPLACE, or tiles shorter
// than one vector) the copy (DENSE only) is followed by a record-by-record patch.
cudaError_t launch_decode(const Prm& pr, int n_mod, const DecodeMod* mods, int64_t T, int64_t L,
                          int64_t h, const uint8_t* stream, int64_t K, int64_t kmax, int out_dtype, int mode,
                          uint64_t* masks, void* scratch, uint32_t* status, cudaStream_t st) {
  const bool fused = decode_clears_status(pr, mode) && scratch != nullptr;
  unsigned long long* map = nullptr;
  uint4* codes = nullptr;
  uint4* nib = nullptr;
  // the record-by-record patch with a workspace claims tiles first (without
  // one, as for the no-allocation entry point, the stream must name each tile
  // at most once)
  uint32_t* claim = (!fused && scratch != nullptr) ? static_cast<uint32_t*>(scratch) : nullptr;
  if (fused) {
    const DenseScratch ds = dense_scratch(pr, T);
    map = static_cast<unsigned long long*>(scratch);
    codes = reinterpret_cast<uint4*>(static_cast<uint8_t*>(scratch) + ds.slots_off);
    if (code_tables(pr)) nib = reinterpret_cast<uint4*>(static_cast<uint8_t*>(scratch) + ds.nib_off);
    const cudaError_t e = launch_dense_prep(pr, T, L, h, stream, K, kmax, masks, scratch, status, st);
    if (e != cudaSuccess) return e;
  }
  if (claim) {
    const int64_t work = K >= 0 ? std::min(K, kmax) : kmax;
    cudaError_t e = cudaMemsetAsync(claim, 0, (size_t)T * sizeof(uint32_t), st);
    if (e != cudaSuccess) return e;
    if (work > 0) {
      DecArgs a;
      a.n_mod = 0;
      a.T = T; a.L = L; a.h = h; a.K = K; a.kmax = kmax;
      a.claim = nullptr;
      const unsigned gx = (unsigned)std::max<int64_t>(1, std::min<int64_t>((work + 255) / 256, 1 << 20));
      claim_kernel<<<gx, 256, 0, st>>>(pr, a, stream, claim, status);
      note_launches(1);
      if ((e = cudaGetLastError()) != cudaSuccess) return e;
    }
  }
  int i0 = 0;
  while (i0 < n_mod) {
    int i1 = i0 + 1;
    while (i1 < n_mod && i1 - i0 < kMaxModsPerLaunch && mods[i1].w0_dtype == mods[i0].w0_dtype) ++i1;
    DecArgs a;
    a.n_mod = i1 - i0;
    a.T = T; a.L = L; a.h = h; a.K = K; a.kmax = kmax;
    a.claim = claim;
    for (int i = 0; i < a.n_mod; ++i) a.m[i] = mods[i0 + i];
    const cudaError_t e =
        fused ? launch_fused(pr, a, mods[i0].w0_dtype, out_dtype, map, codes, masks, nib, st)
              : launch_group(pr, a, mods[i0].w0_dtype, out_dtype, mode == AWSRC_DECODE_DENSE, i0 == 0, stream,
                             masks, status, st);
    if (e != cudaSuccess) return e;
    i0 = i1;
  }
  return cudaSuccess;
}

bool decode_clears_status(const Prm& pr, int mode) { return mode == AWSRC_DECODE_DENSE && pr.C >= 8; }

size_t decode_scratch_bytes(const Prm& pr, int64_t T, int mode) {
  // dense: dense_scratch(); in-place: one claim word per tile
  if (mode != AWSRC_DECODE_DENSE) return align_up((size_t)T * 4, 256);
  return dense_scratch(pr, T).bytes;
}

}  // namespace awsrc
