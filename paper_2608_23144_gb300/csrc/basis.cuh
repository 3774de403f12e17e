// basis.cuh — GenBasis(s, C, P) of Eq. 2 (Sec. 3.1) for four selectors by one
// warp, shared by the stand-alone mask kernel and the decoder's kernels.
#pragma once

#include "common.cuh"

namespace awsrc {

// Selectors per warp of basis_warp4 and its shared memory per warp: draw
// indices, permutation and column pool, one padded row of kMaxC + 4 bytes per
// selector (the padding spreads the four rows over different banks).
constexpr int kWarpSeeds = 4;
constexpr int kRowStride = kMaxC + 4;
constexpr size_t kBasisWarp4Smem = 3 * (size_t)kWarpSeeds * kRowStride;

// GenBasis for the selectors s0 .. s0+3 (those below S_out) by one warp. All
// lanes compute the SplitMix64 permutation draws of the four selectors; lane t
// then applies selector s0+t's Fisher-Yates swaps in the documented order and
// draws its P columns; finally the warp assembles each selector's P masks with
// ballots (one bit per lane). Selectors >= S get zero masks.
__device__ __forceinline__ void basis_warp4(const Prm& pr, uint64_t* __restrict__ masks, int s0, int S_out,
                                            uint8_t* sm) {
  const int lane = threadIdx.x & 31;
  const int C = pr.C, P = pr.P, W = pr.W;
  uint8_t* kidx = sm;
  uint8_t* perm = sm + kWarpSeeds * kRowStride;
  uint8_t* pool = sm + 2 * kWarpSeeds * kRowStride;
  const int ns = min(kWarpSeeds, S_out - s0);
  uint64_t key[kWarpSeeds];
#pragma unroll
  for (int t = 0; t < kWarpSeeds; ++t) key[t] = sm64_output(pr.gen_seed, (uint64_t)(s0 + t) + 1);
  const uint64_t n_perm0 = (uint64_t)W + 1;
  const int nperm = pr.permute ? C - 1 : 0;
  for (int idx = lane; idx < ns * nperm; idx += 32) {  // permutation draws of all selectors
    const int t = idx / nperm, m = idx - t * nperm;
    const uint64_t kt = t == 0 ? key[0] : (t == 1 ? key[1] : (t == 2 ? key[2] : key[3]));
    const int i = C - 1 - m;
    const uint64_t x = sm64_output(kt, n_perm0 + (uint64_t)m) >> 32;
    kidx[t * kRowStride + i] = (uint8_t)((x * (uint64_t)(i + 1)) >> 32);
  }
  for (int idx = lane; idx < ns * C; idx += 32) {
    const int t = idx / C, j = idx - t * C;
    perm[t * kRowStride + j] = (uint8_t)j;
    pool[t * kRowStride + j] = (uint8_t)j;
  }
  __syncwarp();
  int cols[kMaxP];
#pragma unroll
  for (int p = 0; p < kMaxP; ++p) cols[p] = 0;
  if (lane < ns && s0 + lane < pr.S) {  // lane t: selector s0 + t
    uint8_t* pm = perm + lane * kRowStride;
    const uint8_t* kx = kidx + lane * kRowStride;
    for (int i = C - 1; i >= 1 && nperm > 0; --i) {
      const int k = kx[i];
      const uint8_t a = pm[i];
      pm[i] = pm[k];
      pm[k] = a;
    }
    uint8_t* pl = pool + lane * kRowStride;
    const uint64_t kt = lane == 0 ? key[0] : (lane == 1 ? key[1] : (lane == 2 ? key[2] : key[3]));
    const uint64_t n_col0 = n_perm0 + (uint64_t)nperm;
#pragma unroll
    for (int p = 0; p < kMaxP; ++p) {
      if (p < P) {
        const uint64_t x = sm64_output(kt, n_col0 + (uint64_t)p) >> 32;
        const int k = p + (int)((x * (uint64_t)(C - p)) >> 32);
        const uint8_t a = pl[p];
        pl[p] = pl[k];
        pl[k] = a;
        cols[p] = pl[p];
      }
    }
  }
  __syncwarp();
  for (int t = 0; t < ns; ++t) {  // the warp assembles selector s0 + t
    uint64_t* out = masks + (size_t)(s0 + t) * P * W;
    if (s0 + t >= pr.S) {  // padding selectors of the last search chunk
      if (lane < P * W) out[lane] = 0ull;
      continue;
    }
    int ct[kMaxP];
#pragma unroll
    for (int p = 0; p < kMaxP; ++p) ct[p] = __shfl_sync(0xffffffffu, cols[p], t);
    const uint64_t kt = t == 0 ? key[0] : (t == 1 ? key[1] : (t == 2 ? key[2] : key[3]));
    const uint8_t* pm = perm + t * kRowStride;
    for (int w = 0; w < W; ++w) {
      const uint64_t sign = sm64_output(kt, (uint64_t)w + 1);
      const int j0 = 64 * w + lane, j1 = j0 + 32;
      const uint32_t sb0 = (uint32_t)(sign >> lane) & 1u, sb1 = (uint32_t)(sign >> (32 + lane)) & 1u;
      const int pj0 = j0 < C ? pm[j0] : 0, pj1 = j1 < C ? pm[j1] : 0;
#pragma unroll
      for (int p = 0; p < kMaxP; ++p) {
        if (p < P) {
          const uint32_t b0 = j0 < C ? (sb0 ^ (uint32_t)(__popc((unsigned)(pj0 & ct[p])) & 1)) : 0u;
          const uint32_t b1 = j1 < C ? (sb1 ^ (uint32_t)(__popc((unsigned)(pj1 & ct[p])) & 1)) : 0u;
          const uint32_t lo = __ballot_sync(0xffffffffu, b0);
          const uint32_t hi = __ballot_sync(0xffffffffu, b1);
          if (lane == p) out[p * W + w] = ((uint64_t)hi << 32) | lo;
        }
      }
    }
  }
}

// GenBasis for one selector s by one warp when C <= 64 (one mask word per
// atom). Lane l owns positions l and l + 32. The Fisher-Yates steps i = C-1 .. 1
// swap positions i and k_i <= i, so position i is final after step i and holds
// what position k_i held just before it. With touch[p] = { i : k_i = p }, the
// latest swap into position p before step i is the smallest i' > i in touch[p];
// with F(q) = the value at position q just before step q (F(i') of the latest
// swap into q, else q itself), perm[i] = F(i) when k_i = i, else F(i') for that
// swap, else k_i, and perm[0] follows from touch[0] alike. F is resolved by
// pointer doubling along q -> smallest i' > q in touch[q]. The P columns are the
// first P steps of a Fisher-Yates shuffle of 0 .. C-1 (lane 0), and the masks
// are assembled with ballots. Selectors >= S get zero masks.
constexpr size_t kBasisWarp1Smem = 64 * 8 + 64;  // touch words, column pool

__device__ __forceinline__ void basis_warp1(const Prm& pr, uint64_t* __restrict__ masks, int s, uint8_t* sm) {
  const int lane = threadIdx.x & 31;
  const int C = pr.C, P = pr.P;
  uint64_t* out = masks + (size_t)s * P;
  if (s >= pr.S) {  // padding selectors of the last search chunk
    if (lane < P) out[lane] = 0ull;
    return;
  }
  unsigned long long* touch = reinterpret_cast<unsigned long long*>(sm);
  uint8_t* pool = sm + 64 * 8;
  const int i0 = lane, i1 = lane + 32;
  const uint64_t key = sm64_output(pr.gen_seed, (uint64_t)s + 1);
  touch[i0] = 0ull;
  touch[i1] = 0ull;
  pool[i0] = (uint8_t)i0;
  pool[i1] = (uint8_t)i1;
  int perm0 = i0, perm1 = i1;
  const int nperm = pr.permute ? C - 1 : 0;
  if (nperm > 0) {
    // draw m = C - 1 - i of the permutation stream gives k_i
    int k0 = i0, k1 = i1;
    if (i0 >= 1 && i0 < C) {
      const uint64_t x = sm64_output(key, 2ull + (uint64_t)(C - 1 - i0)) >> 32;
      k0 = (int)((x * (uint64_t)(i0 + 1)) >> 32);
    }
    if (i1 < C) {
      const uint64_t x = sm64_output(key, 2ull + (uint64_t)(C - 1 - i1)) >> 32;
      k1 = (int)((x * (uint64_t)(i1 + 1)) >> 32);
    }
    __syncwarp();
    if (i0 >= 1 && i0 < C) atomicOr(&touch[k0], 1ull << i0);
    if (i1 < C) atomicOr(&touch[k1], 1ull << i1);
    __syncwarp();
    const uint64_t t00 = touch[i0], t01 = touch[i1];
    // smallest i' > q in touch[q] (bits above q), else q: a root
    const uint64_t u0 = t00 & ~((2ull << i0) - 1ull), u1 = i1 == 63 ? 0ull : (t01 & ~((2ull << i1) - 1ull));
    int f0 = u0 ? __ffsll((long long)u0) - 1 : i0;
    int f1 = u1 ? __ffsll((long long)u1) - 1 : i1;
    for (int r = 1; r < C; r <<= 1) {  // chains are shorter than C
      const int a0 = __shfl_sync(0xffffffffu, f0, f0 & 31), b0 = __shfl_sync(0xffffffffu, f1, f0 & 31);
      const int a1 = __shfl_sync(0xffffffffu, f0, f1 & 31), b1 = __shfl_sync(0xffffffffu, f1, f1 & 31);
      f0 = f0 < 32 ? a0 : b0;
      f1 = f1 < 32 ? a1 : b1;
    }
    // the value each position holds at the end
    int j0 = i0, j1 = i1;   // F index to gather, or own
    int v0 = -1, v1 = -1;   // a value known without gathering
    if (i0 == 0) {
      const uint64_t t = t00 & ~1ull;
      if (t) j0 = __ffsll((long long)t) - 1;
      else v0 = 0;
    } else if (i0 < C) {
      if (k0 != i0) {
        const uint64_t t = touch[k0] & ~((2ull << i0) - 1ull);
        if (t) j0 = __ffsll((long long)t) - 1;
        else v0 = k0;
      }
    }
    if (i1 < C && k1 != i1) {
      const uint64_t t = i1 == 63 ? 0ull : (touch[k1] & ~((2ull << i1) - 1ull));
      if (t) j1 = __ffsll((long long)t) - 1;
      else v1 = k1;
    }
    const int a0 = __shfl_sync(0xffffffffu, f0, j0 & 31), b0 = __shfl_sync(0xffffffffu, f1, j0 & 31);
    const int a1 = __shfl_sync(0xffffffffu, f0, j1 & 31), b1 = __shfl_sync(0xffffffffu, f1, j1 & 31);
    perm0 = v0 >= 0 ? v0 : (j0 < 32 ? a0 : b0);
    perm1 = v1 >= 0 ? v1 : (j1 < 32 ? a1 : b1);
  }
  // columns: draws n_col0 + p in lanes p, then the partial shuffle in lane 0
  int kc = 0;
  if (lane < P) {
    const uint64_t x = sm64_output(key, 2ull + (uint64_t)nperm + (uint64_t)lane) >> 32;
    kc = lane + (int)((x * (uint64_t)(C - lane)) >> 32);
  }
  int kcs[kMaxP];
#pragma unroll
  for (int p = 0; p < kMaxP; ++p) kcs[p] = __shfl_sync(0xffffffffu, kc, p);
  __syncwarp();
  if (lane == 0) {
#pragma unroll
    for (int p = 0; p < kMaxP; ++p) {
      if (p < P) {
        const uint8_t a = pool[p];
        pool[p] = pool[kcs[p]];
        pool[kcs[p]] = a;
      }
    }
  }
  __syncwarp();
  const uint64_t sign = sm64_output(key, 1ull);
  const uint32_t sb0 = (uint32_t)(sign >> i0) & 1u, sb1 = (uint32_t)(sign >> i1) & 1u;
#pragma unroll
  for (int p = 0; p < kMaxP; ++p) {
    if (p < P) {
      const int col = pool[p];
      const uint32_t b0 = i0 < C ? (sb0 ^ (uint32_t)(__popc((unsigned)(perm0 & col)) & 1)) : 0u;
      const uint32_t b1 = i1 < C ? (sb1 ^ (uint32_t)(__popc((unsigned)(perm1 & col)) & 1)) : 0u;
      const uint32_t lo = __ballot_sync(0xffffffffu, b0);
      const uint32_t hi = __ballot_sync(0xffffffffu, b1);
      if (lane == p) out[p] = ((uint64_t)hi << 32) | lo;
    }
  }
}

// Selectors one warp generates: 1 with basis_warp1 (C <= 64), else 4.
__host__ __device__ constexpr int basis_warp_seeds(int C) { return C <= 64 ? 1 : kWarpSeeds; }
constexpr size_t kBasisSmem = kBasisWarp4Smem > kBasisWarp1Smem ? kBasisWarp4Smem : kBasisWarp1Smem;

// GenBasis for the selectors of warp w (global warp index) into masks[0 .. S_out).
__device__ __forceinline__ void basis_warp(const Prm& pr, uint64_t* __restrict__ masks, int64_t w, int S_out,
                                           uint8_t* sm) {
  if (pr.C <= 64) {
    if (w < S_out) basis_warp1(pr, masks, (int)w, sm);
  } else {
    const int64_t s0 = w * kWarpSeeds;
    if (s0 < S_out) basis_warp4(pr, masks, (int)s0, S_out, sm);
  }
}

}  // namespace awsrc
