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

}  // namespace awsrc
