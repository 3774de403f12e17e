// basis.cuh — GenBasis(s, C, P) of Eq. 2 (Sec. 3.1) for one selector by one warp,
// shared by the stand-alone mask kernel and the decoder's fused copy kernel.
#pragma once

#include "common.cuh"

namespace awsrc {

// SplitMix64 is counter-based, so the lanes compute the seed's draws in
// parallel; lane 0 then applies the Fisher-Yates swaps in the documented order,
// and the masks are assembled with ballots (one bit per lane). perm/kidx/pool:
// C bytes of shared memory each, cols: P ints, all private to the warp.
__device__ __forceinline__ void basis_warp(const Prm& pr, uint64_t* __restrict__ masks, int s,
                                           uint8_t* perm, uint8_t* kidx, uint8_t* pool, int* cols) {
  const int lane = threadIdx.x & 31;
  const int C = pr.C, P = pr.P, W = pr.W;
  uint64_t* out = masks + (size_t)s * P * W;
  if (s >= pr.S) {  // padding seeds of the last search chunk: never selected
    for (int i = lane; i < P * W; i += 32) out[i] = 0ull;
    return;
  }
  const uint64_t key = sm64_output(pr.gen_seed, (uint64_t)s + 1);
  // draw numbers: 1..W sign words, W+1..W+C-1 permutation (i = C-1 down to 1),
  // then P column draws
  const uint64_t n_perm0 = (uint64_t)W + 1;
  const int nperm = pr.permute ? C - 1 : 0;
  for (int m = lane; m < nperm; m += 32) {   // m-th permutation draw is for i = C-1-m
    const int i = C - 1 - m;
    const uint64_t x = sm64_output(key, n_perm0 + (uint64_t)m) >> 32;
    kidx[i] = (uint8_t)((x * (uint64_t)(i + 1)) >> 32);
  }
  for (int j = lane; j < C; j += 32) {
    perm[j] = (uint8_t)j;
    pool[j] = (uint8_t)j;
  }
  __syncwarp();
  if (lane == 0) {
    for (int i = C - 1; i >= 1 && nperm > 0; --i) {
      const int k = kidx[i];
      const uint8_t t = perm[i];
      perm[i] = perm[k];
      perm[k] = t;
    }
    // P distinct columns by a partial Fisher-Yates over 0..C-1
    const uint64_t n_col0 = n_perm0 + (uint64_t)nperm;
    for (int p = 0; p < P; ++p) {
      const uint64_t x = sm64_output(key, n_col0 + (uint64_t)p) >> 32;
      const int k = p + (int)((x * (uint64_t)(C - p)) >> 32);
      const uint8_t t = pool[p];
      pool[p] = pool[k];
      pool[k] = t;
      cols[p] = pool[p];
    }
  }
  __syncwarp();
  for (int w = 0; w < W; ++w) {
    const uint64_t sign = sm64_output(key, (uint64_t)w + 1);
    const int j0 = 64 * w + lane, j1 = j0 + 32;
    const uint32_t s0 = (uint32_t)(sign >> lane) & 1u, s1 = (uint32_t)(sign >> (32 + lane)) & 1u;
    const int pj0 = j0 < C ? perm[j0] : 0, pj1 = j1 < C ? perm[j1] : 0;
    for (int p = 0; p < P; ++p) {
      const int cp = cols[p];
      const uint32_t b0 = j0 < C ? (s0 ^ (uint32_t)(__popc((unsigned)(pj0 & cp)) & 1)) : 0u;
      const uint32_t b1 = j1 < C ? (s1 ^ (uint32_t)(__popc((unsigned)(pj1 & cp)) & 1)) : 0u;
      const uint32_t lo = __ballot_sync(0xffffffffu, b0);
      const uint32_t hi = __ballot_sync(0xffffffffu, b1);
      if (lane == p) out[p * W + w] = ((uint64_t)hi << 32) | lo;
    }
  }
}

}  // namespace awsrc
