// basis.cu — GenBasis(s, C, P) of Eq. 2 (Sec. 3.1) on the device.
//
// One thread per selector s draws, from the SplitMix64 stream keyed by s, the
// sign pattern, the coordinate permutation (Fisher-Yates) and P distinct
// columns of the order-C Sylvester Hadamard matrix, and writes the P sign masks
// of B_s as bits (bit j set when entry (j, p) is negative). The draw schedule is
// the one the public header documents; it is integer-only, so every device and
// host reproduces it exactly.
#include "basis.cuh"
#include "internal.h"

namespace awsrc {

constexpr int kBasisWarps = 8;  // warps per block of the stand-alone kernel

__global__ void __launch_bounds__(32 * kBasisWarps) gen_basis_kernel(Prm pr, uint64_t* __restrict__ masks,
                                                                     int S_out) {
  __shared__ __align__(16) uint8_t smem[kBasisWarps][kBasisSmem];
  const int warp = threadIdx.x >> 5;
  basis_warp(pr, masks, (int64_t)blockIdx.x * kBasisWarps + warp, S_out, smem[warp]);
}

cudaError_t launch_gen_basis(const Prm& pr, uint64_t* masks, int S_out, cudaStream_t st) {
  const int per = kBasisWarps * basis_warp_seeds(pr.C);
  gen_basis_kernel<<<(S_out + per - 1) / per, 32 * kBasisWarps, 0, st>>>(pr, masks, S_out);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
