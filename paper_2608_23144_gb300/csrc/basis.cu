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

constexpr int kBasisWarps = 4;  // seeds per block of the stand-alone kernel

__global__ void __launch_bounds__(32 * kBasisWarps) gen_basis_kernel(Prm pr, uint64_t* __restrict__ masks,
                                                                     int S_out) {
  __shared__ uint8_t perm_s[kBasisWarps][kMaxC];
  __shared__ uint8_t kidx_s[kBasisWarps][kMaxC];
  __shared__ uint8_t pool_s[kBasisWarps][kMaxC];
  __shared__ int cols_s[kBasisWarps][kMaxP];
  const int warp = threadIdx.x >> 5;
  const int s = blockIdx.x * kBasisWarps + warp;
  if (s >= S_out) return;  // whole warp leaves together
  basis_warp(pr, masks, s, perm_s[warp], kidx_s[warp], pool_s[warp], cols_s[warp]);
}

cudaError_t launch_gen_basis(const Prm& pr, uint64_t* masks, int S_out, cudaStream_t st) {
  gen_basis_kernel<<<(S_out + kBasisWarps - 1) / kBasisWarps, 32 * kBasisWarps, 0, st>>>(pr, masks, S_out);
  note_launches(1);
  return cudaGetLastError();
}

// Expand the bit masks of C = 64, P = 4 into +-1.0f in the layout the
// specialised search streams into shared memory with one bulk copy per chunk:
// out[((chunk*64 + j)*CH + sl)*4 + p], seed = chunk*CH + sl.
__global__ void expand_masks_c64p4_kernel(const uint64_t* __restrict__ masks, float* __restrict__ out,
                                          int S_pad, int CH) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;  // one float4 (4 atoms)
  const int64_t n = (int64_t)S_pad * 64;
  if (i >= n) return;
  const int sl = (int)(i % CH);
  const int j = (int)((i / CH) % 64);
  const int chunk = (int)(i / (CH * 64));
  const int s = chunk * CH + sl;
  float4 v;
  v.x = sign_f(masks[(size_t)s * 4 + 0] >> j);
  v.y = sign_f(masks[(size_t)s * 4 + 1] >> j);
  v.z = sign_f(masks[(size_t)s * 4 + 2] >> j);
  v.w = sign_f(masks[(size_t)s * 4 + 3] >> j);
  reinterpret_cast<float4*>(out)[i] = v;
}

cudaError_t launch_expand_masks_c64p4(const Prm& pr, const uint64_t* masks, float* out,
                                      cudaStream_t st) {
  const int64_t n = (int64_t)pr.S_pad * 64;
  const int tpb = 256;
  expand_masks_c64p4_kernel<<<(unsigned)((n + tpb - 1) / tpb), tpb, 0, st>>>(
      masks, out, pr.S_pad, search_c64p4_chunk());
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
