// basis.cu — GenBasis(s, C, P) of Eq. 2 (Sec. 3.1) on the device.
//
// One thread per selector s draws, from the SplitMix64 stream keyed by s, the
// sign pattern, the coordinate permutation (Fisher-Yates) and P distinct
// columns of the order-C Sylvester Hadamard matrix, and writes the P sign masks
// of B_s as bits (bit j set when entry (j, p) is negative). The draw schedule is
// the one the public header documents; it is integer-only, so every device and
// host reproduces it exactly.
#include "internal.h"

namespace awsrc {

__global__ void gen_basis_kernel(Prm pr, uint64_t* __restrict__ masks, int S_out) {
  const int s = blockIdx.x * blockDim.x + threadIdx.x;
  if (s >= S_out) return;
  const int C = pr.C, P = pr.P, W = pr.W;
  if (s >= pr.S) {  // padding seeds of the last search chunk: never selected
    for (int i = 0; i < P * W; ++i) masks[(size_t)s * P * W + i] = 0ull;
    return;
  }
  const uint64_t key = sm64_output(pr.gen_seed, (uint64_t)s + 1);
  uint64_t n = 1;
  uint64_t sign[kMaxC / 64];
  for (int w = 0; w < W; ++w) sign[w] = sm64_output(key, n++);
  if (C < 64) sign[0] &= (1ull << C) - 1ull;
  uint8_t perm[kMaxC];
  for (int j = 0; j < C; ++j) perm[j] = (uint8_t)j;
  if (pr.permute) {
    for (int i = C - 1; i >= 1; --i) {
      const uint64_t x = sm64_output(key, n++) >> 32;
      const int k = (int)((x * (uint64_t)(i + 1)) >> 32);
      const uint8_t t = perm[i];
      perm[i] = perm[k];
      perm[k] = t;
    }
  }
  uint8_t pool[kMaxC];
  for (int j = 0; j < C; ++j) pool[j] = (uint8_t)j;
  int cols[kMaxP];
  for (int p = 0; p < P; ++p) {
    const uint64_t x = sm64_output(key, n++) >> 32;
    const int k = p + (int)((x * (uint64_t)(C - p)) >> 32);
    const uint8_t t = pool[p];
    pool[p] = pool[k];
    pool[k] = t;
    cols[p] = pool[p];
  }
  for (int p = 0; p < P; ++p) {
    for (int w = 0; w < W; ++w) {
      uint64_t m = 0;
      const int jn = min(64, C - 64 * w);
      for (int jj = 0; jj < jn; ++jj) {
        const int j = 64 * w + jj;
        const uint64_t h = (uint64_t)(__popc((unsigned)(perm[j] & cols[p])) & 1);
        m |= (((sign[w] >> jj) & 1ull) ^ h) << jj;
      }
      masks[((size_t)s * P + p) * W + w] = m;
    }
  }
}

cudaError_t launch_gen_basis(const Prm& pr, uint64_t* masks, int S_out, cudaStream_t st) {
  const int tpb = 128;
  gen_basis_kernel<<<(S_out + tpb - 1) / tpb, tpb, 0, st>>>(pr, masks, S_out);
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
