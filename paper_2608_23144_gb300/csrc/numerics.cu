// numerics.cu — on-device checks of the library's own arithmetic primitives.
#include "internal.h"

namespace awsrc {

namespace {

// Counts the binary32 bit patterns in [first, last) where rcp_rn differs from
// __frcp_rn (bit for bit; NaN results compare as equal when both are NaN).
__global__ void verify_rcp_kernel(uint32_t first, uint32_t last, unsigned long long* __restrict__ bad) {
  unsigned long long n = 0;
  const uint64_t stride = (uint64_t)gridDim.x * blockDim.x;
  for (uint64_t i = (uint64_t)first + (uint64_t)blockIdx.x * blockDim.x + threadIdx.x; i < last; i += stride) {
    const float x = __uint_as_float((uint32_t)i);
    const float a = rcp_rn(x), b = __frcp_rn(x);
    const bool same = __float_as_uint(a) == __float_as_uint(b) || (a != a && b != b);
    n += same ? 0ull : 1ull;
  }
  for (int o = 16; o > 0; o >>= 1) n += __shfl_xor_sync(0xffffffffu, n, o);
  if ((threadIdx.x & 31) == 0 && n) atomicAdd(bad, n);
}

}  // namespace

cudaError_t launch_verify_rcp(uint32_t first, uint32_t last, unsigned long long* bad, cudaStream_t st) {
  verify_rcp_kernel<<<152 * 8, 256, 0, st>>>(first, last, bad);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace awsrc
