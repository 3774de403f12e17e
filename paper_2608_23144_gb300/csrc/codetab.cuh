// codetab.cuh — code tables of the dense decoder and the packed GEMV: the
// integer sums k_j = sum_p code_p (1 - 2 bit_p(j)) of a record (Sec. 3.2)
// from a per-record table and a per-seed nibble table, by byte permutes.
#pragma once

#include "common.cuh"

namespace awsrc {

// Code tables of the dense decoder for P = 4 and C in {8, 16, 32, 64}
// (code_tables()). With n_j = sum_p bit_p(j) 2^p the sign pattern of the four
// atoms at element j (bit set: -1), k_j = sum_p code_p (1 - 2 bit_p(j)) is
// T[n_j & 7] - 2 code_3 [n_j >= 8], with T[m] = code_3 + sum_{p<3} code_p
// (1 - 2 bit_p(m)): eight signed bytes per record. Per seed and
// window of 8 elements, nib holds (n_j & 7) in nibble j of x and, for elements
// 0..3 and 4..7, a byte mask (0xFF where n_j >= 8) in y and z. A vector's k_j
// then come from two byte permutes and two byte-wise subtractions, exactly.
// With codes of at most 6 bits |k_j| <= 128, so T and k fit in signed bytes.
__host__ __device__ __forceinline__ bool code_tables(const Prm& pr) {
  return pr.P == 4 && pr.b <= 6 && pr.C <= 64 && (pr.C & 7) == 0;
}

// The nibble-major table of seed s from its four mask words (C <= 64, one
// word per atom): window w of C / 8, lanes 0 .. C/8 - 1 of a warp.
__device__ __forceinline__ void nib_window(const uint64_t* __restrict__ mk, int w, uint4* __restrict__ out) {
  uint32_t lo = 0u, h0 = 0u, h1 = 0u;
#pragma unroll
  for (int e = 0; e < 8; ++e) {
    const int j = 8 * w + e;
    uint32_t n = 0u;
#pragma unroll
    for (int p = 0; p < 4; ++p) n |= (uint32_t)((mk[p] >> j) & 1ull) << p;
    lo |= (n & 7u) << (4 * e);
    if (n & 8u) {
      if (e < 4) h0 |= 0xFFu << (8 * e);
      else h1 |= 0xFFu << (8 * (e - 4));
    }
  }
  *out = make_uint4(lo, h0, h1, 0u);
}

// Four consecutive k_j from the record slot's table: sel holds (n_j & 7) in
// its four low nibbles, hm the byte mask of n_j >= 8.
__device__ __forceinline__ void table_k4(const uint4& slot, uint32_t sel, uint32_t hm, float* k) {
  const uint32_t c3x2 = ((slot.x >> 24) * 2u & 0xFFu) * 0x01010101u;  // 2 code_3, each byte
  const uint32_t kb = __vsub4(__byte_perm(slot.z, slot.w, sel & 0xFFFFu), hm & c3x2);
  const uint32_t ub = __vadd4(kb, 0x80808080u);  // k + 128 in [0, 255]
#pragma unroll
  for (int e = 0; e < 4; ++e)
    k[e] = __fsub_rn(__uint_as_float(__byte_perm(ub, 0x4B000000u, 0x7650u + e)), 8388736.0f);  // 2^23 + 128
}

}  // namespace awsrc
