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
// then come from three byte permutes, a byte select and one subtraction each,
// exactly. With codes of at most 5 bits (any stream's, -16 included)
// |T[m]|, |k_j| <= 64, so T fits in signed bytes and k_j + 128 in a byte.
__host__ __device__ __forceinline__ bool code_tables(const Prm& pr) {
  return pr.P == 4 && pr.b <= 5 && pr.C <= 64 && (pr.C & 7) == 0;
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

// The record's two byte tables for table_k4, offset by 128 (the offset flips
// the top bit of a byte): T[m] + 128 and T[m] - 2 code_3 + 128, the value of
// k_j + 128 for n_j = m and n_j = m + 8.
struct KTab {
  uint32_t t0, t1, u0, u1;
};

__device__ __forceinline__ KTab k_tables(const uint4& slot) {
  const uint32_t c3x2 = ((slot.x >> 24) * 2u & 0xFFu) * 0x01010101u;  // 2 code_3, each byte
  return {slot.z ^ 0x80808080u, slot.w ^ 0x80808080u, __vsub4(slot.z, c3x2) ^ 0x80808080u,
          __vsub4(slot.w, c3x2) ^ 0x80808080u};
}

// The constants of table_k4 for k_j 2^-S: the magic 2^(23-S), whose
// mantissa unit is 2^-S, and the offset 2^(23-S) + 128 2^-S. S = 3 (C = 64)
// and 2 (C = 16) give k_j c at once (c = 2^-S, and k_j c is exact); S = 0
// (C = 32) gives k_j.
struct KMagic {
  uint32_t bits;
  float off;
  bool folded;  // c folded in
};

__host__ __device__ __forceinline__ KMagic k_magic(const Prm& pr) {
  const int S = pr.c == 0.125f ? 3 : (pr.c == 0.25f ? 2 : 0);
  return {0x4B000000u - ((uint32_t)S << 23), (float)(1u << (23 - S)) + (float)(128u >> S), S != 0};
}

// Four consecutive k_j 2^-S from a record's tables: sel holds (n_j & 7) in
// its four low nibbles, hm the byte mask of n_j >= 8. The byte k + 128 goes
// into the low mantissa bits of the magic and one subtraction leaves k 2^-S
// exactly.
__device__ __forceinline__ void table_k4(const KTab& t, uint32_t sel, uint32_t hm, const KMagic& km, float* k) {
  const uint32_t a = __byte_perm(t.t0, t.t1, sel & 0xFFFFu), b = __byte_perm(t.u0, t.u1, sel & 0xFFFFu);
  const uint32_t ub = (a & ~hm) | (b & hm);
#pragma unroll
  for (int e = 0; e < 4; ++e) k[e] = __fsub_rn(__uint_as_float(__byte_perm(ub, km.bits, 0x7650u + e)), km.off);
}

}  // namespace awsrc
