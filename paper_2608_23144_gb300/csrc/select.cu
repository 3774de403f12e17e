// select.cu — byte-aware allocation (Sec. 3.3) and serialisation (Sec. 3.4, Eq. 5).
//
// Every candidate becomes a 64-bit key that sorts ascending into the stream
// order: rho_t = gain_t / L with one L for all records, so gain descending,
// ties by tile ascending. Non-positive or non-finite gains get the largest gain
// field and sort behind every eligible record. U prefixes the module index so
// one sort yields each module's ranking in its own contiguous segment; PF keeps
// one global ranking whose prefixes are the rate cuts.
//
// The sort is a stable LSD radix sort with 8-bit digits over the module and
// gain fields (the keys are made in tile order, which the stable passes keep
// among equal fields, so the tile field needs no pass): per pass a block
// histogram, a per-digit scan over blocks, and a scatter whose in-block ranks
// come from __match_any_sync over each warp plus per-warp digit counters.
// Counts, cuts, packing and the header are device kernels, so the whole step
// is asynchronous on the caller's stream.
#include <cfloat>

#include "internal.h"

namespace awsrc {

namespace {

constexpr int RT = 256;        // radix threads
constexpr int IPT = 8;         // keys per thread per block
constexpr int ITEMS = RT * IPT;
constexpr int kMaxSelMods = 1024;
constexpr int kMaxRates = 64;

struct SelArgs {
  int n_mod, n_rates, variant;
  int tbl;                       // U: local tile bits; PF: global tile bits
  int mshift;                    // U: shift of the module index
  int64_t T, L, h;
  int64_t tile_off[kMaxSelMods + 1];
  int64_t kcap[kMaxSelMods];     // U: per module; PF: per rate
};

struct SelWs {                   // device scratch after the status word
  int64_t npos;
  int64_t kstream;
  int64_t K[kMaxSelMods];        // records per module in the stream
  int64_t rec_off[kMaxSelMods + 1];
};

__device__ __forceinline__ uint32_t gain_field(float g) {
  const bool ok = (g > 0.0f) && (g <= FLT_MAX);
  return ok ? (0x7F7FFFFFu - __float_as_uint(g)) : 0x7FFFFFFFu;
}

__global__ void make_keys_kernel(const awsrc_candidate* __restrict__ cands, uint64_t* __restrict__ keys,
                                 const __grid_constant__ SelArgs a) {
  const int64_t t = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (t >= a.T) return;
  const uint64_t gf = gain_field(cands[t].gain);
  uint64_t key;
  if (a.variant == AWSRC_VARIANT_U) {
    int lo = 0, hi = a.n_mod - 1;  // module containing t
    while (lo < hi) {
      const int mid = (lo + hi + 1) / 2;
      if (t >= a.tile_off[mid]) lo = mid; else hi = mid - 1;
    }
    key = ((uint64_t)lo << a.mshift) | (gf << a.tbl) | (uint64_t)(t - a.tile_off[lo]);
  } else {
    key = (gf << a.tbl) | (uint64_t)t;
  }
  keys[t] = key;
}

__global__ void __launch_bounds__(RT) radix_hist_kernel(const uint64_t* __restrict__ keys, int64_t n,
                                                        int shift, uint32_t* __restrict__ hist,
                                                        int64_t nblocks) {
  __shared__ uint32_t cnt[256];
  cnt[threadIdx.x] = 0;
  __syncthreads();
  const int64_t base = (int64_t)blockIdx.x * ITEMS;
#pragma unroll
  for (int r = 0; r < IPT; ++r) {
    const int64_t i = base + r * RT + threadIdx.x;
    if (i < n) atomicAdd(&cnt[(keys[i] >> shift) & 255u], 1u);
  }
  __syncthreads();
  hist[(int64_t)threadIdx.x * nblocks + blockIdx.x] = cnt[threadIdx.x];
}

// Block-wide exclusive scan of one value per thread (blockDim.x multiple of 32).
__device__ __forceinline__ uint32_t block_exclusive_scan(uint32_t v, uint32_t* total,
                                                          uint32_t* warp_sums) {
  const int lane = threadIdx.x & 31, w = threadIdx.x >> 5, nw = blockDim.x >> 5;
  uint32_t x = v;
#pragma unroll
  for (int o = 1; o < 32; o <<= 1) {
    const uint32_t y = __shfl_up_sync(0xffffffffu, x, o);
    if (lane >= o) x += y;
  }
  if (lane == 31) warp_sums[w] = x;
  __syncthreads();
  if (w == 0) {
    uint32_t s = lane < nw ? warp_sums[lane] : 0u;
#pragma unroll
    for (int o = 1; o < 32; o <<= 1) {
      const uint32_t y = __shfl_up_sync(0xffffffffu, s, o);
      if (lane >= o) s += y;
    }
    if (lane < nw) warp_sums[lane] = s;
  }
  __syncthreads();
  const uint32_t before = (w > 0 ? warp_sums[w - 1] : 0u) + x - v;
  if (total) *total = warp_sums[nw - 1];
  __syncthreads();
  return before;
}

// One block per digit: exclusive scan of that digit's per-block counts.
__global__ void __launch_bounds__(1024) radix_scan_rows_kernel(uint32_t* __restrict__ hist,
                                                               int64_t nblocks,
                                                               uint32_t* __restrict__ totals) {
  __shared__ uint32_t ws[32];
  uint32_t* row = hist + (int64_t)blockIdx.x * nblocks;
  const int64_t per = (nblocks + blockDim.x - 1) / blockDim.x;
  const int64_t b0 = threadIdx.x * per;
  uint32_t s = 0;
  for (int64_t i = b0; i < b0 + per && i < nblocks; ++i) s += row[i];
  uint32_t tot;
  uint32_t run = block_exclusive_scan(s, &tot, ws);
  for (int64_t i = b0; i < b0 + per && i < nblocks; ++i) {
    const uint32_t v = row[i];
    row[i] = run;
    run += v;
  }
  if (threadIdx.x == 0) totals[blockIdx.x] = tot;
}

__global__ void __launch_bounds__(RT) radix_scatter_kernel(const uint64_t* __restrict__ in,
                                                           uint64_t* __restrict__ out, int64_t n,
                                                           int shift, const uint32_t* __restrict__ hist,
                                                           int64_t nblocks,
                                                           const uint32_t* __restrict__ totals) {
  __shared__ uint32_t ws[32];
  __shared__ uint32_t base[256];
  __shared__ uint32_t wcnt[RT / 32][256];
  const int tid = threadIdx.x, lane = tid & 31, w = tid >> 5;
  const uint32_t tot = totals[tid];
  const uint32_t dbase = block_exclusive_scan(tot, nullptr, ws);
  base[tid] = dbase + hist[(int64_t)tid * nblocks + blockIdx.x];
  const int64_t b0 = (int64_t)blockIdx.x * ITEMS;
  for (int r = 0; r < IPT; ++r) {
    for (int i = tid; i < (RT / 32) * 256; i += RT) (&wcnt[0][0])[i] = 0;
    __syncthreads();
    const int64_t idx = b0 + r * RT + tid;
    const bool valid = idx < n;
    const uint64_t key = valid ? in[idx] : 0ull;
    const uint32_t dg = valid ? (uint32_t)((key >> shift) & 255u) : 256u;
    const uint32_t peers = __match_any_sync(0xffffffffu, dg);
    const uint32_t rank = __popc(peers & ((1u << lane) - 1u));
    if (valid && rank == 0) wcnt[w][dg] = __popc(peers);
    __syncthreads();
    {  // per digit: exclusive prefix over warps, then advance the running base
      uint32_t run = 0;
#pragma unroll
      for (int ww = 0; ww < RT / 32; ++ww) {
        const uint32_t c = wcnt[ww][tid];
        wcnt[ww][tid] = run;
        run += c;
      }
      __syncthreads();
      if (valid) out[base[dg] + wcnt[w][dg] + rank] = key;
      __syncthreads();
      base[tid] += run;
    }
    __syncthreads();
  }
}

// First index in [lo, hi) whose key is ineligible (eligible keys form a prefix
// of the range), by one warp: each round the lanes test 32 evenly spaced
// positions and the range shrinks to the gap where eligibility ends.
__device__ __forceinline__ int64_t first_ineligible(const uint64_t* __restrict__ keys, int64_t lo,
                                                    int64_t hi, int tbl) {
  const int lane = threadIdx.x & 31;
  while (hi - lo > 1) {
    const int64_t span = (hi - lo + 31) / 32;
    const int64_t pos = lo + lane * span;
    bool valid = false;
    if (pos < hi) valid = ((keys[pos] >> tbl) & 0x7FFFFFFFull) != 0x7FFFFFFFull;
    const int cnt = __popc(__ballot_sync(0xffffffffu, valid));  // valid starts form a prefix of lanes
    if (cnt == 0) return lo;                                      // keys[lo] already ineligible
    const int64_t last_valid = lo + (int64_t)(cnt - 1) * span;
    lo = last_valid + 1;
    hi = min(hi, lo - 1 + span);
  }
  if (lo < hi) {
    const bool v = ((keys[lo] >> tbl) & 0x7FFFFFFFull) != 0x7FFFFFFFull;
    return v ? hi : lo;
  }
  return lo;
}

// Count eligible keys and cut: U per module (one warp per module), PF per rate.
__global__ void __launch_bounds__(256) cut_kernel(const uint64_t* __restrict__ keys,
                                                  const __grid_constant__ SelArgs a,
                                                  SelWs* __restrict__ sw, int64_t* __restrict__ d_counts,
                                                  int64_t* __restrict__ d_bytes) {
  const int warp = threadIdx.x >> 5, lane = threadIdx.x & 31;
  if (a.variant == AWSRC_VARIANT_U) {
    for (int m = warp; m < a.n_mod; m += blockDim.x >> 5) {
      const int64_t beg = a.tile_off[m], end = a.tile_off[m + 1];
      const int64_t f = first_ineligible(keys, beg, end, a.tbl);
      if (lane == 0) sw->K[m] = min(f - beg, a.kcap[m]);
    }
    __syncthreads();
    if (threadIdx.x == 0) {
      int64_t off = 0;
      for (int m = 0; m < a.n_mod; ++m) {
        sw->rec_off[m] = off;
        d_counts[m] = sw->K[m];
        off += sw->K[m];
      }
      sw->rec_off[a.n_mod] = off;
      sw->kstream = off;
      d_bytes[0] = a.h + off * a.L;
    }
  } else {
    if (warp == 0) {
      const int64_t npos = first_ineligible(keys, 0, a.T, a.tbl);
      if (lane == 0) {
        sw->npos = npos;
        int64_t kmax = 0;
        for (int r = 0; r < a.n_rates; ++r) {
          const int64_t K = min(npos, a.kcap[r]);
          d_counts[r] = K;
          d_bytes[r] = a.h + K * a.L;
          kmax = max(kmax, K);
        }
        sw->kstream = kmax;
      }
    }
    for (int m = threadIdx.x; m < a.n_mod; m += blockDim.x) sw->K[m] = 0;
  }
}

__device__ __forceinline__ int ceil_log2_dev(uint64_t x) {
  return x <= 1 ? 0 : 64 - __clzll((long long)(x - 1));
}

// Append the low nbits (<= 64) of v at bit *pos of the 128-bit record (w1:w0).
__device__ __forceinline__ void put_bits(uint64_t* w0, uint64_t* w1, int* pos, uint64_t v, int nbits) {
  if (nbits == 0) return;
  v &= nbits >= 64 ? ~0ull : ((1ull << nbits) - 1ull);
  const int p = *pos;
  if (p >= 64) {
    *w1 |= v << (p - 64);
  } else {
    *w0 |= v << p;
    if (p + nbits > 64) *w1 |= v >> (64 - p);
  }
  *pos += nbits;
}

__global__ void pack_kernel(const uint64_t* __restrict__ keys, const awsrc_candidate* __restrict__ cands,
                            const __grid_constant__ SelArgs a, Prm pr, SelWs* __restrict__ sw,
                            uint8_t* __restrict__ stream, int64_t cap_records) {
  const int64_t i = (int64_t)blockIdx.x * blockDim.x + threadIdx.x;
  if (i >= cap_records || i >= sw->kstream) return;
  int64_t tile;
  if (a.variant == AWSRC_VARIANT_U) {
    int lo = 0, hi = a.n_mod - 1;  // module whose record range holds i
    while (lo < hi) {
      const int mid = (lo + hi + 1) / 2;
      if (i >= sw->rec_off[mid]) lo = mid; else hi = mid - 1;
    }
    const uint64_t key = keys[a.tile_off[lo] + (i - sw->rec_off[lo])];
    tile = a.tile_off[lo] + (int64_t)(key & ((1ull << a.tbl) - 1ull));
  } else {
    const uint64_t key = keys[i];
    tile = (int64_t)(key & ((a.tbl >= 64) ? ~0ull : ((1ull << a.tbl) - 1ull)));
    int lo = 0, hi = a.n_mod - 1;
    while (lo < hi) {
      const int mid = (lo + hi + 1) / 2;
      if (tile >= a.tile_off[mid]) lo = mid; else hi = mid - 1;
    }
    atomicAdd(reinterpret_cast<unsigned long long*>(&sw->K[lo]), 1ull);
  }
  const awsrc_candidate cd = cands[tile];
  uint64_t w0 = 0, w1 = 0;
  int pos = 0;
  put_bits(&w0, &w1, &pos, (uint64_t)tile, ceil_log2_dev((uint64_t)a.T));
  put_bits(&w0, &w1, &pos, cd.seed, ceil_log2_dev((uint64_t)pr.S));
  uint64_t sf;
  if (pr.scale_mode == AWSRC_SCALE_POW2) sf = (uint64_t)(int64_t)(cd.scale - pr.e_bias);
  else sf = (uint16_t)cd.scale;
  put_bits(&w0, &w1, &pos, sf, pr.b_e);
  for (int p = 0; p < pr.P; ++p) put_bits(&w0, &w1, &pos, (uint64_t)(int64_t)cd.code[p], pr.b);
  uint8_t* dst = stream + a.h + i * a.L;
  for (int k = 0; k < a.L; ++k) dst[k] = (uint8_t)(k < 8 ? (w0 >> (8 * k)) : (w1 >> (8 * (k - 8))));
}

__device__ __forceinline__ void put_le(uint8_t* p, uint64_t v, int n) {
  for (int i = 0; i < n; ++i) p[i] = (uint8_t)(v >> (8 * i));
}

__global__ void header_kernel(const __grid_constant__ SelArgs a, Prm pr, const SelWs* __restrict__ sw,
                              uint8_t* __restrict__ stream) {
  const int i = blockIdx.x * blockDim.x + threadIdx.x;
  if (i == 0) {
    for (int k = 0; k < 40; ++k) stream[k] = 0;
    put_le(stream + 0, 0x52535741u, 4);
    put_le(stream + 4, 1, 2);
    stream[6] = (uint8_t)pr.variant;
    stream[7] = (uint8_t)pr.scale_mode;
    put_le(stream + 8, (uint64_t)pr.C, 2);
    stream[10] = (uint8_t)pr.P;
    stream[11] = (uint8_t)pr.b;
    stream[12] = (uint8_t)pr.b_e;
    stream[13] = (uint8_t)(int8_t)pr.e_bias;
    stream[14] = (uint8_t)pr.permute;
    put_le(stream + 16, (uint64_t)pr.S, 4);
    put_le(stream + 20, (uint64_t)a.n_mod, 4);
    put_le(stream + 24, pr.gen_seed, 8);
    put_le(stream + 32, (uint64_t)sw->kstream, 8);
  }
  if (i < a.n_mod) {
    put_le(stream + 40 + 8 * i, (uint64_t)(a.tile_off[i + 1] - a.tile_off[i]), 4);
    put_le(stream + 44 + 8 * i, (uint64_t)sw->K[i], 4);
  }
}

}  // namespace

size_t select_ws_bytes(const SelectPlan& sp) {
  size_t b = kStatusBytes;
  b += align_up(sizeof(SelWs), 256);
  b += 2 * align_up((size_t)sp.T * 8, 256);          // keys ping-pong
  b += align_up((size_t)256 * sp.nblocks * 4, 256);  // histograms
  b += align_up(256 * 4, 256);                        // digit totals
  return b;
}

awsrc_status select_run(const Prm& pr, const SelectPlan& sp, const int64_t* tile_off,
                        const int64_t* mod_tiles, const int64_t* kcap,
                        const awsrc_candidate* cands, uint8_t* stream_out, int64_t* d_counts,
                        int64_t* d_bytes, void* ws, size_t ws_bytes, cudaStream_t st) {
  (void)mod_tiles;
  if (sp.n_mod > kMaxSelMods || sp.n_rates > kMaxRates) return AWSRC_ERR_UNSUPPORTED;
  if (ws_bytes < select_ws_bytes(sp)) return AWSRC_ERR_WORKSPACE;
  SelArgs a;
  a.n_mod = sp.n_mod;
  a.n_rates = sp.n_rates;
  a.variant = pr.variant;
  a.tbl = sp.tile_bits_local;
  a.mshift = sp.mod_shift;
  a.T = sp.T;
  a.L = sp.L;
  a.h = sp.h;
  for (int m = 0; m <= sp.n_mod; ++m) a.tile_off[m] = tile_off[m];
  const int nk = pr.variant == AWSRC_VARIANT_U ? sp.n_mod : sp.n_rates;
  for (int i = 0; i < nk; ++i) a.kcap[i] = kcap[i];

  uint8_t* p = static_cast<uint8_t*>(ws) + kStatusBytes;
  SelWs* sw = reinterpret_cast<SelWs*>(p);
  p += align_up(sizeof(SelWs), 256);
  uint64_t* ka = reinterpret_cast<uint64_t*>(p);
  p += align_up((size_t)sp.T * 8, 256);
  uint64_t* kb = reinterpret_cast<uint64_t*>(p);
  p += align_up((size_t)sp.T * 8, 256);
  uint32_t* hist = reinterpret_cast<uint32_t*>(p);
  p += align_up((size_t)256 * sp.nblocks * 4, 256);
  uint32_t* totals = reinterpret_cast<uint32_t*>(p);

  if (sp.T > 0) {
    make_keys_kernel<<<(unsigned)((sp.T + 255) / 256), 256, 0, st>>>(cands, ka, a);
    note_launches(1);
    if (cudaGetLastError() != cudaSuccess) return check_launch("select: keys");
    // the tile field (the low bits) needs no pass: the keys start in tile
    // order and every pass is stable, so equal (module, gain) keys keep it
    const int low = sp.tile_bits_local;
    const int passes = (sp.key_bits - low + 7) / 8;
    for (int ps = 0; ps < passes; ++ps) {
      const int shift = low + 8 * ps;
      radix_hist_kernel<<<(unsigned)sp.nblocks, RT, 0, st>>>(ka, sp.T, shift, hist, sp.nblocks);
      radix_scan_rows_kernel<<<256, 1024, 0, st>>>(hist, sp.nblocks, totals);
      radix_scatter_kernel<<<(unsigned)sp.nblocks, RT, 0, st>>>(ka, kb, sp.T, shift, hist,
                                                                 sp.nblocks, totals);
      note_launches(3);
      uint64_t* t = ka;
      ka = kb;
      kb = t;
    }
    if (cudaGetLastError() != cudaSuccess) return check_launch("select: sort");
  }
  cut_kernel<<<1, 256, 0, st>>>(ka, a, sw, d_counts, d_bytes);
  note_launches(1);
  if (sp.cap_records > 0)
    pack_kernel<<<(unsigned)((sp.cap_records + 127) / 128), 128, 0, st>>>(ka, cands, a, pr, sw,
                                                                           stream_out, sp.cap_records);
  if (sp.cap_records > 0) note_launches(1);
  header_kernel<<<(sp.n_mod + 127) / 128 + 1, 128, 0, st>>>(a, pr, sw, stream_out);
  note_launches(1);
  return check_launch("select: pack");
}

}  // namespace awsrc
