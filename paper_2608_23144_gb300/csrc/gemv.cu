// gemv.cu — the decoded weights of a module applied to M vectors without
// forming them: y[m] = (W0 + r_hat) x[m], with W0 = q * s_eff read from the
// packed RTN-INT4 backbone (binary16 or SDQ scales, Sec. 3.3) and r_hat the
// decoder's residual (Sec. 3.2) on the tiles a prepared sidecar names. This is
// the packed-inference use the paper leaves to future work (Sec. 5).
//
// One launch serves a batch of tasks (module, x, y). The tasks whose x fits in
// shared memory: gemv_warp_kernel below, warps per output row, the tasks'
// blocks side by side in one grid. Otherwise one block per output row,
// 8 warps taking interleaved runs of 4 groups of 128 inputs (lane l: elements
// 4l .. 4l + 3 of each group; its 4 codes are 16 bits). Per element, w =
// fl(q * s_eff) as in W0 and r = fl(fl(k * C^-1/2) * scale) as in the decoder;
// both are accumulated into binary32 sums with fma, reduced over lanes and
// warps.
#include "codetab.cuh"
#include "internal.h"

namespace awsrc {

namespace {

constexpr int kGemvWarps = 8;
constexpr size_t kGemvSmemMax = 96 * 1024;  // x staged in shared memory up to this size
constexpr int kRun = 4;  // groups per warp iteration

__device__ __forceinline__ int code4(uint32_t packed, int i) {  // 4-bit two's complement
  return (int)((int32_t)(packed << (28 - 4 * i)) >> 28);
}

__device__ __forceinline__ float sidecar_scale(const Prm& pr, int16_t s) {
  if (pr.scale_mode == AWSRC_SCALE_POW2) return __int_as_float((s + 127) << 23);
  return __half2float(__ushort_as_half((unsigned short)s));
}

__device__ __forceinline__ float group_scale(const GemvTask& t, int64_t gid) {
  if (t.sdq) {
    const float2 ms = __ldg(reinterpret_cast<const float2*>(t.sdq_consts) + (gid >> 8));
    return __fadd_rn(ms.x, __fmul_rn((float)__ldg(t.sdq_codes + gid), ms.y));
  }
  return __half2float(__ushort_as_half(__ldg(t.scales + gid)));
}

// One block per output row of task ti (x too large for shared memory).
template <int M>
__global__ void __launch_bounds__(32 * kGemvWarps) gemv_kernel(Prm pr, const __grid_constant__ GemvArgs a,
                                                               int ti) {
  __shared__ float part[kGemvWarps][M];
  const GemvTask& tk = a.t[ti];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  const int64_t i = blockIdx.x;  // output row
  const int64_t gpr = tk.cols >> 7;
  float acc[M];
#pragma unroll
  for (int m = 0; m < M; ++m) acc[m] = 0.0f;
  for (int64_t gb = (int64_t)warp * kRun; gb < gpr; gb += (int64_t)kGemvWarps * kRun) {
    uint32_t pk[kRun];
    float s[kRun];
    unsigned long long ent[kRun];
    float4 xv[kRun][M];
#pragma unroll
    for (int u = 0; u < kRun; ++u) {
      const int64_t g = gb + u;
      pk[u] = 0u;
      s[u] = 0.0f;
      ent[u] = 0ull;
#pragma unroll
      for (int m = 0; m < M; ++m) xv[u][m] = make_float4(0.0f, 0.0f, 0.0f, 0.0f);  // runs past the row end
      if (g < gpr) {
        const int64_t gid = i * gpr + g;
        pk[u] = __ldg(tk.codes + gid * 32 + lane);
        s[u] = group_scale(tk, gid);
        const int64_t j0 = g * 128 + 4 * lane;
        if (a.map) ent[u] = __ldg(a.map + tk.tile_off + (i * tk.cols + j0) / pr.C);
#pragma unroll
        for (int m = 0; m < M; ++m) xv[u][m] = __ldg(reinterpret_cast<const float4*>(tk.x + m * tk.cols + j0));
      }
    }
#pragma unroll
    for (int u = 0; u < kRun; ++u) {
      float w[4], r[4] = {0.0f, 0.0f, 0.0f, 0.0f};
#pragma unroll
      for (int e = 0; e < 4; ++e) w[e] = __fmul_rn((float)code4(pk[u], e), s[u]);
      if (ent[u] != 0ull) {  // a recorded tile: its residual on these 4 elements
        const unsigned long long en = ent[u];
        const int64_t k = (int64_t)(en >> 32) - 1;
        const uint32_t seed = (uint32_t)(en >> 16) & 0xFFFFu;
        const float sc = sidecar_scale(pr, (int16_t)(uint16_t)(en & 0xFFFFull));
        const uint2 cw = __ldg(reinterpret_cast<const uint2*>(a.slots + k));  // the slot's codes
        const int jt = (int)(((gb + u) * 128 + 4 * lane) & (pr.C - 1));  // position in the tile
        const uint64_t* mk = a.masks + (size_t)seed * pr.P * pr.W + (jt >> 6);
        int kj[4] = {0, 0, 0, 0};
        for (int p = 0; p < pr.P; ++p) {
          const uint32_t bits = (uint32_t)(__ldg(mk + (size_t)p * pr.W) >> (jt & 63));
          const int cp = (int)(int8_t)((p < 4 ? cw.x : cw.y) >> (8 * (p & 3)));
#pragma unroll
          for (int e = 0; e < 4; ++e) kj[e] += ((bits >> e) & 1u) ? -cp : cp;
        }
#pragma unroll
        for (int e = 0; e < 4; ++e) r[e] = __fmul_rn(__fmul_rn((float)kj[e], pr.c), sc);
      }
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float xe[4] = {xv[u][m].x, xv[u][m].y, xv[u][m].z, xv[u][m].w};
#pragma unroll
        for (int e = 0; e < 4; ++e) {
          acc[m] = __fmaf_rn(w[e], xe[e], acc[m]);
          acc[m] = __fmaf_rn(r[e], xe[e], acc[m]);
        }
      }
    }
  }
#pragma unroll
  for (int m = 0; m < M; ++m) {
#pragma unroll
    for (int off = 16; off > 0; off >>= 1) acc[m] = __fadd_rn(acc[m], __shfl_xor_sync(0xffffffffu, acc[m], off));
    if (lane == 0) part[warp][m] = acc[m];
  }
  __syncthreads();
  if (threadIdx.x < M) {
    float t = 0.0f;
#pragma unroll
    for (int w = 0; w < kGemvWarps; ++w) t = __fadd_rn(t, part[w][threadIdx.x]);
    tk.y[(int64_t)threadIdx.x * tk.rows + i] = t;
  }
}

// One warp per output row (8 rows per block); block b serves the task whose
// block range holds b. The block first stages the task's x in shared memory,
// lane-major per 1024-column chunk: element 1024c + 32l + 4q + e at float
// index 4((8c + q) 32 + l) + e, so that lane l's 16-byte reads of its 32
// consecutive inputs of chunk c are conflict-free. Lane l then streams
// 16-byte code words (32 weights of one group) chunk by chunk, kUnroll chunks
// in flight: nibble pairs become floats through a byte permute into 2^23 + u
// (u the offset-binary code) and one packed subtraction, and are accumulated
// with packed FMAs; each chunk's sum is scaled by its group's s. The row's
// recorded tiles follow, 32 tiles at a time (one map entry per lane). With
// code tables (P = 4, C in {16, 32, 64}) C/16 lanes share a tile, 16 elements
// each, so 512/C recorded tiles go at once: the k_j come from the record's
// table and the seed's nibble table, and r x is accumulated with packed FMAs.
// Otherwise the recorded lanes fetch their record codes and mask words and the
// warp walks the tiles together (elements lane + 32e). The residual terms have
// their own accumulator, added to the backbone's before the lane reduction.
constexpr int kUnroll = 2;
constexpr float kNibbleBias = 8388616.0f;  // 2^23 + 8
constexpr int kPrefetchWords = 4;          // mask words (P * W) a recorded lane prefetches

__device__ __forceinline__ int xs_index(int j) {  // permuted position of input j
  return (((j >> 10) * 8 + ((j >> 2) & 7)) * 32 + ((j >> 5) & 31)) * 4 + (j & 3);
}

// The two codes of byte b of `lo` (even elements) and `hi` (odd elements), both
// offset binary, as floats.
__device__ __forceinline__ float2 nibble_pair(uint32_t lo, uint32_t hi, int b) {
  const float2 v = make_float2(__uint_as_float(__byte_perm(lo, 0x4B000000u, 0x7540u + b)),
                               __uint_as_float(__byte_perm(hi, 0x4B000000u, 0x7540u + b)));
  return __fadd2_rn(v, make_float2(-kNibbleBias, -kNibbleBias));
}

// Loads of one row that do not depend on anything else: the first kUnroll
// chunks' code words and scales, and the first 32 tile-map entries.
struct RowHead {
  uint4 pk[kUnroll];
  float s[kUnroll];
  unsigned long long ent;
};

// Chunks c0, c0 + cs, ... (kUnroll of them) of a row.
__device__ __forceinline__ void load_chunks(const GemvTask& t, int64_t row, int c0, int cs, int nch, int lane,
                                            uint4* pk, float* s) {
  const int64_t rowe = row * t.cols;
  const uint4* cp = reinterpret_cast<const uint4*>(t.codes) + (rowe >> 5) + lane;
  const int lim = (int)t.cols - 32 * lane;  // chunk c is active for this lane when 1024c < lim
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    const int c = c0 + u * cs;
    pk[u] = make_uint4(0u, 0u, 0u, 0u);
    s[u] = 0.0f;
    if (c < nch && 1024 * c < lim) {
      pk[u] = __ldg(cp + 32 * c);
      s[u] = group_scale(t, (rowe >> 7) + 8 * c + (lane >> 2));
    }
  }
}

// The first loads of warp `part` of the wpr warps sharing a row: its chunks
// part, part + wpr and the map entries of tiles 32 part .. 32 part + 31.
__device__ __forceinline__ void load_head(const GemvArgs& a, const GemvTask& t, int64_t row, int nch, int n_cb,
                                          int lane, int part, int wpr, RowHead& h) {
  load_chunks(t, row, part, wpr, nch, lane, h.pk, h.s);
  h.ent = 0ull;
  if (a.map && 32 * part + lane < n_cb) h.ent = __ldg(a.map + t.tile_off + row * n_cb + 32 * part + lane);
}

template <int M>
__device__ __forceinline__ void dense_chunks(const float* xb, int xs_stride, int c0, int cs, const uint4* pk,
                                             const float* s, float* acc) {
#pragma unroll
  for (int u = 0; u < kUnroll; ++u) {
    if (s[u] == 0.0f) continue;  // beyond the row, or an all-zero group (all codes 0)
    const float* xc = xb + 1024 * (c0 + u * cs);
    const uint32_t wd[4] = {pk[u].x, pk[u].y, pk[u].z, pk[u].w};
    float2 part[M];
#pragma unroll
    for (int m = 0; m < M; ++m) part[m] = make_float2(0.0f, 0.0f);
#pragma unroll
    for (int k = 0; k < 4; ++k) {  // word k: inputs 8k .. 8k + 7 of the lane's 32
      const uint32_t lo = (wd[k] & 0x0F0F0F0Fu) ^ 0x08080808u;
      const uint32_t hi = ((wd[k] >> 4) & 0x0F0F0F0Fu) ^ 0x08080808u;
#pragma unroll
      for (int m = 0; m < M; ++m) {
        const float4 x0 = *reinterpret_cast<const float4*>(xc + m * xs_stride + 256 * k);
        const float4 x1 = *reinterpret_cast<const float4*>(xc + m * xs_stride + 256 * k + 128);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 0), make_float2(x0.x, x0.y), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 1), make_float2(x0.z, x0.w), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 2), make_float2(x1.x, x1.y), part[m]);
        part[m] = __ffma2_rn(nibble_pair(lo, hi, 3), make_float2(x1.z, x1.w), part[m]);
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) acc[m] = __fmaf_rn(__fadd_rn(part[m].x, part[m].y), s[u], acc[m]);
  }
}

// The recorded tiles of a row with code tables, in rounds of up to 256 tiles:
// the lanes load the round's map entries at once (tile r0 + 32 i + lane in
// e[i]; the first 32 come with the row head), compact the recorded ones into
// the warp's list (map entry and tile), then take them 512/C per pass, C/16
// lanes per tile and 16 elements per lane: the k_j from the record's table and
// the seed's nibble table, r x accumulated with packed FMAs.
constexpr int kWalkRound = 8;  // batches of 32 tiles per round

struct WalkList {
  unsigned long long en[32 * kWalkRound];
  uint16_t tile[32 * kWalkRound];
};

template <int M, int NB>
__device__ __forceinline__ void walk_tables(const Prm& pr, const GemvArgs& a, const unsigned long long* mrow,
                                            int n_cb, unsigned long long ent0, const float* xsm, int xs_stride,
                                            int lane, WalkList& wl, float2* racc) {
  const int lshift = pr.logC - 4;  // log2 of the lanes per tile
  const int tp = 32 >> lshift;     // tiles per pass
  const int q = lane >> lshift, sub = lane & ((1 << lshift) - 1);
  const KMagic km = k_magic(pr);
  for (int r0 = 0; r0 < n_cb; r0 += 32 * NB) {
    const int nb = min(NB, (n_cb - r0 + 31) >> 5);
    unsigned long long e[NB];
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      const int t = r0 + 32 * i + lane;
      e[i] = (r0 == 0 && i == 0) ? ent0 : ((i < nb && t < n_cb) ? __ldg(mrow + t) : 0ull);
    }
    int n = 0;
#pragma unroll
    for (int i = 0; i < NB; ++i) {
      if (i < nb) {
        const unsigned rec = __ballot_sync(0xffffffffu, e[i] != 0ull);
        if (e[i] != 0ull) {
          const int pos = n + __popc(rec & ((1u << lane) - 1u));
          wl.en[pos] = e[i];
          wl.tile[pos] = (uint16_t)(32 * i + lane);
        }
        n += __popc(rec);
      }
    }
    __syncwarp();
    for (int p0 = 0; p0 < n; p0 += tp) {
      if (p0 + q < n) {
        const unsigned long long en = wl.en[p0 + q];
        const int tile = r0 + wl.tile[p0 + q];
        const uint4 slot = __ldg(a.slots + ((int64_t)(en >> 32) - 1));
        const uint4* nbp = a.nib + (size_t)((uint32_t)(en >> 16) & 0xFFFFu) * (pr.C >> 3) + 2 * sub;
        const uint4 n0 = __ldg(nbp), n1 = __ldg(nbp + 1);
        const float sc = sidecar_scale(pr, (int16_t)(uint16_t)(en & 0xFFFFull));
        const KTab kt = k_tables(slot);
        float k[16];  // k_j c when c is a power of two, else k_j
        table_k4(kt, n0.x, n0.y, km, k);
        table_k4(kt, n0.x >> 16, n0.z, km, k + 4);
        table_k4(kt, n1.x, n1.y, km, k + 8);
        table_k4(kt, n1.x >> 16, n1.z, km, k + 12);
        if (!km.folded) {
#pragma unroll
          for (int i = 0; i < 16; ++i) k[i] = __fmul_rn(k[i], pr.c);
        }
        const float2 s2 = make_float2(sc, sc);
        float2 r[8];
#pragma unroll
        for (int i = 0; i < 8; ++i) r[i] = __fmul2_rn(make_float2(k[2 * i], k[2 * i + 1]), s2);
        // inputs col0 .. col0 + 15 (col0 a multiple of 16): four float4 128 floats apart
        const float* xq = xsm + xs_index(tile * pr.C + 16 * sub);
#pragma unroll
        for (int m = 0; m < M; ++m) {
#pragma unroll
          for (int i = 0; i < 4; ++i) {
            const float4 xv = *reinterpret_cast<const float4*>(xq + m * xs_stride + 128 * i);
            racc[m] = __ffma2_rn(r[2 * i], make_float2(xv.x, xv.y), racc[m]);
            racc[m] = __ffma2_rn(r[2 * i + 1], make_float2(xv.z, xv.w), racc[m]);
          }
        }
      }
    }
    __syncwarp();  // the list is written again by the next round
  }
}

// The same tiles without code tables: the recorded lanes fetch their record
// codes and mask words, and the warp walks the tiles one by one.
template <int M>
__device__ __forceinline__ void walk_masks(const Prm& pr, const GemvArgs& a, unsigned long long ent, int tb,
                                           const float* xsm, int xs_stride, int lane, float2* racc) {
  const bool pre = pr.P * pr.W <= kPrefetchWords;  // recorded lanes prefetch their mask words
  unsigned rec = __ballot_sync(0xffffffffu, ent != 0ull);
  if (!rec) return;
  uint2 cw = make_uint2(0u, 0u);
  unsigned long long mw[kPrefetchWords];
#pragma unroll
  for (int i = 0; i < kPrefetchWords; ++i) mw[i] = 0ull;
  if (ent != 0ull) {
    cw = __ldg(reinterpret_cast<const uint2*>(a.slots + ((int64_t)(ent >> 32) - 1)));
    if (pre) {
      const uint64_t* mk = a.masks + (size_t)((uint32_t)(ent >> 16) & 0xFFFFu) * pr.P * pr.W;
#pragma unroll
      for (int i = 0; i < kPrefetchWords; ++i)
        if (i < pr.P * pr.W) mw[i] = __ldg(mk + i);
    }
  }
  while (rec) {
    const int src = __ffs(rec) - 1;
    rec &= rec - 1;
    const unsigned long long en = __shfl_sync(0xffffffffu, ent, src);
    const uint32_t cx = __shfl_sync(0xffffffffu, cw.x, src), cy = __shfl_sync(0xffffffffu, cw.y, src);
    unsigned long long wv[kPrefetchWords];
#pragma unroll
    for (int i = 0; i < kPrefetchWords; ++i) wv[i] = pre ? __shfl_sync(0xffffffffu, mw[i], src) : 0ull;
    const uint32_t seed = (uint32_t)(en >> 16) & 0xFFFFu;
    const float sc = sidecar_scale(pr, (int16_t)(uint16_t)(en & 0xFFFFull));
    const uint64_t* mk = a.masks + (size_t)seed * pr.P * pr.W;
    const int col0 = (int)(tb + src) * pr.C;
    for (int j = lane; j < pr.C; j += 32) {
      const int wj = j >> 6, sh = j & 63;
      int kj = 0;
#pragma unroll
      for (int p = 0; p < kMaxP; ++p) {
        if (p < pr.P) {
          // prefetched words are indexed statically (one word per atom when C <= 64)
          const unsigned long long word = (pre && pr.W == 1) ? wv[p] : __ldg(mk + p * pr.W + wj);
          const int cpv = (int)(int8_t)((p < 4 ? cx : cy) >> (8 * (p & 3)));
          kj += ((word >> sh) & 1ull) ? -cpv : cpv;
        }
      }
      const float r = __fmul_rn(__fmul_rn((float)kj, pr.c), sc);
#pragma unroll
      for (int m = 0; m < M; ++m) racc[m].x = __fmaf_rn(r, xsm[m * xs_stride + xs_index(col0 + j)], racc[m].x);
    }
  }
}

template <int M>
__global__ void __launch_bounds__(32 * kGemvWarps, M <= 2 ? 3 : 1) gemv_warp_kernel(Prm pr, const __grid_constant__ GemvArgs a) {
  extern __shared__ float4 xs4[];
  __shared__ WalkList wlist[kGemvWarps];
  const int lane = threadIdx.x & 31, warp = threadIdx.x >> 5;
  int ti = 0;
  for (int i = 1; i < a.n_task; ++i)
    if ((int)blockIdx.x >= a.t[i].block0) ti = i;
  const GemvTask& tk = a.t[ti];
  const int nblk = (ti + 1 < a.n_task ? a.t[ti + 1].block0 : (int)gridDim.x) - tk.block0;
  const int xs_stride = (int)((tk.cols + 1023) / 1024 * 1024);
  {
    float* xw = reinterpret_cast<float*>(xs4);
    const int n4 = (int)(tk.cols >> 2), tot = M * n4;
    for (int base = 0; base < tot; base += 4 * blockDim.x) {
      float4 v[4];
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int idx = base + threadIdx.x + i * blockDim.x;
        if (idx < tot) v[i] = __ldg(reinterpret_cast<const float4*>(tk.x) + idx);
      }
#pragma unroll
      for (int i = 0; i < 4; ++i) {
        const int idx = base + threadIdx.x + i * blockDim.x;
        if (idx < tot) {
          const int m = idx / n4, r = idx - m * n4;
          *reinterpret_cast<float4*>(xw + m * xs_stride + xs_index(4 * r)) = v[i];
        }
      }
    }
  }
  __syncthreads();
  const int n_cb = (int)(tk.cols / pr.C);
  const int nch = (int)((tk.cols + 1023) >> 10);
  const float* xsm = reinterpret_cast<const float*>(xs4);  // x in shared memory (permuted)
  const float* xb = xsm + 4 * lane;
  const bool tables = a.nib != nullptr;
  const int64_t stride = (int64_t)nblk * kGemvWarps;
  int64_t row = (int64_t)(blockIdx.x - tk.block0) * kGemvWarps + warp;
  RowHead cur;
  if (row < tk.rows) load_head(a, tk, row, nch, n_cb, lane, 0, 1, cur);
  for (; row < tk.rows; row += stride) {
    // the next row's head is in flight while this row is computed
    RowHead nxt;
    if (row + stride < tk.rows) load_head(a, tk, row + stride, nch, n_cb, lane, 0, 1, nxt);
    float acc[M];
    float2 racc[M];
#pragma unroll
    for (int m = 0; m < M; ++m) {
      acc[m] = 0.0f;
      racc[m] = make_float2(0.0f, 0.0f);
    }
    if (nch <= kUnroll) {
      dense_chunks<M>(xb, xs_stride, 0, 1, cur.pk, cur.s, acc);
    } else {  // wide rows: the next kUnroll chunks are in flight while these are summed
      uint4 pk[kUnroll];
      float s[kUnroll];
      load_chunks(tk, row, kUnroll, 1, nch, lane, pk, s);
      dense_chunks<M>(xb, xs_stride, 0, 1, cur.pk, cur.s, acc);
      for (int c0 = kUnroll; c0 < nch; c0 += kUnroll) {
        uint4 pk2[kUnroll];
        float s2[kUnroll];
        load_chunks(tk, row, c0 + kUnroll, 1, nch, lane, pk2, s2);  // zeros past the row end
        dense_chunks<M>(xb, xs_stride, c0, 1, pk, s, acc);
#pragma unroll
        for (int u = 0; u < kUnroll; ++u) {
          pk[u] = pk2[u];
          s[u] = s2[u];
        }
      }
    }
    if (a.map) {
      const unsigned long long* mrow = a.map + tk.tile_off + row * n_cb;
      if (tables) {
        if (n_cb <= 32)  // one batch of map entries, already loaded with the row head
          walk_tables<M, 1>(pr, a, mrow, n_cb, cur.ent, xsm, xs_stride, lane, wlist[warp], racc);
        else
          walk_tables<M, kWalkRound>(pr, a, mrow, n_cb, cur.ent, xsm, xs_stride, lane, wlist[warp], racc);
      } else {
        for (int tb = 0; tb < n_cb; tb += 32) {
          const unsigned long long ent =
              tb == 0 ? cur.ent : ((tb + lane < n_cb) ? __ldg(mrow + tb + lane) : 0ull);
          walk_masks<M>(pr, a, ent, tb, xsm, xs_stride, lane, racc);
        }
      }
    }
#pragma unroll
    for (int m = 0; m < M; ++m) {
      float v = __fadd_rn(acc[m], __fadd_rn(racc[m].x, racc[m].y));
#pragma unroll
      for (int off = 16; off > 0; off >>= 1) v = __fadd_rn(v, __shfl_xor_sync(0xffffffffu, v, off));
      if (lane == 0) tk.y[(int64_t)m * tk.rows + row] = v;
    }
    cur = nxt;
  }
}

// Relative cost of a task: its weights.
double task_cost(const GemvTask& t) { return (double)t.rows * (double)t.cols; }

size_t x_smem_bytes(const GemvTask& t, int M) { return (size_t)M * ((t.cols + 1023) / 1024 * 1024) * 4; }

template <int M>
cudaError_t launch_gemv_m(const Prm& pr, const GemvArgs& a, cudaStream_t st) {
  const dim3 block(32 * kGemvWarps);
  // tasks whose x fits in shared memory share one launch; the others take a
  // block per output row each
  GemvArgs b = a;
  b.n_task = 0;
  size_t smem = 0;
  double work = 0.0;
  for (int i = 0; i < a.n_task; ++i) {
    const size_t need = x_smem_bytes(a.t[i], M);
    if (need <= kGemvSmemMax) {
      b.t[b.n_task++] = a.t[i];
      smem = need > smem ? need : smem;
      work += task_cost(a.t[i]);
    } else {
      gemv_kernel<M><<<dim3((unsigned)a.t[i].rows), block, 0, st>>>(pr, a, i);
      note_launches(1);
      const cudaError_t e = cudaGetLastError();
      if (e != cudaSuccess) return e;
    }
  }
  if (b.n_task == 0) return cudaSuccess;
  int dev = 0, nsm = 0, per_sm = 0;
  cudaError_t e = cudaGetDevice(&dev);
  if (e == cudaSuccess) e = cudaDeviceGetAttribute(&nsm, cudaDevAttrMultiProcessorCount, dev);
  if (e == cudaSuccess)
    e = cudaFuncSetAttribute(gemv_warp_kernel<M>, cudaFuncAttributeMaxDynamicSharedMemorySize, (int)kGemvSmemMax);
  if (e == cudaSuccess) e = cudaOccupancyMaxActiveBlocksPerMultiprocessor(&per_sm, gemv_warp_kernel<M>,
                                                                          32 * kGemvWarps, smem);
  if (e != cudaSuccess) return e;
  // one wave of resident blocks shared out in proportion to each task's cost
  // (largest remainders first), each task at least one block and at most one
  // per 8 rows
  const int64_t slots = (int64_t)nsm * (per_sm > 0 ? per_sm : 1);
  int64_t nb[kMaxGemvTasks], most[kMaxGemvTasks], used = 0;
  double frac[kMaxGemvTasks];
  for (int i = 0; i < b.n_task; ++i) {
    most[i] = (b.t[i].rows + kGemvWarps - 1) / kGemvWarps;
    const double share = (double)slots * task_cost(b.t[i]) / work;
    nb[i] = (int64_t)share;
    frac[i] = share - (double)nb[i];
    nb[i] = nb[i] < 1 ? 1 : (nb[i] > most[i] ? most[i] : nb[i]);
    used += nb[i];
  }
  while (used < slots) {
    int best = -1;
    for (int i = 0; i < b.n_task; ++i)
      if (nb[i] < most[i] && (best < 0 || frac[i] > frac[best])) best = i;
    if (best < 0) break;
    ++nb[best];
    frac[best] -= 1.0;
    ++used;
  }
  int blocks = 0;
  for (int i = 0; i < b.n_task; ++i) {
    b.t[i].block0 = blocks;
    blocks += (int)nb[i];
  }
  gemv_warp_kernel<M><<<dim3((unsigned)blocks), block, smem, st>>>(pr, b);
  note_launches(1);
  return cudaGetLastError();
}

}  // namespace

cudaError_t launch_gemv(const Prm& pr, const GemvArgs& a, int M, cudaStream_t st) {
  switch (M) {
    case 1: return launch_gemv_m<1>(pr, a, st);
    case 2: return launch_gemv_m<2>(pr, a, st);
    case 3: return launch_gemv_m<3>(pr, a, st);
    case 4: return launch_gemv_m<4>(pr, a, st);
    case 5: return launch_gemv_m<5>(pr, a, st);
    case 6: return launch_gemv_m<6>(pr, a, st);
    case 7: return launch_gemv_m<7>(pr, a, st);
    case 8: return launch_gemv_m<8>(pr, a, st);
    default: return cudaErrorInvalidValue;
  }
}

bool gemv_tables(const Prm& pr) { return code_tables(pr) && pr.C >= 16; }

}  // namespace awsrc
