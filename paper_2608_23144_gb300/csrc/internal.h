// internal.h — host-side declarations shared by the library's translation units.
#pragma once

#include <cstddef>
#include <cstdint>
#include <cuda_runtime.h>

#include "common.cuh"

namespace awsrc {

// Validated parameters -> Prm (derived constants). Returns AWSRC_OK or an error.
awsrc_status make_prm(const awsrc_params* prm, Prm* out);

// Records the CUDA error text for awsrc_last_error_message() and maps it.
awsrc_status cuda_fail(cudaError_t e, const char* where);
awsrc_status check_launch(const char* where);
// Sets the text awsrc_last_error_message() returns (printf-style).
void set_error_message(const char* fmt, ...);

inline size_t align_up(size_t x, size_t a) { return (x + a - 1) / a * a; }

// Launch counter behind awsrc_kernel_launches(): every launch site adds its kernels.
void note_launches(int n);

// masks[(s*P + p)*W + w] for s in [0, S_pad); seeds >= S get zero masks.
cudaError_t launch_gen_basis(const Prm& pr, uint64_t* masks, int S_out, cudaStream_t st);


// encode.cu
// Writes the Gram table and, when `pairs` is not null, the paired table
// (pair_stride(P) float2 per seed pair) the C = 64, P = 4 search reads.
cudaError_t launch_gram_u(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                          float* gram, float2* pairs, cudaStream_t st);
// The generic search (any C, P, variant): blocks of gen_shape(pr).tiles
// consecutive tiles, `lanes` threads per tile; writes whole candidates to
// cands[z * T + t] like the specialised kernels.
struct GenShape {
  int lanes, tiles;
};
GenShape gen_shape(const Prm& pr);
cudaError_t launch_search_generic(const Prm& pr, const LaunchDesc& ld, const uint64_t* masks,
                                  const float* gram, int64_t n_blocks, awsrc_candidate* cands,
                                  cudaStream_t st);
// search_c64p4.cu
// FP16 table of the +-1 atoms in MMA operand order, then the tcgen05 search.
size_t search_c64p4_table_bytes(int S_pad);
cudaError_t launch_bfrag_c64p4(const Prm& pr, const uint64_t* masks, void* out, cudaStream_t st);
// Writes each tile's best candidate (codes included) to cands[z * T + t] for
// seed split z; launch_merge_candidates reduces the splits of tiles [t0, t1).
cudaError_t launch_search_c64p4(const Prm& pr, const LaunchDesc& ld, const void* table,
                                const float2* pairs, const uint64_t* masks, int64_t n_blocks,
                                awsrc_candidate* cands,
                                uint32_t* status, cudaStream_t st);
cudaError_t launch_merge_candidates(const awsrc_candidate* pc, int nsplit, int64_t T, int64_t t0, int64_t t1,
                                   awsrc_candidate* out, cudaStream_t st);
int search_c64p4_rows();   // rows per block of the specialised kernel
int search_c64p4_chunk();  // seeds per chunk of the specialised kernel
// search_pf_c64p4.cu: P_F with C = 64, P = 4 on tcgen05 (atoms from the table
// above, plus a table of atom products), same candidate output.
int search_pf_c64p4_chunk();
size_t search_pf_c64p4_table_bytes(int S_pad);
cudaError_t launch_products_pf_c64p4(const Prm& pr, const uint64_t* masks, void* out, cudaStream_t st);
cudaError_t launch_search_pf_c64p4(const Prm& pr, const LaunchDesc& ld, const void* atoms, const void* prods,
                                   const uint64_t* masks, int64_t n_blocks, awsrc_candidate* cands,
                                   uint32_t* status, cudaStream_t st);

// select.cu
struct SelectPlan {
  int n_mod, n_rates;
  int64_t T, L, h;
  int key_bits, tile_bits_local, mod_shift;
  int64_t cap_records;      // upper bound on records written
  int64_t nblocks;          // radix blocks
};
awsrc_status select_run(const Prm& pr, const SelectPlan& sp, const int64_t* tile_off,
                        const int64_t* mod_tiles, const int64_t* kcap /* U: per module; PF: per rate */,
                        const awsrc_candidate* cands, uint8_t* stream_out, int64_t* d_counts,
                        int64_t* d_bytes, void* ws, size_t ws_bytes, cudaStream_t st);
size_t select_ws_bytes(const SelectPlan& sp);

// decode.cu
struct DecodeMod {
  const void* W0;
  void* out;
  int64_t rows, cols, tile_off;
  int32_t w0_dtype, pad_;
};
cudaError_t launch_decode(const Prm& pr, int n_mod, const DecodeMod* mods, int64_t T, int64_t L,
                          int64_t h, const uint8_t* stream, int64_t K, int64_t kmax, int out_dtype, int mode,
                          uint64_t* masks, void* scratch, uint32_t* status, cudaStream_t st);
size_t decode_scratch_bytes(const Prm& pr, int64_t T, int mode);
// Dense scratch: the tile map (8 B per tile, from offset 0), then one 16-byte
// slot per record (codes x, y; code tables z, w) at slots_off, then (P = 4,
// C <= 64) the nibble tables at nib_off.
struct DenseScratch {
  size_t slots_off, nib_off, bytes;
};
DenseScratch dense_scratch(const Prm& pr, int64_t T);
cudaError_t launch_dense_prep(const Prm& pr, int64_t T, int64_t L, int64_t h, const uint8_t* stream, int64_t K,
                              int64_t kmax, uint64_t* masks, void* scratch, uint32_t* status, cudaStream_t st);
// The dense fused decoder clears the fault word itself (no separate memset).
bool decode_clears_status(const Prm& pr, int mode);

// gemv.cu: y[m] = (W0 + r_hat) x[m] for a batch of (module, x, y) tasks of a
// prepared sidecar, one launch for the tasks whose x fits in shared memory.
struct GemvTask {
  int64_t rows, cols, tile_off;  // tile_off: the module's first global tile
  int32_t sdq, block0;           // block0: the task's first block (set by launch_gemv)
  const uint16_t* codes;         // 4 codes per uint16, element 2i in the low nibble of byte i
  const uint16_t* scales;        // binary16 per group (sdq == 0)
  const int8_t* sdq_codes;       // per group (sdq)
  const float* sdq_consts;       // (mean, step) per 256 groups (sdq)
  const float* x;                // M x cols
  float* y;                      // M x rows
};
constexpr int kMaxGemvTasks = 16;
struct GemvArgs {
  int n_task;
  const unsigned long long* map; // tile map of the prepared sidecar, or null (no residual)
  const uint4* slots;            // per-record slots of the prepared sidecar (codes in x, y)
  const uint64_t* masks;         // basis masks of the prepared sidecar
  const uint4* nib;              // nibble tables of the prepared sidecar when gemv_tables(), else null
  GemvTask t[kMaxGemvTasks];
};
// Whether the GEMV walks recorded tiles with the decoder's code tables.
bool gemv_tables(const Prm& pr);
cudaError_t launch_gemv(const Prm& pr, const GemvArgs& a, int M, cudaStream_t st);

// backbone.cu: RTN-INT4 groups of rtn_group() inputs, SDQ blocks of sdq_block() groups.
int rtn_group();
int sdq_block();
// One launch for a batch of modules sharing (w_dtype, w0_dtype).
struct RtnTask {
  const void* W;
  int64_t G;            // groups of 128
  int32_t sdq, block0;  // block0: the task's first block (set by launch_rtn)
  uint32_t* codes;
  uint16_t* scales;
  int8_t* sdq_codes;
  float* sdq_consts;
  void* W0;
};
constexpr int kMaxRtnTasks = 16;
struct RtnArgs {
  int n;
  RtnTask t[kMaxRtnTasks];
};
cudaError_t launch_rtn(const RtnArgs& a, int w_dtype, int w0_dtype, cudaStream_t st);
int64_t rtn_max_blocks();  // blocks one launch may take

// numerics.cu: bit patterns in [first, last) where rcp_rn differs from __frcp_rn
// are added to *bad (device).
cudaError_t launch_verify_rcp(uint32_t first, uint32_t last, unsigned long long* bad, cudaStream_t st);

}  // namespace awsrc
