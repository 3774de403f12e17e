/*
 * awsrc.h — C ABI of the GB300 (sm_103a) implementation of the hot path of
 * Activation-Weighted Seeded Residual Coding (AWSRC, arXiv 2608.23144):
 * per-(tile, seed) search over the residual R = W - W0 of a fixed backbone,
 * byte-aware record selection, and decode-apply.
 *
 * Conventions shared by every entry point
 * ---------------------------------------
 *  - Every array argument documented as "device" is caller-owned device memory
 *    on the current CUDA device; "host" arguments are caller-owned host memory.
 *    The library never allocates device memory: scratch space is the caller's
 *    `workspace`, whose size is queried with the matching *_workspace_bytes call.
 *  - `stream` is a cudaStream_t passed as void* (NULL = legacy default stream).
 *    Every launch is asynchronous on that stream; no entry point synchronises
 *    unless its comment says so.
 *  - Errors are returned as awsrc_status, never thrown. Arguments are validated
 *    on the host before any launch; on error nothing is launched and no output
 *    is written. A CUDA runtime failure returns AWSRC_ERR_CUDA, and
 *    awsrc_last_error_message() gives the runtime's text (thread-local).
 *  - Inputs are never modified; the only exception is W_hat aliasing W0 in
 *    AWSRC_DECODE_INPLACE mode.
 *  - Matrices are row-major: element (i, j) of a rows x cols module is at
 *    i*cols + j (output row i, input channel j). Tiles are C contiguous input
 *    channels of one output row (Sec. 3.1): tile t = i*(cols/C) + cb covers
 *    columns [cb*C, cb*C + C). Global tile indices concatenate modules in the
 *    order given: module m's tiles start at sum_{m'<m} rows*cols/C.
 *
 * Numeric convention
 * ------------------
 * Encoder and decoder share the generator and the numeric convention (Sec. 3.1);
 * basis generation and tie breaking are fixed (Sec. 4). The convention is IEEE
 * binary32, round-to-nearest-even, in exactly this order (fma = one rounding,
 * every other operation rounds once; sums run j = 0..C-1 ascending):
 *
 *  GenBasis(s) (Eq. 2). SplitMix64 (Steele, Lea & Flood 2014): the n-th output
 *   (n >= 1) of the stream started at state x is mix64(x + n*0x9E3779B97F4A7C15).
 *   key_s = output s+1 of the stream at gen_seed; draws are outputs 1, 2, ... of
 *   the stream at key_s, consumed in this order: ceil(C/64) sign words (bit j%64
 *   of word j/64 is sigma_j, 1 = negative); if permute, for i = C-1 down to 1 one
 *   draw, k = ((draw >> 32) * (i+1)) >> 32, swap(pi[i], pi[k]) starting from the
 *   identity; then for p = 0..P-1 one draw, k = p + (((draw >> 32) * (C-p)) >> 32),
 *   swap(col[p], col[k]) on the identity array, c_p = col[p]. Entry (j, p) of
 *   B_s is C^-1/2 * (-1)^(sigma_j + popcount(pi[j] & c_p)) (Sylvester Hadamard).
 *   m_p(j) denotes the sign (+-1) of that entry.
 *  Weights. r_j = W - W0 (after exact widening to f32); U: d_j = a_j; PF:
 *   d_j = w_act*a_j + w_fisher*F_ij; y_j = d_j * r_j. A tile is invalid (gain
 *   -inf) unless every r_j is finite with |r_j| <= 2^16 and every d_j is in [0, 2^32].
 *  Fit (Eq. 3). c = RN(C^-1/2), c2 = 1/C. The +-1 correlations are exact
 *   integer sums on a per-tile fixed-point grid: for a vector x (y or d) let
 *   q = ilogb(max_j |x_j|) - 20 and X_j = rint(x_j*2^-q), so |X_j| <= 2^21 (x is
 *   all zero, q = 0, when max |x| < 2^-100). Then u_p = 2^qy * RN(sum_j m_p(j) Y_j)
 *   and b_p = c*u_p; gd = c2 * 2^qd * RN(sum_j D_j); G_pp = gd;
 *   G_pq = c2 * 2^qd * RN(sum_j m_p(j)m_q(j) D_j) (each sum exact, rounded once).
 *   eps = ridge_rel*gd; A = G + eps*I. LDL^T, k = 0..P-1: for j < k:
 *   v = A_kj, v = fma(-L_ki, E_ji, v) for i < j, E_kj = v, L_kj = v*invD_j;
 *   D_k = A_kk, D_k = fma(-L_ki, E_ki, D_k) for i < k; the candidate is invalid
 *   unless 0 < D_k <= FLT_MAX; invD_k = 1/D_k. Solve: z_k = b_k then
 *   z_k = fma(-L_ki, z_i, z_k) for i < k; w_k = z_k*invD_k; for k = P-1 down to 0:
 *   alpha_k = w_k then alpha_k = fma(-L_ik, alpha_i, alpha_k) for i = k+1..P-1.
 *  Quantisation (Sec. 3.2). amax = max_p |alpha_p| (NaN propagates); invalid
 *   unless 2^-100 <= amax <= 2^32. POW2: e = smallest integer with
 *   amax <= qmax*2^e, clamped to the exponent range; code_p =
 *   clamp(rint(alpha_p*2^-e), -qmax, qmax); sc = 2^e. FP16: sc = binary16_RN(
 *   amax/qmax) (invalid if 0 or inf), code_p = clamp(rint(alpha_p/sc), -qmax, qmax).
 *  Gain (Eq. 4, unregularised G). Aq = fma(code_p, b_p, Aq) over p; Qq over p
 *   ascending: Qq = fma(code_p^2, G_pp, Qq), then for q > p
 *   Qq = fma(2*code_p*code_q, G_pq, Qq); gain = sc * (2*Aq - sc*Qq).
 *  Selection. s* = argmax_s gain (strictly greater replaces: ties keep the
 *   smallest s); a tile whose every candidate is invalid has gain -inf.
 * Integer outputs (seed selectors, exponents, codes, record order, byte counts)
 * are therefore reproducible bit for bit by any implementation of this recipe.
 */
#ifndef AWSRC_H
#define AWSRC_H

#include <stddef.h>
#include <stdint.h>

#ifdef __cplusplus
extern "C" {
#endif

typedef enum awsrc_status {
  AWSRC_OK = 0,
  AWSRC_ERR_INVALID_ARG = 1,  /* null pointer, bad enum, n_mod < 1, K out of range */
  AWSRC_ERR_SHAPE = 2,        /* cols % C != 0, rows/cols < 1, C not a power of two */
  AWSRC_ERR_UNSUPPORTED = 3,  /* parameter outside the supported ranges below */
  AWSRC_ERR_BUDGET = 4,       /* a byte budget is smaller than the stream header */
  AWSRC_ERR_CUDA = 5,         /* CUDA runtime error; see awsrc_last_error_message() */
  AWSRC_ERR_WORKSPACE = 6,    /* workspace NULL or smaller than the queried size */
  AWSRC_ERR_CAPACITY = 7,     /* output stream buffer smaller than awsrc_stream_capacity() */
  AWSRC_ERR_DEVICE = 8        /* a kernel reported a fault in its inputs (corrupt stream) */
} awsrc_status;

enum { AWSRC_VARIANT_U = 0, AWSRC_VARIANT_PF = 1 };
enum { AWSRC_SCALE_POW2 = 0, AWSRC_SCALE_FP16 = 1 };
enum { AWSRC_DTYPE_F32 = 0, AWSRC_DTYPE_BF16 = 1 };
enum { AWSRC_DECODE_DENSE = 0, AWSRC_DECODE_INPLACE = 1 };

/*
 * Codec parameters (Sec. 3.1: C locality, P subspace dimension, b coefficient
 * precision, S basis diversity; Eq. 5: b_e scale-exponent width).
 *   C          tile length; power of two in [4, 256] (Sylvester Hadamard order).
 *   P          atoms (basis columns) per tile, 1 <= P <= min(8, C).
 *   b          coefficient bits, 2 <= b <= 8. Codes are symmetric round-to-
 *              nearest-even integers in [-qmax, qmax], qmax = 2^(b-1) - 1 (Sec. 3.2).
 *   S          seeds searched per tile, 1 <= S <= 65536; selector s in [0, S).
 *   b_e        scale field width. POW2: 1..8 bits holding e - e_bias in two's
 *              complement (the paper's power-of-two scale exponent, Sec. 3.2);
 *              FP16: must be 16 (binary16 scale, the small synthetic workload's option).
 *   e_bias     POW2 only: exponents are clamped to
 *              [max(e_bias - 2^(b_e-1), -126), min(e_bias + 2^(b_e-1) - 1, 126)],
 *              which must be non-empty.
 *   scale_mode AWSRC_SCALE_POW2 or AWSRC_SCALE_FP16.
 *   permute    1: each seed draws a coordinate permutation (Sec. 3.1); 0: identity.
 *   variant    AWSRC_VARIANT_U (activation weights, per-module quotas) or
 *              AWSRC_VARIANT_PF (blended activation/Fisher weights, global
 *              progressive prefixes) (Sec. 3.3).
 *   ridge_rel  ridge of Eq. 3 relative to the tile's mean weight:
 *              eps = ridge_rel * (1/C) * sum_j d_{t,j}; finite, >= 0.
 *   gen_seed   key of the shared deterministic basis generator (Sec. 3.1).
 */
typedef struct awsrc_params {
  int32_t C, P, b, S;
  int32_t b_e, e_bias;
  int32_t scale_mode, permute, variant;
  float ridge_rel;
  uint64_t gen_seed;
} awsrc_params;

/*
 * Pointer alignment (checked; a violation returns AWSRC_ERR_INVALID_ARG before
 * any launch): device arrays at least at their element size; workspaces at 256
 * bytes (as cudaMalloc returns them); W0 and W_hat of the decoder at 16 bytes.
 *
 * One linear module (a weight matrix W with backbone reconstruction W0 = Q(W),
 * Eq. 1) and its per-input-channel statistics (Sec. 3.2).
 *   rows, cols  output and input dimensions; cols % C == 0. The tiles of all
 *               modules of one call, sum rows*cols/C, must number below 2^32
 *               (tile indices are 32-bit), else AWSRC_ERR_UNSUPPORTED.
 *   W, W0       device, rows*cols elements of w_dtype / w0_dtype (F32 or BF16).
 *               The encoder reads both; the decoder reads W0 only (W may be NULL).
 *   act         device, cols floats: activation second moments a_j = E[x_j^2].
 *   fisher      device, rows*cols floats: Fisher diagonal (PF only; NULL for U).
 *   w_act, w_fisher  PF blend weights including their normalisers: the element
 *               weight is d_ij = w_act*a_j + w_fisher*F_ij (Sec. 3.3). Ignored by U,
 *               where d_ij = a_j (the activation diagonal is shared by rows, Sec. 3.2).
 */
typedef struct awsrc_module {
  int64_t rows, cols;
  int32_t w_dtype, w0_dtype;
  const void* W;
  const void* W0;
  const float* act;
  const float* fisher;
  float w_act, w_fisher;
} awsrc_module;

/*
 * Best candidate of one tile (Sec. 3.2: the seed with the lowest post-quantisation
 * weighted error, i.e. the largest gain). 16 bytes, device arrays of these are
 * indexed by global tile.
 *   gain   weighted error reduction of Eq. 4 (numerator), computed from the
 *          quantised coefficients; -inf when no seed yields a valid fit.
 *   seed   selector s_t* in [0, S) (0 when gain is -inf).
 *   scale  POW2: exponent e (scale 2^e); FP16: raw binary16 bits of the scale.
 *   code   the P signed b-bit codes; entries p >= P are 0.
 */
typedef struct awsrc_candidate {
  float gain;
  uint16_t seed;
  int16_t scale;
  int8_t code[8];
} awsrc_candidate;

/* ---------------------------------------------------------------- encoder -- */

/*
 * awsrc_encode_workspace_bytes — device scratch needed by awsrc_encode_tiles for
 * these parameters and modules (basis masks, per-(seed, column block) Gram
 * factors for U, per-split partial results). Host-only; launches nothing.
 */
awsrc_status awsrc_encode_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, size_t* bytes);

/*
 * awsrc_encode_tiles — the seed search of Sec. 3.2 for every tile of every
 * module. For each tile t and each seed s it regenerates B_s = GenBasis(s, C, P)
 * (Eq. 2), fits alpha*_{t,s} by the weighted ridge least squares of Eq. 3,
 * quantises it coefficient-wise with one scale per tile, scores the quantised
 * reconstruction by the weighted error reduction of Eq. 4, and keeps the best
 * seed (ties: smallest s).
 *   out        device, sum_m rows_m*cols_m/C candidates, indexed by global tile.
 *   workspace  device, >= awsrc_encode_workspace_bytes(); contents are scratch.
 * Errors: INVALID_ARG, SHAPE, UNSUPPORTED, WORKSPACE, CUDA.
 */
awsrc_status awsrc_encode_tiles(const awsrc_params* prm, int32_t n_mod,
                                const awsrc_module* mods, awsrc_candidate* out,
                                void* workspace, size_t workspace_bytes, void* stream);

/*
 * awsrc_rtn_quantize — the RTN-INT4 backbone W0 = Q(W) of Eq. 1 that the
 * residual R = W - W0 is coded against: symmetric round to nearest with groups
 * of 128 consecutive input coordinates of a row (Sec. 4), optionally with scale
 * double quantisation (SDQ, Sec. 3.3, after QLoRA's double quantisation; the
 * paper gives no format, this is the library's). All binary32, one rounding per
 * operation:
 *   group g (row-major, cols % 128 == 0): s_g = binary16(max|w| / 7);
 *     q = clamp(rint(w / s_g), -8, 7), q = 0 when s_g == 0 (|q| <= 7 in fact);
 *   SDQ block b of 256 consecutive groups (the last may be shorter, n groups):
 *     mu = binary32((sum of the block's s_g, exact in double) / n);
 *     step = max_g |s_g - mu| / 127;
 *     c_g = clamp(rint((s_g - mu) / step), -127, 127), 0 when step == 0;
 *     s~_g = mu + c_g * step;
 *   W0 = q * s_eff with s_eff = s_g, or s~_g under SDQ (codes stay those of s_g).
 * Metadata: binary16 scales cost 2 bytes per group (0.125 bits/weight); SDQ
 * 1 byte per group plus 8 per block (0.0645 bits/weight on whole blocks), see
 * awsrc_backbone_metadata_bytes and awsrc_rate_with_sdq_savings. W must be finite.
 *   W           device, rows*cols elements of w_dtype, 16-byte aligned.
 *   codes       device, rows*cols/2 bytes (4-byte aligned): element 2i in the
 *               low nibble of byte i, 4-bit two's complement.
 *   scales      device, G = rows*cols/128 binary16 s_g, or NULL.
 *   sdq_codes   device, G int8 c_g (SDQ), or NULL.
 *   sdq_consts  device, 2*ceil(G/256) floats (mu, step) per block (SDQ), or NULL.
 *   W0          device, rows*cols elements of w0_dtype (16-byte aligned), or NULL.
 * Errors: INVALID_ARG, SHAPE (cols % 128), UNSUPPORTED (rows*cols > 2^46),
 * CUDA.
 */
awsrc_status awsrc_rtn_quantize(int64_t rows, int64_t cols, const void* W, int32_t w_dtype, int32_t sdq,
                                uint8_t* codes, uint16_t* scales, int8_t* sdq_codes, float* sdq_consts,
                                void* W0, int32_t w0_dtype, void* stream);

/*
 * awsrc_rtn_quantize_batch — awsrc_rtn_quantize for n_task >= 1 modules in as
 * few launches as their dtypes allow (one when all share w_dtype and
 * w0_dtype and there are at most 16): every output is bit-identical to the
 * single call's. Arguments per task as for awsrc_rtn_quantize; the output
 * arrays of different tasks must not overlap. Errors: as awsrc_rtn_quantize
 * (the first failing task decides; nothing is launched then).
 */
typedef struct awsrc_rtn_task {
  int64_t rows, cols;
  const void* W;
  int32_t w_dtype, sdq;
  uint8_t* codes;
  uint16_t* scales;
  int8_t* sdq_codes;
  float* sdq_consts;
  void* W0;
  int32_t w0_dtype, pad_;
} awsrc_rtn_task;

awsrc_status awsrc_rtn_quantize_batch(int32_t n_task, const awsrc_rtn_task* tasks, void* stream);

/*
 * awsrc_backbone_metadata_bytes — scale metadata of a rows x cols RTN-INT4
 * backbone: 2 bytes per group of 128, or with SDQ 1 per group plus 8 per block
 * of 256 groups. Under a fixed total budget the bytes SDQ saves can go to the
 * residual records (Sec. 3.3): awsrc_rate_with_sdq_savings gives the rate for
 * awsrc_select_records that does so exactly. Returns -1 for a bad shape or
 * rows*cols above 2^46.
 */
int64_t awsrc_backbone_metadata_bytes(int64_t rows, int64_t cols, int32_t sdq);

/*
 * awsrc_rate_with_sdq_savings — the rate to give awsrc_select_records when the
 * backbone's scales are double quantised and the metadata bytes SDQ saves go
 * to the residual records (Sec. 3.3) under an unchanged total budget. With
 * binary16 scales the scope holds meta_fp16 + B bytes, B = floor(rate_bpw *
 * N_scope / 8) (Eq. 5, header included); with SDQ the sidecar may then take
 * B + saved bytes, saved = sum_m (awsrc_backbone_metadata_bytes(m, 0) -
 * awsrc_backbone_metadata_bytes(m, 1)). *rate_out is a rate whose budget
 * floor(rate_out * N_scope / 8) is exactly B + saved, so that backbone
 * metadata plus stream never exceed meta_fp16 + B; *saved_bytes (may be NULL)
 * receives saved. On modules of a few groups SDQ's 8-byte block constants
 * cost more than it saves: saved is then negative and the budget shrinks.
 * Reads rows and cols of each module (cols % 128 == 0). Host-only.
 * Errors: INVALID_ARG, SHAPE, BUDGET (B + saved < 0), UNSUPPORTED
 * (N_scope >= 2^52).
 */
awsrc_status awsrc_rate_with_sdq_savings(int32_t n_mod, const awsrc_module* mods, double rate_bpw,
                                         double* rate_out, int64_t* saved_bytes);

/*
 * awsrc_gen_basis — writes the sign masks of GenBasis (Eq. 2) for seeds [0, S):
 * masks[(s*P + p)*W + w], W = ceil(C/64) words, bit j%64 of word j/64 set when
 * entry (j, p) of B_s is negative. Device array of S*P*W uint64. Used by the
 * decoder and exposed for tests.
 */
awsrc_status awsrc_gen_basis(const awsrc_params* prm, uint64_t* masks, void* stream);

/* ------------------------------------------------------------- selection -- */

/* Serialized record size L of Eq. 5 in bytes for T candidate tiles:
 * ceil((ceil(log2 T) + ceil(log2 S) + b_e + P*b) / 8). Host-only. Returns -1 on
 * invalid parameters. */
int64_t awsrc_record_bytes(const awsrc_params* prm, int64_t T);

/* Stream header size h of Eq. 5: 40 bytes + 8 bytes per module. Host-only. */
int64_t awsrc_header_bytes(int32_t n_mod);

/*
 * awsrc_stream_capacity — bytes the stream buffer of awsrc_select_records must
 * hold: h + K_max*L, K_max the largest record count any of the rates allows.
 * Host-only.
 */
awsrc_status awsrc_stream_capacity(const awsrc_params* prm, int32_t n_mod,
                                   const awsrc_module* mods, const double* rates_bpw,
                                   int32_t n_rates, size_t* bytes);

awsrc_status awsrc_select_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, size_t* bytes);

/*
 * awsrc_select_records — byte-aware allocation (Sec. 3.3) and serialisation
 * (Sec. 3.4, Eq. 5). Candidates with gain <= 0 (or non-finite) are discarded.
 * Records are ranked by rho_t = gain_t / L (Eq. 4); L is the same for every
 * record, so the order is gain descending, ties by global tile ascending.
 * Budgets are B = floor(rate * N_scope / 8) bytes including the header, with
 * N_scope = sum_m rows*cols.
 *   U  (n_rates == 1): module m receives quota_m = floor((B - h) * N_m / N_scope)
 *      bytes and keeps K_m = min(#positive_m, floor(quota_m / L)) records; the
 *      stream holds module 0's records, then module 1's, ..., each block in
 *      rank order. d_counts[m] = K_m (n_mod entries), d_bytes[0] = stream bytes.
 *   PF (n_rates >= 1): one global ranking; rate r keeps the longest prefix
 *      K_r = min(#positive, floor((B_r - h) / L)); the stream holds the longest
 *      prefix and every shorter one decodes as it stands. d_counts[r] = K_r,
 *      d_bytes[r] = h + K_r*L.
 *   stream_out  device, >= awsrc_stream_capacity() bytes: header + records.
 *   d_counts, d_bytes  device int64 arrays as above.
 * Stream layout (little-endian): header of 40 + 8*n_mod bytes, then fixed-width
 * records of L bytes. Record bits are LSB-first from bit 0: tile (ceil(log2 T)
 * bits), seed (ceil(log2 S)), scale field (b_e), codes 0..P-1 (b bits each, two's
 * complement); remaining bits zero. Header: u32 magic 0x52535741, u16 version 1,
 * u8 variant, u8 scale_mode, u16 C, u8 P, u8 b, u8 b_e, i8 e_bias, u8 permute,
 * u8 0, u32 S, u32 n_mod, u64 gen_seed, u64 K (records in this stream), then per
 * module u32 tiles, u32 records.
 * Errors: INVALID_ARG, UNSUPPORTED (U with n_rates != 1), BUDGET, CAPACITY,
 * WORKSPACE, CUDA.
 */
awsrc_status awsrc_select_records(const awsrc_params* prm, int32_t n_mod,
                                  const awsrc_module* mods, const awsrc_candidate* cands,
                                  const double* rates_bpw, int32_t n_rates,
                                  uint8_t* stream_out, size_t stream_capacity,
                                  int64_t* d_counts, int64_t* d_bytes,
                                  void* workspace, size_t workspace_bytes, void* stream);

/* ---------------------------------------------------------------- decoder -- */

awsrc_status awsrc_decode_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, int32_t mode,
                                          size_t* bytes);

/*
 * awsrc_decode_apply — the decoder of Sec. 3.2: for each of the first K records
 * it regenerates B_s (Eq. 2) and adds r_hat = B_s * alpha_hat to W0 (Eq. 1);
 * tiles without a record keep W0 unchanged, so K == 0 returns W0 exactly.
 * Any prefix of a progressive stream decodes against the same W0 (Sec. 3.3).
 *   stream   device, header + records as written by awsrc_select_records.
 *   stream_len  bytes readable at `stream`; records beyond it are never read.
 *   K        records to apply (0 <= K <= header's K). K < 0 applies all the
 *            header's records (read on the device; no synchronisation). Either
 *            way at most (stream_len - h) / L records are applied; an explicit
 *            K above that returns AWSRC_ERR_INVALID_ARG.
 *   W_hat    host array of n_mod device pointers, rows*cols elements of out_dtype.
 *   mode     DENSE: every element of W_hat is written (W0 copied, corrected where
 *            a record exists). INPLACE: only the tiles named by records are
 *            written; W_hat must already hold W0 (it may be W0 itself when
 *            out_dtype == w0_dtype).
 * Each corrected element is fl(W0 + fl(fl(k_j * C^-1/2) * scale)) with the exact
 * integer k_j = sum_p sign_{j,p} * code_p, rounded once more to BF16 when
 * out_dtype is BF16. Records naming a tile >= T or a seed >= S are skipped and
 * reported through awsrc_workspace_status(). A stream names each tile at most
 * once (the encoder never repeats one); decoding a stream that does, in either
 * mode, applies only the tile's later record and reports it the same way.
 * Requires the same params as the encoder.
 * Workspace (awsrc_decode_workspace_bytes): the basis masks, plus for DENSE a
 * tile -> record map and the unpacked records, 24 bytes per tile (and, for
 * P = 4 with C <= 64 and b <= 5, 2*C bytes per seed of code tables); for
 * INPLACE one claim word per tile (4 bytes).
 */
awsrc_status awsrc_decode_apply(const awsrc_params* prm, int32_t n_mod,
                                const awsrc_module* mods, const uint8_t* stream,
                                size_t stream_len, int64_t K, void* const* W_hat, int32_t out_dtype,
                                int32_t mode, void* workspace, size_t workspace_bytes,
                                void* stream_handle);

/*
 * awsrc_decode_apply_inplace_noalloc — the in-place decode of awsrc_decode_apply
 * (mode AWSRC_DECODE_INPLACE) for callers that may not allocate device memory:
 * a model loader inside an engine that has handed all device memory to its own
 * pool, a plain C program without an allocator, a recovery path that must not
 * allocate. The paper has no counterpart; this is an interface convenience.
 * It takes no workspace: its scratch (the basis mask table and a fault word)
 * is a static device array of this library, about 1 MiB that every GPU which
 * loads the library keeps until the process exits. It allocates nothing (no
 * cudaMalloc, cudaFree or allocating library call).
 *   W_hat   host array of n_mod device pointers; each must already hold that
 *           module's W0 (dtype mods[m].w0_dtype, the same for all modules) and
 *           receives W0 + r_hat on the tiles the first K records name.
 *   mods    rows, cols and w0_dtype are read; W, W0 and the statistics are not.
 *   stream, stream_len, K  as in awsrc_decode_apply.
 * Limits: S * P * ceil(C/64) <= 131072 (else AWSRC_ERR_UNSUPPORTED, with the
 * numbers in awsrc_last_error_message()); at most 16 modules per call.
 * All calls share the one array per device and leave their contents in it;
 * calls whose kernels overlap on the GPU race on it, so the caller serialises
 * them. Every call looks up the array's address on the current device (the
 * device that holds W_hat and the stream must be current); the first call on a
 * device should come before any stream capture. Records naming a tile or seed
 * out of range are skipped; this entry point does not report them. The stream
 * must name each tile at most once, as the encoder's streams do: there is no
 * room for per-tile claims here, so a tile named twice is left unspecified.
 */
awsrc_status awsrc_decode_apply_inplace_noalloc(const awsrc_params* prm, int32_t n_mod,
                                                const awsrc_module* mods, const uint8_t* stream,
                                                size_t stream_len, int64_t K, void* const* W_hat,
                                                void* stream_handle);

/* ------------------------------------------------------------------ misc -- */

/*
 * Serving with the sidecar applied on the fly (the fused packed inference the
 * paper leaves to future work, Sec. 5): a stream is unpacked once for a model,
 * then each module's product with a few vectors reads the packed RTN-INT4
 * backbone and the sidecar, never a dense W_hat.
 *
 * awsrc_sidecar_workspace_bytes — device bytes of a prepared sidecar for the
 *   stream's module list (the dense decoder's workspace: basis masks, tile ->
 *   record map, per-record codes).
 * awsrc_sidecar_prepare — unpacks the first K records of `stream` (K < 0: the
 *   header's count) into `workspace`, as awsrc_decode_apply's first step does;
 *   faults are reported through awsrc_workspace_status(workspace).
 * awsrc_packed_gemv — y[m][i] = sum_j (W0_ij + r_ij) x[m][j] for module `m` of
 *   the list and the M <= 8 vectors x[m] (rows of x, M x cols, 16-byte
 *   aligned; y is M x rows): W0_ij = fl(q_ij * s_eff) from the packed backbone
 *   (awsrc_rtn_quantize's outputs; binary16 scales or SDQ), r_ij =
 *   fl(fl(k_j * C^-1/2) * scale) on the tiles the sidecar names (none when
 *   `sidecar` is NULL), both accumulated in binary32 with fma (the residual
 *   terms in their own sums). The result equals the double-precision product
 *   sum_j (W0_ij + r_ij) x_j, r_ij = k_j C^-1/2 scale, within
 *   (cols / min(C, 32) + 32) * 2^-24 * sum_j (|W0_ij x_j| + |r_ij x_j|).
 *   The module needs cols % 128 == 0.
 * Errors: INVALID_ARG, SHAPE, UNSUPPORTED, WORKSPACE, CUDA.
 */
typedef struct awsrc_packed_weights {
  const uint8_t* codes;      /* rows*cols/2 bytes, 4-byte aligned */
  const uint16_t* scales;    /* binary16 per group (sdq == 0) */
  const int8_t* sdq_codes;   /* per group (sdq == 1) */
  const float* sdq_consts;   /* (mean, step) per 256 groups (sdq == 1), 8-byte aligned */
  int32_t sdq;
  int32_t pad_;
} awsrc_packed_weights;

awsrc_status awsrc_sidecar_workspace_bytes(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                           size_t* bytes);
awsrc_status awsrc_sidecar_prepare(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                   const uint8_t* stream, size_t stream_len, int64_t K, void* workspace,
                                   size_t workspace_bytes, void* stream_handle);
awsrc_status awsrc_packed_gemv(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods, int32_t m,
                               const awsrc_packed_weights* pw, const void* sidecar, size_t sidecar_bytes,
                               int32_t M, const float* x, float* y, void* stream);

/*
 * awsrc_packed_gemv_batch — awsrc_packed_gemv for 1 <= n_task <= 16 tasks in
 * one launch (tasks whose M x cols inputs exceed 96 KB take one more launch
 * each): task i computes y_i = (W0 + r_hat) x_i for module tasks[i].m with
 * its packed backbone tasks[i].pw, all with the same sidecar and M. Tasks may
 * name the same module and share x (the q/k/v or gate/up projections of one
 * input); y arrays must not overlap each other or any input. Each y_i is
 * bit-identical to the single call's. Errors: as awsrc_packed_gemv;
 * UNSUPPORTED for n_task > 16.
 */
typedef struct awsrc_gemv_task {
  int32_t m;                 /* module index in the list */
  int32_t pad_;
  awsrc_packed_weights pw;   /* module m's packed backbone */
  const float* x;            /* M x cols, 16-byte aligned */
  float* y;                  /* M x rows */
} awsrc_gemv_task;

awsrc_status awsrc_packed_gemv_batch(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                     int32_t n_task, const awsrc_gemv_task* tasks, const void* sidecar,
                                     size_t sidecar_bytes, int32_t M, void* stream);

/*
 * awsrc_workspace_status — synchronises `stream`, then reads and clears the
 * device fault word kept in the first bytes of an encode/select/decode
 * workspace. Each of those entry points clears the word when it starts, so the
 * flags describe the last call made with this workspace; 0 means no fault.
 * Bit 0 (1): a record named a tile or seed out of range (decoder; skipped), or
 *            a tile a second time (dense decoder).
 * Bit 1 (2): encoder self-check — recomputing the winning candidate of a tile
 *            (for its codes) gave a different gain than the search found
 *            (never expected).
 * Bit 2 (4): a bounded wait inside a kernel gave up (never expected).
 */
awsrc_status awsrc_workspace_status(void* workspace, void* stream, uint32_t* flags);

const char* awsrc_status_string(awsrc_status st);
const char* awsrc_last_error_message(void);

/* -------------------------------------------------------------- diagnostics --
 * Measurement hooks with no counterpart in the paper. */

/*
 * awsrc_set_timing_events — for the calling host thread, makes every later
 * awsrc_encode_tiles record `before_search` (a cudaEvent_t) on its stream
 * immediately before its first seed-search kernel and `after_search`
 * immediately after its last one. NULL, NULL switches it off. The events are
 * owned by the caller and must outlive the calls that record them.
 */
void awsrc_set_timing_events(void* before_search, void* after_search);

/* Number of kernels this library has launched in the process so far. */
uint64_t awsrc_kernel_launches(void);

/*
 * awsrc_set_search_pruning — for the calling host thread, enabled = 0 makes
 * every later awsrc_encode_tiles score every (tile, seed) candidate; 1 (the
 * default) restores the exact pruning of the C = 64, P = 4, AWSRC-U search.
 * That search skips a candidate whose upper bound on the Eq. 4 gain (the
 * maximum b^T G^-1 b of the unquantised fit, inflated by a per-seed margin for
 * binary32 rounding) lies below the best gain its row has already reached, so
 * its candidates are by design identical either way; this switch exists to
 * check that on real inputs. The other searches never prune.
 */
void awsrc_set_search_pruning(int32_t enabled);

/*
 * awsrc_set_wait_test — a test of the kernels' failure handling, for the
 * calling host thread (no counterpart in the paper). Every wait inside the
 * tcgen05 search kernels (for bulk copies, tensor-core results and the release
 * of shared buffers) gives up after a time limit, 2 s by default; the block
 * then records bit 2 of the workspace's fault word, waits (with the same
 * limit) for its own copies and tensor-core work still in flight, frees its
 * tensor memory and exits, so the GPU context stays usable.
 *   wait_ns      the limit of every such wait in later awsrc_encode_tiles
 *                calls (0: the default 2 s).
 *   stall_chunk  >= 0: the C = 64, P = 4, AWSRC-U search issues no copies of
 *                its seed chunks from this one (counted within each block's
 *                range of 32-seed chunks) on, so its waits for that chunk run
 *                out; -1: normal operation.
 * The call's candidates are then undefined and awsrc_workspace_status reports
 * bit 2. awsrc_set_wait_test(0, -1) restores normal operation.
 */
void awsrc_set_wait_test(uint64_t wait_ns, int32_t stall_chunk);

/*
 * awsrc_verify_reciprocal — a check of the library's own arithmetic (no
 * counterpart in the paper): the LDL^T factorisations take 1/D_k correctly
 * rounded from a cheaper sequence on [2^-125, 2^125); this compares that
 * sequence with CUDA's correctly rounded reciprocal on every binary32 bit
 * pattern in [first, last) and adds the number that differ to *mismatches
 * (device, 8-byte aligned; the caller zeroes it). Asynchronous on `stream`.
 * Errors: INVALID_ARG (null, misaligned, first > last), CUDA.
 */
awsrc_status awsrc_verify_reciprocal(uint32_t first, uint32_t last, uint64_t* mismatches, void* stream);

#ifdef __cplusplus
}
#endif

#endif /* AWSRC_H */
