// api.cu — the extern "C" entry points declared in include/awsrc.h: argument
// validation, workspace layout and the launch sequence of each step.
#include <algorithm>
#include <atomic>
#include <cmath>
#include <cstdarg>
#include <cstdio>
#include <cstring>
#include <vector>

#include "internal.h"

namespace awsrc {

namespace {
thread_local char g_err[512] = "";
thread_local cudaEvent_t g_ev_before = nullptr, g_ev_after = nullptr;
thread_local int g_prune = 1;
thread_local uint64_t g_wait_ns = 0;  // 0: the default limit
thread_local int g_stall_chunk = -1;
std::atomic<uint64_t> g_launches{0};
constexpr int64_t kTargetBlocks = 1216;  // enough blocks to fill a GB300 (152 SMs) several times
// one RTN launch has a block per 256 groups of 128 weights: 2^46 weights keep
// its grid far inside gridDim.x and every size product inside int64
constexpr int64_t kMaxBackboneWeights = 1ll << 46;

int ceil_log2_host(uint64_t x) {
  int n = 0;
  while (n < 64 && (1ull << n) < x) ++n;
  return n;
}

bool is_pow2(int64_t x) { return x > 0 && (x & (x - 1)) == 0; }

bool use_c64p4(const Prm& pr) {
  return pr.C == 64 && pr.P == 4 && pr.variant == AWSRC_VARIANT_U;
}

bool use_c64p4_pf(const Prm& pr) {
  return pr.C == 64 && pr.P == 4 && pr.variant == AWSRC_VARIANT_PF;
}

bool aligned(const void* p, uintptr_t a) { return (reinterpret_cast<uintptr_t>(p) & (a - 1)) == 0; }
uintptr_t elt_bytes(int32_t dtype) { return dtype == AWSRC_DTYPE_BF16 ? 2 : 4; }

// Shapes, dtypes and, for the encoder, pointers: it reads W, W0 and the
// statistics element by element (natural alignment).
awsrc_status check_modules(const Prm& pr, int32_t n_mod, const awsrc_module* mods, bool encoder,
                           int64_t* T_out) {
  if (n_mod < 1 || mods == nullptr) return AWSRC_ERR_INVALID_ARG;
  int64_t T = 0;
  for (int m = 0; m < n_mod; ++m) {
    const awsrc_module& md = mods[m];
    if (md.rows < 1 || md.cols < 1) return AWSRC_ERR_SHAPE;
    if (md.cols % pr.C != 0) return AWSRC_ERR_SHAPE;
    if (md.w0_dtype != AWSRC_DTYPE_F32 && md.w0_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
    if (encoder) {
      if (md.w_dtype != AWSRC_DTYPE_F32 && md.w_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
      if (!md.W || !md.W0 || !md.act) return AWSRC_ERR_INVALID_ARG;
      if (pr.variant == AWSRC_VARIANT_PF && !md.fisher) return AWSRC_ERR_INVALID_ARG;
      if (!aligned(md.W, elt_bytes(md.w_dtype)) || !aligned(md.W0, elt_bytes(md.w0_dtype)) ||
          !aligned(md.act, 4) || !aligned(md.fisher, 4))
        return AWSRC_ERR_INVALID_ARG;
    }
    // tile indices are 32-bit: refuse before rows * n_cb can overflow
    const int64_t n_cb = md.cols / pr.C;
    if (md.rows > ((1ll << 32) - 1 - T) / n_cb) return AWSRC_ERR_UNSUPPORTED;
    T += md.rows * n_cb;
  }
  *T_out = T;
  return AWSRC_OK;
}

struct EncodeLayout {
  size_t masks, gram, pairs, mexp, ptab, pcands, total;
  int nsplit;
  bool spec;     // U, C = 64, P = 4: tcgen05 search
  bool spec_pf;  // P_F, C = 64, P = 4: tcgen05 search
};

EncodeLayout encode_layout(const Prm& pr, int32_t n_mod, const awsrc_module* mods, int64_t T) {
  EncodeLayout L{};
  L.spec = use_c64p4(pr);
  L.spec_pf = use_c64p4_pf(pr);
  const GenShape gs = gen_shape(pr);
  int64_t base_blocks = 0, ncb = 0;
  for (int m = 0; m < n_mod; ++m) {
    const int64_t n_cb = mods[m].cols / pr.C;
    ncb += n_cb;
    if (L.spec || L.spec_pf) base_blocks += n_cb * ((mods[m].rows + search_c64p4_rows() - 1) / search_c64p4_rows());
  }
  if (!(L.spec || L.spec_pf)) base_blocks = (T + gs.tiles - 1) / gs.tiles;
  const int64_t units = L.spec ? pr.S_pad / search_c64p4_chunk()
                       : L.spec_pf ? pr.S_pad / search_pf_c64p4_chunk()
                                   : (pr.S + gs.lanes - 1) / gs.lanes;
  int64_t ns = (kTargetBlocks + base_blocks - 1) / base_blocks;
  ns = std::max<int64_t>(1, std::min<int64_t>(ns, units));
  L.nsplit = (int)ns;
  size_t off = kStatusBytes;
  L.masks = off;
  off += align_up((size_t)pr.S_pad * pr.P * pr.W * 8, 256);
  L.gram = off;  // read by the generic U search
  if (pr.variant == AWSRC_VARIANT_U && !L.spec)
    off += align_up((size_t)ncb * pr.S_pad * gram_stride(pr.P) * 4, 256);
  L.pairs = off;
  if (L.spec) off += align_up((size_t)ncb * (pr.S_pad / 2) * pair_stride(pr.P) * 8, 256);
  L.mexp = off;
  if (L.spec || L.spec_pf) off += align_up(search_c64p4_table_bytes(pr.S_pad), 256);
  L.ptab = off;
  if (L.spec_pf) off += align_up(search_pf_c64p4_table_bytes(pr.S_pad), 256);
  L.pcands = off;  // candidates per tile and seed split, merged when nsplit > 1
  if (L.nsplit > 1) off += align_up((size_t)L.nsplit * T * sizeof(awsrc_candidate), 256);
  L.total = off;
  return L;
}

}  // namespace

void note_launches(int n) { g_launches.fetch_add((uint64_t)n, std::memory_order_relaxed); }

awsrc_status cuda_fail(cudaError_t e, const char* where) {
  snprintf(g_err, sizeof g_err, "%s: %s (%s)", where, cudaGetErrorString(e), cudaGetErrorName(e));
  return AWSRC_ERR_CUDA;
}

void set_error_message(const char* fmt, ...) {
  va_list ap;
  va_start(ap, fmt);
  vsnprintf(g_err, sizeof g_err, fmt, ap);
  va_end(ap);
}

awsrc_status check_launch(const char* where) {
  const cudaError_t e = cudaGetLastError();
  if (e != cudaSuccess) return cuda_fail(e, where);
  return AWSRC_OK;
}

awsrc_status make_prm(const awsrc_params* p, Prm* out) {
  if (!p) return AWSRC_ERR_INVALID_ARG;
  if (!is_pow2(p->C) || p->C < 4 || p->C > kMaxC) return AWSRC_ERR_SHAPE;
  if (p->P < 1 || p->P > kMaxP || p->P > p->C) return AWSRC_ERR_UNSUPPORTED;
  if (p->b < 2 || p->b > 8) return AWSRC_ERR_UNSUPPORTED;
  if (p->S < 1 || p->S > 65536) return AWSRC_ERR_UNSUPPORTED;
  if (p->variant != AWSRC_VARIANT_U && p->variant != AWSRC_VARIANT_PF) return AWSRC_ERR_INVALID_ARG;
  if (p->permute != 0 && p->permute != 1) return AWSRC_ERR_INVALID_ARG;
  if (!(p->ridge_rel >= 0.0f) || !std::isfinite(p->ridge_rel)) return AWSRC_ERR_INVALID_ARG;
  Prm r{};
  r.C = p->C; r.P = p->P; r.b = p->b; r.S = p->S; r.b_e = p->b_e; r.e_bias = p->e_bias;
  r.scale_mode = p->scale_mode; r.permute = p->permute; r.variant = p->variant;
  r.ridge_rel = p->ridge_rel; r.gen_seed = p->gen_seed;
  if (p->scale_mode == AWSRC_SCALE_POW2) {
    if (p->b_e < 1 || p->b_e > 8) return AWSRC_ERR_UNSUPPORTED;
    r.e_lo = std::max(p->e_bias - (1 << (p->b_e - 1)), -126);
    r.e_hi = std::min(p->e_bias + (1 << (p->b_e - 1)) - 1, 126);
    if (r.e_lo > r.e_hi) return AWSRC_ERR_UNSUPPORTED;
  } else if (p->scale_mode == AWSRC_SCALE_FP16) {
    if (p->b_e != 16) return AWSRC_ERR_UNSUPPORTED;
    r.e_lo = r.e_hi = 0;
  } else {
    return AWSRC_ERR_INVALID_ARG;
  }
  r.qmax = (1 << (p->b - 1)) - 1;
  r.qmaxf = (float)r.qmax;
  r.c = (float)(1.0 / std::sqrt((double)p->C));
  r.c2 = 1.0f / (float)p->C;
  r.W = (p->C + 63) / 64;
  // selectors padded to whole search chunks: 32 seeds (U, C = 64, P = 4) or 12
  // (P_F, C = 64, P = 4; then a multiple of 96, which keeps the atom table of
  // 32-seed chunks whole), padding selectors having all-zero masks
  r.S_pad = (p->S + 31) / 32 * 32;
  if (p->variant == AWSRC_VARIANT_PF && p->C == 64 && p->P == 4) r.S_pad = (p->S + 95) / 96 * 96;
  r.logC = ceil_log2_host((uint64_t)p->C);
  {
    const float qf = r.qmaxf;
    uint32_t qb;
    std::memcpy(&qb, &qf, 4);
    r.mant_q = qb & 0x007FFFFFu;
  }
  // valid candidates have 2^-100 <= amax <= 2^32, so e lies in
  // [-100 - (b-2), 33 - (b-2)]; if the range covers that, it never binds
  r.fast_pow2 = (p->scale_mode == AWSRC_SCALE_POW2) && r.e_lo <= -100 - (p->b - 2) &&
                r.e_hi >= 33 - (p->b - 2);
  r.prune = 1;
  r.stall_chunk = -1;
  r.wait_ns = kWaitLimitNs;
  *out = r;
  return AWSRC_OK;
}

namespace {

// One GEMV task: module m of the list with its packed backbone, x and y.
awsrc_status gemv_task(const Prm& pr, int32_t n_mod, const awsrc_module* mods, int32_t m,
                       const awsrc_packed_weights* pw, const float* x, float* y, GemvTask* t) {
  if (m < 0 || m >= n_mod || !pw || !x || !y) return AWSRC_ERR_INVALID_ARG;
  if (mods[m].cols % rtn_group() != 0) return AWSRC_ERR_SHAPE;
  if (pw->sdq != 0 && pw->sdq != 1) return AWSRC_ERR_INVALID_ARG;
  if (!pw->codes || (pw->sdq ? (!pw->sdq_codes || !pw->sdq_consts) : !pw->scales)) return AWSRC_ERR_INVALID_ARG;
  if (!aligned(pw->codes, 4) || !aligned(pw->scales, 2) || !aligned(pw->sdq_consts, 8) || !aligned(x, 16) ||
      !aligned(y, 4))
    return AWSRC_ERR_INVALID_ARG;
  *t = GemvTask{};
  t->rows = mods[m].rows;
  t->cols = mods[m].cols;
  for (int i = 0; i < m; ++i) t->tile_off += mods[i].rows * (mods[i].cols / pr.C);
  t->sdq = pw->sdq;
  t->codes = reinterpret_cast<const uint16_t*>(pw->codes);
  t->scales = pw->scales;
  t->sdq_codes = pw->sdq_codes;
  t->sdq_consts = pw->sdq_consts;
  t->x = x;
  t->y = y;
  return AWSRC_OK;
}

// The sidecar's arrays (none when `sidecar` is null).
awsrc_status gemv_sidecar(const awsrc_params* prm, const Prm& pr, int32_t n_mod, const awsrc_module* mods,
                          int64_t T, const void* sidecar, size_t sidecar_bytes, GemvArgs* a) {
  a->map = nullptr;
  a->slots = nullptr;
  a->masks = nullptr;
  a->nib = nullptr;
  if (!sidecar) return AWSRC_OK;
  size_t need;
  const awsrc_status s = awsrc_sidecar_workspace_bytes(prm, n_mod, mods, &need);
  if (s != AWSRC_OK) return s;
  if (sidecar_bytes < need) return AWSRC_ERR_WORKSPACE;
  if (!aligned(sidecar, 256)) return AWSRC_ERR_INVALID_ARG;
  const uint8_t* ws = static_cast<const uint8_t*>(sidecar);
  const uint8_t* scratch = ws + kStatusBytes + align_up((size_t)pr.S * pr.P * pr.W * 8, 256);
  const DenseScratch ds = dense_scratch(pr, T);
  a->masks = reinterpret_cast<const uint64_t*>(ws + kStatusBytes);
  a->map = reinterpret_cast<const unsigned long long*>(scratch);
  a->slots = reinterpret_cast<const uint4*>(scratch + ds.slots_off);
  if (gemv_tables(pr)) a->nib = reinterpret_cast<const uint4*>(scratch + ds.nib_off);
  return AWSRC_OK;
}

}  // namespace

}  // namespace awsrc

using namespace awsrc;

extern "C" {

const char* awsrc_status_string(awsrc_status st) {
  switch (st) {
    case AWSRC_OK: return "ok";
    case AWSRC_ERR_INVALID_ARG: return "invalid argument";
    case AWSRC_ERR_SHAPE: return "unsupported shape (C must be a power of two in [4, 256] dividing cols)";
    case AWSRC_ERR_UNSUPPORTED: return "parameter outside the supported range";
    case AWSRC_ERR_BUDGET: return "byte budget smaller than the stream header";
    case AWSRC_ERR_CUDA: return "CUDA runtime error";
    case AWSRC_ERR_WORKSPACE: return "workspace missing or too small";
    case AWSRC_ERR_CAPACITY: return "output stream buffer too small";
    case AWSRC_ERR_DEVICE: return "a kernel reported a fault in its inputs";
  }
  return "unknown status";
}

const char* awsrc_last_error_message(void) { return g_err; }

void awsrc_set_timing_events(void* before_search, void* after_search) {
  g_ev_before = (cudaEvent_t)before_search;
  g_ev_after = (cudaEvent_t)after_search;
}

uint64_t awsrc_kernel_launches(void) { return g_launches.load(std::memory_order_relaxed); }

void awsrc_set_search_pruning(int32_t enabled) { g_prune = enabled ? 1 : 0; }

void awsrc_set_wait_test(uint64_t wait_ns, int32_t stall_chunk) {
  g_wait_ns = wait_ns;
  g_stall_chunk = stall_chunk < 0 ? -1 : stall_chunk;
}

int64_t awsrc_header_bytes(int32_t n_mod) { return n_mod < 0 ? -1 : 40 + 8 * (int64_t)n_mod; }

int64_t awsrc_record_bytes(const awsrc_params* prm, int64_t T) {
  Prm pr;
  if (make_prm(prm, &pr) != AWSRC_OK || T < 1) return -1;
  const int64_t bits = ceil_log2_host((uint64_t)T) + ceil_log2_host((uint64_t)pr.S) + pr.b_e +
                       (int64_t)pr.P * pr.b;
  return (bits + 7) / 8;
}

awsrc_status awsrc_encode_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, size_t* bytes) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (!bytes) return AWSRC_ERR_INVALID_ARG;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  *bytes = encode_layout(pr, n_mod, mods, T).total;
  return AWSRC_OK;
}

awsrc_status awsrc_rtn_quantize(int64_t rows, int64_t cols, const void* W, int32_t w_dtype, int32_t sdq,
                                uint8_t* codes, uint16_t* scales, int8_t* sdq_codes, float* sdq_consts,
                                void* W0, int32_t w0_dtype, void* stream) {
  const awsrc_rtn_task t{rows, cols, W, w_dtype, sdq, codes, scales, sdq_codes, sdq_consts, W0, w0_dtype, 0};
  return awsrc_rtn_quantize_batch(1, &t, stream);
}

awsrc_status awsrc_rtn_quantize_batch(int32_t n_task, const awsrc_rtn_task* tasks, void* stream) {
  if (n_task < 1 || !tasks) return AWSRC_ERR_INVALID_ARG;
  for (int i = 0; i < n_task; ++i) {
    const awsrc_rtn_task& t = tasks[i];
    if (t.rows < 1 || t.cols < 1 || t.cols % rtn_group() != 0) return AWSRC_ERR_SHAPE;
    if (t.rows > kMaxBackboneWeights / t.cols) return AWSRC_ERR_UNSUPPORTED;
    if (t.w_dtype != AWSRC_DTYPE_F32 && t.w_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
    if (t.w0_dtype != AWSRC_DTYPE_F32 && t.w0_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
    if (t.sdq != 0 && t.sdq != 1) return AWSRC_ERR_INVALID_ARG;
    if (!t.W || !t.codes || !aligned(t.W, 16) || !aligned(t.codes, 4) || !aligned(t.scales, 2) ||
        !aligned(t.sdq_consts, 4) || !aligned(t.W0, 16))
      return AWSRC_ERR_INVALID_ARG;
  }
  // one launch per run of tasks with the same dtypes, at most kMaxRtnTasks
  // pieces and rtn_max_blocks() blocks of 256 groups each; a module larger than
  // that is cut into pieces on block boundaries (the blocks are independent)
  const int64_t gpb = sdq_block(), maxg = rtn_max_blocks() * gpb, grp = rtn_group();
  RtnArgs a{};
  int64_t blocks = 0;
  int dt_in = -1, dt_out = -1;
  auto flush = [&]() -> cudaError_t {
    cudaError_t e = cudaSuccess;
    if (a.n > 0) e = launch_rtn(a, dt_in, dt_out, (cudaStream_t)stream);
    a.n = 0;
    blocks = 0;
    return e;
  };
  for (int i = 0; i < n_task; ++i) {
    const awsrc_rtn_task& t = tasks[i];
    const int64_t G = t.rows * t.cols / grp;
    for (int64_t off = 0; off < G;) {
      const int64_t len = std::min(G - off, maxg);
      const int64_t nb = (len + gpb - 1) / gpb;
      if (a.n == kMaxRtnTasks || blocks + nb > rtn_max_blocks() || t.w_dtype != dt_in || t.w0_dtype != dt_out) {
        const cudaError_t e = flush();
        if (e != cudaSuccess) return cuda_fail(e, "rtn_quantize");
        dt_in = t.w_dtype;
        dt_out = t.w0_dtype;
      }
      const size_t wi = t.w_dtype == AWSRC_DTYPE_F32 ? 4 : 2, wo = t.w0_dtype == AWSRC_DTYPE_F32 ? 4 : 2;
      RtnTask& r = a.t[a.n++];
      r.W = static_cast<const uint8_t*>(t.W) + (size_t)(off * grp) * wi;
      r.G = len;
      r.sdq = t.sdq;
      r.codes = reinterpret_cast<uint32_t*>(t.codes) + off * (grp / 8);
      r.scales = t.scales ? t.scales + off : nullptr;
      r.sdq_codes = t.sdq_codes ? t.sdq_codes + off : nullptr;
      r.sdq_consts = t.sdq_consts ? t.sdq_consts + 2 * (off / gpb) : nullptr;
      r.W0 = t.W0 ? static_cast<uint8_t*>(t.W0) + (size_t)(off * grp) * wo : nullptr;
      blocks += nb;
      off += len;
    }
  }
  const cudaError_t e = flush();
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "rtn_quantize");
}

int64_t awsrc_backbone_metadata_bytes(int64_t rows, int64_t cols, int32_t sdq) {
  if (rows < 1 || cols < 1 || cols % rtn_group() != 0 || rows > kMaxBackboneWeights / cols) return -1;
  const int64_t G = rows * cols / rtn_group();
  return sdq ? G + 8 * ((G + sdq_block() - 1) / sdq_block()) : 2 * G;
}

awsrc_status awsrc_rate_with_sdq_savings(int32_t n_mod, const awsrc_module* mods, double rate_bpw,
                                         double* rate_out, int64_t* saved_bytes) {
  if (n_mod < 1 || !mods || !rate_out) return AWSRC_ERR_INVALID_ARG;
  if (!(rate_bpw >= 0.0) || !std::isfinite(rate_bpw)) return AWSRC_ERR_INVALID_ARG;
  int64_t N = 0, saved = 0;
  for (int m = 0; m < n_mod; ++m) {
    const int64_t fp16 = awsrc_backbone_metadata_bytes(mods[m].rows, mods[m].cols, 0);
    const int64_t sdq = awsrc_backbone_metadata_bytes(mods[m].rows, mods[m].cols, 1);
    if (fp16 < 0 || sdq < 0) return AWSRC_ERR_SHAPE;
    if (N > (1ll << 52) - mods[m].rows * mods[m].cols) return AWSRC_ERR_UNSUPPORTED;
    N += mods[m].rows * mods[m].cols;
    saved += fp16 - sdq;
  }
  // the budget awsrc_select_records derives from a rate, B = floor(rate N / 8)
  auto budget = [N](double r) { return (int64_t)std::floor(r * (double)N / 8.0); };
  const int64_t target = budget(rate_bpw) + saved;
  if (target < 0) return AWSRC_ERR_BUDGET;  // SDQ's block constants cost more than it saves
  double r = 8.0 * (double)target / (double)N;
  for (int i = 0; i < 64 && budget(r) < target; ++i) r = std::nextafter(r, INFINITY);
  for (int i = 0; i < 64 && budget(r) > target; ++i) r = std::nextafter(r, 0.0);
  if (budget(r) != target) return AWSRC_ERR_UNSUPPORTED;
  *rate_out = r;
  if (saved_bytes) *saved_bytes = saved;
  return AWSRC_OK;
}

awsrc_status awsrc_gen_basis(const awsrc_params* prm, uint64_t* masks, void* stream) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (!masks) return AWSRC_ERR_INVALID_ARG;
  const cudaError_t e = launch_gen_basis(pr, masks, pr.S, (cudaStream_t)stream);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "gen_basis");
}

awsrc_status awsrc_encode_tiles(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                awsrc_candidate* out, void* workspace, size_t workspace_bytes,
                                void* stream) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  pr.prune = g_prune;
  if (g_wait_ns) pr.wait_ns = g_wait_ns;
  pr.stall_chunk = g_stall_chunk;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, true, &T)) != AWSRC_OK) return s;
  if (!out || !aligned(out, 4)) return AWSRC_ERR_INVALID_ARG;
  const EncodeLayout lay = encode_layout(pr, n_mod, mods, T);
  if (!workspace || workspace_bytes < lay.total) return AWSRC_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return AWSRC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint32_t* status = reinterpret_cast<uint32_t*>(ws);
  uint64_t* masks = reinterpret_cast<uint64_t*>(ws + lay.masks);
  float* gram = lay.spec ? nullptr : reinterpret_cast<float*>(ws + lay.gram);
  awsrc_candidate* pcands = lay.nsplit > 1 ? reinterpret_cast<awsrc_candidate*>(ws + lay.pcands) : out;
  float2* pairs = lay.spec ? reinterpret_cast<float2*>(ws + lay.pairs) : nullptr;
  void* mexp = ws + lay.mexp;
  cudaError_t e = cudaMemsetAsync(status, 0, sizeof(uint32_t), st);
  if (e != cudaSuccess) return cuda_fail(e, "encode: clear status");
  e = launch_gen_basis(pr, masks, pr.S_pad, st);
  if (e != cudaSuccess) return cuda_fail(e, "encode: gen_basis");
  void* ptab = ws + lay.ptab;
  if ((lay.spec || lay.spec_pf) && (e = launch_bfrag_c64p4(pr, masks, mexp, st)) != cudaSuccess)
    return cuda_fail(e, "encode: atom table");
  if (lay.spec_pf && (e = launch_products_pf_c64p4(pr, masks, ptab, st)) != cudaSuccess)
    return cuda_fail(e, "encode: atom product table");
  const bool spec = lay.spec || lay.spec_pf;
  const int rb = search_c64p4_rows();
  const GenShape gs = gen_shape(pr);
  int64_t tile_off = 0, gram_off = 0;
  for (int g0 = 0; g0 < n_mod; g0 += kMaxModsPerLaunch) {
    LaunchDesc ld;
    std::memset(&ld, 0, sizeof ld);
    ld.n = std::min(kMaxModsPerLaunch, n_mod - g0);
    ld.T = T;
    int64_t blocks = 0;
    for (int i = 0; i < ld.n; ++i) {
      const awsrc_module& md = mods[g0 + i];
      ModDesc& d = ld.m[i];
      d.W = md.W; d.W0 = md.W0; d.act = md.act; d.fisher = md.fisher;
      d.rows = md.rows; d.cols = md.cols; d.n_cb = md.cols / pr.C;
      d.n_rb = (md.rows + rb - 1) / rb;
      d.tile_off = tile_off;
      d.gram_off = gram_off;
      d.block_off = blocks;
      d.w_dtype = md.w_dtype; d.w0_dtype = md.w0_dtype;
      d.nsplit = lay.nsplit;
      d.w_act = md.w_act; d.w_fisher = md.w_fisher;
      blocks += d.n_cb * d.n_rb * d.nsplit;
      tile_off += d.rows * d.n_cb;
      gram_off += d.n_cb * pr.S_pad;
    }
    if (!spec) {  // the generic search takes runs of consecutive tiles
      const int64_t tiles = tile_off - ld.m[0].tile_off;
      blocks = (tiles + gs.tiles - 1) / gs.tiles * lay.nsplit;
    }
    if (pr.variant == AWSRC_VARIANT_U && (e = launch_gram_u(pr, ld, masks, gram, pairs, st)) != cudaSuccess)
      return cuda_fail(e, "encode: gram");
    if (g0 == 0 && g_ev_before && (e = cudaEventRecord(g_ev_before, st)) != cudaSuccess)
      return cuda_fail(e, "encode: timing event");
    if (lay.spec) e = launch_search_c64p4(pr, ld, mexp, pairs, masks, blocks, pcands, status, st);
    else if (lay.spec_pf) e = launch_search_pf_c64p4(pr, ld, mexp, ptab, masks, blocks, pcands, status, st);
    else e = launch_search_generic(pr, ld, masks, gram, blocks, pcands, st);
    if (e != cudaSuccess) return cuda_fail(e, "encode: search");
    if (g0 + kMaxModsPerLaunch >= n_mod && g_ev_after && (e = cudaEventRecord(g_ev_after, st)) != cudaSuccess)
      return cuda_fail(e, "encode: timing event");
    if (lay.nsplit > 1) {  // best of the seed splits of each tile
      const int64_t t0 = ld.m[0].tile_off;
      const int64_t t1 = ld.m[ld.n - 1].tile_off + ld.m[ld.n - 1].rows * ld.m[ld.n - 1].n_cb;
      if ((e = launch_merge_candidates(pcands, lay.nsplit, T, t0, t1, out, st)) != cudaSuccess)
        return cuda_fail(e, "encode: merge");
    }
  }
  return AWSRC_OK;
}

// ------------------------------------------------------------------ select --

static awsrc_status select_plan(const Prm& pr, int32_t n_mod, const awsrc_module* mods,
                                const double* rates, int32_t n_rates, SelectPlan* sp,
                                std::vector<int64_t>* tile_off, std::vector<int64_t>* kcap) {
  int64_t T;
  awsrc_status s = check_modules(pr, n_mod, mods, false, &T);
  if (s != AWSRC_OK) return s;
  if (!rates || n_rates < 1) return AWSRC_ERR_INVALID_ARG;
  if (pr.variant == AWSRC_VARIANT_U && n_rates != 1) return AWSRC_ERR_UNSUPPORTED;
  if (n_rates > 64 || n_mod > 1024) return AWSRC_ERR_UNSUPPORTED;
  sp->n_mod = n_mod;
  sp->n_rates = n_rates;
  sp->T = T;
  sp->h = 40 + 8 * (int64_t)n_mod;
  sp->L = (ceil_log2_host((uint64_t)T) + ceil_log2_host((uint64_t)pr.S) + pr.b_e +
           (int64_t)pr.P * pr.b + 7) / 8;
  int64_t N = 0;
  tile_off->assign(n_mod + 1, 0);
  int64_t maxTm = 1;
  for (int m = 0; m < n_mod; ++m) {
    const int64_t Tm = mods[m].rows * (mods[m].cols / pr.C);
    (*tile_off)[m + 1] = (*tile_off)[m] + Tm;
    maxTm = std::max(maxTm, Tm);
    N += mods[m].rows * mods[m].cols;
  }
  for (int r = 0; r < n_rates; ++r)
    if (!(rates[r] >= 0.0) || !std::isfinite(rates[r])) return AWSRC_ERR_INVALID_ARG;
  kcap->clear();
  if (pr.variant == AWSRC_VARIANT_U) {
    const int64_t B = (int64_t)std::floor(rates[0] * (double)N / 8.0);
    if (B < sp->h) return AWSRC_ERR_BUDGET;
    int64_t cap = 0;
    for (int m = 0; m < n_mod; ++m) {
      const unsigned __int128 q = (unsigned __int128)(uint64_t)(B - sp->h) *
                                  (uint64_t)(mods[m].rows * mods[m].cols);
      const int64_t quota = (int64_t)(q / (uint64_t)N);
      const int64_t k = std::min(quota / sp->L, (*tile_off)[m + 1] - (*tile_off)[m]);
      kcap->push_back(k);
      cap += k;
    }
    sp->cap_records = cap;
    sp->tile_bits_local = ceil_log2_host((uint64_t)maxTm);
    sp->mod_shift = 31 + sp->tile_bits_local;
    sp->key_bits = sp->mod_shift + ceil_log2_host((uint64_t)n_mod);
  } else {
    int64_t cap = 0;
    for (int r = 0; r < n_rates; ++r) {
      const int64_t B = (int64_t)std::floor(rates[r] * (double)N / 8.0);
      if (B < sp->h) return AWSRC_ERR_BUDGET;
      const int64_t k = std::min((B - sp->h) / sp->L, T);
      kcap->push_back(k);
      cap = std::max(cap, k);
    }
    sp->cap_records = cap;
    sp->tile_bits_local = ceil_log2_host((uint64_t)T);
    sp->mod_shift = 0;
    sp->key_bits = 31 + sp->tile_bits_local;
  }
  if (sp->key_bits > 64) return AWSRC_ERR_UNSUPPORTED;
  sp->nblocks = (T + 2047) / 2048;
  return AWSRC_OK;
}

awsrc_status awsrc_stream_capacity(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                   const double* rates_bpw, int32_t n_rates, size_t* bytes) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (!bytes) return AWSRC_ERR_INVALID_ARG;
  SelectPlan sp;
  std::vector<int64_t> to, kc;
  if ((s = select_plan(pr, n_mod, mods, rates_bpw, n_rates, &sp, &to, &kc)) != AWSRC_OK) return s;
  *bytes = (size_t)(sp.h + sp.cap_records * sp.L);
  return AWSRC_OK;
}

awsrc_status awsrc_select_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, size_t* bytes) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (!bytes) return AWSRC_ERR_INVALID_ARG;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  SelectPlan sp{};
  sp.T = T;
  sp.nblocks = (T + 2047) / 2048;
  *bytes = select_ws_bytes(sp);
  return AWSRC_OK;
}

awsrc_status awsrc_select_records(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                  const awsrc_candidate* cands, const double* rates_bpw,
                                  int32_t n_rates, uint8_t* stream_out, size_t stream_capacity,
                                  int64_t* d_counts, int64_t* d_bytes, void* workspace,
                                  size_t workspace_bytes, void* stream) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  SelectPlan sp;
  std::vector<int64_t> to, kc;
  if ((s = select_plan(pr, n_mod, mods, rates_bpw, n_rates, &sp, &to, &kc)) != AWSRC_OK) return s;
  if (!cands || !stream_out || !d_counts || !d_bytes) return AWSRC_ERR_INVALID_ARG;
  if (!aligned(cands, 4) || !aligned(d_counts, 8) || !aligned(d_bytes, 8)) return AWSRC_ERR_INVALID_ARG;
  if (stream_capacity < (size_t)(sp.h + sp.cap_records * sp.L)) return AWSRC_ERR_CAPACITY;
  if (!workspace || workspace_bytes < select_ws_bytes(sp)) return AWSRC_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return AWSRC_ERR_INVALID_ARG;
  std::vector<int64_t> mt(n_mod);
  for (int m = 0; m < n_mod; ++m) mt[m] = to[m + 1] - to[m];
  const cudaError_t e = cudaMemsetAsync(workspace, 0, sizeof(uint32_t), (cudaStream_t)stream);
  if (e != cudaSuccess) return cuda_fail(e, "select: clear status");
  return select_run(pr, sp, to.data(), mt.data(), kc.data(), cands, stream_out, d_counts, d_bytes,
                    workspace, workspace_bytes, (cudaStream_t)stream);
}

// ------------------------------------------------------------------ decode --

awsrc_status awsrc_decode_workspace_bytes(const awsrc_params* prm, int32_t n_mod,
                                          const awsrc_module* mods, int32_t mode, size_t* bytes) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (!bytes) return AWSRC_ERR_INVALID_ARG;
  if (mode != AWSRC_DECODE_DENSE && mode != AWSRC_DECODE_INPLACE) return AWSRC_ERR_INVALID_ARG;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  *bytes = kStatusBytes + align_up((size_t)pr.S * pr.P * pr.W * 8, 256) + decode_scratch_bytes(pr, T, mode);
  return AWSRC_OK;
}

awsrc_status awsrc_decode_apply(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                const uint8_t* stream, size_t stream_len, int64_t K, void* const* W_hat,
                                int32_t out_dtype, int32_t mode, void* workspace,
                                size_t workspace_bytes, void* stream_handle) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  if (!stream || !W_hat) return AWSRC_ERR_INVALID_ARG;
  if (out_dtype != AWSRC_DTYPE_F32 && out_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
  if (mode != AWSRC_DECODE_DENSE && mode != AWSRC_DECODE_INPLACE) return AWSRC_ERR_INVALID_ARG;
  std::vector<DecodeMod> dm(n_mod);
  int64_t off = 0;
  for (int m = 0; m < n_mod; ++m) {
    if (!W_hat[m] || !aligned(W_hat[m], 16)) return AWSRC_ERR_INVALID_ARG;
    // the decoder moves W0 and W_hat in 16-byte vectors
    if (mode == AWSRC_DECODE_DENSE && (!mods[m].W0 || !aligned(mods[m].W0, 16))) return AWSRC_ERR_INVALID_ARG;
    if (mode == AWSRC_DECODE_INPLACE && mods[m].w0_dtype != out_dtype) return AWSRC_ERR_INVALID_ARG;
    dm[m].W0 = mods[m].W0;
    dm[m].out = W_hat[m];
    dm[m].rows = mods[m].rows;
    dm[m].cols = mods[m].cols;
    dm[m].tile_off = off;
    dm[m].w0_dtype = mods[m].w0_dtype;
    dm[m].pad_ = 0;
    off += mods[m].rows * (mods[m].cols / pr.C);
  }
  size_t need;
  if ((s = awsrc_decode_workspace_bytes(prm, n_mod, mods, mode, &need)) != AWSRC_OK) return s;
  if (!workspace || workspace_bytes < need) return AWSRC_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return AWSRC_ERR_INVALID_ARG;
  const int64_t L = awsrc_record_bytes(prm, T), h = awsrc_header_bytes(n_mod);
  if (stream_len < (size_t)h) return AWSRC_ERR_INVALID_ARG;
  const int64_t kmax = std::min<int64_t>(((int64_t)stream_len - h) / L, T);
  if (K > kmax) return AWSRC_ERR_INVALID_ARG;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint32_t* status = reinterpret_cast<uint32_t*>(ws);
  uint64_t* masks = reinterpret_cast<uint64_t*>(ws + kStatusBytes);
  void* scratch = ws + kStatusBytes + align_up((size_t)pr.S * pr.P * pr.W * 8, 256);
  cudaStream_t st = (cudaStream_t)stream_handle;
  cudaError_t e = cudaSuccess;
  if (!decode_clears_status(pr, mode) && (e = cudaMemsetAsync(status, 0, sizeof(uint32_t), st)) != cudaSuccess)
    return cuda_fail(e, "decode: clear status");
  e = launch_decode(pr, n_mod, dm.data(), T, L, h, stream, K, kmax, out_dtype, mode, masks, scratch, status, st);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "decode");
}

// ----------------------------------------------------------------- serving --

awsrc_status awsrc_sidecar_workspace_bytes(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                           size_t* bytes) {
  return awsrc_decode_workspace_bytes(prm, n_mod, mods, AWSRC_DECODE_DENSE, bytes);
}

awsrc_status awsrc_sidecar_prepare(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                   const uint8_t* stream, size_t stream_len, int64_t K, void* workspace,
                                   size_t workspace_bytes, void* stream_handle) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  if (!stream) return AWSRC_ERR_INVALID_ARG;
  size_t need;
  if ((s = awsrc_sidecar_workspace_bytes(prm, n_mod, mods, &need)) != AWSRC_OK) return s;
  if (!workspace || workspace_bytes < need) return AWSRC_ERR_WORKSPACE;
  if (!aligned(workspace, 256)) return AWSRC_ERR_INVALID_ARG;
  const int64_t L = awsrc_record_bytes(prm, T), h = awsrc_header_bytes(n_mod);
  if (stream_len < (size_t)h) return AWSRC_ERR_INVALID_ARG;
  const int64_t kmax = std::min<int64_t>(((int64_t)stream_len - h) / L, T);
  if (K > kmax) return AWSRC_ERR_INVALID_ARG;
  uint8_t* ws = static_cast<uint8_t*>(workspace);
  uint64_t* masks = reinterpret_cast<uint64_t*>(ws + kStatusBytes);
  void* scratch = ws + kStatusBytes + align_up((size_t)pr.S * pr.P * pr.W * 8, 256);
  const cudaError_t e = launch_dense_prep(pr, T, L, h, stream, K, kmax, masks, scratch,
                                          reinterpret_cast<uint32_t*>(ws), (cudaStream_t)stream_handle);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "sidecar_prepare");
}

awsrc_status awsrc_packed_gemv(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods, int32_t m,
                               const awsrc_packed_weights* pw, const void* sidecar, size_t sidecar_bytes,
                               int32_t M, const float* x, float* y, void* stream) {
  awsrc_gemv_task task{};
  task.m = m;
  if (pw) task.pw = *pw;
  task.x = x;
  task.y = y;
  if (!pw) return AWSRC_ERR_INVALID_ARG;
  return awsrc_packed_gemv_batch(prm, n_mod, mods, 1, &task, sidecar, sidecar_bytes, M, stream);
}

awsrc_status awsrc_packed_gemv_batch(const awsrc_params* prm, int32_t n_mod, const awsrc_module* mods,
                                     int32_t n_task, const awsrc_gemv_task* tasks, const void* sidecar,
                                     size_t sidecar_bytes, int32_t M, void* stream) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  int64_t T;
  if ((s = check_modules(pr, n_mod, mods, false, &T)) != AWSRC_OK) return s;
  if (!tasks || n_task < 1 || M < 1 || M > 8) return AWSRC_ERR_INVALID_ARG;
  if (n_task > kMaxGemvTasks) return AWSRC_ERR_UNSUPPORTED;
  GemvArgs a{};
  a.n_task = n_task;
  for (int i = 0; i < n_task; ++i)
    if ((s = gemv_task(pr, n_mod, mods, tasks[i].m, &tasks[i].pw, tasks[i].x, tasks[i].y, &a.t[i])) != AWSRC_OK)
      return s;
  if ((s = gemv_sidecar(prm, pr, n_mod, mods, T, sidecar, sidecar_bytes, &a)) != AWSRC_OK) return s;
  const cudaError_t e = launch_gemv(pr, a, M, (cudaStream_t)stream);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "packed_gemv");
}

awsrc_status awsrc_verify_reciprocal(uint32_t first, uint32_t last, uint64_t* mismatches, void* stream) {
  if (!mismatches || !aligned(mismatches, 8) || first > last) return AWSRC_ERR_INVALID_ARG;
  const cudaError_t e = launch_verify_rcp(first, last, reinterpret_cast<unsigned long long*>(mismatches),
                                          (cudaStream_t)stream);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "verify_reciprocal");
}

awsrc_status awsrc_workspace_status(void* workspace, void* stream, uint32_t* flags) {
  if (!workspace || !flags) return AWSRC_ERR_INVALID_ARG;
  cudaStream_t st = (cudaStream_t)stream;
  cudaError_t e = cudaStreamSynchronize(st);
  if (e != cudaSuccess) return cuda_fail(e, "workspace_status: sync");
  uint32_t v = 0;
  if ((e = cudaMemcpy(&v, workspace, sizeof v, cudaMemcpyDeviceToHost)) != cudaSuccess)
    return cuda_fail(e, "workspace_status: read");
  if ((e = cudaMemset(workspace, 0, sizeof v)) != cudaSuccess) return cuda_fail(e, "workspace_status: clear");
  *flags = v;
  return AWSRC_OK;
}

}  // extern "C"
