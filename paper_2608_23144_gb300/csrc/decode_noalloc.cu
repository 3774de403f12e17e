// decode_noalloc.cu — the in-place decoder for callers that cannot allocate
// device memory.
//
// Some callers of a weight-repair decoder are not allowed to call cudaMalloc:
// a model loader running inside an inference engine that has already handed
// every byte of device memory to its own pool, a C host program with no
// allocator of its own, or a recovery path that must not allocate while it
// restores weights. awsrc_decode_apply_inplace_noalloc serves them: it runs the
// same two kernels as the in-place mode of awsrc_decode_apply (basis masks,
// then the patch of the recorded tiles), but its scratch — the fault word and the basis
// mask table — lives in the file-scope device array below instead of a
// caller-supplied workspace. It calls no cudaMalloc, cudaFree or allocating
// library routine.
//
// Consequences a caller must know:
//  * every GPU that loads this library holds kScratchWords * 8 bytes (about
//    1 MiB) for this array until the process exits;
//  * the table holds at most kMaxMaskWords = S * P * ceil(C/64) 64-bit words;
//    larger parameters are rejected with AWSRC_ERR_UNSUPPORTED;
//  * every call shares the one array per device and leaves its contents there;
//    calls whose work overlaps on the GPU (other streams, other host threads)
//    race on it and must be serialised by the caller;
//  * every call looks up the array's device address on the current device
//    (cudaGetSymbolAddress, which allocates nothing), so the address is never
//    stale after a device reset; make the first call on a device before any
//    stream capture, since that lookup may load the library's module there;
//  * the stream must name each tile at most once (the encoder never repeats
//    one); this entry point has no room for per-tile claims, so a tile named
//    twice is left unspecified.
#include <algorithm>

#include "internal.h"

namespace awsrc {

namespace {

constexpr int kStatusWords = (int)(kStatusBytes / sizeof(uint64_t));  // 32 words = 256 B
constexpr int kMaxMaskWords = 131072;                                   // 1 MiB of masks
constexpr int kScratchWords = kStatusWords + kMaxMaskWords;

// The scratch: [fault word + padding (256 B)] [basis masks (up to 1 MiB)].
static __device__ __align__(256) uint64_t g_noalloc_scratch[kScratchWords];

// Device address of the scratch array on the current device, looked up on
// every call: a cached address would outlive a device reset or a recreated
// primary context. Host code must not use the array's name as an address: on
// the host it is only a stand-in symbol.
awsrc_status scratch_for_current_device(uint64_t** out) {
  void* p = nullptr;
  const cudaError_t e = cudaGetSymbolAddress(&p, g_noalloc_scratch);
  if (e != cudaSuccess) return cuda_fail(e, "decode_noalloc: cudaGetSymbolAddress");
  if (!p) {
    set_error_message("decode_noalloc: no device address for the scratch array");
    return AWSRC_ERR_CUDA;
  }
  *out = static_cast<uint64_t*>(p);
  return AWSRC_OK;
}

}  // namespace

}  // namespace awsrc

using namespace awsrc;

extern "C" awsrc_status awsrc_decode_apply_inplace_noalloc(const awsrc_params* prm, int32_t n_mod,
                                                           const awsrc_module* mods,
                                                           const uint8_t* stream, size_t stream_len,
                                                           int64_t K, void* const* W_hat,
                                                           void* stream_handle) {
  Prm pr;
  awsrc_status s = make_prm(prm, &pr);
  if (s != AWSRC_OK) return s;
  if (n_mod < 1 || !mods || !stream || !W_hat) return AWSRC_ERR_INVALID_ARG;
  const int64_t mask_words = (int64_t)pr.S * pr.P * pr.W;
  if (mask_words > kMaxMaskWords) {
    set_error_message("decode_noalloc: the basis table needs S*P*ceil(C/64) = %lld words; "
                      "this entry point holds at most %d",
                      (long long)mask_words, kMaxMaskWords);
    return AWSRC_ERR_UNSUPPORTED;
  }
  if (n_mod > kMaxModsPerLaunch) return AWSRC_ERR_UNSUPPORTED;
  DecodeMod dm[kMaxModsPerLaunch];
  int64_t T = 0;
  for (int m = 0; m < n_mod; ++m) {
    const awsrc_module& md = mods[m];
    if (md.rows < 1 || md.cols < 1 || md.cols % pr.C != 0) return AWSRC_ERR_SHAPE;
    if (md.w0_dtype != AWSRC_DTYPE_F32 && md.w0_dtype != AWSRC_DTYPE_BF16) return AWSRC_ERR_INVALID_ARG;
    if (!W_hat[m] || (reinterpret_cast<uintptr_t>(W_hat[m]) & 15) != 0) return AWSRC_ERR_INVALID_ARG;
    dm[m].W0 = W_hat[m];
    dm[m].out = W_hat[m];
    dm[m].rows = md.rows;
    dm[m].cols = md.cols;
    dm[m].tile_off = T;
    dm[m].w0_dtype = md.w0_dtype;
    dm[m].pad_ = 0;
    if (m > 0 && md.w0_dtype != mods[0].w0_dtype) return AWSRC_ERR_INVALID_ARG;
    const int64_t n_cb = md.cols / pr.C;
    if (md.rows > ((1ll << 32) - 1 - T) / n_cb) return AWSRC_ERR_UNSUPPORTED;  // 32-bit tile indices
    T += md.rows * n_cb;
  }
  const int64_t L = awsrc_record_bytes(prm, T), h = awsrc_header_bytes(n_mod);
  if (stream_len < (size_t)h) return AWSRC_ERR_INVALID_ARG;
  const int64_t kmax = std::min<int64_t>(((int64_t)stream_len - h) / L, T);
  if (K > kmax) return AWSRC_ERR_INVALID_ARG;

  uint64_t* scratch = nullptr;
  if ((s = scratch_for_current_device(&scratch)) != AWSRC_OK) return s;
  uint32_t* status = reinterpret_cast<uint32_t*>(scratch);
  uint64_t* masks = scratch + kStatusWords;
  cudaStream_t st = (cudaStream_t)stream_handle;
  cudaError_t e = cudaMemsetAsync(status, 0, sizeof(uint32_t), st);  // the fault word starts at 0
  if (e != cudaSuccess) return cuda_fail(e, "decode_noalloc: clear");
  e = launch_decode(pr, n_mod, dm, T, L, h, stream, K, kmax, mods[0].w0_dtype, AWSRC_DECODE_INPLACE,
                    masks, nullptr, status, st);
  return e == cudaSuccess ? AWSRC_OK : cuda_fail(e, "decode_noalloc");
}
