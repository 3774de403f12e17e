"""GB300 (sm_103a) implementation of the hot path of AWSRC — Activation-Weighted
Seeded Residual Coding for low-bit LLM weight repair (arXiv 2608.23144).

The work runs in hand-written CUDA kernels behind the C ABI of
``include/awsrc.h`` (``_lib/libawsrc.so``); this package is its thin Python
binding with the same entry-point names:

* ``awsrc_encode_tiles``   per-(tile, seed) search of Sec. 3.2 (Eqs. 2-4)
* ``awsrc_select_records`` byte-aware allocation and stream (Sec. 3.3-3.4, Eq. 5)
* ``awsrc_decode_apply``   decoder, W_hat = W0 + B_s alpha_hat (Eq. 1)
* ``awsrc_rtn_quantize``   the RTN-INT4 backbone W0 = Q(W) with optional scale
  double quantisation (Sec. 3.3)
* ``awsrc_sidecar_prepare`` / ``awsrc_packed_gemv`` / ``awsrc_packed_gemv_batch``  the
  sidecar applied inside a packed INT4 product, W_hat never formed
"""
from ._binding import (  # noqa: F401
    CANDIDATE_DTYPE,
    DECODE_DENSE,
    DECODE_INPLACE,
    DTYPE_BF16,
    DTYPE_F32,
    LIB_PATH,
    SCALE_FP16,
    SCALE_POW2,
    VARIANT_PF,
    VARIANT_U,
    AwsrcError,
    Module,
    Params,
    awsrc_decode_apply,
    awsrc_decode_apply_inplace_noalloc,
    awsrc_encode_tiles,
    awsrc_encode_workspace_bytes,
    awsrc_gen_basis,
    awsrc_rtn_quantize,
    awsrc_rtn_quantize_batch,
    awsrc_backbone_metadata_bytes,
    awsrc_rate_with_sdq_savings,
    awsrc_sidecar_prepare,
    awsrc_packed_gemv,
    awsrc_packed_gemv_batch,
    shape_modules,
    awsrc_header_bytes,
    awsrc_kernel_launches,
    awsrc_verify_reciprocal,
    awsrc_record_bytes,
    awsrc_select_records,
    awsrc_set_search_pruning,
    awsrc_set_timing_events,
    awsrc_set_wait_test,
    awsrc_stream_capacity,
    awsrc_workspace_status,
    candidates_to_numpy,
    lib,
    module_array,
    params,
)
