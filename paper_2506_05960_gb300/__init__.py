"""GB300-native AQ x A8 layer library (AQUATIC-Diff inference hot path).

The compute lives in the sm_103a shared library ``lib/libaq_gb300.so`` (C ABI
in ``include/aq.h``).  This package is a thin ctypes binding with the same
function names: it converts tensors to device pointers and sizes, passes the
current CUDA stream, and raises :class:`AQError` on a non-zero status.  There
is no Python or CPU fallback: if the library is missing, importing the binding
raises.
"""

from ._binding import (  # noqa: F401
    AQ_DTYPE_F16, AQ_DTYPE_F32, AQ_DTYPE_I8, AQ_DTYPE_F16_CODES, AQ_PATH_AUTO, AQ_PATH_DENSE, AQ_PATH_FUSED, AQ_PATH_LUT, AQ_PATH_FEW_TOKENS, AQ_PATH_PREDECODED,
    AQError, aq_abi_version, aq_codebook_grad, aq_code_update, aq_conv2d_ex_plan, aq_conv2d_ex_workspace_size, aq_conv2d_f16_plan, aq_conv2d_f16_workspace_size, aq_conv2d_nhwc, aq_conv2d_nhwc_ex, aq_conv2d_nhwc_f16, aq_conv2d_nhwc_q8, aq_conv2d_plan, aq_conv2d_workspace_size, aq_decode,
    aq_device_error, aq_last_error_string, aq_linear, aq_linear_f16, aq_linear_f16_workspace_size,
    aq_linear_f16_plan, aq_linear_a16, aq_linear_a16_plan, aq_linear_a16_workspace_size,
    aq_linear_ex, aq_linear_ex_plan, aq_linear_ex_workspace_size, aq_linear_noalloc, aq_linear_q8,
    aq_linear_plan, aq_linear_workspace_size, aq_pack, aq_set_plan_override,
    aq_set_wait_limit_ns, aq_linear_input_grad, aq_linear_input_grad_workspace_size, AQ_DEVERR_TIMEOUT_FULL,
    AQ_DEVERR_TIMEOUT_EMPTY, AQ_DEVERR_TIMEOUT_CONV, AQ_DEVERR_TIMEOUT_ACCUM, AQ_DEVERR_TIMEOUT_DRAIN,
    AQ_DEVERR_SMEM_LAYOUT,
    aq_packed_size, aq_profile_enable, aq_profile_read, aq_quant_act, library_path,
    load_library, PROFILE_KINDS,
)
