"""GB300-native rolling action-expert step of RAVEL (asynchronous rolling
inference for flow-based VLAs).

The compute path is the CUDA library ``libravel.so`` (C ABI in
``include/ravel.h``); this package is its thin Python binding plus a small
session helper that owns the device tensors of one rollout.  PyTorch is used
for device memory and streams only.
"""
from ._binding import (  # noqa: F401
    RAVEL_BF16, RAVEL_FP32, RAVEL_MASK_FULL, RAVEL_MASK_SLOT_ISOLATED, RavelError, load, lib_path,
    ravel_create, ravel_destroy, ravel_reset, ravel_set_context, ravel_set_context_robots, ravel_roll_step, ravel_roll_step_rel, ravel_set_relative_dims,
    ravel_denoise_chunk, ravel_get_state,
    ravel_set_state, ravel_step_kernel_count, ravel_profile_step, ravel_gemm, ravel_gemm_noalloc,
    ravel_gemm_noalloc_status, ravel_debug_inject, RAVEL_FAULT_PREFIX_LEN, RAVEL_FAULT_WITHHOLD_ARRIVAL,
    ravel_status_string, ravel_last_error,
)
from .session import RollingSession  # noqa: F401
