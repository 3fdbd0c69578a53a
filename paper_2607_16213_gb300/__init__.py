"""SelKV on GB300: Python binding of the C-ABI library libselkv.so (include/selkv.h).

The binding only marshals arguments: every step of compression and decode runs in the
library's CUDA kernels.  Tensors may be passed as torch tensors (their data_ptr() is used) or
as raw integer addresses.  Importing the package does not load the library; the first call
does, and raises if the library has not been built (`__graft_entry__.build()`), so a missing
extension fails loudly instead of falling back to anything else.
"""
from ._binding import (  # noqa: F401
    SELKV_OK, SELKV_ERR_INVALID_ARG, SELKV_ERR_UNSUPPORTED, SELKV_ERR_WORKSPACE, SELKV_ERR_CUDA,
    SELKV_ERR_DEVICE, SELKV_BF16, SELKV_FP32, SELKV_GATE_COSINE, SELKV_GATE_OPEN,
    SELKV_GATE_CLOSED, SELKV_EMPTY_EXPAND, SELKV_EMPTY_DROP, SELKV_SELECT_SHARED,
    SELKV_SELECT_PER_HEAD, SELKV_ROPE_OFF, SELKV_ROPE_HALF, SELKV_ROPE_INTERLEAVED,
    SELKV_BIAS_RATIO, SELKV_BIAS_COUNT, SELKV_ROUTE_BUCKET, SELKV_ROUTE_COSINE,
    SELKV_SCORE_ROWSTATS, SELKV_SCORE_COLSUMS, SELKV_SCORE_ALL,
    SELKV_DEVERR_CAPACITY,
    SELKV_DEVERR_TIMEOUT, SELKV_DEVERR_LENGTH, SELKV_DEVERR_COUNT, SELKV_MAX_BATCH,
    SelKVError, selkv_shape, selkv_params, selkv_compress_debug, library, library_path,
    exported_symbols, check, selkv_status_string, selkv_last_cuda_error, selkv_kernel_launches,
    selkv_workspace_init,
    selkv_workspace_error, selkv_compress_workspace_size, selkv_compress,
    selkv_decode_workspace_size, selkv_decode_attn, selkv_decode_attn_static,
    selkv_layer_average_workspace_size, selkv_layer_average_bias, selkv_score_workspace_size,
    selkv_score,
    SELKV_STATIC_SCRATCH_BYTES,
)
